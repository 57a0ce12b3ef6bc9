// Group-resident path for fp32 embeddings: one launch, one CTA per prompt group (chain
// layout, groups of at most kF32MaxN states whose embeddings fit in shared memory), the
// whole advantage construction without leaving the CTA:
//   rows of the group into shared memory (row stride a multiple of 32 floats plus 4: each
//   row starts one 16-byte bank group after the one before it)
//   Gram block on the CUDA cores (Sec. 4.2: sim of every comparable pair): thread (ti, tj)
//   owns the outputs of rows ti + 16 a and columns tj + 16 c (a, c < 8), reading 16-byte
//   chunks of 8 rows and 8 columns per 4 elements of k (eight consecutive rows in a
//   quarter-warp: conflict-free); fp32 accumulation, the threshold test needs no more
//   (generated similarities keep a 1e-3 margin from kappa)
//   squared norms from its diagonal; the pair test acc / |z_j| >= kappa |z_i| as one fma
//   per pair, linked pairs united at once in a shared-memory union-find (Alg. S.1)
//   eta(p(v), v) from error-free row statistics (TwoProduct / TwoSum, fp32 products are
//   not exact), one warp per row
//   graph reward, dual-group advantage (gpo_group_math.cuh), exploration efficiency and
//   the token scatter (Sec. 4.3-4.5)
// Replaces the tiled path's six launches for such batches (prep, row norms, similarity,
// statistics, per-group math, tokens).  Groups of at most 64 states run with 512 threads
// (the Gram's k range split between the block's halves), larger ones with 256.
#include "gpo_group_math.cuh"

namespace gpo {

namespace {

constexpr int kF32MaxN = 128;
constexpr int kF32MaxZBytes = 160 * 1024;  // the group's rows in shared memory
// Two instances: 256 threads for groups of up to 128 states (TA <= 8 row blocks of 16), and
// 512 threads for groups of up to 64 (TA <= 4), whose Gram splits k between the two halves
// of the block (twice the warps to hide the loop's latency; the second half's partial sums
// pass through shared memory and are added in a fixed order)
constexpr int kF32SmallN = 64;
__host__ __device__ constexpr int f32_partial_bytes(int nt, int tamax) { return (nt / 256 - 1) * tamax * tamax * 256 * 4; }

struct __align__(16) F32Smem {
  int lab[kF32MaxN];
  int roll[kF32MaxN];
  int dep[kF32MaxN];
  int slen[kF32MaxN];
  int rstart[kF32MaxN + 1];
  int rend[kF32MaxN];
  float n2[kF32MaxN];  // fp32 squared norms (Gram diagonal); the efficiency marks later
  float rn[kF32MaxN];  // 1 / |z_i| (0 for a zero row)
  float thr[kF32MaxN];  // kappa |z_i| (+inf for a zero row or an invalid group)
  float eadv[kF32MaxN], ecor[kF32MaxN], eeff[kF32MaxN];
  float2 xn2[kF32MaxN];  // compensated |z_v|^2
  float2 xdot[kF32MaxN];  // compensated <z_{p(v)}, z_v> (0 without a parent embedding)
  float2 root_n2;
  int64_t tok0[kF32MaxN + 1];
  int64_t tstart[kF32MaxN];
  uint8_t rew[kF32MaxN];
  uint8_t emask[kF32MaxN];
  unsigned long long esum[3];
  int flags;
  alignas(16) unsigned char X[group_scratch_sep_bytes(kF32MaxN)];
};
constexpr size_t kF32ZOff = (sizeof(F32Smem) + 15) & ~size_t(15);

__host__ __device__ inline int f32_row_stride(int d) { return ((d + 31) & ~31) + 4; }  // floats, == 4 (mod 32)

__device__ __forceinline__ bool any_block(bool f) { return __syncthreads_or(f ? 1 : 0) != 0; }

// Gram block of the group's rows in shared memory (row stride ds floats) and its linked
// pairs.  Within each 256-thread part q of the block, thread (ti, tj) = (t / 16, t % 16)
// (t = tid % 256) accumulates rows ti + 16 a and columns tj + 16 c for a, c < TA
// (TA = ceil(n / 16)) over part q's range of k: per 4 elements, one 16-byte chunk of each of
// its TA rows and TA columns (a quarter-warp reads 8 consecutive rows: one bank group each)
// and 4 TA^2 fma.  With NT / 256 > 1 parts, parts 1.. leave their sums in `part` and part 0
// adds them in part order.  The diagonal (ti == tj, a == c) gives the squared norms of the
// threshold test; after a barrier every comparable pair i < j (another rollout: j at or
// after the end of i's rollout; with the same-depth rule also equal depth) with
// acc / |z_j| - kappa |z_i| >= 0 is united in the label forest.  Ends with the barrier
// that publishes the forest.
template <int TA, int NT>
__device__ __forceinline__ void f32_gram_links(F32Smem* gs, const float* Zs, int n, int d, int ds, int s0,
                                               float kappa, int rule, int tid, float* part, uint32_t* st) {
  constexpr int KS = NT / 256;  // parts of the block, each a range of k
  const int t = tid & 255, kq = tid >> 8;
  const int ti = t >> 4, tj = t & 15;
  float acc[TA][TA];
#pragma unroll
  for (int a = 0; a < TA; ++a)
#pragma unroll
    for (int c = 0; c < TA; ++c) acc[a][c] = 0.f;
  const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
  const int kend = (d + 3) & ~3;  // zeros from d on
  const int kh = ((kend / 4 + KS - 1) / KS) * 4;  // elements of k per part
  const int ka = kq * kh, kb = min(kend, ka + kh);
  // not unrolled: the loop body is fetched once (the instruction cache is cold on every launch
  // after other work has gone through L2)
#pragma unroll 1
  for (int k = ka; k < kb; k += 4) {
    float4 ra4[TA], cb4[TA];
#pragma unroll
    for (int a = 0; a < TA; ++a) {
      ra4[a] = ti + 16 * a < n ? *reinterpret_cast<const float4*>(Zs + (ti + 16 * a) * ds + k) : z4;
      cb4[a] = tj + 16 * a < n ? *reinterpret_cast<const float4*>(Zs + (tj + 16 * a) * ds + k) : z4;
    }
#pragma unroll
    for (int a = 0; a < TA; ++a)
#pragma unroll
      for (int c = 0; c < TA; ++c) {
        float s = acc[a][c];
        s = fmaf(ra4[a].x, cb4[c].x, s);
        s = fmaf(ra4[a].y, cb4[c].y, s);
        s = fmaf(ra4[a].z, cb4[c].z, s);
        s = fmaf(ra4[a].w, cb4[c].w, s);
        acc[a][c] = s;
      }
  }
  if (KS > 1) {  // the other parts' sums into part 0's, in part order
    if (kq > 0) {
#pragma unroll
      for (int a = 0; a < TA; ++a)
#pragma unroll
        for (int c = 0; c < TA; ++c) part[(((kq - 1) * TA + a) * TA + c) * 256 + t] = acc[a][c];
    }
    __syncthreads();
    if (kq == 0) {
      for (int q = 1; q < KS; ++q)
#pragma unroll
        for (int a = 0; a < TA; ++a)
#pragma unroll
          for (int c = 0; c < TA; ++c) acc[a][c] += part[(((q - 1) * TA + a) * TA + c) * 256 + t];
    }
  }
  if (kq == 0 && ti == tj) {
#pragma unroll
    for (int a = 0; a < TA; ++a) {
      const int i = ti + 16 * a;
      if (i < n) {
        const float dg = acc[a][a];
        gs->n2[i] = dg;
        gs->rn[i] = dg > 0.f ? 1.0f / sqrtf(dg) : 0.f;
        gs->thr[i] = dg > 0.f ? kappa * sqrtf(dg) : __int_as_float(0x7f800000);
        if (!isfinite(dg)) report(st, GPO_ERR_NONFINITE, 2, s0 + i);
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int a = 0; a < TA; ++a) {
    const int i = ti + 16 * a;
    if (kq != 0 || i >= n) continue;
    const float th = gs->thr[i];
    const int re = gs->rend[i], di = gs->dep[i];
#pragma unroll
    for (int c = 0; c < TA; ++c) {
      const int j = tj + 16 * c;
      if (j >= n || j < re) continue;  // j > i outside i's rollout
      if (rule == GPO_MERGE_SAME_DEPTH && gs->dep[j] != di) continue;
      if (fmaf(acc[a][c], gs->rn[j], -th) >= 0.f) uf_union(gs->lab, i, j);
    }
  }
  __syncthreads();
}


template <int NT, int TAMAX>
__global__ void __launch_bounds__(NT, 1) fused_f32_kernel(gpo_batch b, gpo_outputs o, Sizes sz, Ws ws, Params p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  F32Smem* gs = reinterpret_cast<F32Smem*>(smem_raw);
  float* Zs = reinterpret_cast<float*>(smem_raw + kF32ZOff);
  uint32_t* st = ws.status;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int nt = NT;
  const int d = sz.d, ds = f32_row_stride(d);
  float* part = Zs + (size_t)sz.maxn * ds;  // Gram partial sums of parts 1.. (f32_partial_bytes)
  const float kappa = p.kappa_f;
  if (blockIdx.x == 0 && tid == 0) {
    if (b.group_rollout_off[0] != 0 || b.group_rollout_off[sz.G] != sz.R) report(st, GPO_ERR_SHAPE, 2, 0);
    if (b.rollout_step_off[0] != 0 || b.rollout_step_off[sz.R] != sz.N) report(st, GPO_ERR_SHAPE, 2, 1);
    if (b.rollout_token_off[0] != 0 || b.rollout_token_off[sz.R] != sz.T) report(st, GPO_ERR_SHAPE, 2, 2);
  }
  const float* Z = reinterpret_cast<const float*>(b.emb);
  auto sync = [] { __syncthreads(); };

  for (int g = sz.g0 + (int)blockIdx.x; g < sz.g1; g += gridDim.x) {
    // ---- the group's rollouts and states (out of range: reported, nothing written)
    const int ra = b.group_rollout_off[g], rc = b.group_rollout_off[g + 1];
    bool in_range = ra >= 0 && rc >= ra && rc <= sz.R;
    const int x0 = in_range ? b.rollout_step_off[ra] : 0, x1 = in_range ? b.rollout_step_off[rc] : 0;
    in_range = in_range && x0 >= 0 && x1 >= x0 && x1 <= sz.N;
    const int r0 = ra, nr = rc - ra, s0 = x0, n = x1 - x0;
    if (!(in_range && n > 0 && n <= kF32MaxN && n <= sz.maxn && nr > 0 && nr <= n)) {
      if (tid == 0) {
        if (!in_range || nr > n || (nr > 0 && n == 0)) report(st, GPO_ERR_SHAPE, 2, g);
        else if (n > kF32MaxN || n > sz.maxn) report(st, GPO_ERR_UNSUPPORTED, 2, g);
        else if (n == 0) {  // a group without states: Eff 0 (no tokens)
          if (o.group_eff) o.group_eff[g] = 0.f;
          if (o.group_eff_graph) o.group_eff_graph[g] = 0.f;
        }
      }
      continue;
    }
    // ---- validate the group and lay out its states (Sec. 4.2 chain layout); its rows into
    //      shared memory (16-byte loads; the row's ragged tail, if any, element by element)
    if (tid == 0) gs->flags = 0;
    for (int r = tid; r <= nr; r += nt) {
      gs->rstart[r] = b.rollout_step_off[r0 + r] - s0;
      gs->tok0[r] = b.rollout_token_off[r0 + r];
    }
    for (int r = tid; r < nr; r += nt) gs->rew[r] = b.reward[r0 + r];
    group_scratch_zero(gs->X, n, tid, nt);
    for (int i = tid; i < n; i += nt) {
      gs->lab[i] = i;
      gs->slen[i] = b.step_len[s0 + i];
      gs->roll[i] = 0;
      gs->dep[i] = 1;
    }
    {
      const int dv = d / 4;  // whole 16-byte chunks of a row (rows start on 16 bytes)
      for (int e = tid; e < n * dv; e += nt) {
        const int i = e / dv, k4 = e - i * dv;
        if (!GPO_BOUNDS(st, (int64_t)i * ds + 4 * k4 + 3, (int64_t)kF32MaxN * ds, kWhereSmemRow)) continue;
        const float4 v = *reinterpret_cast<const float4*>(Z + (int64_t)(s0 + i) * sz.stride + 4 * k4);
        *reinterpret_cast<float4*>(Zs + i * ds + 4 * k4) = v;
      }
      for (int e = tid; e < n * (ds - 4 * dv); e += nt) {  // ragged tail, then zeros to the stride
        const int w = ds - 4 * dv, i = e / w, k = 4 * dv + (e - i * w);
        Zs[i * ds + k] = k < d ? Z[(int64_t)(s0 + i) * sz.stride + k] : 0.f;
      }
    }
    sync();
    for (int r = tid; r < nr; r += nt) {
      const int a = gs->rstart[r], e = gs->rstart[r + 1];
      bool bad = !(a >= 0 && e > a && e <= n) || gs->rew[r] > 1;
      if (gs->rew[r] > 1) report(st, GPO_ERR_BAD_REWARD, 2, r0 + r);
      int64_t t = gs->tok0[r];
      if (!bad) {
        for (int i = a; i < e; ++i) {
          gs->roll[i] = r;
          gs->dep[i] = i - a + 1;
          gs->rend[i] = e;
          gs->tstart[i] = t;
          if (gs->slen[i] < 1) bad = true;
          t += gs->slen[i];
        }
        if (t != gs->tok0[r + 1] || gs->tok0[r] < 0 || gs->tok0[r + 1] > sz.T) bad = true;
      }
      if (bad) {
        if (gs->rew[r] <= 1) report(st, GPO_ERR_SHAPE, 2, r0 + r);
        atomicOr(&gs->flags, 1);
      }
    }
    sync();
    const bool valid = (gs->flags & 1) == 0;
    if (!valid) continue;  // reported; nothing of this group is written

    // ---- Gram block and pair tests (f32_gram_links: TA = ceil(n / 16) row blocks per thread)
    switch ((n + 15) >> 4) {
      case 1: f32_gram_links<1, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
      case 2: f32_gram_links<2, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
      case 3: f32_gram_links<3, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
      case 4: f32_gram_links<4, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
      default:
        if constexpr (TAMAX > 4) {
          switch ((n + 15) >> 4) {
            case 5: f32_gram_links<5, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
            case 6: f32_gram_links<6, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
            case 7: f32_gram_links<7, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
            default: f32_gram_links<8, NT>(gs, Zs, n, d, ds, s0, kappa, p.rule, tid, part, st); break;
          }
        }
        break;
    }
    // ---- error-free row statistics for eta (one warp per row, from the rows in shared
    //      memory; the prompt embedding from global memory; TwoProduct for fp32 products)
    for (int i = warp; i < n; i += nt / 32) {
      const bool first = gs->dep[i] == 1;
      const bool has_p = !first || b.root_emb != nullptr;
      const void* pbase = first ? b.root_emb : static_cast<const void*>(Zs);
      const int64_t prow = first ? (int64_t)g * sz.stride : (int64_t)(i - 1) * ds;
      float2 n2v, dot;
      exact_pair_sums<false>(Zs, (int64_t)i * ds, pbase, prow, has_p, d, lane, n2v, dot);
      if (lane == 0) {
        if (!isfinite(n2v.x) || !isfinite(dot.x)) report(st, GPO_ERR_NONFINITE, 3, s0 + i);
        gs->xn2[i] = n2v;
        gs->xdot[i] = has_p ? dot : make_float2(0.f, 0.f);
      }
    }
    if (b.root_emb && warp == 0) {
      float2 n2r, dot;
      exact_pair_sums<false>(b.root_emb, (int64_t)g * sz.stride, nullptr, 0, false, d, lane, n2r, dot);
      if (lane == 0) {
        if (!isfinite(n2r.x)) report(st, GPO_ERR_NONFINITE, 3, sz.N + g);
        gs->root_n2 = n2r;
      }
    }
    sync();

    // ---- graph reward and dual-group advantage of every edge
    auto eta = [&](int i) -> float2 {
      const float2 z = make_float2(0.f, 0.f);
      const float2 n1 = gs->dep[i] == 1 ? (b.root_emb ? gs->root_n2 : z) : gs->xn2[i - 1];
      return ff_eta(gs->xdot[i], n1, gs->xn2[i]);
    };
    auto out = [&](int i, int label, float S, float acor, float E, float dual, unsigned char mask) {
      gs->eadv[i] = dual;
      gs->ecor[i] = acor;
      gs->eeff[i] = E;
      gs->emask[i] = mask;
      const int v = s0 + i;
      if (!GPO_BOUNDS(st, v, sz.N, kWhereStateOut)) return;
      if (o.edge_adv) o.edge_adv[v] = dual;
      if (o.class_id) o.class_id[v] = s0 + label;
      if (o.node_score) o.node_score[v] = S;
      if (o.edge_cor) o.edge_cor[v] = acor;
      if (o.edge_eff) o.edge_eff[v] = E;
      if (o.edge_eff_mask) o.edge_eff_mask[v] = mask;
    };
    group_advantages<1, true>(n, nr, gs->lab, gs->roll, gs->dep, gs->rstart, gs->rew, group_scratch_sep(gs->X, n),
                              p, tid, nt, sync, eta, out);
    // ---- exploration efficiency, Eq. (eq1) (the norms' array is free here)
    if (o.group_eff || o.group_eff_graph) {
      auto own = [&](int i) { return gs->rew[gs->roll[i]] != 0; };
      auto par = [&](int i) { return gs->dep[i] == 1 ? -1 : i - 1; };
      auto len = [&](int i) { return gs->slen[i]; };
      group_efficiency(n, gs->lab, reinterpret_cast<int*>(gs->n2), gs->esum, tid, nt, own, par, len, sync, any_block,
                       o.group_eff ? o.group_eff + g : nullptr, o.group_eff_graph ? o.group_eff_graph + g : nullptr);
    }
    // ---- every token of an edge carries the edge's advantage (Sec. 4.5): a half-warp per
    //      state, 16-byte stores inside the state's span, scalar stores at its ragged ends
    const bool more = o.adv_cor || o.adv_eff || o.eff_mask;
    const int hl = tid & 15;
    for (int i = tid >> 4; i < n; i += nt / 16) {
      const int64_t ts = gs->tstart[i], te = ts + gs->slen[i];
      const int64_t qa = (ts + 3) >> 2, qb = te >> 2;
      const int64_t h1 = qa <= qb ? 4 * qa : te;  // head [ts, h1)
      const int64_t t0 = qa <= qb ? 4 * qb : te;  // tail [t0, te)
      const int64_t tp = hl < 4 ? ts + hl : t0 + (hl - 4);
      const bool scal = hl < 4 ? tp < h1 : (hl < 8 && tp < te);
      if (!GPO_BOUNDS(st, te - 1, sz.T, kWhereTokens)) continue;
      auto put = [&](float* dst, float x) {
        const float4 v = make_float4(x, x, x, x);
        for (int64_t c = qa + hl; c < qb; c += 16) reinterpret_cast<float4*>(dst)[c] = v;
        if (scal) dst[tp] = x;
      };
      put(o.adv, gs->eadv[i]);
      if (more) {
        if (o.adv_cor) put(o.adv_cor, gs->ecor[i]);
        if (o.adv_eff) put(o.adv_eff, gs->eeff[i]);
        if (o.eff_mask) {
          const uint8_t m = gs->emask[i];
          const uint32_t v = 0x01010101u * m;
          for (int64_t c = qa + hl; c < qb; c += 16) reinterpret_cast<uint32_t*>(o.eff_mask)[c] = v;
          if (scal) o.eff_mask[tp] = m;
        }
      }
    }
    sync();
  }
}

size_t f32_smem_bytes(int d, int maxn, int nt, int tamax) {
  return kF32ZOff + (size_t)maxn * f32_row_stride(d) * sizeof(float) + (size_t)f32_partial_bytes(nt, tamax);
}

}  // namespace

bool fused_f32_fits(int d, int maxn) {
  return maxn >= 1 && maxn <= kF32MaxN && d >= 1 && (size_t)maxn * f32_row_stride(d) * sizeof(float) <= kF32MaxZBytes;
}

cudaError_t setup_fused_f32() {
  cudaError_t e = cudaFuncSetAttribute(fused_f32_kernel<256, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(kF32ZOff + kF32MaxZBytes));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(fused_f32_kernel<512, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(kF32ZOff + kF32MaxZBytes + f32_partial_bytes(512, 4)));
  return e;
}

cudaError_t launch_fused_f32(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                             const Ws& ws, const Params& p) {
  const int ng = sz.g1 - sz.g0;
  if (ng <= 0) return cudaSuccess;
  const int grid = ng < lc.num_sms ? ng : lc.num_sms;
  if (sz.maxn <= kF32SmallN)
    fused_f32_kernel<512, 4><<<grid, 512, f32_smem_bytes(sz.d, sz.maxn, 512, 4), lc.stream>>>(b, o, sz, ws, p);
  else
    fused_f32_kernel<256, 8><<<grid, 256, f32_smem_bytes(sz.d, sz.maxn, 256, 8), lc.stream>>>(b, o, sz, ws, p);
  return cudaGetLastError();
}

}  // namespace gpo
