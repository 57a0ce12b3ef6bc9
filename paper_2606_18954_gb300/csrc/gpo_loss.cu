// Policy loss of GraphPO (Sec. 4.5 objective J_GraphPO; Algorithm S.1 Stage 4 split
// form) on per-token log-probabilities, and the plan it runs on.
//
//   plan      loss_plan_kernel (a CTA per prompt group): validates the token layout,
//             writes the first token of every edge (an exclusive scan of step_len per
//             rollout, or per group in the tree layout) and counts the groups with
//             states; loss_weights_kernel: every edge's token weight 1/(G' |E_g| |e|)
//             and the edge holding the first token of every tile of kLossTile tokens.
//   loss      token_loss_kernel: persistent CTAs over token tiles; a tile's edges (first
//             token, weight x advantages; at most one per token) are staged in shared
//             memory with a token -> edge map of the tile; each thread takes four 16-byte
//             chunks of tokens (coalesced across the CTA; all four loaded before the
//             edges are staged) and reads each token's edge from the map; per token the
//             ratio, the
//             clipped surrogate, the k3 KL estimate, the gradient (one 16-byte store per
//             chunk); sums in fp32 per tile, fp64 across tiles, per-CTA partials combined
//             by the last CTA in a fixed order (deterministic).
// HBM-bound: 12 bytes per token (16 with the KL term) plus ~16 bytes per edge.
#include "gpo_internal.cuh"

namespace gpo {

namespace {

constexpr int kPlanThreads = 256;
constexpr int kLossThreads = 256;
constexpr int kLossChunks = kLossTile / (4 * kLossThreads);  // 16-byte chunks per thread and tile
static_assert(kLossChunks * 4 * kLossThreads == kLossTile, "loss tile shape");

__device__ __forceinline__ int64_t warp_incl_scan(int64_t x, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  return x;
}

// First tokens of the edges [v0, v1) of one token segment starting at `base` (one warp):
// chunks of 32 states, an inclusive scan each.  Returns the segment's token count and
// whether every step length is >= 1.
__device__ __forceinline__ int64_t segment_starts(const int32_t* step_len, int v0, int v1, int64_t base, float ng,
                                                  const LossPlan& lp, int lane, bool& ok) {
  int64_t carry = 0;
  for (int i0 = v0; i0 < v1; i0 += 32) {
    const int i = i0 + lane;
    const int64_t len = i < v1 ? (int64_t)step_len[i] : 0;
    if (i < v1 && len < 1) ok = false;
    const int64_t incl = warp_incl_scan(len, lane);
    if (i < v1) {
      lp.start[i] = base + carry + incl - len;
      lp.w[i] = ng;  // |E_g| for now; loss_weights_kernel turns it into the weight
    }
    carry += __shfl_sync(0xffffffffu, incl, 31);
  }
  return carry;
}

__global__ void __launch_bounds__(kPlanThreads) loss_plan_kernel(gpo_batch b, Sizes sz, LossPlan lp) {
  uint32_t* st = lp.status;
  const int g = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const bool tree = b.parent != nullptr;
  const int32_t* go = b.group_rollout_off;
  const int r0 = go[g], r1 = go[g + 1];
  if (r0 < 0 || r1 < r0 || r1 > sz.R) {
    if (threadIdx.x == 0) report(st, GPO_ERR_SHAPE, 6, g);
    return;
  }
  const int s0 = tree ? b.group_state_off[g] : (r1 > r0 ? b.rollout_step_off[r0] : 0);
  const int s1 = tree ? b.group_state_off[g + 1] : (r1 > r0 ? b.rollout_step_off[r1] : 0);
  if (s0 < 0 || s1 < s0 || s1 > sz.N) {
    if (threadIdx.x == 0) report(st, GPO_ERR_SHAPE, 6, g);
    return;
  }
  const int n = s1 - s0;
  if (threadIdx.x == 0) {
    if (n > 0) atomicAdd(&st[kLossWordGroups], 1u);
    if (g == 0) {  // the groups, states and tokens of the layout cover [0, R), [0, N) and [0, T)
      const int64_t first = tree ? b.group_token_off[0] : b.rollout_token_off[0];
      const int64_t last = tree ? b.group_token_off[sz.G] : b.rollout_token_off[sz.R];
      const int sf = tree ? b.group_state_off[0] : b.rollout_step_off[0];
      const int sl = tree ? b.group_state_off[sz.G] : b.rollout_step_off[sz.R];
      if (first != 0 || last != sz.T || sf != 0 || sl != sz.N || go[0] != 0 || go[sz.G] != sz.R)
        report(st, GPO_ERR_SHAPE, 6, g);
      lp.dims[0] = sz.N;
      lp.dims[1] = sz.T;
    }
  }
  bool ok = true;
  if (!tree) {
    // one warp per rollout: its states' spans follow each other from rollout_token_off[r]
    for (int r = r0 + warp; r < r1; r += nw) {
      const int v0 = b.rollout_step_off[r], v1 = b.rollout_step_off[r + 1];
      if (v0 < s0 || v1 < v0 || v1 > s1) {
        ok = false;
        continue;
      }
      const int64_t base = b.rollout_token_off[r];
      const int64_t tot = segment_starts(b.step_len, v0, v1, base, (float)n, lp, lane, ok);
      if (base + tot != b.rollout_token_off[r + 1]) ok = false;
    }
  } else {
    // the whole group is one span from group_token_off[g]: each warp scans a slice, the
    // slices' totals are combined through shared memory, then each warp writes its slice
    __shared__ int64_t s_tot[kPlanThreads / 32];
    const int slice = ((n + nw - 1) / nw + 31) & ~31;
    const int v0 = min(s1, s0 + warp * slice), v1 = min(s1, v0 + slice);
    int64_t part = 0;
    for (int i = v0 + lane; i < v1; i += 32) part += (int64_t)b.step_len[i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    if (lane == 0) s_tot[warp] = part;
    __syncthreads();
    int64_t before = 0, all = 0;
    for (int k = 0; k < nw; ++k) {
      if (k < warp) before += s_tot[k];
      all += s_tot[k];
    }
    const int64_t base = b.group_token_off[g];
    segment_starts(b.step_len, v0, v1, base + before, (float)n, lp, lane, ok);
    if (warp == 0 && lane == 0 && base + all != b.group_token_off[g + 1]) ok = false;
  }
  if (!ok) report(st, GPO_ERR_SHAPE, 6, g);
}

__global__ void __launch_bounds__(256) loss_weights_kernel(Sizes sz, LossPlan lp) {
  if (aborted(lp.status)) return;
  const double groups = (double)lp.status[kLossWordGroups];
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < sz.N; v += stride) {
    const int64_t a = lp.start[v], e = v + 1 < sz.N ? lp.start[v + 1] : sz.T;
    const double ng = (double)lp.w[v];
    lp.w[v] = e > a && ng > 0.0 ? (float)(1.0 / (groups * ng * (double)(e - a))) : 0.f;
    // tiles whose first token k * kLossTile lies in [a, e)
    const int64_t k0 = (a + kLossTile - 1) / kLossTile, k1 = min((e + kLossTile - 1) / kLossTile, lp.ntiles);
    for (int64_t k = max(k0, (int64_t)0); k < k1; ++k) lp.tile_edge[k] = (int32_t)v;
    if (v == sz.N - 1) {
      lp.tile_edge[lp.ntiles] = (int32_t)v;
      lp.start[sz.N] = sz.T;
    }
  }
}

// e^x - 1 (em1) and e^x - 1 - x (k3) of x = log pi_ref - log pi_theta: for |x| < 1/2 from
// the Taylor series of e^x (terms up to x^10 / 10!: truncation below 1e-10 relative), else
// from the fast exponential (|e^x - 1| >= 0.39 and k3 >= 0.1 there, so its few-ulp error
// stays a few ulp)
__device__ __forceinline__ void kl_terms(float x, float& em1, float& k3) {
  if (fabsf(x) < 0.5f) {
    float p = 1.f / 3628800.f;
    p = fmaf(p, x, 1.f / 362880.f);
    p = fmaf(p, x, 1.f / 40320.f);
    p = fmaf(p, x, 1.f / 5040.f);
    p = fmaf(p, x, 1.f / 720.f);
    p = fmaf(p, x, 1.f / 120.f);
    p = fmaf(p, x, 1.f / 24.f);
    p = fmaf(p, x, 1.f / 6.f);
    p = fmaf(p, x, 0.5f);
    k3 = x * x * p;
    em1 = x + k3;
  } else {
    em1 = __expf(x) - 1.f;
    k3 = em1 - x;
  }
}

// w min(r A, clip(r) A) = min(r wA, clip(r) wA) for the edge's wA = w A (w > 0), its
// derivative with respect to log r (r wA where the unclipped term is the minimum, else 0);
// true if the clipped term was strictly smaller
__device__ __forceinline__ bool surrogate(float r, float rc, float wa, float& f, float& df) {
  const float u = r * wa, c = rc * wa;
  const bool take = u <= c;
  f = fminf(u, c);
  df = take ? u : 0.f;
  return !take;
}

// Shared memory of one CTA: the tile's edges (at most one per token)
template <bool kSplit, bool kKL>
struct LossSmem {
  uint16_t map[kLossTile];                // edge (tile-local) of every token of the tile
  int16_t start[kLossTile + 2];           // first token of each edge, relative to the tile
  float wa[kLossTile];                    // w A (dual) or w A_cor (split)
  float we[kSplit ? kLossTile : 1];       // split: w lambda m_eff A_eff
  float w[kKL ? kLossTile : 1];           // KL: w
  float2 red[kLossThreads / 32][3];
  long long redn[kLossThreads / 32];
  int last;
};

template <bool kSplit, bool kKL>
__global__ void __launch_bounds__(kLossThreads, kKL ? 3 : 4) token_loss_kernel(LossArgs a, LossPlan lp) {
  extern __shared__ __align__(16) unsigned char loss_smem[];
  LossSmem<kSplit, kKL>& sm = *reinterpret_cast<LossSmem<kSplit, kKL>*>(loss_smem);
  if (aborted(lp.status)) return;  // the plan found a layout error (read before any block ran)
  if (lp.dims[0] != a.N || lp.dims[1] != a.T) {  // a plan of another batch shape
    if (threadIdx.x == 0) report(lp.status, GPO_ERR_SHAPE, 7, 0);
    return;
  }
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float inv_t = a.inv_t;
  // across tiles: float pairs for the policy term, the KL term and the sum of r (every
  // addition's rounding error kept in the low word), an integer count of clipped tokens
  float2 acc[3] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  long long nclip_all = 0;
  const int64_t ntiles = a.N > 0 ? lp.ntiles : 0;  // (a valid plan has no tokens without edges)
  for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const int64_t t0 = tile * kLossTile;
    const int tn = (int)min((int64_t)kLossTile, a.T - t0);  // tokens of this tile
    // this thread's token chunks first (streaming loads, all in flight together), then the
    // tile's edges: the two memory latencies overlap
    float x[kLossChunks][4], y[kLossChunks][4], z[kLossChunks][4];
#pragma unroll
    for (int k = 0; k < kLossChunks; ++k) {
      const int rel = 4 * (tid + k * kLossThreads);
      const int64_t q = t0 + rel;
      if (rel + 4 <= tn) {
        const float4 u = __ldcs(reinterpret_cast<const float4*>(a.logp + q));
        const float4 v = __ldcs(reinterpret_cast<const float4*>(a.old_logp + q));
        x[k][0] = u.x, x[k][1] = u.y, x[k][2] = u.z, x[k][3] = u.w;
        y[k][0] = v.x, y[k][1] = v.y, y[k][2] = v.z, y[k][3] = v.w;
        if (kKL) {
          const float4 w4 = __ldcs(reinterpret_cast<const float4*>(a.ref_logp + q));
          z[k][0] = w4.x, z[k][1] = w4.y, z[k][2] = w4.z, z[k][3] = w4.w;
        }
      } else {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const bool in = rel + c < tn;
          x[k][c] = in ? a.logp[q + c] : 0.f;
          y[k][c] = in ? a.old_logp[q + c] : 0.f;
          if (kKL) z[k][c] = in ? a.ref_logp[q + c] : 0.f;
        }
      }
    }
    // edges [e_lo, e_hi] hold the tile's tokens (each edge has >= 1 token: at most kLossTile)
    const int e_lo = min(max(lp.tile_edge[tile], 0), a.N - 1);
    const int e_hi = min(max(lp.tile_edge[tile + 1], e_lo), min(a.N - 1, e_lo + kLossTile - 1));
    const int ne = e_hi - e_lo + 1;
    __syncthreads();  // the previous tile's readers are done
    for (int j = tid; j <= ne; j += kLossThreads) {
      const int64_t st = lp.start[e_lo + j] - t0;
      sm.start[j] = (int16_t)max(min(st, (int64_t)kLossTile), (int64_t)0);  // clamped to the tile
      if (j < ne) {
        const float w = a.norm_token ? inv_t : lp.w[e_lo + j];
        sm.wa[j] = w * a.adv[e_lo + j];
        if (kSplit) sm.we[j] = a.mask[e_lo + j] ? w * (a.lambda * a.eff[e_lo + j]) : 0.f;
        if (kKL) sm.w[j] = w;
      }
    }
    __syncthreads();
    // the token -> edge map of the tile: warp w fills the spans of edges w, w + 8, ...
    for (int j = warp; j < ne; j += kLossThreads / 32)
      for (int t = sm.start[j] + lane; t < sm.start[j + 1]; t += 32) sm.map[t] = (uint16_t)j;
    __syncthreads();
    float pg = 0.f, kl = 0.f, rs = 0.f;
    int nclip = 0;
#pragma unroll
    for (int k = 0; k < kLossChunks; ++k) {
      const int rel = 4 * (tid + k * kLossThreads);  // first token of this chunk in the tile
      if (rel >= tn) continue;
      const uint2 m4 = *reinterpret_cast<const uint2*>(sm.map + rel);  // the 4 tokens' edges
      const int jj[4] = {(int)(m4.x & 0xFFFFu), (int)(m4.x >> 16), (int)(m4.y & 0xFFFFu), (int)(m4.y >> 16)};
      float gr[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const bool in = rel + c < tn;
        const int j = in ? min(jj[c], ne - 1) : 0;  // tokens past the tile's end read edge 0
        const float r = __expf(x[k][c] - y[k][c]);
        const float rc = fminf(fmaxf(r, a.lo), a.hi);
        float f, df;
        const bool clipped = surrogate(r, rc, sm.wa[j], f, df);
        if (kSplit) {
          float f2, df2;
          surrogate(r, rc, sm.we[j], f2, df2);
          f += f2;
          df += df2;
        }
        float g = -df;
        if (kKL) {
          float em1, k3;
          kl_terms(z[k][c] - x[k][c], em1, k3);
          const float w = sm.w[j];
          kl = in ? fmaf(w, k3, kl) : kl;
          g = fmaf(-a.beta * w, em1, g);  // beta w (1 - e^x)
        }
        if (in) {
          pg += f;
          rs += r;
          nclip += clipped ? 1 : 0;
        }
        gr[c] = g;
      }
      if (a.grad) {
        const int64_t q = t0 + rel;
        if (rel + 4 <= tn) __stcs(reinterpret_cast<float4*>(a.grad + q), make_float4(gr[0], gr[1], gr[2], gr[3]));
        else
          for (int c = 0; rel + c < tn; ++c) a.grad[q + c] = gr[c];
      }
    }
    ff_acc(acc[0].x, acc[0].y, pg);
    ff_acc(acc[1].x, acc[1].y, kl);
    ff_acc(acc[2].x, acc[2].y, rs);
    nclip_all += nclip;
  }
  // CTA sums in a fixed tree of pair additions, then the last CTA adds the partials in a
  // fixed order; the slots of lp.partial hold float pairs (and the clip count as an integer)
  float2* part = reinterpret_cast<float2*>(lp.partial);
  long long* part_n = reinterpret_cast<long long*>(lp.partial);
  auto warp_tree = [&](float2 (&v)[3], long long& n) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
      for (int i = 0; i < 3; ++i) {
        const float2 u = make_float2(__shfl_xor_sync(0xffffffffu, v[i].x, o), __shfl_xor_sync(0xffffffffu, v[i].y, o));
        v[i] = ff_add(v[i], u);
      }
      n += __shfl_xor_sync(0xffffffffu, n, o);
    }
  };
  warp_tree(acc, nclip_all);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < 3; ++i) sm.red[warp][i] = acc[i];
    sm.redn[warp] = nclip_all;
  }
  __syncthreads();
  if (tid == 0) {
    float2 t[3] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    long long n = 0;
    for (int k = 0; k < kLossThreads / 32; ++k) {
#pragma unroll
      for (int i = 0; i < 3; ++i) t[i] = ff_add(t[i], sm.red[k][i]);
      n += sm.redn[k];
    }
#pragma unroll
    for (int i = 0; i < 3; ++i) part[4 * blockIdx.x + i] = t[i];
    part_n[4 * blockIdx.x + 3] = n;
    __threadfence();
    sm.last = atomicAdd(&lp.status[kLossWordTicket], 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!sm.last) return;
  // the last CTA: every thread loads the partials of CTAs tid, tid + 256, ... (all loads in
  // flight together), then the same fixed trees as above
  __threadfence();
  constexpr int kMaxPer = kLossMaxBlocks / kLossThreads;
  float2 pt[kMaxPer][3];
  long long pn[kMaxPer];
#pragma unroll
  for (int m = 0; m < kMaxPer; ++m) {
    const int blk = tid + m * kLossThreads;
    const bool have = blk < (int)gridDim.x;
#pragma unroll
    for (int i = 0; i < 3; ++i) pt[m][i] = have ? __ldcg(&part[4 * blk + i]) : make_float2(0.f, 0.f);
    pn[m] = have ? __ldcg(&part_n[4 * blk + 3]) : 0ll;
  }
  float2 t[3] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  long long n = 0;
#pragma unroll
  for (int m = 0; m < kMaxPer; ++m) {
#pragma unroll
    for (int i = 0; i < 3; ++i) t[i] = ff_add(t[i], pt[m][i]);
    n += pn[m];
  }
  warp_tree(t, n);
  __syncthreads();  // every thread has read sm.red above
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < 3; ++i) sm.red[warp][i] = t[i];
    sm.redn[warp] = n;
  }
  __syncthreads();
  if (tid == 0) {
    float2 u[3] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    long long nn = 0;
    for (int k = 0; k < kLossThreads / 32; ++k) {
#pragma unroll
      for (int i = 0; i < 3; ++i) u[i] = ff_add(u[i], sm.red[k][i]);
      nn += sm.redn[k];
    }
    const double pg = (double)u[0].x + (double)u[0].y;
    const double kl_term = kKL ? (double)u[1].x + (double)u[1].y : 0.0;
    const double rsum = (double)u[2].x + (double)u[2].y;
    *a.loss = (float)(-(pg - (double)a.beta * kl_term));
    if (a.stats) {
      a.stats[0] = pg;
      a.stats[1] = kl_term;
      a.stats[2] = (double)nn;
      a.stats[3] = a.T > 0 ? rsum / (double)a.T : 0.0;
    }
    lp.status[kLossWordTicket] = 0u;  // ready for the next call on this plan
  }
}

template <bool kSplit, bool kKL>
cudaError_t setup_loss_variant() {
  return cudaFuncSetAttribute(token_loss_kernel<kSplit, kKL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)sizeof(LossSmem<kSplit, kKL>));
}

template <bool kSplit, bool kKL>
cudaError_t launch_loss_variant(const LaunchCtx& lc, const LossPlan& lp, const LossArgs& a) {
  const int bytes = (int)sizeof(LossSmem<kSplit, kKL>);
  const int per_sm = kKL ? 3 : 4;  // resident CTAs (registers, shared memory)
  const int64_t cap = min((int64_t)lc.num_sms * per_sm, (int64_t)kLossMaxBlocks);
  const int grid = (int)max((int64_t)1, min(lp.ntiles, cap));
  token_loss_kernel<kSplit, kKL><<<grid, kLossThreads, bytes, lc.stream>>>(a, lp);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_loss_plan(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const LossPlan& lp) {
  if (sz.G > 0) loss_plan_kernel<<<sz.G, kPlanThreads, 0, lc.stream>>>(b, sz, lp);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess && sz.N > 0) {
    const int64_t want = (sz.N + 255) / 256;
    const int blocks = (int)min(want, (int64_t)lc.num_sms * 8);
    loss_weights_kernel<<<blocks, 256, 0, lc.stream>>>(sz, lp);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t setup_loss() {
  cudaError_t e = setup_loss_variant<false, false>();
  if (e == cudaSuccess) e = setup_loss_variant<false, true>();
  if (e == cudaSuccess) e = setup_loss_variant<true, false>();
  if (e == cudaSuccess) e = setup_loss_variant<true, true>();
  return e;
}

cudaError_t launch_token_loss(const LaunchCtx& lc, const LossPlan& lp, const LossArgs& a) {
  if (a.split) return a.kl ? launch_loss_variant<true, true>(lc, lp, a) : launch_loss_variant<true, false>(lc, lp, a);
  return a.kl ? launch_loss_variant<false, true>(lc, lp, a) : launch_loss_variant<false, false>(lc, lp, a);
}

}  // namespace gpo
