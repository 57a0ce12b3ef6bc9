// Validation and planning (first kernel), per-state row statistics, and the
// per-token advantage scatter (last kernel) of the GraphPO path.
#include "gpo_internal.cuh"

namespace gpo {

constexpr int kPlanThreads = 1024;

// Similarity work items of a group with n states, in row blocks of 128 states: one
// diagonal item per block (the block against itself; it also yields the block's
// norms), and off-diagonal items (the block against the columns after it, in chunks
// of 256).
__host__ __device__ inline int blocks_for(int n) { return (n + kTileM - 1) / kTileM; }

__host__ __device__ inline int offdiag_chunks(int n, int rb) {
  const int rem = n - (rb + 1) * kTileM;
  return rem > 0 ? (rem + kTileN - 1) / kTileN : 0;
}

__host__ __device__ inline int offdiag_for(int n) {
  int c = 0;
  for (int rb = 0; rb * kTileM < n; ++rb) c += offdiag_chunks(n, rb);
  return c;
}

// Inclusive scan of one int per thread across a block of kPlanThreads.
__device__ int block_incl_scan(int x, int* warp_tot) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[wid] = x;
  __syncthreads();
  if (wid == 0) {
    int t = warp_tot[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    warp_tot[lane] = t;
  }
  __syncthreads();
  const int add = wid > 0 ? warp_tot[wid - 1] : 0;
  const int res = x + add;
  __syncthreads();
  return res;
}

// ---------------------------------------------------------------------------
// K0: validate the offset arrays, rewards and step lengths; write per-state
// (rollout, depth) and per-rollout group; the last block to finish plans the
// similarity work items.  Nothing is dereferenced before its range is checked.
__global__ void __launch_bounds__(kPlanThreads) prep_kernel(gpo_batch b, Sizes sz, Ws ws) {
  uint32_t* st = ws.status;
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int nth = gridDim.x * blockDim.x;
  const int32_t* go = b.group_rollout_off;
  const int32_t* so = b.rollout_step_off;
  const int64_t* to = b.rollout_token_off;

  if (tid == 0) {
    if (go[0] != 0 || go[sz.G] != sz.R) report(st, GPO_ERR_SHAPE, 0, 0);
    if (so[0] != 0 || so[sz.R] != sz.N) report(st, GPO_ERR_SHAPE, 0, 1);
    if (to[0] != 0 || to[sz.R] != sz.T) report(st, GPO_ERR_SHAPE, 0, 2);
  }
  for (int g = tid; g < sz.G; g += nth) {
    const int a = go[g], c = go[g + 1];
    if (a < 0 || c < a || c > sz.R) {
      report(st, GPO_ERR_SHAPE, 0, 3);
      continue;
    }
    for (int r = a; r < c; ++r) ws.rollout_group[r] = g;
  }
  // one warp per rollout: its lanes stride over the rollout's steps
  const int lane = threadIdx.x & 31;
  for (int r = tid >> 5; r < sz.R; r += nth >> 5) {
    const int s = so[r], e = so[r + 1];
    if (s < 0 || e <= s || e > sz.N) {  // every rollout has at least one step
      if (lane == 0) report(st, GPO_ERR_SHAPE, 0, 4);
      continue;
    }
    if (lane == 0 && b.reward[r] > 1) report(st, GPO_ERR_BAD_REWARD, 0, r);
    int64_t sum = 0;
    bool bad = false;
    for (int v = s + lane; v < e; v += 32) {
      const int L = b.step_len[v];
      bad |= L < 1;
      sum += L;
      ws.state_meta[v] = make_int2(r, v - s + 1);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    bad = __any_sync(0xffffffffu, bad);
    if (lane == 0) {
      if (bad) report(st, GPO_ERR_SHAPE, 0, 5);
      const int64_t t0 = to[r], t1 = to[r + 1];
      if (t0 < 0 || t1 > sz.T || t1 - t0 != sum) report(st, GPO_ERR_SHAPE, 0, 6);
    }
  }

  // ---- last block: plan the work items
  __shared__ int s_last;
  __shared__ int s_warp[32];
  __shared__ int s_carry;
  __shared__ int s_incl[kPlanThreads], s_s0[kPlanThreads], s_n[kPlanThreads];
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(&st[kStTicket], 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (threadIdx.x == 0) s_carry = 0;
  __syncthreads();
  const bool ok = !aborted(st);
  // items group by group: a group's diagonal items (one per row block, block order), then
  // its off-diagonal ones; every item an off-diagonal item waits for thus comes before it
  for (int base = 0; base < sz.G; base += kPlanThreads) {
    const int g = base + threadIdx.x;
    int cnt = 0, nb = 0, s0 = 0, n = 0;
    if (ok && g < sz.G) {
      const int r0 = go[g], r1 = go[g + 1];
      s0 = so[r0];
      n = so[r1] - s0;
      if (n > sz.maxn || n > GPO_MAX_GROUP_STATES) report(st, GPO_ERR_UNSUPPORTED, 0, g);
      nb = blocks_for(n);
      cnt = nb + offdiag_for(n);
    }
    const int incl = block_incl_scan(cnt, s_warp);
    if (ok && g < sz.G) {
      GroupInfo gi;
      gi.s0 = s0;
      gi.n = n;
      gi.r0 = go[g];
      gi.nr = go[g + 1] - gi.r0;
      gi.blk0 = s_carry + incl - cnt;
      gi.nblk = nb;
      gi.off0 = gi.blk0 + nb;
      gi.noff = cnt - nb;
      ws.groups[g] = gi;
    }
    s_incl[threadIdx.x] = incl;
    s_s0[threadIdx.x] = s0;
    s_n[threadIdx.x] = n;
    __syncthreads();
    const int batch = s_incl[kPlanThreads - 1];
    for (int j = threadIdx.x; j < batch && ok; j += kPlanThreads) {
      int lo = 0, hi = kPlanThreads - 1;  // first t with s_incl[t] > j
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (s_incl[mid] > j) hi = mid;
        else lo = mid + 1;
      }
      const int gn = s_n[lo], gs0 = s_s0[lo], gnb = blocks_for(gn);
      int idx = j - (s_incl[lo] - gnb - offdiag_for(gn));  // item index within the group
      const int k = s_carry + j;
      if (k >= ws.max_items) continue;
      Item it;
      it.group = base + lo;
      if (idx < gnb) {  // diagonal item of row block idx
        it.row0 = it.col0 = gs0 + idx * kTileM;
        it.ncols = min(kTileM, gn - idx * kTileM);
        ws.blk_ready[k] = 0;
      } else {
        idx -= gnb;
        int rb = 0;
        for (;; ++rb) {
          const int c = offdiag_chunks(gn, rb);
          if (idx < c) break;
          idx -= c;
        }
        it.row0 = gs0 + rb * kTileM;
        it.col0 = gs0 + (rb + 1) * kTileM + idx * kTileN;
        it.ncols = min(kTileN, gn - (rb + 1) * kTileM - idx * kTileN);
      }
      ws.items[k] = it;
      ws.edge_count[k] = 0;
    }
    __syncthreads();
    if (threadIdx.x == kPlanThreads - 1) s_carry += incl;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const int total = s_carry;
    if (total > ws.max_items) report(st, GPO_ERR_WORKSPACE, 0, total);
    st[kStItems] = aborted(st) ? 0u : (uint32_t)total;
  }
}

cudaError_t launch_prep(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws) {
  const int64_t work = 32 * ((int64_t)sz.R + 1);  // a warp per rollout
  int blocks = (int)((work + kPlanThreads - 1) / kPlanThreads);
  blocks = blocks < 1 ? 1 : (blocks > 4 * lc.num_sms ? 4 * lc.num_sms : blocks);
  prep_kernel<<<blocks, kPlanThreads, 0, lc.stream>>>(b, sz, ws);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// K1a: per state, |z_v|^2 and <z_{p(v)}, z_v> with fp32 accumulation (one warp
// per row: lane partial sums over a strided set of elements, then a shuffle
// tree).  p(v) is the previous state of the rollout, or the prompt embedding
// for the first step when one is given.  Extra warps compute |root|^2.

template <bool kBf16>
__device__ __forceinline__ void load8(const void* base, int64_t elem, float (&x)[8]) {
  if (kBf16) {
    const uint4 u = *reinterpret_cast<const uint4*>(reinterpret_cast<const uint16_t*>(base) + elem);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[2 * i] = __uint_as_float(w[i] << 16);
      x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  } else {
    const float4* p = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(base) + elem);
    const float4 a = p[0], c = p[1];
    x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
    x[4] = c.x; x[5] = c.y; x[6] = c.z; x[7] = c.w;
  }
}

template <bool kBf16>
__device__ __forceinline__ float load1(const void* base, int64_t elem) {
  if (kBf16) return __uint_as_float((uint32_t)(reinterpret_cast<const uint16_t*>(base)[elem]) << 16);
  return reinterpret_cast<const float*>(base)[elem];
}

// kRootsOnly: only what the tcgen05 similarity kernel does not produce itself, i.e. the
// dots of first steps with the prompt embeddings and |root|^2.
template <bool kBf16, bool kRootsOnly>
__global__ void __launch_bounds__(256) row_stats_kernel(gpo_batch b, Sizes sz, Ws ws) {
  if (aborted(ws.status)) return;
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int nroot = b.root_emb ? sz.G : 0;
  const int d = sz.d, nvec = d / 8;
  for (int64_t job = warp; job < (int64_t)sz.N + nroot; job += nwarps) {
    const void* rowp;
    const void* parp = nullptr;
    int64_t row, prow = 0;
    if (job < sz.N) {
      row = job;
      rowp = b.emb;
      const int2 m = ws.state_meta[job];
      if (kRootsOnly && m.y > 1) continue;
      if (m.y > 1) {
        parp = b.emb;
        prow = job - 1;
      } else if (b.root_emb) {
        parp = b.root_emb;
        prow = ws.rollout_group[m.x];
      }
    } else {
      row = job - sz.N;
      rowp = b.root_emb;
    }
    const int64_t rb = row * sz.stride, pb = prow * sz.stride;
    float s2 = 0.f, sd = 0.f;
#pragma unroll 2
    for (int k = lane; k < nvec; k += 32) {
      float x[8];
      load8<kBf16>(rowp, rb + 8 * k, x);
      if (parp) {
        float y[8];
        load8<kBf16>(parp, pb + 8 * k, y);
#pragma unroll
        for (int i = 0; i < 8; ++i) sd = fmaf(x[i], y[i], sd);
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) s2 = fmaf(x[i], x[i], s2);
    }
    for (int k = nvec * 8 + lane; k < d; k += 32) {
      const float x = load1<kBf16>(rowp, rb + k);
      s2 = fmaf(x, x, s2);
      if (parp) sd = fmaf(x, load1<kBf16>(parp, pb + k), sd);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      s2 += __shfl_xor_sync(0xffffffffu, s2, o);
      sd += __shfl_xor_sync(0xffffffffu, sd, o);
    }
    if (lane == 0) {
      if (!isfinite(s2) || !isfinite(sd)) report(ws.status, GPO_ERR_NONFINITE, 1, (int)job);
      if (job < sz.N) {
        if (!kRootsOnly) {
          ws.nrm2[row] = s2;
          ws.rn[row] = s2 > 0.f ? 1.0f / sqrtf(s2) : 0.f;
        }
        ws.dotp[row] = sd;
      } else {
        ws.root_n2[row] = s2;
      }
    }
  }
}

// bf16 rows of d = 8 * 32 * kNV elements at most: one warp walks a run of 32
// consecutive rows (one coalesced metadata load for the run), holds a whole row in
// registers (kNV 16-byte chunks per lane) and keeps it as the parent of the next
// row, so every row is read once.  The prompt rows (|root|^2) and the dots of first
// steps against them come from the generic kernel's formula with plain loads.
template <int kNV>
__global__ void __launch_bounds__(256) row_stats_run_kernel(gpo_batch b, Sizes sz, Ws ws) {
  if (aborted(ws.status)) return;
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int nvec = sz.d / 8;
  const uint4* Z = reinterpret_cast<const uint4*>(b.emb);
  const int64_t rs = sz.stride / 8;  // row stride in 16-byte chunks
  auto load_row = [&](int64_t r, uint4 (&x)[kNV]) {
#pragma unroll
    for (int c = 0; c < kNV; ++c) {
      const int k = lane + 32 * c;
      x[c] = k < nvec ? Z[r * rs + k] : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  auto dot2 = [](uint32_t a, uint32_t b) {  // two bf16 pairs, fp32 products
    return __uint_as_float(a << 16) * __uint_as_float(b << 16) +
           __uint_as_float(a & 0xFFFF0000u) * __uint_as_float(b & 0xFFFF0000u);
  };
  for (int64_t base = warp * 32; base < sz.N; base += nwarps * 32) {
    const int64_t nrun = min((int64_t)32, (int64_t)sz.N - base);
    const int2 m = lane < nrun ? ws.state_meta[base + lane] : make_int2(0, 1);
    uint4 prev[kNV], cur[kNV], nxt[kNV];
    const int d0 = __shfl_sync(0xffffffffu, m.y, 0);
    if (d0 > 1) load_row(base - 1, prev);
    load_row(base, nxt);
    for (int i = 0; i < nrun; ++i) {
      const int dep = __shfl_sync(0xffffffffu, m.y, i);
      const int rol = __shfl_sync(0xffffffffu, m.x, i);
#pragma unroll
      for (int c = 0; c < kNV; ++c) cur[c] = nxt[c];
      if (i + 1 < nrun) load_row(base + i + 1, nxt);  // next row in flight during this one
      float s2 = 0.f, sd = 0.f;
#pragma unroll
      for (int c = 0; c < kNV; ++c) {
        const uint32_t w[4] = {cur[c].x, cur[c].y, cur[c].z, cur[c].w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const float lo = __uint_as_float(w[h] << 16), hi = __uint_as_float(w[h] & 0xFFFF0000u);
          s2 = fmaf(lo, lo, s2);
          s2 = fmaf(hi, hi, s2);
        }
      }
      if (dep > 1) {
#pragma unroll
        for (int c = 0; c < kNV; ++c) {
          sd += dot2(cur[c].x, prev[c].x) + dot2(cur[c].y, prev[c].y);
          sd += dot2(cur[c].z, prev[c].z) + dot2(cur[c].w, prev[c].w);
        }
      } else if (b.root_emb) {
        const uint16_t* R = reinterpret_cast<const uint16_t*>(b.root_emb) + (int64_t)ws.rollout_group[rol] * sz.stride;
        const uint16_t* X = reinterpret_cast<const uint16_t*>(b.emb) + (base + i) * sz.stride;
        for (int k = lane; k < sz.d; k += 32)
          sd = fmaf(__uint_as_float((uint32_t)X[k] << 16), __uint_as_float((uint32_t)R[k] << 16), sd);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        s2 += __shfl_xor_sync(0xffffffffu, s2, o);
        sd += __shfl_xor_sync(0xffffffffu, sd, o);
      }
      if (lane == 0) {
        const int64_t row = base + i;
        if (!isfinite(s2) || !isfinite(sd)) report(ws.status, GPO_ERR_NONFINITE, 1, (int)row);
        ws.nrm2[row] = s2;
        ws.dotp[row] = sd;
        ws.rn[row] = s2 > 0.f ? 1.0f / sqrtf(s2) : 0.f;
      }
#pragma unroll
      for (int c = 0; c < kNV; ++c) prev[c] = cur[c];
    }
  }
  // |root|^2 of every prompt embedding
  if (b.root_emb) {
    const uint16_t* R = reinterpret_cast<const uint16_t*>(b.root_emb);
    for (int64_t g = warp; g < sz.G; g += nwarps) {
      float s2 = 0.f;
      for (int k = lane; k < sz.d; k += 32) {
        const float x = __uint_as_float((uint32_t)R[g * sz.stride + k] << 16);
        s2 = fmaf(x, x, s2);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s2 += __shfl_xor_sync(0xffffffffu, s2, o);
      if (lane == 0) {
        if (!isfinite(s2)) report(ws.status, GPO_ERR_NONFINITE, 1, (int)(sz.N + g));
        ws.root_n2[g] = s2;
      }
    }
  }
}

cudaError_t launch_root_stats(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws) {
  const int64_t jobs = (int64_t)sz.N + sz.G;
  if (!b.root_emb || jobs == 0) return cudaSuccess;
  int64_t blocks = (jobs * 32 + 255) / 256;
  if (blocks > (int64_t)lc.num_sms * 8) blocks = (int64_t)lc.num_sms * 8;
  row_stats_kernel<true, true><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
  return cudaGetLastError();
}

cudaError_t launch_row_stats(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws) {
  const int64_t jobs = (int64_t)sz.N + (b.root_emb ? sz.G : 0);
  if (jobs == 0) return cudaSuccess;
  int64_t blocks = (jobs * 32 + 255) / 256;
  const int64_t cap = (int64_t)lc.num_sms * 8;
  if (blocks > cap) blocks = cap;
  const bool aligned16 = (reinterpret_cast<uintptr_t>(b.emb) & 15u) == 0 && sz.stride % 8 == 0 && sz.d % 8 == 0;
  if (b.emb_dtype == GPO_EMB_BF16 && aligned16 && sz.d <= 8 * 32 * 8) {
    int64_t rblocks = ((int64_t)sz.N + 255) / 256;  // a warp per 32 rows
    if (rblocks < 1) rblocks = 1;
    if (rblocks > (int64_t)lc.num_sms * 8) rblocks = (int64_t)lc.num_sms * 8;
    if (sz.d <= 8 * 32 * 4)
      row_stats_run_kernel<4><<<(int)rblocks, 256, 0, lc.stream>>>(b, sz, ws);
    else
      row_stats_run_kernel<8><<<(int)rblocks, 256, 0, lc.stream>>>(b, sz, ws);
  } else if (b.emb_dtype == GPO_EMB_BF16)
    row_stats_kernel<true, false><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
  else
    row_stats_kernel<false, false><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// K3: every token of edge e receives e's advantage (Sec. 4.5).  One warp
// writes whole edge spans: the metadata of 32 consecutive edges is fetched in
// one coalesced round trip and broadcast by shuffles; each span is written
// with 16-byte stores in its aligned middle and scalar stores at the ends.

__global__ void __launch_bounds__(256) tokens_kernel(gpo_batch b, gpo_outputs o, Sizes sz, Ws ws) {
  if (aborted(ws.status)) return;
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t base = warp * 32; base < sz.N; base += nwarps * 32) {
    const int64_t v = base + lane;
    int64_t ts = 0;
    int L = 0;
    float va = 0.f, vc = 0.f, ve = 0.f;
    uint32_t vm = 0;
    if (v < sz.N) {
      ts = ws.tok_start[v];
      L = b.step_len[v];
      va = ws.e_adv[v];
      if (o.adv_cor) vc = ws.e_cor[v];
      if (o.adv_eff) ve = ws.e_eff[v];
      if (o.eff_mask) vm = ws.e_mask[v];
    }
    const int cnt = (int)(sz.N - base < 32 ? sz.N - base : 32);
    for (int j = 0; j < cnt; ++j) {
      const int64_t s = __shfl_sync(0xffffffffu, ts, j);
      const int64_t e = s + __shfl_sync(0xffffffffu, L, j);
      write_span(o.adv, s, e, __shfl_sync(0xffffffffu, va, j), lane);
      if (o.adv_cor) write_span(o.adv_cor, s, e, __shfl_sync(0xffffffffu, vc, j), lane);
      if (o.adv_eff) write_span(o.adv_eff, s, e, __shfl_sync(0xffffffffu, ve, j), lane);
      if (o.eff_mask) write_span_u8(o.eff_mask, s, e, (uint8_t)__shfl_sync(0xffffffffu, vm, j), lane);
    }
  }
}

cudaError_t launch_tokens(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                          const Ws& ws) {
  if (sz.T == 0 || sz.N == 0) return cudaSuccess;
  int64_t blocks = (sz.N + 255) / 256;  // one warp per 32 edges
  const int64_t cap = (int64_t)lc.num_sms * 8;
  if (blocks > cap) blocks = cap;
  tokens_kernel<<<(unsigned)blocks, 256, 0, lc.stream>>>(b, o, sz, ws);
  return cudaGetLastError();
}

}  // namespace gpo
