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
  const bool tree = b.parent != nullptr;  // tree layout: tree_prep_kernel checks the groups and lays out their states

  if (tid == 0) {
    if (go[0] != 0 || go[sz.G] != sz.R) report(st, GPO_ERR_SHAPE, 0, 0);
    if (tree) {
      if (b.group_state_off[0] != 0 || b.group_state_off[sz.G] != sz.N) report(st, GPO_ERR_SHAPE, 0, 1);
      if (b.group_token_off[0] != 0 || b.group_token_off[sz.G] != sz.T) report(st, GPO_ERR_SHAPE, 0, 2);
    } else {
      if (so[0] != 0 || so[sz.R] != sz.N) report(st, GPO_ERR_SHAPE, 0, 1);
      if (to[0] != 0 || to[sz.R] != sz.T) report(st, GPO_ERR_SHAPE, 0, 2);
    }
  }
  for (int g = tid; g < sz.G; g += nth) {
    const int a = go[g], c = go[g + 1];
    if (a < 0 || c < a || c > sz.R) report(st, GPO_ERR_SHAPE, 0, 3);
  }
  // one warp per rollout: its lanes stride over the rollout's steps
  const int lane = threadIdx.x & 31;
  for (int r = tid >> 5; r < (tree ? 0 : sz.R); r += nth >> 5) {
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
      s0 = tree ? b.group_state_off[g] : so[r0];
      n = (tree ? b.group_state_off[g + 1] : so[r1]) - s0;
      if (tree && (s0 < 0 || n < 0 || s0 + n > sz.N)) {  // reported by tree_prep_kernel
        s0 = 0;
        n = 0;
      }
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

// ---------------------------------------------------------------------------
// K0 (tree layout, before the planning kernel): one CTA per prompt group.  Checks the
// group's offsets, parents (earlier states of the group, depth-first pre-order), step
// lengths, leaf count and rewards; writes per state {group, depth}, the global parent,
// the end of its subtree, its own terminal statistics (Sec. 4.3: c_own / t_own = the
// rewards / the number of the leaves of its subtree, bottom-up along direct edges) and
// the first token of its edge.
constexpr int kTreeThreads = 1024;

// Exclusive scan of (a, b) over the block; returns the block totals too.
__device__ void block_excl_scan2(int& a, long long& b, int& ta, long long& tb, int* wa, long long* wb) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = a;
  long long y = b;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, x, o);
    const long long v = __shfl_up_sync(0xffffffffu, y, o);
    if (lane >= o) {
      x += u;
      y += v;
    }
  }
  if (lane == 31) {
    wa[wid] = x;
    wb[wid] = y;
  }
  __syncthreads();
  int pa = 0;
  long long pb = 0;
  ta = 0;
  tb = 0;
  for (int w = 0; w < nw; ++w) {
    if (w < wid) {
      pa += wa[w];
      pb += wb[w];
    }
    ta += wa[w];
    tb += wb[w];
  }
  a = pa + x - a;
  b = pb + y - b;
  __syncthreads();
}

__host__ __device__ inline size_t tree_prep_smem(int maxn) { return 4 * sizeof(int) * (size_t)(maxn < 1 ? 1 : maxn); }

__global__ void __launch_bounds__(kTreeThreads) tree_prep_kernel(gpo_batch b, Sizes sz, Ws ws) {
  extern __shared__ int tsm[];
  __shared__ int s_wa[32];
  __shared__ long long s_wb[32];
  uint32_t* st = ws.status;
  const int g = blockIdx.x, tid = threadIdx.x, nt = blockDim.x;
  const int r0 = b.group_rollout_off[g], r1 = b.group_rollout_off[g + 1];
  const int s0 = b.group_state_off[g], s1 = b.group_state_off[g + 1];
  const int64_t t0 = b.group_token_off[g], t1 = b.group_token_off[g + 1];
  if (r0 < 0 || r1 < r0 || r1 > sz.R || s0 < 0 || s1 < s0 || s1 > sz.N || t0 < 0 || t1 < t0 || t1 > sz.T ||
      r1 - r0 > s1 - s0 || (s1 == s0 && (r1 != r0 || t1 != t0)) || (s1 > s0 && r1 == r0)) {
    if (tid == 0) report(st, GPO_ERR_SHAPE, 0, 7);
    return;
  }
  const int n = s1 - s0, nr = r1 - r0;
  if (n == 0) return;
  if (n > sz.maxn || n > GPO_MAX_GROUP_STATES) return;  // the planning kernel reports it
  int* par = tsm;
  int* end = tsm + n;
  int* cown = tsm + 2 * n;
  int* town = tsm + 3 * n;
  bool bad = false;
  for (int i = tid; i < n; i += nt) {
    const int pp = b.parent[s0 + i], L = b.step_len[s0 + i];
    par[i] = pp;
    end[i] = i + 1;
    cown[i] = town[i] = 0;
    bad = bad || pp < -1 || pp >= i || L < 1;
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) report(st, GPO_ERR_SHAPE, 0, 8);
    return;
  }
  for (int i = tid; i < n; i += nt) {
    const int pp = par[i];
    if (pp >= 0) {  // pre-order: p(v) lies on the path from the root to the state before v
      int x = i - 1;
      while (x > pp) x = par[x];
      bad = bad || x != pp;
    }
    int d = 1;
    for (int x = pp; x >= 0; x = par[x]) {  // par[x] < x: at most i steps
      ++d;
      atomicMax(&end[x], i + 1);
    }
    ws.state_meta[s0 + i] = make_int2(g, d);
    ws.tree_par[s0 + i] = pp < 0 ? -1 : s0 + pp;
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) report(st, GPO_ERR_SHAPE, 0, 9);
    return;
  }
  // leaves in state order are the group's rollouts; edge spans follow in state order.  Each
  // thread takes a contiguous run of states; one block scan over the runs.
  const int per = (n + nt - 1) / nt, a0 = min(n, tid * per), a1 = min(n, a0 + per);
  int lc = 0;
  long long tc = 0;
  for (int i = a0; i < a1; ++i) {
    lc += end[i] == i + 1;
    tc += b.step_len[s0 + i];
  }
  int ltot;
  long long ttot;
  block_excl_scan2(lc, tc, ltot, ttot, s_wa, s_wb);
  if (ltot != nr || ttot != t1 - t0) {
    if (tid == 0) report(st, GPO_ERR_SHAPE, 0, 10);
    return;
  }
  for (int i = a0; i < a1; ++i) {
    ws.tok_start[s0 + i] = t0 + tc;
    tc += b.step_len[s0 + i];
    if (end[i] == i + 1) {
      const int rw = b.reward[r0 + lc];
      ++lc;
      if (rw > 1) {
        report(st, GPO_ERR_BAD_REWARD, 0, r0 + lc - 1);
        bad = true;
      } else {
        for (int x = i; x >= 0; x = par[x]) {
          atomicAdd(&cown[x], rw);
          atomicAdd(&town[x], 1);
        }
      }
    }
  }
  if (__syncthreads_or(bad)) return;
  for (int i = tid; i < n; i += nt) {
    ws.tree_end[s0 + i] = s0 + end[i];
    ws.tree_own[s0 + i] = make_int2(cown[i], town[i]);
  }
}

cudaError_t setup_tree_prep() {
  return cudaFuncSetAttribute(tree_prep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)tree_prep_smem(GPO_MAX_GROUP_STATES));
}

cudaError_t launch_tree_prep(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws) {
  if (sz.G == 0) return cudaSuccess;
  int threads = (sz.maxn + 31) & ~31;
  threads = threads < 64 ? 64 : (threads > kTreeThreads ? kTreeThreads : threads);
  tree_prep_kernel<<<sz.G, threads, tree_prep_smem(sz.maxn), lc.stream>>>(b, sz, ws);
  return cudaGetLastError();
}

cudaError_t launch_prep(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws) {
  const int64_t work = 32 * ((int64_t)sz.R + 1);  // a warp per rollout
  int blocks = (int)((work + kPlanThreads - 1) / kPlanThreads);
  blocks = blocks < 1 ? 1 : (blocks > 4 * lc.num_sms ? 4 * lc.num_sms : blocks);
  prep_kernel<<<blocks, kPlanThreads, 0, lc.stream>>>(b, sz, ws);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// K1a (CUDA-core similarity only): |z_v|^2 and 1/|z_v| with fp32 accumulation for the
// threshold test, one warp per row (lane partial sums over a strided set of elements, then
// a shuffle tree).  eta takes its norms from exact_stats instead.

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

template <bool kBf16, bool kVec>
__global__ void __launch_bounds__(256) row_stats_kernel(gpo_batch b, Sizes sz, Ws ws) {
  if (aborted(ws.status)) return;
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int d = sz.d, nvec = kVec ? d / 8 : 0;
  for (int64_t row = warp; row < sz.N; row += nwarps) {
    const int64_t rb = row * sz.stride;
    float s2 = 0.f;
#pragma unroll 2
    for (int k = lane; k < nvec; k += 32) {
      float x[8];
      load8<kBf16>(b.emb, rb + 8 * k, x);
#pragma unroll
      for (int i = 0; i < 8; ++i) s2 = fmaf(x[i], x[i], s2);
    }
    for (int k = nvec * 8 + lane; k < d; k += 32) {
      const float x = load1<kBf16>(b.emb, rb + k);
      s2 = fmaf(x, x, s2);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s2 += __shfl_xor_sync(0xffffffffu, s2, o);
    if (lane == 0) {
      if (!isfinite(s2)) report(ws.status, GPO_ERR_NONFINITE, 1, (int)row);
      ws.nrm2[row] = s2;
      ws.rn[row] = s2 > 0.f ? 1.0f / sqrtf(s2) : 0.f;
    }
  }
}

cudaError_t launch_row_stats(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws) {
  if (sz.N == 0) return cudaSuccess;
  int64_t blocks = ((int64_t)sz.N * 32 + 255) / 256;
  const int64_t cap = (int64_t)lc.num_sms * 8;
  if (blocks > cap) blocks = cap;
  const bool vec = (reinterpret_cast<uintptr_t>(b.emb) & 15u) == 0 && sz.stride % 8 == 0 && sz.d % 8 == 0;
  if (b.emb_dtype == GPO_EMB_BF16) {
    if (vec) row_stats_kernel<true, true><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
    else row_stats_kernel<true, false><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
  } else {
    if (vec) row_stats_kernel<false, true><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
    else row_stats_kernel<false, false><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Accurate row statistics for eta(p(v), v) = max(0, cos(z_{p(v)}, z_v)) (Sec. 4.3): |z_v|^2
// and <z_{p(v)}, z_v> as float pairs, one warp per state.  p(v) is the previous state of
// the rollout (chain layout) or the parent (tree layout); a root child is dotted with its
// group's prompt embedding when one is given.  bf16 products are exact in fp32, fp32
// products are split exactly by TwoProduct, and every sum is compensated (Sum2), so the
// cosine keeps ~1e-12 absolute accuracy even for nearly orthogonal rows, where a plain
// fp32 (or tensor-core) accumulation loses it: the standardisation of Sec. 4.4 then
// amplifies that loss in groups of nearly equal step rewards.
// Nothing outside the arrays is read whatever the offsets hold: rollout and group come
// from binary searches, and a parent outside [start of the group, v) counts as the root
// (the validating kernels report such inputs).

__device__ __forceinline__ int upper_idx(const int32_t* off, int n, int v) {  // last r < n with off[r] <= v
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= v) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// The same as upper_idx, for a value common to the warp: rounds of 32 probes (one
// coalesced load per round, log32(n) rounds) instead of log2(n) dependent loads.
__device__ __forceinline__ int warp_upper_idx(const int32_t* off, int n, int v, int lane) {
  int lo = 0, hi = n;  // the answer lies in [lo, hi)
  while (hi - lo > 1) {
    const int step = (hi - lo + 31) / 32;  // probes at lo, lo + step, ...
    const int k = lo + lane * step;
    const uint32_t m = __ballot_sync(0xffffffffu, k < hi && off[k] <= v);
    lo += (m ? 31 - __clz(m) : 0) * step;
    hi = min(hi, lo + step);
  }
  return lo;
}

template <bool kBf16>
__global__ void __launch_bounds__(256) exact_stats_kernel(gpo_batch b, Sizes sz, Ws ws) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const bool tree = b.parent != nullptr;
  // the states and prompt embeddings of groups [g0, g1) (the whole batch but for range calls)
  int v0 = 0, v1 = sz.N;
  if (sz.g0 != 0 || sz.g1 != sz.G) {
    const int32_t* go = b.group_rollout_off;
    if (tree) {
      v0 = b.group_state_off[sz.g0];
      v1 = b.group_state_off[sz.g1];
    } else {
      const int ra = go[sz.g0], rb = go[sz.g1];
      v0 = ra >= 0 && ra <= sz.R ? b.rollout_step_off[ra] : 0;
      v1 = rb >= 0 && rb <= sz.R ? b.rollout_step_off[rb] : 0;
    }
    v0 = max(0, min(v0, sz.N));
    v1 = max(v0, min(v1, sz.N));
  }
  const int nstate = v1 - v0, nroot = b.root_emb ? sz.g1 - sz.g0 : 0;
  for (int64_t jj = warp; jj < (int64_t)nstate + nroot; jj += nwarps) {
    const int64_t job = jj < nstate ? v0 + jj : sz.N + sz.g0 + (jj - nstate);
    if (job >= sz.N) {  // |prompt embedding|^2
      const int64_t g = job - sz.N;
      float2 n2, dot;
      exact_pair_sums<kBf16>(b.root_emb, g * sz.stride, nullptr, 0, false, sz.d, lane, n2, dot);
      if (lane == 0) {
        if (!isfinite(n2.x)) report(ws.status, GPO_ERR_NONFINITE, 3, (int)job);
        ws.x_root_n2[g] = n2;
      }
      continue;
    }
    const int v = (int)job;
    int prow = -1, g = -1;  // parent row, or the group whose prompt embedding is the parent
    if (tree) {
      if (sz.G > 0) {
        g = upper_idx(b.group_state_off, sz.G, v);
        const int s0 = b.group_state_off[g], pl = b.parent[v];
        if (pl >= 0 && s0 >= 0 && (int64_t)s0 + pl < v) prow = s0 + pl;
      }
    } else if (sz.R > 0) {
      const int r = upper_idx(b.rollout_step_off, sz.R, v);
      if (v > b.rollout_step_off[r]) prow = v - 1;
      else if (sz.G > 0) g = upper_idx(b.group_rollout_off, sz.G, r);
    }
    const bool root_parent = prow < 0 && b.root_emb && g >= 0;
    const void* pbase = prow >= 0 ? b.emb : (root_parent ? b.root_emb : nullptr);
    const int64_t poff = prow >= 0 ? (int64_t)prow * sz.stride : (root_parent ? (int64_t)g * sz.stride : 0);
    float2 n2, dot;
    exact_pair_sums<kBf16>(b.emb, (int64_t)v * sz.stride, pbase, poff, pbase != nullptr, sz.d, lane, n2, dot);
    if (lane == 0) {
      if (!isfinite(n2.x) || !isfinite(dot.x)) report(ws.status, GPO_ERR_NONFINITE, 3, v);
      ws.x_n2[v] = n2;
      ws.x_dot[v] = dot;
    }
  }
}

// bf16 rows (16-byte aligned, d a multiple of 32): a warp takes 8 consecutive rows, lane
// 4 r + j summing quarter j of row base + r in 16-byte chunks, four chunks in flight.  In the
// chain layout the parent of a row is the row before, whose chunk the lane 4 below already
// holds (a shuffle); the first row's parent chunk, a tree parent or a prompt embedding is
// loaded.  Compensated sums per lane, two fp32 lanes per instruction, then a fixed butterfly
// over the 4 quarters: the accuracy of exact_stats_kernel with every row read once.
//   kNorms = false: TwoSum per product (f2_acc).
//   kNorms = true (after the similarity stage, which leaves fp32 squared norms in ws.nrm2,
//   accurate to far better than 1 %): biased error-free sums with one bias per row and sum,
//   sigma = 2^ceil(log2 (4.04 |z_v|^2)) for |z_v|^2 and 2^ceil(log2 (2.02 (|z_v|^2 + |z_p|^2)))
//   for <z_p, z_v> (|x y| <= (x^2 + y^2) / 2), so that each running sum stays in
//   [sigma/2, 3 sigma/2] and every product is Fast2Sum's case (see BiasedSum): four fp32
//   operations per product, two independent chains per sum, no bound pass.  A lane whose sum
//   ends outside the range (a norm that was not what the similarity stage reported) sends its
//   row through the TwoSum path instead.
template <bool kNorms>
__global__ void __launch_bounds__(256) exact_stats_lane_kernel(gpo_batch b, Sizes sz, Ws ws) {
  const int lane = threadIdx.x & 31, r = lane >> 2, j = lane & 3;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const bool tree = b.parent != nullptr;
  const int nq = sz.d / 32;          // 16-byte chunks per quarter
  const int64_t rs = sz.stride / 8;  // row stride in 16-byte chunks
  const uint4* Z = reinterpret_cast<const uint4*>(b.emb);
  const uint4* RZ = reinterpret_cast<const uint4*>(b.root_emb);
  int v0 = 0, v1 = sz.N;  // states of groups [g0, g1)
  if (sz.g0 != 0 || sz.g1 != sz.G) {
    if (tree) {
      v0 = b.group_state_off[sz.g0];
      v1 = b.group_state_off[sz.g1];
    } else {
      const int ra = b.group_rollout_off[sz.g0], rb = b.group_rollout_off[sz.g1];
      v0 = ra >= 0 && ra <= sz.R ? b.rollout_step_off[ra] : 0;
      v1 = rb >= 0 && rb <= sz.R ? b.rollout_step_off[rb] : 0;
    }
    v0 = max(0, min(v0, sz.N));
    v1 = max(v0, min(v1, sz.N));
  }
  auto quad = [&](float2 P) -> float2 {  // the 4 quarters' pairs, fixed order
#pragma unroll
    for (int o = 1; o < 4; o <<= 1) {
      const float a = __shfl_xor_sync(0xffffffffu, P.x, o), c = __shfl_xor_sync(0xffffffffu, P.y, o);
      float t, u;
      two_sum(P.x, a, t, u);
      P.x = t;
      P.y = P.y + c + u;
    }
    float h, l;
    two_sum(P.x, P.y, h, l);
    return make_float2(h, l);
  };
  auto finish4 = [&](uint64_t s, uint64_t e) -> float2 { return quad(f2_finish(s, e)); };
  // TwoSum sums of this lane's quarter of row zb and its parent pb (chunks loaded here)
  auto twosum_quarter = [&](const uint4* zb, const uint4* pb, bool on, float2& n2, float2& dot) {
    uint64_t ns = 0ull, ne = 0ull, ds = 0ull, de = 0ull;
    for (int c = 0; on && c < nq; ++c) {
      const int k = j * nq + c;
      const uint4 x = zb[k], y = pb ? pb[k] : make_uint4(0u, 0u, 0u, 0u);
      const uint32_t xw[4] = {x.x, x.y, x.z, x.w}, yw[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const uint64_t xx = bf16x2_f32x2(xw[h]), yy = bf16x2_f32x2(yw[h]);
        f2_acc(ns, ne, f2mul(xx, xx));
        f2_acc(ds, de, f2mul(xx, yy));
      }
    }
    n2 = finish4(ns, ne);
    dot = finish4(ds, de);
  };
  for (int64_t base = v0 + warp * 8; base < v1; base += nwarps * 8) {
    const int64_t v = base + r;
    const bool live = v < v1;
    // the rollout (chain) or group (tree) of the warp's first row by a 32-ary search, then each
    // row's from a window of 32 offsets and one ballot per row
    const int32_t* off = tree ? b.group_state_off : b.rollout_step_off;
    const int cnt = tree ? sz.G : sz.R;
    int k_row = 0, start = 0;
    if (cnt > 0) {
      const int k0 = warp_upper_idx(off, cnt, (int)base, lane);
      const int win = k0 + lane < cnt ? off[k0 + lane] : 0x7fffffff;
      for (int q = 0; q < 8; ++q) {
        const int vq = (int)min(base + q, (int64_t)v1 - 1);
        const uint32_t m = __ballot_sync(0xffffffffu, win <= vq);
        int k = k0 + (m ? 31 - __clz(m) : 0);
        if (m == 0xffffffffu)
          while (k + 1 < cnt && off[k + 1] <= vq) ++k;
        const int st_k = k - k0 < 32 ? __shfl_sync(0xffffffffu, win, (k - k0) & 31) : off[k];
        if (q == r) {
          k_row = k;
          start = st_k;
        }
      }
    }
    // parent: p >= 0 a state row, -2 - g the prompt embedding of group g, -1 none
    int p = -1;
    if (live && cnt > 0) {
      int g = -1;
      if (tree) {
        g = k_row;
        const int pl = b.parent[v];
        if (pl >= 0 && start >= 0 && (int64_t)start + pl < v) p = start + pl;
      } else {
        if (v > start) p = (int)v - 1;
        else if (b.root_emb && sz.G > 0) g = upper_idx(b.group_rollout_off, sz.G, k_row);
      }
      if (p < 0 && b.root_emb && g >= 0) p = -2 - g;
    }
    // the parent chunk comes from the lane 4 below when it holds the parent's row
    const bool from_left = p >= 0 && p == v - 1 && r > 0;
    const uint4* pb = p >= 0 ? Z + (int64_t)p * rs : (p <= -2 ? RZ + (int64_t)(-2 - p) * rs : nullptr);
    const uint4* zb = Z + (live ? v : base) * rs;
    float2 n2, dot;
    if (!kNorms) {
      uint64_t ns = 0ull, ne = 0ull, ds = 0ull, de = 0ull;
      constexpr int kU = 4;  // chunks loaded ahead of their arithmetic (memory-level parallelism)
      for (int c0 = 0; c0 < nq; c0 += kU) {
        uint4 x[kU], y[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int k = j * nq + c0 + u;
          x[u] = live && c0 + u < nq ? zb[k] : make_uint4(0u, 0u, 0u, 0u);
          y[u] = (!from_left && pb && c0 + u < nq) ? pb[k] : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          uint4 t;
          t.x = __shfl_up_sync(0xffffffffu, x[u].x, 4);
          t.y = __shfl_up_sync(0xffffffffu, x[u].y, 4);
          t.z = __shfl_up_sync(0xffffffffu, x[u].z, 4);
          t.w = __shfl_up_sync(0xffffffffu, x[u].w, 4);
          if (from_left) y[u] = t;
          const uint32_t xw[4] = {x[u].x, x[u].y, x[u].z, x[u].w}, yw[4] = {y[u].x, y[u].y, y[u].z, y[u].w};
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            const uint64_t xx = bf16x2_f32x2(xw[h]), yy = bf16x2_f32x2(yw[h]);
            f2_acc(ns, ne, f2mul(xx, xx));  // bf16 products are exact in fp32
            f2_acc(ds, de, f2mul(xx, yy));
          }
        }
      }
      n2 = finish4(ns, ne);
      dot = finish4(ds, de);
    } else {
      // the biases: fp32 squared norms of the row and its parent (ws.nrm2; the prompt
      // embedding's from root_norms_kernel, which ran first)
      float nv = 0.f, np = 0.f;
      if (live) {
        nv = ws.nrm2[v];
        if (p >= 0) np = ws.nrm2[p];
        else if (p <= -2) np = ws.x_root_n2[-2 - p].x;
      }
      const float sgn = pow2_ceil(4.04f * nv), sgd = pow2_ceil(2.02f * (nv + np));
      const uint64_t sn0 = f2splat(sgn), sd0 = f2splat(sgd);
      uint64_t a0 = sn0, a1 = sn0, b0 = sd0, b1 = sd0, ea0 = 0ull, ea1 = 0ull, eb0 = 0ull, eb1 = 0ull;
      constexpr int kU = 4;
      for (int c0 = 0; c0 < nq; c0 += kU) {
        uint4 x[kU], y[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int k = j * nq + c0 + u;
          x[u] = live && c0 + u < nq ? zb[k] : make_uint4(0u, 0u, 0u, 0u);
          y[u] = (!from_left && pb && c0 + u < nq) ? pb[k] : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          uint4 t;
          t.x = __shfl_up_sync(0xffffffffu, x[u].x, 4);
          t.y = __shfl_up_sync(0xffffffffu, x[u].y, 4);
          t.z = __shfl_up_sync(0xffffffffu, x[u].z, 4);
          t.w = __shfl_up_sync(0xffffffffu, x[u].w, 4);
          if (from_left) y[u] = t;
          const uint32_t xw[4] = {x[u].x, x[u].y, x[u].z, x[u].w}, yw[4] = {y[u].x, y[u].y, y[u].z, y[u].w};
#pragma unroll
          for (int h = 0; h < 4; h += 2) {
            const uint64_t x0 = bf16x2_f32x2(xw[h]), y0 = bf16x2_f32x2(yw[h]);
            const uint64_t x1 = bf16x2_f32x2(xw[h + 1]), y1 = bf16x2_f32x2(yw[h + 1]);
            biased_add(a0, ea0, x0, x0);
            biased_add(b0, eb0, x0, y0);
            biased_add(a1, ea1, x1, x1);
            biased_add(b1, eb1, x1, y1);
          }
        }
      }
      // every running sum still in [sigma/2, 3 sigma/2]: then each step was error-free
      auto in_range = [](uint64_t s, float sg) {
        uint32_t lo, hi;
        unpack_f2(s, lo, hi);
        return fabsf(__uint_as_float(lo) - sg) <= 0.5f * sg && fabsf(__uint_as_float(hi) - sg) <= 0.5f * sg;
      };
      int okv = !live || (in_range(a0, sgn) && in_range(a1, sgn) && in_range(b0, sgd) && in_range(b1, sgd));
      // the row's 4 lanes agree (lanes 4 r .. 4 r + 3); every lane takes part in both shuffles
      okv &= __shfl_xor_sync(0xffffffffu, okv, 1);
      okv &= __shfl_xor_sync(0xffffffffu, okv, 2);
      const bool ok = okv != 0;
      // (s - sigma) is exact in each lane; the lane's pair: both chains' parts and errors
      auto lane_pair = [](uint64_t s0, uint64_t e0, uint64_t s1, uint64_t e1, float sg) {
        uint64_t h = 0ull, l = 0ull;
        f2_acc(h, l, f2sub(s0, f2splat(sg)));
        f2_acc(h, l, f2sub(s1, f2splat(sg)));
        return f2_finish(h, f2add(l, f2add(e0, e1)));
      };
      n2 = quad(lane_pair(a0, ea0, a1, ea1, sgn));
      dot = quad(lane_pair(b0, eb0, b1, eb1, sgd));
      if (__any_sync(0xffffffffu, !ok)) {  // rare: the rows out of range, by TwoSum
        float2 n2b, dotb;
        twosum_quarter(zb, pb ? pb : nullptr, live && !ok, n2b, dotb);
        if (!ok) {
          n2 = n2b;
          dot = dotb;
        }
      }
    }
    if (p == -1) dot = make_float2(0.f, 0.f);
    if (live && j == 0) {
      if (!isfinite(n2.x) || !isfinite(dot.x)) report(ws.status, GPO_ERR_NONFINITE, 3, (int)v);
      ws.x_n2[v] = n2;
      ws.x_dot[v] = dot;
    }
  }
}

// |prompt embedding|^2 of groups [g0, g1), one warp each (the streamed kernel covers the states).
__global__ void __launch_bounds__(256) root_norms_kernel(gpo_batch b, Sizes sz, Ws ws) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t g = sz.g0 + warp; g < sz.g1; g += nwarps) {
    float2 n2, dot;
    exact_pair_sums<true>(b.root_emb, g * sz.stride, nullptr, 0, false, sz.d, lane, n2, dot);
    if (lane == 0) {
      if (!isfinite(n2.x)) report(ws.status, GPO_ERR_NONFINITE, 3, (int)(sz.N + g));
      ws.x_root_n2[g] = n2;
    }
  }
}

cudaError_t launch_exact_stats(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws,
                               bool with_norms) {
  const int64_t jobs = (int64_t)sz.N + (b.root_emb ? sz.G : 0);  // at most (range calls take fewer)
  if (jobs == 0) return cudaSuccess;
  const bool aligned16 = (reinterpret_cast<uintptr_t>(b.emb) & 15u) == 0 && sz.stride % 8 == 0 && sz.d % 8 == 0 &&
                         (!b.root_emb || (reinterpret_cast<uintptr_t>(b.root_emb) & 15u) == 0);
  if (b.emb_dtype == GPO_EMB_BF16 && aligned16 && sz.d % 32 == 0) {
    int64_t blocks = ((int64_t)sz.N + 63) / 64;  // a warp per 8 rows
    const int64_t bcap = (int64_t)lc.num_sms * 32;
    blocks = blocks < 1 ? 1 : (blocks > bcap ? bcap : blocks);
    if (b.root_emb && sz.g1 > sz.g0) {  // first: the norms-based path reads them
      int64_t rblocks = ((int64_t)(sz.g1 - sz.g0) + 7) / 8;
      if (rblocks > (int64_t)lc.num_sms * 8) rblocks = (int64_t)lc.num_sms * 8;
      root_norms_kernel<<<(int)rblocks, 256, 0, lc.stream>>>(b, sz, ws);
    }
    if (with_norms)
      exact_stats_lane_kernel<true><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
    else
      exact_stats_lane_kernel<false><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
    return cudaGetLastError();
  }
  int64_t blocks = (jobs + 7) / 8;  // a warp per row
  const int64_t cap = (int64_t)lc.num_sms * 16;
  if (blocks > cap) blocks = cap;
  if (b.emb_dtype == GPO_EMB_BF16)
    exact_stats_kernel<true><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
  else
    exact_stats_kernel<false><<<(int)blocks, 256, 0, lc.stream>>>(b, sz, ws);
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
      const float a = __shfl_sync(0xffffffffu, va, j);
      if (!GPO_BOUNDS(ws.status, e - 1, sz.T, kWhereTokens) || !GPO_BOUNDS(ws.status, s, sz.T, kWhereTokens)) continue;
      write_span(o.adv, s, e, a, lane);
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
