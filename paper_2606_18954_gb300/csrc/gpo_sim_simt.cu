// Cosine-similarity merge on the CUDA cores (fp32 embeddings; also selectable
// for bf16 to cross-check the tensor-core kernel).  Same work items and same
// per-item spanning-forest output as the tcgen05 kernel: GraphPO Sec. 4.2,
// pairs of states of one group that are not ancestor-related and have
// cosine >= kappa are linked.  fp32 fused multiply-add accumulation.
#include "gpo_internal.cuh"

namespace gpo {

namespace {

constexpr int kThreads = 256;          // 16 x 16 threads, each 8 rows x 16 columns
constexpr int kKc = 16;                // k-chunk staged in shared memory
constexpr int kSlots = kTileM + kTileN;

__device__ __forceinline__ int sfind(int* p, int x) {
  volatile int* vp = p;
  while (true) {
    const int y = vp[x];
    if (y == x) return x;
    x = y;
  }
}

__device__ __forceinline__ void sunion(int* p, int a, int b) {
  while (true) {
    a = sfind(p, a);
    b = sfind(p, b);
    if (a == b) return;
    if (a > b) {
      const int t = a;
      a = b;
      b = t;
    }
    if (atomicCAS(&p[b], b, a) == b) return;
  }
}

template <bool kBf16>
__device__ __forceinline__ float ld_elem(const void* base, int64_t i) {
  if (kBf16) return __uint_as_float((uint32_t)(reinterpret_cast<const uint16_t*>(base)[i]) << 16);
  return reinterpret_cast<const float*>(base)[i];
}

constexpr int kSmall = 64;   // rows and columns of a small item
constexpr int kKs = 32;      // k-chunk of a small item (kKs x kSmall floats fit in As and in Bs)
static_assert(kKs * kSmall <= kKc * (kTileM + 4) && kKs * kSmall <= kKc * (kTileN + 4), "small-item staging");

// A small item: the same products, pair test and unions as the general path below, with
// every thread on a 4 x 4 micro-tile of the 64 x 64 block (all 256 threads busy) and
// k-chunks of kKs elements (fewer barriers and load round trips per item).  As / Bs are
// the general path's staging arrays, viewed as [kKs][kSmall].
template <bool kBf16>
__device__ __forceinline__ void small_item(const gpo_batch& b, const Sizes& sz, const Item& item, int nrows, int send,
                                           float* As, float* Bs, const int* rm_roll, const int* rm_depth,
                                           const int* rm_end, const float* rm_rn, const int* cm_roll,
                                           const int* cm_depth, const float* cm_rn, int* lp, bool tree, float kappa,
                                           int rule) {
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;  // columns 4 tx.., rows 4 ty..
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < sz.d; k0 += kKs) {
    __syncthreads();
    for (int e = threadIdx.x; e < kKs * nrows; e += kThreads) {
      const int r = e / kKs, k = e % kKs;
      const int row = item.row0 + r;
      As[k * kSmall + r] = (row < send && k0 + k < sz.d) ? ld_elem<kBf16>(b.emb, (int64_t)row * sz.stride + k0 + k) : 0.f;
    }
    for (int e = threadIdx.x; e < kKs * item.ncols; e += kThreads) {
      const int c = e / kKs, k = e % kKs;
      Bs[k * kSmall + c] = k0 + k < sz.d ? ld_elem<kBf16>(b.emb, (int64_t)(item.col0 + c) * sz.stride + k0 + k) : 0.f;
    }
    __syncthreads();
    if (ty * 4 < nrows && tx * 4 < item.ncols) {
      const int kn = min(kKs, sz.d - k0);
      for (int k = 0; k < kn; ++k) {
        const float4 a = *reinterpret_cast<const float4*>(As + k * kSmall + ty * 4);
        const float4 bv = *reinterpret_cast<const float4*>(Bs + k * kSmall + tx * 4);
        const float av[4] = {a.x, a.y, a.z, a.w}, bw[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bw[j], acc[i][j]);
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = ty * 4 + i;
    if (r >= nrows || rm_roll[r] < 0) continue;
    const int row = item.row0 + r;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = tx * 4 + j;
      const int col = item.col0 + c;
      // comparable: not the row's own rollout (tree layout: outside the row's subtree)
      if (c >= item.ncols || col <= row || (tree ? col < rm_end[r] : cm_roll[c] == rm_roll[r])) continue;
      if (rule == GPO_MERGE_SAME_DEPTH && cm_depth[c] != rm_depth[r]) continue;
      if (acc[i][j] * rm_rn[r] * cm_rn[c] >= kappa) {
        const int sc = (col < item.row0 + kTileM) ? col - item.row0 : kTileM + (col - item.col0);
        sunion(lp, r, sc);
      }
    }
  }
}

template <bool kBf16>
__global__ void __launch_bounds__(kThreads) sim_simt_kernel(gpo_batch b, Sizes sz, Ws ws, float kappa, int rule) {
  __shared__ __align__(16) float As[kKc][kTileM + 4];
  __shared__ __align__(16) float Bs[kKc][kTileN + 4];
  __shared__ int lp[kSlots];
  __shared__ int cm_roll[kTileN], cm_depth[kTileN];
  __shared__ float cm_rn[kTileN];
  __shared__ int rm_roll[kTileM], rm_depth[kTileM], rm_end[kTileM];
  __shared__ float rm_rn[kTileM];
  __shared__ int edge_n;
  uint32_t* st = ws.status;
  const bool tree = ws.tree_end != nullptr;
  const int nitems = (int)*((volatile uint32_t*)&st[kStItems]);
  if (aborted(st)) return;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  for (int i = threadIdx.x; i < kSlots; i += kThreads) lp[i] = i;

  for (int it = blockIdx.x; it < nitems; it += gridDim.x) {
    const Item item = ws.items[it];
    const GroupInfo gi = ws.groups[item.group];
    const int send = gi.s0 + gi.n;
    __syncthreads();
    for (int c = threadIdx.x; c < kTileN; c += kThreads) {
      if (c < item.ncols) {
        const int2 mt = ws.state_meta[item.col0 + c];
        cm_roll[c] = mt.x;
        cm_depth[c] = mt.y;
        cm_rn[c] = ws.rn[item.col0 + c];
      }
    }
    for (int r = threadIdx.x; r < kTileM; r += kThreads) {
      const int row = item.row0 + r;
      if (row < send) {
        const int2 mt = ws.state_meta[row];
        rm_roll[r] = mt.x;
        rm_depth[r] = mt.y;
        rm_rn[r] = ws.rn[row];
        rm_end[r] = tree ? ws.tree_end[row] : 0;
      } else {
        rm_roll[r] = -1;
      }
    }
    if (threadIdx.x == 0) edge_n = 0;

    const int nrows = min(kTileM, send - item.row0);
    if (nrows <= kSmall && item.ncols <= kSmall) {
      // a small item (groups of at most 64 states): every thread one 4 x 4 micro-tile of the
      // 64 x 64 block, k-chunks of kKs staged at once
      small_item<kBf16>(b, sz, item, nrows, send, &As[0][0], &Bs[0][0], rm_roll, rm_depth, rm_end, rm_rn, cm_roll,
                        cm_depth, cm_rn, lp, tree, kappa, rule);
    } else {
    float acc[8][16];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 16; ++j) acc[i][j] = 0.f;
    // only the tile's valid rows and columns are staged and multiplied (a thread's rows
    // and columns past them accumulate stale values that the epilogue never reads)
    const bool busy = ty * 8 < nrows && tx * 16 < item.ncols;

    for (int k0 = 0; k0 < sz.d; k0 += kKc) {
      __syncthreads();
      for (int e = threadIdx.x; e < kKc * nrows; e += kThreads) {
        const int r = e / kKc, k = e % kKc;
        const int row = item.row0 + r;
        As[k][r] = (row < send && k0 + k < sz.d) ? ld_elem<kBf16>(b.emb, (int64_t)row * sz.stride + k0 + k) : 0.f;
      }
      for (int e = threadIdx.x; e < kKc * item.ncols; e += kThreads) {
        const int c = e / kKc, k = e % kKc;
        Bs[k][c] = (c < item.ncols && k0 + k < sz.d)
                       ? ld_elem<kBf16>(b.emb, (int64_t)(item.col0 + c) * sz.stride + k0 + k)
                       : 0.f;
      }
      __syncthreads();
      if (busy) {
#pragma unroll 4
      for (int k = 0; k < kKc; ++k) {
        float a[8], bv[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) a[i] = As[k][ty * 8 + i];
#pragma unroll
        for (int j = 0; j < 16; ++j) bv[j] = Bs[k][tx * 16 + j];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int j = 0; j < 16; ++j) acc[i][j] = fmaf(a[i], bv[j], acc[i][j]);
      }
      }
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = ty * 8 + i;
      const int row = item.row0 + r;
      if (rm_roll[r] < 0) continue;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int c = tx * 16 + j;
        const int col = item.col0 + c;
        // comparable: not the row's own rollout (tree layout: outside the row's subtree)
        if (c >= item.ncols || col <= row || (tree ? col < rm_end[r] : cm_roll[c] == rm_roll[r])) continue;
        if (rule == GPO_MERGE_SAME_DEPTH && cm_depth[c] != rm_depth[r]) continue;
        if (acc[i][j] * rm_rn[r] * cm_rn[c] >= kappa) {
          const int sc = (col < item.row0 + kTileM) ? col - item.row0 : kTileM + (col - item.col0);
          sunion(lp, r, sc);
        }
      }
    }
    }
    __syncthreads();
    int2* out = ws.edges + (size_t)it * kEdgeCap;
    for (int s = threadIdx.x; s < kSlots; s += kThreads) {
      const int root = sfind(lp, s);
      if (root != s) {
        const int gs = s < kTileM ? item.row0 + s : item.col0 + (s - kTileM);
        const int gr = root < kTileM ? item.row0 + root : item.col0 + (root - kTileM);
        const int k = atomicAdd(&edge_n, 1);
        if (k < kEdgeCap) out[k] = make_int2(gr, gs);
      }
    }
    __syncthreads();
    for (int s = threadIdx.x; s < kSlots; s += kThreads) lp[s] = s;
    if (threadIdx.x == 0) ws.edge_count[it] = min(edge_n, kEdgeCap);
  }
}

}  // namespace

cudaError_t launch_sim_simt(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws,
                            const Params& p) {
  int grid = ws.max_items < 4 * lc.num_sms ? ws.max_items : 4 * lc.num_sms;
  if (grid < 1) return cudaSuccess;
  if (b.emb_dtype == GPO_EMB_BF16)
    sim_simt_kernel<true><<<grid, kThreads, 0, lc.stream>>>(b, sz, ws, (float)p.kappa, p.rule);
  else
    sim_simt_kernel<false><<<grid, kThreads, 0, lc.stream>>>(b, sz, ws, (float)p.kappa, p.rule);
  return cudaGetLastError();
}

}  // namespace gpo
