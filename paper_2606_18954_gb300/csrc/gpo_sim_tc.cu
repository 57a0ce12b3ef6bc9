// Cosine-similarity merge on the tcgen05 tensor cores (bf16 embeddings).
//
// GraphPO Sec. 4.2 / Algorithm S.1: every pair of states of a prompt group
// that is not in an ancestor-descendant relation (chain layout: different
// rollouts; optionally also the same step depth) and whose cosine similarity
// is >= kappa is linked; the equivalence classes are the connected components.
//
// Work item = 128 rows of one group x up to 256 columns of the same group
// (col0 >= row0, so each unordered pair is visited once).  Persistent CTAs
// (one per SM) walk the item list.  Warp roles:
//   warp 0 (one lane)  TMA producer: 128-row boxes of Z, 64 bf16 wide, 128B swizzle
//   warp 1 (one lane)  MMA issuer: D[128 x N] += A[128 x 64] * B[N x 64]^T per k-step,
//                      fp32 accumulators in TMEM, two buffers of 256 columns
//   warps 4..7         epilogue: TMEM -> registers, cos = acc / (|z_i||z_j|),
//                      pair mask + threshold, union into a shared-memory
//                      union-find of the item's <=384 states, then the item's
//                      spanning forest (<=383 edges) is written out.
// The Gram block Z_g Z_g^T is never written to memory.
#include "gpo_internal.cuh"

namespace gpo {

namespace {

constexpr int kStages = 4;
constexpr int kThreads = 256;
constexpr int kBoxBytes = kTileM * 128;            // one 128-row x 128-byte box
constexpr int kStageBytes = 3 * kBoxBytes;         // A box + two B boxes
constexpr int kSlots = kTileM + kTileN;            // local union-find slots
constexpr int kTmemCols = 512;                     // two accumulators of 256 columns
constexpr int kEpiBarrier = 1;                     // named barrier of the 4 epilogue warps

struct __align__(8) SmemCtl {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int edge_n;
  int lp[kSlots];
  int cm_roll[kTileN];
  int cm_depth[kTileN];
  float cm_rn[kTileN];
};

__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync %0, 128;" ::"n"(kEpiBarrier) : "memory"); }

// Barrier of the 4 epilogue warps that also ORs a flag across them, so that
// they all take the same early exit.
__device__ __forceinline__ bool epi_any(bool flag) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(out)
      : "r"((uint32_t)flag), "n"(kEpiBarrier)
      : "memory");
  return out != 0;
}

__device__ __forceinline__ int lfind(int* p, int x) {
  volatile int* vp = p;
  while (true) {
    const int y = vp[x];
    if (y == x) return x;
    x = y;
  }
}

// Hook the larger root under the smaller one; parent[x] <= x always holds.
__device__ __forceinline__ void lunion(int* p, int a, int b) {
  while (true) {
    a = lfind(p, a);
    b = lfind(p, b);
    if (a == b) return;
    if (a > b) {
      const int t = a;
      a = b;
      b = t;
    }
    if (atomicCAS(&p[b], b, a) == b) return;
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    sim_tc_kernel(const __grid_constant__ CUtensorMap zmap, Sizes sz, Ws ws, float kappa, int rule) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // control block first, then the tiles on a 1024-byte boundary (128B swizzle); both are
  // smem_raw plus an offset, so the compiler keeps the shared address space
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem_raw);
  const uint32_t sbase = smem_u32(smem_raw);
  constexpr uint32_t kCtlBytes = (sizeof(SmemCtl) + 15) & ~15u;
  unsigned char* tiles = smem_raw + (((sbase + kCtlBytes + 1023u) & ~1023u) - sbase);
  uint32_t* st = ws.status;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nitems = (int)*((volatile uint32_t*)&st[kStItems]);
  if (aborted(st) || nitems == 0 || (int)blockIdx.x >= nitems) return;
  const int KT = (sz.d + kTileK - 1) / kTileK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&ctl->full[s], 1);
      mbar_init(&ctl->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl->tfull[b], 1);
      mbar_init(&ctl->tempty[b], 4);
    }
    mbar_init(&ctl->drain, 1);
    fence_mbar_init();
    tma_prefetch_desc(&zmap);
  }
  for (int i = threadIdx.x; i < kSlots; i += kThreads) ctl->lp[i] = i;
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (lane 0)
    if (lane == 0) {
    int stage = 0;
    uint32_t phase = 0;
    int last_parity[kStages];
    for (int s = 0; s < kStages; ++s) last_parity[s] = -1;
    bool ok = true;
    for (int it = blockIdx.x; it < nitems && ok; it += gridDim.x) {
      const Item item = ws.items[it];
      const bool diag = item.col0 == item.row0;
      const int nbox = diag ? (item.ncols > kTileM ? 2 : 1) : (item.ncols > kTileM ? 3 : 2);
      for (int k = 0; k < KT; ++k) {
        if (!mbar_wait(&ctl->empty[stage], phase ^ 1u, st, 10)) {
          ok = false;
          break;
        }
        unsigned char* sa = tiles + stage * kStageBytes;
        unsigned char* sb = sa + kBoxBytes;
        mbar_arrive_expect_tx(&ctl->full[stage], (uint32_t)(nbox * kBoxBytes));
        last_parity[stage] = (int)phase;
        const int x = k * kTileK;
        tma_load_2d(sa, &zmap, &ctl->full[stage], x, item.row0);
        if (diag) {
          if (item.ncols > kTileM) tma_load_2d(sb, &zmap, &ctl->full[stage], x, item.row0 + kTileM);
        } else {
          tma_load_2d(sb, &zmap, &ctl->full[stage], x, item.col0);
          if (item.ncols > kTileM) tma_load_2d(sb + kBoxBytes, &zmap, &ctl->full[stage], x, item.col0 + kTileM);
        }
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    // wind-down: every issued copy must land before the CTA may exit
    for (int s = 0; s < kStages; ++s)
      if (last_parity[s] >= 0) mbar_wait(&ctl->full[s], (uint32_t)last_parity[s], st, 11, 200000000ull, false);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (lane 0)
    if (lane == 0) {
    int stage = 0;
    uint32_t phase = 0;
    int m = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < nitems && ok; it += gridDim.x, ++m) {
      const Item item = ws.items[it];
      const bool diag = item.col0 == item.row0;
      const int nn = (item.ncols + 15) & ~15;
      const uint32_t idesc = idesc_bf16_f32(kTileM, nn);
      const int buf = m & 1;
      if (!mbar_wait(&ctl->tempty[buf], ((uint32_t)(m >> 1) & 1u) ^ 1u, st, 12)) break;
      tc_fence_after();
      const uint32_t dt = tmem + (uint32_t)(buf * kTileN);
      for (int k = 0; k < KT; ++k) {
        if (!mbar_wait(&ctl->full[stage], phase, st, 13)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(tiles + stage * kStageBytes);
        const uint32_t sb = diag ? sa : sa + kBoxBytes;
        const uint64_t ad = smem_desc_k128(sa), bd = smem_desc_k128(sb);
#pragma unroll
        for (int kk = 0; kk < kTileK / 16; ++kk)
          mma_bf16_ss(dt, ad + 2u * kk, bd + 2u * kk, idesc, (k | kk) != 0);
        mma_commit(&ctl->empty[stage]);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (ok) mma_commit(&ctl->tfull[buf]);
    }
    // wind-down: all issued MMAs complete before TMEM is released
    mma_commit(&ctl->drain);
    mbar_wait(&ctl->drain, 0, st, 14, 200000000ull, false);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;
    const int t = q * 32 + lane;  // accumulator row = TMEM lane
    int m = 0;
    for (int it = blockIdx.x; it < nitems; it += gridDim.x, ++m) {
      const Item item = ws.items[it];
      const GroupInfo gi = ws.groups[item.group];
      const int send = gi.s0 + gi.n;
      const int buf = m & 1;
      epi_sync();  // previous item finished with the column metadata
      for (int c = t; c < item.ncols; c += 128) {
        const int2 mt = ws.state_meta[item.col0 + c];
        ctl->cm_roll[c] = mt.x;
        ctl->cm_depth[c] = mt.y;
        ctl->cm_rn[c] = ws.rn[item.col0 + c];
      }
      if (t == 0) ctl->edge_n = 0;
      const int row = item.row0 + t;
      const bool vrow = row < send;
      int2 rmeta = make_int2(-1, -1);
      float rn_i = 0.f;
      if (vrow) {
        rmeta = ws.state_meta[row];
        rn_i = ws.rn[row];
      }
      epi_sync();
      const bool got = mbar_wait(&ctl->tfull[buf], (uint32_t)(m >> 1) & 1u, st, 15);
      if (epi_any(!got)) break;
      tc_fence_after();
      // pass masks first (branch-free), unions afterwards over the few set bits
      const int nchunks = (item.ncols + 31) >> 5;
      uint32_t masks[kTileN / 32];
#pragma unroll
      for (int ch = 0; ch < kTileN / 32; ++ch) masks[ch] = 0u;
#pragma unroll
      for (int ch = 0; ch < kTileN / 32; ++ch) {
        if (ch >= nchunks) break;
        // a chunk whose last column is at or above no row of this warp holds no pair col > row
        if (item.col0 + ch * 32 + 31 <= item.row0 + q * 32) continue;
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kTileN + ch * 32), r);
        tmem_wait_ld();
        uint32_t mk = 0u;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int c = ch * 32 + j;
          const bool ok = (c < item.ncols) & (item.col0 + c > row) & (ctl->cm_roll[c] != rmeta.x) &
                          ((rule != GPO_MERGE_SAME_DEPTH) | (ctl->cm_depth[c] == rmeta.y)) &
                          (__uint_as_float(r[j]) * rn_i * ctl->cm_rn[c] >= kappa);
          mk |= (uint32_t)ok << j;
        }
        masks[ch] = vrow ? mk : 0u;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->tempty[buf]);  // accumulator free for the next item
#pragma unroll
      for (int ch = 0; ch < kTileN / 32; ++ch) {
        uint32_t mk = masks[ch];
        while (mk) {
          const int j = __ffs(mk) - 1;
          mk &= mk - 1u;
          const int col = item.col0 + ch * 32 + j;
          const int slot_col = (col < item.row0 + kTileM) ? col - item.row0 : kTileM + (col - item.col0);
          lunion(ctl->lp, t, slot_col);
        }
      }
      epi_sync();
      // spanning forest of this item: one edge per non-root slot
      int2* out = ws.edges + (size_t)it * kEdgeCap;
      for (int s = t; s < kSlots; s += 128) {
        const int root = lfind(ctl->lp, s);
        if (root != s) {
          const int gs = s < kTileM ? item.row0 + s : item.col0 + (s - kTileM);
          const int gr = root < kTileM ? item.row0 + root : item.col0 + (root - kTileM);
          const int k = atomicAdd(&ctl->edge_n, 1);
          if (k < kEdgeCap) out[k] = make_int2(gr, gs);
        }
      }
      epi_sync();
      for (int s = t; s < kSlots; s += 128) ctl->lp[s] = s;
      if (t == 0) ws.edge_count[it] = min(ctl->edge_n, kEdgeCap);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

size_t sim_tc_smem_bytes() { return ((sizeof(SmemCtl) + 15) & ~size_t(15)) + 1023 + (size_t)kStages * kStageBytes; }

cudaError_t setup_sim_tc() {
  return cudaFuncSetAttribute(sim_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)sim_tc_smem_bytes());
}

cudaError_t launch_sim_tc(const LaunchCtx& lc, const CUtensorMap& map, const Sizes& sz, const Ws& ws,
                          const Params& p) {
  int grid = ws.max_items < lc.num_sms ? ws.max_items : lc.num_sms;
  if (grid < 1) return cudaSuccess;
  sim_tc_kernel<<<grid, kThreads, sim_tc_smem_bytes(), lc.stream>>>(map, sz, ws, (float)p.kappa, p.rule);
  return cudaGetLastError();
}

}  // namespace gpo
