// Cosine-similarity merge on the tcgen05 tensor cores (bf16 embeddings).
//
// GraphPO Sec. 4.2 / Algorithm S.1: every pair of states of a prompt group
// that is not in an ancestor-descendant relation (chain layout: different
// rollouts; optionally also the same step depth) and whose cosine similarity
// is >= kappa is linked; the equivalence classes are the connected components.
//
// Work items: per 128-row block of a group, a diagonal item (the block against
// itself) and off-diagonal items (the block against up to 256 later columns), so
// each unordered pair is visited once.  A group's diagonal items precede its
// off-diagonal ones in the list.  A diagonal item takes the block's squared norms from
// the diagonal of its Gram tile (for the threshold test; eta uses the compensated
// statistics), writes them to the workspace and raises the block's ready flag; an off-diagonal
// item waits (bounded) for the flags of its row and column blocks before its
// epilogue reads them.  Every wait is on an item earlier in the list, diagonal items
// never wait, and each CTA takes its items in list order, so every wait ends.
// Persistent CTAs (one per SM) walk the item list.
// Warp roles:
//   warp 0 (one lane)  TMA producer: 128-row boxes of Z, 64 bf16 wide, 128B swizzle
//   warp 1 (one lane)  MMA issuer: D[128 x N] += A[128 x 64] * B[N x 64]^T per k-step,
//                      fp32 accumulators in TMEM, two buffers of 256 columns
//   warps 4..15        epilogue, three warps per TMEM lane quarter splitting the
//                      32-column chunks: pair test acc / |z_j| >= kappa |z_i| (one
//                      fma per pair, comparable columns by one range mask per
//                      chunk), linked pairs into per-warp edge lists, accumulator
//                      released, then classes of the item's <= 384 states by
//                      hook-and-shortcut rounds in shared memory, and the item's
//                      spanning forest (<= 383 edges, state -> smallest state of
//                      its class) written out.
// The Gram block Z_g Z_g^T is never written to memory.
#include "gpo_internal.cuh"

namespace gpo {

namespace {

constexpr int kStages = 4;
constexpr int kThreads = 512;
constexpr int kBoxBytes = kTileM * 128;            // one 128-row x 128-byte box
constexpr int kStageBytes = 3 * kBoxBytes;         // A box + two B boxes
constexpr int kSlots = kTileM + kTileN;            // local union-find slots
constexpr int kTmemCols = 512;                     // two accumulators of 256 columns
constexpr int kEpiBarrier = 1;                     // named barrier of the epilogue warps
constexpr int kEpiThreads = 384;                   // warps 4..15
constexpr int kEpiWarps = kEpiThreads / 32;
constexpr int kWarpEdges = 256;                    // linked pairs listed per epilogue warp and item

struct __align__(8) SmemCtl {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int edge_n;
  int overflow;                    // some warp found more pairs than its list holds
  int lp[kSlots];                  // label forest of the item's slots (rows, then columns)
  int cm_depth[kTileN];
  alignas(16) float cm_rn[kTileN];  // 1 / |z| of the item's columns
  uint32_t elist[kEpiWarps][kWarpEdges];  // slot pairs (row slot | column slot << 16)
};

__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync %0, %1;" ::"n"(kEpiBarrier), "n"(kEpiThreads) : "memory");
}

// Bits a..31 of a word (all for a <= 0, none for a >= 32).
__device__ __forceinline__ uint32_t bits_from(int a) { return a <= 0 ? 0xFFFFFFFFu : (a >= 32 ? 0u : 0xFFFFFFFFu << a); }

// Barrier of the 4 epilogue warps that also ORs a flag across them, so that
// they all take the same early exit.
__device__ __forceinline__ bool epi_any(bool flag) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(out)
      : "r"((uint32_t)flag), "n"(kEpiBarrier), "n"(kEpiThreads)
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
    sim_tc_kernel(const __grid_constant__ CUtensorMap zmap, const int32_t* __restrict__ rollout_step_off, Sizes sz,
                  Ws ws, float kappa, int rule, int debug_timeout) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // control block first, then the tiles on a 1024-byte boundary (128B swizzle); both are
  // smem_raw plus an offset, so the compiler keeps the shared address space
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem_raw);
  const uint32_t sbase = smem_u32(smem_raw);
  constexpr uint32_t kCtlBytes = (sizeof(SmemCtl) + 15) & ~15u;
  unsigned char* tiles = smem_raw + (((sbase + kCtlBytes + 1023u) & ~1023u) - sbase);
  uint32_t* st = ws.status;
  const bool tree = ws.tree_end != nullptr;

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
      mbar_init(&ctl->tempty[b], kEpiWarps);
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
    // GPO_FLAG_DEBUG_TIMEOUT: the first wait runs out (nothing arrives on `drain` before the
    // commit below), and the CTA winds down as after any timeout
    if (debug_timeout) {
      mbar_wait(&ctl->drain, 0, st, 17, kDebugTimeoutNs);  // returns false: reports GPO_ERR_TIMEOUT
      ok = false;
    }
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
    const int q = warp & 3;            // TMEM lane quarter
    const int rep = (warp - 4) >> 2;   // 0..2: which of the quarter's three warps
    const int ew = warp - 4;           // epilogue warp 0..11
    const int te = threadIdx.x - 128;  // 0..383
    const int t = q * 32 + lane;       // accumulator row = TMEM lane
    uint32_t* wlist = ctl->elist[ew];
    int m = 0;
    for (int it = blockIdx.x; it < nitems; it += gridDim.x, ++m) {
      const Item item = ws.items[it];
      const GroupInfo gi = ws.groups[item.group];
      const int send = gi.s0 + gi.n;
      const bool diag = item.col0 == item.row0;
      const int blk_row = gi.blk0 + (item.row0 - gi.s0) / kTileM;
      const int buf = m & 1;
      epi_sync();  // previous item finished with the metadata, lists and forest
      for (int c = te; c < item.ncols; c += kEpiThreads) {
        ctl->cm_depth[c] = ws.state_meta[item.col0 + c].y;
      }
      for (int c = item.ncols + te; c < kTileN; c += kEpiThreads) ctl->cm_rn[c] = 0.f;
      if (te == 0) {
        ctl->edge_n = 0;
        ctl->overflow = 0;
      }
      // row constants: end of the row's rollout (tree layout: of its subtree; the comparable
      // columns right of row i are exactly those at or after it) and depth
      const int row = item.row0 + t;
      int re = send, di = -1;
      if (row < send) {
        const int2 mt = ws.state_meta[row];
        re = tree ? ws.tree_end[row] : rollout_step_off[mt.x + 1];
        di = mt.y;
      }
      float thr = __int_as_float(0x7f800000);  // kappa |z_i|; +inf for a zero or absent row
      if (!diag) {
        // the norms of the row block and of the column blocks come from their diagonal items
        bool ready = true;
        if (te == 0) {
          const int bc = gi.blk0 + (item.col0 - gi.s0) / kTileM;
          ready = wait_flag(ws.blk_ready + blk_row, st, 16) && wait_flag(ws.blk_ready + bc, st, 16) &&
                  (item.col0 + kTileM >= send || item.ncols <= kTileM || wait_flag(ws.blk_ready + bc + 1, st, 16));
        }
        if (epi_any(!ready)) break;
        for (int c = te; c < item.ncols; c += kEpiThreads) ctl->cm_rn[c] = __ldcg(ws.rn + item.col0 + c);
        if (row < send) {
          const float rni = __ldcg(ws.rn + row);
          if (rni > 0.f) thr = kappa / rni;
        }
      }
      epi_sync();
      const bool got = mbar_wait(&ctl->tfull[buf], (uint32_t)(m >> 1) & 1u, st, 15);
      if (epi_any(!got)) break;
      tc_fence_after();
      if (diag) {
        // the block's squared norms (threshold test): the diagonal of its Gram tile, read by
        // one warp per lane quarter; published before the flag that releases the block
        if (rep == 0 && q * 32 < item.ncols) {
          const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kTileN + q * 32);
          uint32_t r[32];
          tmem_ld_32x32b_x32(base, r);
          tmem_wait_ld();
          float dg = 0.f;
#pragma unroll
          for (int k = 0; k < 32; ++k)
            if (k == lane) dg = __uint_as_float(r[k]);
          if (t < item.ncols && GPO_BOUNDS(st, row, sz.N, kWhereNorms)) {
            const float rni = dg > 0.f ? 1.0f / sqrtf(dg) : 0.f;
            ws.nrm2[row] = dg;
            ws.rn[row] = rni;
            ctl->cm_rn[t] = rni;
            if (!isfinite(dg)) report(st, GPO_ERR_NONFINITE, 1, row);
          }
          __threadfence();
        }
        epi_sync();
        if (te == 0) st_release_gpu(ws.blk_ready + blk_row, 1);
        if (t < item.ncols && ctl->cm_rn[t] > 0.f) thr = kappa / ctl->cm_rn[t];
      }
      // linked pairs: chunks holding a column right of some row of the warp, dealt
      // round-robin to the quarter's three warps; one pair per lane per step into the
      // warp's list (slots by ballot), past its capacity straight into the forest
      const int nchunks = (item.ncols + 31) >> 5;
      const int cend = item.col0 + item.ncols;
      int wcount = 0, dealt = 0;
      for (int ch = 0; ch < nchunks; ++ch) {
        const int cb = item.col0 + ch * 32;
        if (cb + 31 <= item.row0 + q * 32) continue;
        if (dealt++ % 3 != rep) continue;
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kTileN + ch * 32), r);
        tmem_wait_ld();
        // <z of the block's last row, z of the next block's first row>: the parent dot of
        // the next block's first state when it continues the same rollout
        uint32_t mp[4] = {0u, 0u, 0u, 0u};
        const float4* rn4 = reinterpret_cast<const float4*>(ctl->cm_rn + ch * 32);
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {
          const float4 c = rn4[j4];
          const float cc[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = 4 * j4 + u;
            mp[u] |= (__float_as_uint(fmaf(__uint_as_float(r[j]), cc[u], -thr)) >> 31) << j;
          }
        }
        const uint32_t miss = (mp[0] | mp[1]) | (mp[2] | mp[3]);
        uint32_t mk = ~miss & bits_from(re - cb) & ~bits_from(cend - cb);
        if (rule == GPO_MERGE_SAME_DEPTH && mk) {
          uint32_t m2 = 0u;
          for (uint32_t x = mk; x; x &= x - 1u) {
            const int j = __ffs(x) - 1;
            if (ctl->cm_depth[ch * 32 + j] == di) m2 |= 1u << j;
          }
          mk = m2;
        }
        for (uint32_t act = __ballot_sync(0xffffffffu, mk != 0); act; act = __ballot_sync(0xffffffffu, mk != 0)) {
          const int slot = wcount + __popc(act & ((1u << lane) - 1u));
          if (mk) {
            const int col = cb + __ffs(mk) - 1;
            mk &= mk - 1u;
            const int sc = col < item.row0 + kTileM ? col - item.row0 : kTileM + (col - item.col0);
            if (slot < kWarpEdges) wlist[slot] = (uint32_t)t | ((uint32_t)sc << 16);
            else lunion(ctl->lp, t, sc);
          }
          wcount += __popc(act);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&ctl->tempty[buf]);  // accumulator free for the next item
        if (wcount > kWarpEdges) ctl->overflow = 1;
      }
      epi_sync();
      // classes of the item's slots: hook-and-shortcut rounds over the listed pairs (the
      // larger of two current labels is pointed at the smaller) until every pair has
      // equal labels and every label is a root; lock-free root unions if a list overflowed
      const int nw = min(wcount, kWarpEdges);
      if (!ctl->overflow) {
        bool conv = false;
        for (int round = 0; round <= kSlots && !conv; ++round) {
          bool chg = false;
          for (int e = lane; e < nw; e += 32) {
            const uint32_t ij = wlist[e];
            const int lu = ctl->lp[ij & 0xFFFFu], lv = ctl->lp[ij >> 16];
            if (lu != lv) {
              atomicMin(&ctl->lp[max(lu, lv)], min(lu, lv));
              chg = true;
            }
          }
          for (int x = te; x < kSlots; x += kEpiThreads) {
            const int l = ctl->lp[x], ll = ctl->lp[l];
            if (ll != l) {
              ctl->lp[x] = ll;
              chg = true;
            }
          }
          conv = !epi_any(chg);
        }
        if (!conv) {
          for (int e0 = 0; e0 < nw; e0 += 32) {
            if (e0 + lane < nw) lunion(ctl->lp, (int)(wlist[e0 + lane] & 0xFFFFu), (int)(wlist[e0 + lane] >> 16));
            __syncwarp();
          }
          epi_sync();
        }
      } else {
        for (int e0 = 0; e0 < nw; e0 += 32) {
          if (e0 + lane < nw) lunion(ctl->lp, (int)(wlist[e0 + lane] & 0xFFFFu), (int)(wlist[e0 + lane] >> 16));
          __syncwarp();
        }
        epi_sync();
      }
      // spanning forest of this item: one edge per non-root slot, to its class's root
      int2* out = ws.edges + (size_t)it * kEdgeCap;
      for (int s0 = 0; s0 < kSlots; s0 += kEpiThreads) {
        const int sl = s0 + te;
        int root = sl;
        if (sl < kSlots) root = lfind(ctl->lp, sl);
        const bool edge = sl < kSlots && root != sl;
        const uint32_t act = __ballot_sync(0xffffffffu, edge);
        int base = 0;
        if (lane == 0 && act) base = atomicAdd(&ctl->edge_n, __popc(act));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (edge) {
          const int k = base + __popc(act & ((1u << lane) - 1u));
          const int gs = sl < kTileM ? item.row0 + sl : item.col0 + (sl - kTileM);
          const int gr = root < kTileM ? item.row0 + root : item.col0 + (root - kTileM);
          if (k < kEdgeCap && GPO_BOUNDS(st, gr, sz.N, kWhereEdges) && GPO_BOUNDS(st, gs, sz.N, kWhereEdges))
            out[k] = make_int2(gr, gs);
        }
      }
      epi_sync();
      for (int x = te; x < kSlots; x += kEpiThreads) ctl->lp[x] = x;
      if (te == 0) ws.edge_count[it] = min(ctl->edge_n, kEdgeCap);
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

cudaError_t launch_sim_tc(const LaunchCtx& lc, const CUtensorMap& map, const gpo_batch& b, const Sizes& sz,
                          const Ws& ws, const Params& p) {
  int grid = ws.max_items < lc.num_sms ? ws.max_items : lc.num_sms;
  if (grid < 1) return cudaSuccess;
  sim_tc_kernel<<<grid, kThreads, sim_tc_smem_bytes(), lc.stream>>>(map, b.rollout_step_off, sz, ws, (float)p.kappa,
                                                                      p.rule, p.debug_timeout);
  return cudaGetLastError();
}

}  // namespace gpo
