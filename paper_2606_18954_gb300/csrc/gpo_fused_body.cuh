// Body of the group-resident kernel (gpo_fused.cu includes it once per capacity, each
// time inside its own namespace after defining kMaxN (largest group), kThreads (a
// multiple of 128, at least 256), kMinBlocks (CTAs per SM the launch bounds ask for),
// kRingBytes (the tile ring) and kTmemCols (accumulator columns, a power of two >= 32
// that holds every segment of a one-pass group of kMaxN states, or 512)).

constexpr int kMaxSlots = 8;                    // k-slices in flight at most (mbarrier pairs)
constexpr int kPlaceBytes = kRingBytes - 96 * 128;  // slices lie below this: the MMA of a group's last
                                                    // 128-row block reads its A operand up to 96 rows
                                                    // past the slice (rows that feed unused lanes)
constexpr int kBoxBytes = kTileM * 128;         // 128 rows x 128 bytes
constexpr int kTailRows = 32;                   // rows of the second tensor map's box
constexpr int kGThreads = kThreads - 64;        // warps 2..: group work
constexpr int kEpiThreads = kThreads - 128;     // warps 4..: accumulator drain
constexpr int kReps = kEpiThreads / 128;        // drain warps per accumulator lane quarter
constexpr int kWarpEdges = 256;                 // linked pairs listed per epilogue warp and group
constexpr int kEdgeList = kWarpEdges * (kEpiThreads / 32);
constexpr int kBarGroup = 1;                    // named barrier of the group warps
constexpr int kBarEpi = 2;                      // named barrier of the drain warps
constexpr int kBarSetup = 3;                    // named barrier of warps 2 and 3 (early set-up)
static_assert(kThreads % 128 == 0 && kThreads >= 256 && kGThreads >= kMaxN, "fused kernel shape");

struct Seg {
  int b, c0, len, tcol;  // row block, first column (local), columns, TMEM column
};

struct Plan {
  int npass;
  int nseg[2];
  Seg seg[2][4];
};

__device__ __forceinline__ int r16(int x) { return (x + 15) & ~15; }

// Byte offset in the ring of the next k-slice of `bytes`: right after the previous
// one, or back at 0 if it would reach past kPlaceBytes.  Producer and MMA warp
// place the same sequence of slices with this rule.
__device__ __forceinline__ int ring_place(int head, int bytes) { return head + bytes <= kPlaceBytes ? head : 0; }
__device__ __forceinline__ int r32(int x) { return (x + 31) & ~31; }

// Segments of the upper triangle: row block b against columns [128 b, n) in
// chunks of at most 256 (one MMA each).  Each segment owns a multiple of 32
// TMEM columns (the epilogue reads 32 columns at a time).  One pass if they
// fit 512 TMEM columns, else pass 0 = blocks >= 1 (at most 256 + 128 columns)
// and pass 1 = block 0 (at most 256 + 128), so that the norms of every column
// a pass needs come from its own or an earlier pass.
__device__ __forceinline__ void make_plan(int n, Plan& pl) {
  Seg all[4];
  int na = 0, tot = 0;
  for (int b = 0; b * kTileM < n; ++b)
    for (int c0 = b * kTileM; c0 < n && na < 4; c0 += kTileN) {
      all[na].b = b;
      all[na].c0 = c0;
      all[na].len = min(kTileN, n - c0);
      tot += r32(all[na].len);
      ++na;
    }
  pl.nseg[0] = pl.nseg[1] = 0;
  if (tot <= kTmemCols) {
    pl.npass = 1;
    int col = 0;
    for (int i = 0; i < na; ++i) {
      Seg s = all[i];
      s.tcol = col;
      col += r32(s.len);
      pl.seg[0][pl.nseg[0]++] = s;
    }
  } else {
    pl.npass = 2;
    int col0 = 0, col1 = 0;
    for (int i = 0; i < na; ++i) {
      Seg s = all[i];
      if (s.b >= 1) {
        s.tcol = col0;
        col0 += r32(s.len);
        pl.seg[0][pl.nseg[0]++] = s;
      } else {
        s.tcol = col1;
        col1 += r32(s.len);
        pl.seg[1][pl.nseg[1]++] = s;
      }
    }
  }
}

// The group's rollout and state ranges; false if they are out of range.  Tree layout:
// the rollouts are the group's leaves and the states come from group_state_off.
__device__ __forceinline__ bool group_range(const gpo_batch& b, const Sizes& sz, int g, int& r0, int& nr, int& s0,
                                            int& n) {
  const int a = b.group_rollout_off[g], c = b.group_rollout_off[g + 1];
  if (a < 0 || c < a || c > sz.R) return false;
  const int x = b.parent ? b.group_state_off[g] : b.rollout_step_off[a];
  const int y = b.parent ? b.group_state_off[g + 1] : b.rollout_step_off[c];
  if (x < 0 || y < x || y > sz.N) return false;
  r0 = a;
  nr = c - a;
  s0 = x;
  n = y - x;
  return true;
}

// Group handled here (all roles agree, they read the same inputs).
__device__ __forceinline__ bool group_active(const gpo_batch& b, const Sizes& sz, int g, int& r0, int& nr, int& s0,
                                             int& n) {
  return group_range(b, sz, g, r0, nr, s0, n) && n > 0 && n <= kMaxN && n <= sz.maxn && nr > 0 && nr <= n;
}

struct __align__(16) GroupSmem {
  int lab[kMaxN];
  union {
    int roll[kMaxN];     // chain layout: rollout of each state (local)
    int par[kMaxN];      // tree layout: parent of each state (local, -1 = the prompt root)
  };
  int dep[kMaxN];
  int slen[kMaxN];
  union {
    int rstart[kMaxN + 1];  // chain layout: local state offsets of the rollouts
    int cown[kMaxN + 1];    // tree layout: c_own, rewards of the subtree's leaves
  };
  float n2[kMaxN];
  alignas(16) float rn[kMaxN];  // 1 / |z_i| (0 for a zero row), read four at a time
  float thr[kMaxN];      // kappa |z_i| (+inf for a zero row or a row that is not tested)
  int rend[kMaxN];       // end (local, exclusive) of the rollout (tree: of the subtree) of state i;
                         // the columns right of i that are not its descendants are [rend, n)
  float eadv[kMaxN], ecor[kMaxN], eeff[kMaxN];
  union {
    int64_t tok0[kMaxN + 1];   // chain layout: token offsets of the rollouts
    int town[2 * kMaxN + 2];   // tree layout: t_own, leaves of the subtree
  };
  int64_t tstart[kMaxN];
  uint8_t rew[kMaxN];
  uint8_t emask[kMaxN];
  unsigned long long esum[3];  // exploration efficiency: token sums
  int flags;             // bit 0: group invalid
  int overflow;          // some warp found more pairs than its part of elist holds
  int stats_next;        // next block of 8 rows for the row statistics (claimed by warps)
  Plan plan;
  uint32_t elist[kEdgeList];  // linked pairs of the group, kWarpEdges per epilogue warp: i | j << 16
  alignas(16) unsigned char X[group_scratch_sep_bytes(kMaxN)];  // group-math sums (separate layout)
};
// Tree layout: the group math's sums (tree_scratch) take elist and X, free once the drain
// has built the classes; during the set-up elist holds the scan's warp totals.
constexpr size_t kTreeXOff = offsetof(GroupSmem, elist);
static_assert(offsetof(GroupSmem, X) + sizeof(GroupSmem::X) - kTreeXOff >= tree_scratch_bytes(kMaxN),
              "tree scratch does not fit");

struct __align__(8) Ctl {
  uint64_t full[kMaxSlots];
  uint64_t empty[kMaxSlots];
  uint64_t tfull;
  uint64_t tempty;
  uint64_t drain;
  uint32_t tmem_base;
};

constexpr uint32_t kCtlOff = (sizeof(GroupSmem) + 15) & ~15u;
constexpr uint32_t kTilesOff = kCtlOff + ((sizeof(Ctl) + 15) & ~15u);
static_assert(kTilesOff + 1023 + kRingBytes <= 232448, "fused kernel exceeds 227 KB of shared memory");

__device__ __forceinline__ void bar_group() { asm volatile("bar.sync %0, %1;" ::"n"(kBarGroup), "n"(kGThreads) : "memory"); }
__device__ __forceinline__ void bar_epi() { asm volatile("bar.sync %0, %1;" ::"n"(kBarEpi), "n"(kEpiThreads) : "memory"); }
__device__ __forceinline__ void bar_setup() { asm volatile("bar.sync %0, %1;" ::"n"(kBarSetup), "n"(64) : "memory"); }

// Bits a..31 of a word (all for a <= 0, none for a >= 32).
__device__ __forceinline__ uint32_t bits_from(int a) { return a <= 0 ? 0xFFFFFFFFu : (a >= 32 ? 0u : 0xFFFFFFFFu << a); }

template <int kBar, int kCount>
__device__ __forceinline__ bool bar_any(bool flag) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(out)
      : "r"((uint32_t)flag), "n"(kBar), "n"(kCount)
      : "memory");
  return out != 0;
}

__device__ __forceinline__ float pick(const uint32_t (&r)[32], int j) {
  float v = 0.f;
#pragma unroll
  for (int k = 0; k < 32; ++k)
    if (k == j) v = __uint_as_float(r[k]);
  return v;
}

// Compensated |z_v|^2 and <z_{p(v)}, z_v> of the group's states [s0, s0 + n) into
// ws.x_n2 / ws.x_dot (float pairs).  The calling warps claim blocks of 8 rows from
// gs->stats_next until none is left, so that warps that join late or run slower take
// fewer.  Parents: with `early` (chain layout, before the group's set-up) the previous
// state for every state but the group's first (the set-up fixes the rollouts' first
// states afterwards: their parent is the prompt root); otherwise from the group layout
// in shared memory (chain: the previous state unless the state is a rollout's first; tree:
// gs->par; the prompt embedding for a root child when there is one).
__device__ __forceinline__ void group_row_stats(const gpo_batch& b, const Sizes& sz, const Ws& ws, GroupSmem* gs,
                                                int g, int s0, int n, bool tree, bool early, int lane, uint32_t* st) {
  const int r = lane >> 2, c = lane & 3;
  const int nch = sz.d / 8;          // whole 16-byte chunks of a row
  const int64_t rs = sz.stride / 8;  // row stride in 16-byte chunks
  const uint4* Z = reinterpret_cast<const uint4*>(b.emb);
  const uint4* RZ = reinterpret_cast<const uint4*>(b.root_emb);
  auto finish4 = [&](uint64_t s, uint64_t e) -> float2 {  // the row's 4 lanes, fixed order
    float2 P = f2_finish(s, e);
#pragma unroll
    for (int o = 1; o < 4; o <<= 1) {
      const float a = __shfl_xor_sync(0xffffffffu, P.x, o), q = __shfl_xor_sync(0xffffffffu, P.y, o);
      float t, u;
      two_sum(P.x, a, t, u);
      P.x = t;
      P.y = P.y + q + u;
    }
    float h, l;
    two_sum(P.x, P.y, h, l);
    return make_float2(h, l);
  };
  auto claim = [&]() {
    int k = 0;
    if (lane == 0) k = atomicAdd(&gs->stats_next, 1);
    return __shfl_sync(0xffffffffu, k, 0);
  };
  for (int blk = claim(); blk * 8 < n; blk = claim()) {
    const int i = blk * 8 + r;  // local row of this lane
    const bool live = i < n;
    // parent: >= 0 a local row, -2 the prompt embedding, -1 none (eta 0)
    int pl = -1;
    if (live) {
      if (early) {
        pl = i - 1;
      } else {
        pl = tree ? gs->par[i] : (gs->dep[i] > 1 ? i - 1 : -1);
        if (pl < 0) pl = b.root_emb ? -2 : -1;
      }
    }
    const bool from_left = pl >= 0 && pl == i - 1 && r > 0;
    // (debug build) the rows this lane reads; the whole warp skips the block if any is out of
    // range, since the sums below shuffle across all its lanes
    const bool rows_ok =
        GPO_BOUNDS(st, s0 + (live ? i : 0), sz.N, kWhereStats) && GPO_BOUNDS(st, pl >= 0 ? s0 + pl : 0, sz.N, kWhereStats);
    if (!__all_sync(0xffffffffu, rows_ok)) continue;
    const uint4* zb = Z + (int64_t)(s0 + (live ? i : 0)) * rs;
    const uint4* pb = pl >= 0 ? Z + (int64_t)(s0 + pl) * rs : (pl == -2 ? RZ + (int64_t)g * rs : nullptr);
    // error-free sums of the exact bf16 products (BiasedSum: a plain fp32 bound of each
    // segment's |products|, then Fast2Sum against a power-of-two bias, four operations per
    // product); a segment is one stage of kU chunks per lane
    BiasedSum sn, sd;
    bs_init(sn);
    bs_init(sd);
    // two stages of kU chunks per lane, software-pipelined: the next stage's loads are in
    // flight while this one's sums run (no register copies between the stages)
    constexpr int kU = 2;
    auto load = [&](int k0, uint4 (&x)[kU], uint4 (&y)[kU]) {
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int k = k0 + 4 * u + c;
        const bool in = k < nch;
        x[u] = live && in ? zb[k] : make_uint4(0u, 0u, 0u, 0u);
        y[u] = !from_left && pb && in ? pb[k] : make_uint4(0u, 0u, 0u, 0u);
      }
    };
    auto accumulate = [&](uint4 (&x)[kU], uint4 (&y)[kU]) {
      uint64_t xx[4 * kU], yy[4 * kU];
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
          xx[4 * u + h] = bf16x2_f32x2(xw[h]);
          yy[4 * u + h] = bf16x2_f32x2(yw[h]);
        }
      }
      uint64_t px = 0ull, py = 0ull;  // the segment's sums of squares (bounds only)
#pragma unroll
      for (int i = 0; i < 4 * kU; ++i) {
        px = f2fma(xx[i], xx[i], px);
        py = f2fma(yy[i], yy[i], py);
      }
      const float qx = f2_lanes_sum(px), qy = f2_lanes_sum(py);
      bs_reserve(sn, qx);
      bs_reserve(sd, 0.5f * (qx + qy));  // |x y| <= (x^2 + y^2) / 2
#pragma unroll
      for (int i = 0; i < 4 * kU; ++i) {
        bs_add(sn, xx[i], xx[i]);  // bf16 products are exact in fp32
        bs_add(sd, xx[i], yy[i]);
      }
    };
    uint4 xa[kU], ya[kU], xb[kU], yb[kU];
    load(0, xa, ya);
    for (int k0 = 0; k0 < nch; k0 += 8 * kU) {
      load(k0 + 4 * kU, xb, yb);  // past the row's end: zeros, which add nothing
      accumulate(xa, ya);
      load(k0 + 8 * kU, xa, ya);
      accumulate(xb, yb);
    }
    if (sz.d % 8 != 0 && c == 0 && live) {  // the ragged end of the row, one lane per row
      const uint16_t* zr = reinterpret_cast<const uint16_t*>(zb);
      const uint16_t* pr = reinterpret_cast<const uint16_t*>(pb);
      float qx = 0.f, qy = 0.f;
      for (int k = 8 * nch; k < sz.d; ++k) {
        const float x = __uint_as_float((uint32_t)zr[k] << 16), y = pr ? __uint_as_float((uint32_t)pr[k] << 16) : 0.f;
        qx = fmaf(x, x, qx);
        qy = fmaf(y, y, qy);
      }
      bs_reserve(sn, qx);
      bs_reserve(sd, 0.5f * (qx + qy));
      for (int k = 8 * nch; k < sz.d; ++k) {
        const uint64_t xx = pack_f2((uint32_t)zr[k] << 16, 0u);  // one fp32 lane (the other stays 0)
        const uint64_t yy = pack_f2(pr ? (uint32_t)pr[k] << 16 : 0u, 0u);
        bs_add(sn, xx, xx);
        bs_add(sd, xx, yy);
      }
    }
    uint64_t ns, ne, ds, de;
    bs_finish(sn, ns, ne);
    bs_finish(sd, ds, de);
    const float2 n2 = finish4(ns, ne);
    float2 dot = finish4(ds, de);
    if (pl == -1) dot = make_float2(0.f, 0.f);
    if (live && c == 0 && GPO_BOUNDS(st, s0 + i, sz.N, kWhereStats)) {
      if (!isfinite(n2.x) || !isfinite(dot.x)) report(st, GPO_ERR_NONFINITE, 3, s0 + i);
      ws.x_n2[s0 + i] = n2;
      ws.x_dot[s0 + i] = dot;
    }
  }
}


// Tree-layout set-up of group g (Sec. 4.2 branching rollouts: parents precede their
// children, depth-first pre-order): checks, depth, subtree end, own terminal statistics
// (Sec. 4.3: c_own / t_own of a state = the rewards / the number of the leaves of its
// subtree, the leaves in state order being the group's rollouts) and the first token of
// every edge.  One state per group thread (kGThreads >= kMaxN); every group thread calls
// it.  An invalid group gets bit 0 of gs->flags (visible to all on return).
__device__ __forceinline__ void tree_setup(const gpo_batch& b, const Sizes& sz, GroupSmem* gs, int g, int r0, int nr,
                                           int s0, int n, int gt, int wg, int lane, uint32_t* st) {
  const int64_t t0 = b.group_token_off[g], t1 = b.group_token_off[g + 1];
  const int i = gt;
  int pp = -1;
  bool bad = gt == 0 && (t0 < 0 || t1 < t0 || t1 > sz.T);
  if (i < n) {
    pp = b.parent[s0 + i];
    const int L = b.step_len[s0 + i];
    gs->lab[i] = i;
    gs->slen[i] = L;
    gs->par[i] = pp;
    gs->rend[i] = i + 1;
    gs->cown[i] = 0;
    gs->town[i] = 0;
    bad = bad || pp < -1 || pp >= i || L < 1;
  }
  bad = bar_any<kBarGroup, kGThreads>(bad);
  bool bad2 = false;
  if (!bad && i < n) {
    if (pp >= 0) {  // pre-order: p(v) lies on the path from the root to the state before v
      int x = i - 1;
      while (x > pp) x = gs->par[x];
      bad2 = x != pp;
    }
    int d = 1;
    for (int x = pp; x >= 0; x = gs->par[x]) {  // par[x] < x: at most i steps
      ++d;
      atomicMax(&gs->rend[x], i + 1);
    }
    gs->dep[i] = d;
  }
  bad = bar_any<kBarGroup, kGThreads>(bad2) || bad;
  if (bad) {
    if (gt == 0) {
      report(st, GPO_ERR_SHAPE, 2, g);
      atomicOr(&gs->flags, 1);
    }
    bar_group();
    return;
  }
  // leaf index and first token: block-wide scans of (is leaf, step length) in state order
  const bool leaf = i < n && gs->rend[i] == i + 1;
  int lc = leaf ? 1 : 0;
  long long tc = i < n ? gs->slen[i] : 0;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, lc, o);
    const long long z = __shfl_up_sync(0xffffffffu, tc, o);
    if (lane >= o) {
      lc += y;
      tc += z;
    }
  }
  int* wl = reinterpret_cast<int*>(gs->X);             // warp totals (X is free until the group math)
  long long* wt = reinterpret_cast<long long*>(gs->X + 64);
  if (lane == 31) {
    wl[wg] = lc;
    wt[wg] = tc;
  }
  bar_group();
  int lbase = 0, ltot = 0;
  long long tbase = 0, ttot = 0;
  for (int w = 0; w < kGThreads / 32; ++w) {
    if (w < wg) {
      lbase += wl[w];
      tbase += wt[w];
    }
    ltot += wl[w];
    ttot += wt[w];
  }
  if (gt == 0 && (ltot != nr || ttot != t1 - t0)) {
    report(st, GPO_ERR_SHAPE, 2, g);
    atomicOr(&gs->flags, 1);
  }
  if (i < n) gs->tstart[i] = t0 + tbase + tc - gs->slen[i];
  if (leaf) {
    const int li = lbase + lc - 1;  // < ltot
    if (li < nr) {
      const int rw = b.reward[r0 + li];
      if (rw > 1) {
        report(st, GPO_ERR_BAD_REWARD, 2, r0 + li);
        atomicOr(&gs->flags, 1);
      } else {
        for (int x = i; x >= 0; x = gs->par[x]) {
          atomicAdd(&gs->cown[x], rw);
          atomicAdd(&gs->town[x], 1);
        }
      }
    }
  }
  bar_group();
}

__global__ void __launch_bounds__(kThreads, kMinBlocks)
    fused_kernel(const __grid_constant__ CUtensorMap zmap, const __grid_constant__ CUtensorMap zmap32, gpo_batch b,
                 gpo_outputs o, Sizes sz, Ws ws, Params p) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // group state, barriers, then the tiles on a 1024-byte boundary (128B swizzle).  Every
  // pointer is smem_raw plus an offset, so the compiler keeps the shared address space
  // (plain shared loads, stores and atomics rather than generic ones).
  GroupSmem* gs = reinterpret_cast<GroupSmem*>(smem_raw);
  Ctl* ctl = reinterpret_cast<Ctl*>(smem_raw + kCtlOff);
  const uint32_t sbase = smem_u32(smem_raw);
  unsigned char* tiles = smem_raw + (((sbase + kTilesOff + 1023u) & ~1023u) - sbase);
  uint32_t* st = ws.status;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int KT = (sz.d + kTileK - 1) / kTileK;
  const float kappa = p.kappa_f;

  const bool tree = b.parent != nullptr;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    if (b.group_rollout_off[0] != 0 || b.group_rollout_off[sz.G] != sz.R) report(st, GPO_ERR_SHAPE, 2, 0);
    if (tree) {
      if (b.group_state_off[0] != 0 || b.group_state_off[sz.G] != sz.N) report(st, GPO_ERR_SHAPE, 2, 1);
      if (b.group_token_off[0] != 0 || b.group_token_off[sz.G] != sz.T) report(st, GPO_ERR_SHAPE, 2, 2);
    } else {
      if (b.rollout_step_off[0] != 0 || b.rollout_step_off[sz.R] != sz.N) report(st, GPO_ERR_SHAPE, 2, 1);
      if (b.rollout_token_off[0] != 0 || b.rollout_token_off[sz.R] != sz.T) report(st, GPO_ERR_SHAPE, 2, 2);
    }
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kMaxSlots; ++s) {
      mbar_init(&ctl->full[s], 1);
      mbar_init(&ctl->empty[s], 1);
    }
    mbar_init(&ctl->tfull, 1);
    mbar_init(&ctl->tempty, kEpiThreads / 32);
    mbar_init(&ctl->drain, 1);
    fence_mbar_init();
    gs->stats_next = 0;
    tma_prefetch_desc(&zmap);
    tma_prefetch_desc(&zmap32);
  }
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem_base;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer (lane 0)
    if (lane == 0) {
    // A k-slice (64 embedding elements of the rows a pass reads) takes exactly its bytes
    // of the ring; slice `seq` signals mbarrier pair seq % kMaxSlots.  The slices in flight
    // form one run in ring order, from the oldest one's offset o to head (wrapping to 0 at
    // most once), so a new slice at `off` is free to write when fewer than kMaxSlots are in
    // flight and: the run does not wrap (o < head) and the slice follows head, or wraps to
    // end by o; or the run wraps (o >= head) and the slice follows head and ends by o.
    // Otherwise wait for the oldest slice's consumption and look again.
    int head = 0;
    uint32_t seq = 0, oldest = 0;  // slices issued; oldest slice not yet seen consumed
    int f_off[kMaxSlots];
    bool ok = true;
    // L2 policy: pass 0 of a two-pass group keeps its rows (pass 1 reads them again),
    // pass 1 drops them first (their last read)
    const uint64_t keep = l2_policy_evict_last(), drop = l2_policy_evict_first();
    for (int g = sz.g0 + (int)blockIdx.x; g < sz.g1 && ok; g += gridDim.x) {
      int r0, nr, s0, n;
      if (!group_active(b, sz, g, r0, nr, s0, n)) continue;
      Plan pl;
      make_plan(n, pl);
      const int rows = r32(n);  // rows [0, r32(n)) of the group; the MMAs read no further
      for (int pass = 0; pass < pl.npass && ok; ++pass) {
        const int row0 = pl.npass == 2 && pass == 0 ? kTileM : 0;  // pass 0 of two never reads block 0
        const int bytes = (rows - row0) * 128;
        const int hint = pl.npass == 1 ? 0 : (pass == 0 ? 1 : 2);
        for (int k = 0; k < KT && ok; ++k) {
          const int off = ring_place(head, bytes);
          while (oldest < seq) {
            const int o = f_off[oldest % kMaxSlots];
            const bool busy = seq - oldest >= (uint32_t)kMaxSlots ||
                              (o < head ? (off != head && off + bytes > o) : (off != head || head + bytes > o));
            if (!busy) break;
            if (!mbar_wait(&ctl->empty[oldest % kMaxSlots], (oldest / kMaxSlots) & 1u, st, 20)) {
              ok = false;
              break;
            }
            ++oldest;
          }
          if (!ok) break;
          const int bi = (int)(seq % kMaxSlots);
          unsigned char* t = tiles + off;
          mbar_arrive_expect_tx(&ctl->full[bi], (uint32_t)bytes);
          for (int r = row0; r < rows;) {  // 128-row boxes, then 32-row boxes for the tail
            const bool big = rows - r >= kTileM;
            if (hint == 0)
              tma_load_2d(t + (r - row0) * 128, big ? &zmap : &zmap32, &ctl->full[bi], k * kTileK, s0 + r);
            else
              tma_load_2d_hint(t + (r - row0) * 128, big ? &zmap : &zmap32, &ctl->full[bi], k * kTileK, s0 + r,
                               hint == 1 ? keep : drop);
            r += big ? kTileM : kTailRows;
          }
          f_off[bi] = off;
          head = off + bytes;
          ++seq;
        }
      }
    }
    for (uint32_t j = oldest; j < seq; ++j)  // copies still landing in shared memory
      mbar_wait(&ctl->full[j % kMaxSlots], (j / kMaxSlots) & 1u, st, 21, 200000000ull, false);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer (lane 0)
    if (lane == 0) {
    int head = 0;
    uint32_t seq = 0;  // slices consumed (the producer's sequence)
    int u = 0;         // accumulator uses (passes) so far
    bool ok = true;
    // GPO_FLAG_DEBUG_TIMEOUT: the first wait runs out (nothing arrives on `drain` before the
    // commit below), and the CTA winds down as after any timeout
    if (p.debug_timeout) {
      mbar_wait(&ctl->drain, 0, st, 27, kDebugTimeoutNs);  // returns false: reports GPO_ERR_TIMEOUT
      ok = false;
    }
    for (int g = sz.g0 + (int)blockIdx.x; g < sz.g1 && ok; g += gridDim.x) {
      int r0, nr, s0, n;
      if (!group_active(b, sz, g, r0, nr, s0, n)) continue;
      Plan pl;
      make_plan(n, pl);
      const int rows = r32(n);
      for (int pass = 0; pass < pl.npass && ok; ++pass, ++u) {
        const int row0 = pl.npass == 2 && pass == 0 ? kTileM : 0;
        const int bytes = (rows - row0) * 128;
        if (!mbar_wait(&ctl->tempty, ((uint32_t)u & 1u) ^ 1u, st, 22)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int k = 0; k < KT; ++k) {
          const int off = ring_place(head, bytes);
          head = off + bytes;
          const int bi = (int)(seq % kMaxSlots);
          if (!mbar_wait(&ctl->full[bi], (seq / kMaxSlots) & 1u, st, 23)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t t = smem_u32(tiles + off);
          for (int si = 0; si < pl.nseg[pass]; ++si) {
            const Seg sg = pl.seg[pass][si];
            const uint64_t ad = smem_desc_k128(t + (uint32_t)((sg.b * kTileM - row0) * 128));
            const uint64_t bd = smem_desc_k128(t + (uint32_t)((sg.c0 - row0) * 128));
            const uint32_t idesc = idesc_bf16_f32(kTileM, r16(sg.len));
#pragma unroll
            for (int kk = 0; kk < kTileK / 16; ++kk)
              mma_bf16_ss(tmem + (uint32_t)sg.tcol, ad + 2u * kk, bd + 2u * kk, idesc, (k | kk) != 0);
          }
          mma_commit(&ctl->empty[bi]);
          ++seq;
        }
        if (ok) mma_commit(&ctl->tfull);
      }
    }
    mma_commit(&ctl->drain);
    mbar_wait(&ctl->drain, 0, st, 24, 200000000ull, false);
    }
    __syncwarp();
  } else if (warp >= 2) {
    // ---------------------------------------------------------------- group warps
    const int gt = threadIdx.x - 64;  // 0..447
    const bool epi = warp >= 4;
    const int q = warp & 3;           // TMEM lane quarter of an epilogue warp
    const int wg = warp - 2;          // 0..13
    int u = 0;
    for (int g = sz.g0 + (int)blockIdx.x; g < sz.g1; g += gridDim.x) {
      int r0 = 0, nr = 0, s0 = 0, n = 0;
      const bool in_range = group_range(b, sz, g, r0, nr, s0, n);
      if (!(in_range && n > 0 && n <= kMaxN && n <= sz.maxn && nr > 0 && nr <= n)) {
        if (gt == 0) {
          // tree layout: states need leaves, and an empty group has no tokens
          const bool tree_bad = tree && in_range &&
                                ((nr == 0 && n > 0) || (n == 0 && b.group_token_off[g + 1] != b.group_token_off[g]));
          if (!in_range || nr > n || (nr > 0 && n == 0) || tree_bad) report(st, GPO_ERR_SHAPE, 2, g);
          else if (n > kMaxN || n > sz.maxn) report(st, GPO_ERR_UNSUPPORTED, 2, g);
          else if (n == 0) {  // a group without states: Eff 0 (no tokens)
            if (o.group_eff) o.group_eff[g] = 0.f;
            if (o.group_eff_graph) o.group_eff_graph[g] = 0.f;
          }
        }
        continue;
      }
      if (gt == 0) {
        make_plan(n, gs->plan);
        gs->flags = 0;
        gs->overflow = 0;
      }

      // ---- compensated row statistics of the group (eta needs them; the Gram accumulator
      //      is too coarse): |z_v|^2 and <z_{p(v)}, z_v> as float pairs into ws.x_n2 / x_dot,
      //      read from L2 or HBM while the producer streams the same rows, only for each
      //      CTA's first group (its stream has nothing to overlap before it; later groups'
      //      come from a launch of their own).  A warp takes 8 rows, lane 4 r + c every fourth
      //      16-byte chunk of row r starting at chunk c; a parent that is the row before comes
      //      from the lane 4 below, other parents and the prompt embedding are loaded.  bf16
      //      products are exact in fp32, every sum is error-free (BiasedSum), the row's 4
      //      partial pairs are combined in a fixed butterfly.  Chain layout without prompt
      //      embeddings: the drain warps start at once (every state's parent taken as the
      //      state before it; a rollout's first state then has eta 0 whatever its dot) while
      //      warps 2 and 3 lay out the group, then join them; otherwise all group warps
      //      after the set-up.
      const bool stats_here = p.mode == 0 && p.stats_in_kernel && g < sz.g0 + (int)gridDim.x;
      const bool early = stats_here && !tree && b.root_emb == nullptr;
      if (early && epi) group_row_stats(b, sz, ws, gs, g, s0, n, false, true, lane, st);

      if (tree) {
        tree_setup(b, sz, gs, g, r0, nr, s0, n, gt, wg, lane, st);
      } else if (!early || !epi) {
      // ---- validate the group and lay out its states (Sec. 4.2 chain layout): all group
      //      threads, or warps 2 and 3 alone while the drain warps read the statistics
      const int tid = gt, nt = early ? 64 : kGThreads;  // warps 2 and 3: gt = 0..63
      auto sync = [&] {
        if (early) bar_setup();
        else bar_group();
      };
      for (int r = tid; r <= nr; r += nt) {
        gs->rstart[r] = b.rollout_step_off[r0 + r] - s0;
        gs->tok0[r] = b.rollout_token_off[r0 + r];
      }
      for (int r = tid; r < nr; r += nt) gs->rew[r] = b.reward[r0 + r];
      group_scratch_zero(gs->X, n, tid, nt);  // read after the drain
      for (int i = tid; i < n; i += nt) {
        gs->lab[i] = i;
        gs->slen[i] = b.step_len[s0 + i];
        gs->roll[i] = 0;
        gs->dep[i] = 1;
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
      if (early) group_row_stats(b, sz, ws, gs, g, s0, n, false, true, lane, st);  // join the drain warps
      }
      bar_group();  // set-up (and with `early` the row statistics) complete
      const bool valid = (gs->flags & 1) == 0;
      if (!early && valid && stats_here) group_row_stats(b, sz, ws, gs, g, s0, n, tree, false, lane, st);
      if (valid && stats_here && b.root_emb && wg == 0) {  // |prompt embedding|^2, one warp
        float2 n2, dot;
        exact_pair_sums<true>(b.root_emb, (int64_t)g * sz.stride, nullptr, 0, false, sz.d, lane, n2, dot);
        if (lane == 0) {
          if (!isfinite(n2.x)) report(st, GPO_ERR_NONFINITE, 3, sz.N + g);
          ws.x_root_n2[g] = n2;
        }
      }

      // ---- eta(p(v), v) of every state from the finished statistics, by warps 2 and 3 while
      //      the drain warps test the pairs (with `early`: no prompt embedding, a rollout's
      //      first state has eta 0); the group math takes it from ecor / eeff, which it
      //      overwrites only with its own outputs, state by state, after reading it
      if (early && valid && !epi) {
        for (int i = gt; i < n; i += 64) {
          const float2 e = gs->dep[i] == 1 ? make_float2(0.f, 0.f)
                                           : ff_eta(ws.x_dot[s0 + i], ws.x_n2[s0 + i - 1], ws.x_n2[s0 + i]);
          gs->ecor[i] = e.x;
          gs->eeff[i] = e.y;
        }
      }

      // ---- drain the accumulator pass by pass (warps 4..15)
      bool fail = false;
      if (epi) {
        const Plan& pl = gs->plan;
        const int te = threadIdx.x - 128;     // 0..383
        const int t128 = q * 32 + lane;       // accumulator lane = row within a 128-row block
        const int rep = (warp - 4) >> 2;      // which of the quarter's kReps warps
        const int ew = warp - 4;              // epilogue warp 0..11: owns elist[ew * kWarpEdges, ...)
        uint32_t* wlist = gs->elist + ew * kWarpEdges;
        int wcount = 0;                       // pairs this warp found in the group (warp-uniform)
        for (int pass = 0; pass < pl.npass; ++pass, ++u) {
          const bool got = mbar_wait(&ctl->tfull, (uint32_t)u & 1u, st, 25);
          if (bar_any<kBarEpi, kEpiThreads>(!got)) {
            fail = true;
            break;
          }
          tc_fence_after();
          const int nseg = pl.nseg[pass];
          // squared norms (for the threshold test) from the diagonal of the diagonal segments
          // of this pass (row block b is read by the quarter's warp b % 3)
#pragma unroll 1
          for (int si = 0; si < nseg; ++si) {
            const Seg sg = pl.seg[pass][si];
            if (sg.c0 != sg.b * kTileM || sg.b % kReps != rep || q * 32 >= sg.len) continue;
            const int i = sg.b * kTileM + t128;
            const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)sg.tcol;
            uint32_t r[32];
            tmem_ld_32x32b_x32(base + (uint32_t)(q * 32), r);
            tmem_wait_ld();
            const float dg = pick(r, lane);
            if (i < n) {
              gs->n2[i] = dg;
              if (!isfinite(dg)) report(st, GPO_ERR_NONFINITE, 2, s0 + i);
            }
          }
          bar_epi();
#pragma unroll 1
          for (int si = 0; si < nseg; ++si) {
            const Seg sg = pl.seg[pass][si];
            if (sg.c0 != sg.b * kTileM || sg.b % kReps != rep) continue;
            const int i = sg.b * kTileM + t128;
            if (i < n) {
              const float n2i = gs->n2[i];
              gs->rn[i] = n2i > 0.f ? 1.0f / sqrtf(n2i) : 0.f;
              gs->thr[i] = n2i > 0.f && valid ? kappa * sqrtf(n2i) : __int_as_float(0x7f800000);
            }
          }
          bar_epi();
          // linked pairs: comparable (different rollout [, same depth]) with sim >= kappa,
          // tested as acc / |z_j| - kappa |z_i| >= 0 (one fma per pair).  In the chain layout
          // the columns j > i outside i's rollout are exactly j >= rend(i), so one bit mask per
          // 32-column chunk keeps j in [rend(i), n).  The quarter's chunks that hold a column
          // right of some row of the warp are dealt round-robin to its three warps.  Each pair
          // found goes to the edge list (or, past its capacity, straight into the forest).
          {
            int dealt = 0;
#pragma unroll 1
            for (int si = 0; si < nseg; ++si) {
              const Seg sg = pl.seg[pass][si];
              const int rowbase = sg.b * kTileM + q * 32;
              const int i = rowbase + lane;
              const bool vrow = i < n;
              const float thr = vrow ? gs->thr[i] : __int_as_float(0x7f800000);
              const int re = vrow ? gs->rend[i] : n;
              const int di = vrow ? gs->dep[i] : -1;
              const int nch = (sg.len + 31) >> 5;
#pragma unroll 1
              for (int ch = 0; ch < nch; ++ch) {
                const int cbase = sg.c0 + ch * 32;
                if (cbase + 31 <= rowbase) continue;  // no column right of any row of this warp
                if (dealt++ % kReps != rep) continue;
                uint32_t r[32];
                tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(sg.tcol + ch * 32), r);
                tmem_wait_ld();
                // bit j of `miss` = sign of acc_j / |z_j| - kappa |z_i| (one fma, exact product):
                // set when the pair is below the threshold
                // (four partial masks keep the or-chains short)
                uint32_t mp[4] = {0u, 0u, 0u, 0u};
                const float4* rn4 = reinterpret_cast<const float4*>(gs->rn + cbase);
#pragma unroll
                for (int j4 = 0; j4 < 8; ++j4) {
                  const float4 c = rn4[j4];
                  const float cc[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
                  for (int t = 0; t < 4; ++t) {
                    const int j = 4 * j4 + t;
                    mp[t] |= (__float_as_uint(fmaf(__uint_as_float(r[j]), cc[t], -thr)) >> 31) << j;
                  }
                }
                const uint32_t miss = (mp[0] | mp[1]) | (mp[2] | mp[3]);
                uint32_t mk = vrow ? ~miss & bits_from(re - cbase) & ~bits_from(n - cbase) : 0u;
                if (p.rule == GPO_MERGE_SAME_DEPTH && mk) {
                  uint32_t m2 = 0u;
                  for (uint32_t t = mk; t; t &= t - 1u) {
                    const int j = __ffs(t) - 1;
                    if (gs->dep[cbase + j] == di) m2 |= 1u << j;
                  }
                  mk = m2;
                }
                // this warp's part of the edge list: one pair per lane per step, slots by ballot
                for (uint32_t act = __ballot_sync(0xffffffffu, mk != 0); act;
                     act = __ballot_sync(0xffffffffu, mk != 0)) {
                  const int slot = wcount + __popc(act & ((1u << lane) - 1u));
                  if (mk) {
                    const int j = cbase + __ffs(mk) - 1;
                    mk &= mk - 1u;
                    if (slot < kWarpEdges) wlist[slot] = (uint32_t)i | ((uint32_t)j << 16);
                    else uf_union(gs->lab, i, j);
                  }
                  wcount += __popc(act);
                }
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ctl->tempty);  // accumulator free for the next pass
          // classes = connected components of the linked pairs (Alg. S.1) in the label forest
          // lab (lab[x] <= x, within x's class).  Rounds of hooking over every listed pair of
          // the group (the larger of the two current labels is pointed at the smaller) and
          // shortcutting (lab[x] = lab[lab[x]]) until no pair has unequal labels and every
          // label is a root: then each class's label is its smallest member.  The rounds
          // revisit the pairs of earlier passes, whose links a hook may re-point.  If the list
          // overflowed (pairs united directly), the listed pairs are united the same way
          // instead (root-to-root links, which never re-point a link).
          if (lane == 0 && wcount > kWarpEdges) gs->overflow = 1;
          bar_epi();
          const int nw = min(wcount, kWarpEdges);  // this warp's listed pairs
          if (!gs->overflow) {
            bool conv = false;
#pragma unroll 1
            for (int round = 0; round <= kMaxN && !conv; ++round) {
              bool ch = false;
              for (int e = lane; e < nw; e += 32) {
                const uint32_t ij = wlist[e];
                const int lu = gs->lab[ij & 0xFFFFu], lv = gs->lab[ij >> 16];
                if (lu != lv) {
                  atomicMin(&gs->lab[max(lu, lv)], min(lu, lv));
                  ch = true;
                }
              }
              for (int x = te; x < n; x += kEpiThreads) {
                const int l = gs->lab[x], ll = gs->lab[l];
                if (ll != l) {
                  gs->lab[x] = ll;
                  ch = true;
                }
              }
              conv = !bar_any<kBarEpi, kEpiThreads>(ch);
            }
            if (!conv) {  // not reached in practice; the unions below are correct from any state
              for (int e0 = 0; e0 < nw; e0 += 32) {
                if (e0 + lane < nw) {
                  const uint32_t ij = wlist[e0 + lane];
                  uf_union(gs->lab, (int)(ij & 0xFFFFu), (int)(ij >> 16));
                }
                __syncwarp();
              }
            }
          } else {
            for (int e0 = 0; e0 < nw; e0 += 32) {
              if (e0 + lane < nw) {
                const uint32_t ij = wlist[e0 + lane];
                uf_union(gs->lab, (int)(ij & 0xFFFFu), (int)(ij >> 16));
              }
              __syncwarp();
            }
          }
        }
      }
      if (bar_any<kBarGroup, kGThreads>(fail)) break;

      // ---- next-layer budgets of a branching group (gpo_layer_budget)
      if (valid && p.mode == 1) {
        auto active = [&](int i) { return p.active == nullptr || p.active[s0 + i] != 0; };
        auto put = [&](int i, int label, int bud) {
          p.budget[s0 + i] = bud;
          if (o.class_id) o.class_id[s0 + i] = s0 + label;
        };
        group_budget(n, gs->lab, gs->dep, p.layer, p.b_next, reinterpret_cast<int*>(gs->n2),
                     reinterpret_cast<int*>(gs->esum), reinterpret_cast<int*>(gs->elist), gt, kGThreads,
                     active, [] { bar_group(); }, put);
      }
      // ---- graph reward and dual-group advantage of every edge
      else if (valid) {
        // eta(p(v), v) from the compensated row statistics (pairs; see exact_stats_kernel)
        auto eta = [&](int i) -> float2 {
          if (early) return make_float2(gs->ecor[i], gs->eeff[i]);
          const float2 z = make_float2(0.f, 0.f);
          const float2 n1 = gs->dep[i] == 1 ? (b.root_emb ? ws.x_root_n2[g] : z) : ws.x_n2[s0 + i - 1];
          return ff_eta(ws.x_dot[s0 + i], n1, ws.x_n2[s0 + i]);
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
        if (tree) {
          auto eta_t = [&](int i) -> float2 {
            const float2 z = make_float2(0.f, 0.f);
            const int pp = gs->par[i];
            const float2 n1 = pp < 0 ? (b.root_emb ? ws.x_root_n2[g] : z) : ws.x_n2[s0 + pp];
            return ff_eta(ws.x_dot[s0 + i], n1, ws.x_n2[s0 + i]);
          };
          group_advantages_tree<1>(n, nr, gs->lab, gs->par, gs->dep, gs->rend, gs->cown, gs->town,
                                   tree_scratch(smem_raw + kTreeXOff, n), p, gt, kGThreads, [] { bar_group(); },
                                   eta_t, out);
        } else {
          group_advantages<1, true>(n, nr, gs->lab, gs->roll, gs->dep, gs->rstart, gs->rew,
                                    group_scratch_sep(gs->X, n), p, gt, kGThreads, [] { bar_group(); }, eta, out);
        }
        // ---- exploration efficiency, Eq. (eq1) (the threshold norms' array is free here)
        if (o.group_eff || o.group_eff_graph) {
          auto own = [&](int i) { return tree ? gs->cown[i] > 0 : gs->rew[gs->roll[i]] != 0; };
          auto par = [&](int i) { return tree ? gs->par[i] : (gs->dep[i] == 1 ? -1 : i - 1); };
          auto len = [&](int i) { return gs->slen[i]; };
          group_efficiency(n, gs->lab, reinterpret_cast<int*>(gs->n2), gs->esum, gt, kGThreads, own, par, len,
                           [] { bar_group(); }, [](bool f) { return bar_any<kBarGroup, kGThreads>(f); },
                           o.group_eff ? o.group_eff + g : nullptr, o.group_eff_graph ? o.group_eff_graph + g : nullptr);
        }
        // ---- every token of an edge carries the edge's advantage (Sec. 4.5).  State-major:
        //      each half-warp takes a state, its 16 lanes write the whole 16-byte chunks of the
        //      state's token span, then the at most 3 + 3 tokens of its partial first and last
        //      chunk (which neighbour other states' tokens) with scalar stores.
        const bool more = o.adv_cor || o.adv_eff || o.eff_mask;
        const int hl = gt & 15;
#pragma unroll 1
        for (int i = gt >> 4; i < n; i += kGThreads / 16) {
          const int64_t ts = gs->tstart[i], te = ts + gs->slen[i];
          const float x = gs->eadv[i];
          const int64_t qa = (ts + 3) >> 2, qb = te >> 2;
          const int64_t h1 = qa <= qb ? 4 * qa : te;  // head [ts, h1)
          const int64_t t0 = qa <= qb ? 4 * qb : te;  // tail [t0, te)
          const int64_t tp = hl < 4 ? ts + hl : t0 + (hl - 4);
          const bool scal = hl < 4 ? tp < h1 : (hl < 8 && tp < te);
          // (debug build) every store below lies in the state's span [ts, te)
          if (!GPO_BOUNDS(st, ts, sz.T, kWhereTokens) || !GPO_BOUNDS(st, te - 1, sz.T, kWhereTokens)) continue;
          {
            const float4 v = make_float4(x, x, x, x);
            for (int64_t c = qa + hl; c < qb; c += 16) reinterpret_cast<float4*>(o.adv)[c] = v;
            if (scal) o.adv[tp] = x;
          }
          if (more) {
            if (o.adv_cor) {
              const float y = gs->ecor[i];
              const float4 v = make_float4(y, y, y, y);
              for (int64_t c = qa + hl; c < qb; c += 16) reinterpret_cast<float4*>(o.adv_cor)[c] = v;
              if (scal) o.adv_cor[tp] = y;
            }
            if (o.adv_eff) {
              const float y = gs->eeff[i];
              const float4 v = make_float4(y, y, y, y);
              for (int64_t c = qa + hl; c < qb; c += 16) reinterpret_cast<float4*>(o.adv_eff)[c] = v;
              if (scal) o.adv_eff[tp] = y;
            }
            if (o.eff_mask) {
              const uint8_t m = gs->emask[i];
              const uint32_t v = 0x01010101u * m;
              for (int64_t c = qa + hl; c < qb; c += 16) reinterpret_cast<uint32_t*>(o.eff_mask)[c] = v;
              if (scal) o.eff_mask[tp] = m;
            }
          }
        }
      }
      if (gt == 0) gs->stats_next = 0;  // for the next group's row statistics
      bar_group();
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

size_t fused_smem() { return (size_t)kTilesOff + 1023 + (size_t)kRingBytes; }
