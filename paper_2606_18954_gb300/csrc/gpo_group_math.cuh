// Per-group graph reward and dual-group advantage, shared by the per-group
// kernel of the tiled path and by the fused group-resident kernel.
//
// Given the group's union-find forest (parent[x] <= x, built from the linked
// pairs of Sec. 4.2), per-state rollout / depth and per-rollout rewards, it
// computes for every generated edge (p(v), v):
//   S(v)      Eq. (combain), chain layout: c_own(v) = R of v's rollout,
//             t_own(v) = 1, so S(v) = (c + w (C_Q - c)) / (1 + w (|Q| - 1));
//             S(root) = sum R / R_g                                  (Sec. 4.3)
//   r_step    (S(v) - S(p(v))) (1 - eta(p(v), v))                    (Sec. 4.3)
//   A_cor     edges grouped by the class of p(v) (the root is its own group);
//             (r - mean) / (std + eps), groups of one edge get 0     (Sec. 4.4)
//   A_eff     per class |Q| >= 2: Sbar_Q (-l_v - mean(-l)) / (std(-l) + eps),
//             l_v = depth (a_Q is the root), routed onto every edge of
//             root -> v, summed over routes                           (Sec. 4.4)
//   A_dual    A_cor + lambda_eff * routed A_eff                        (Sec. 4.5)
#pragma once

#include "gpo_internal.cuh"

namespace gpo {

__device__ __forceinline__ int uf_find(const int* p, int x) {
  const volatile int* vp = p;
  while (true) {
    const int y = vp[x];
    if (y == x) return x;
    x = y;
  }
}

// Hook the larger root under the smaller one, so parent[x] <= x always holds
// and the final root of a class is its smallest member.
__device__ __forceinline__ void uf_union(int* p, int a, int b) {
  while (true) {
    a = uf_find(p, a);
    b = uf_find(p, b);
    if (a == b) return;
    if (a > b) {
      const int t = a;
      a = b;
      b = t;
    }
    if (atomicCAS(&p[b], b, a) == b) return;
  }
}

// Exact, order-independent integer sums through 32-bit shared-memory atomics (64-bit
// ones are compare-and-swap loops that serialise under contention): a non-negative
// value below 2^(kChunks * kBits) is added as kChunks chunks of kBits bits, one counter
// each.  With kBits <= 19 and at most 4096 terms no counter can overflow.
template <int kChunks, int kBits>
__device__ __forceinline__ void red_chunks(unsigned* acc, unsigned long long v) {
#pragma unroll
  for (int c = 0; c < kChunks; ++c) atomicAdd(&acc[c], (unsigned)((v >> (c * kBits)) & ((1ull << kBits) - 1)));
}

template <int kChunks, int kBits>
__device__ __forceinline__ unsigned long long sum_chunks(const unsigned* acc) {
  unsigned long long s = 0;
#pragma unroll
  for (int c = 0; c < kChunks; ++c) s += (unsigned long long)acc[c] << (c * kBits);
  return s;
}

// Chunk counters of the sums below (per key).
constexpr int kSumWords = 3;   // sum of r on the 2^-50 grid: r * 2^50 + 2^50 in [0, 2^51], 3 x 18 bits
constexpr int kSqhWords = 3;   // sum of (r - mean)^2 on the 2^-36 grid: in [0, 2^38] (|r - mean| <= 2), 3 x 13 bits
constexpr int kSqlWords = 3;   // and its 2^-76 grid remainder + 2^39, in [0, 2^40], 3 x 14 bits

// Exact sum of x = (r - mean)^2 <= 4: each x splits into a 2^-36-grid part and a
// 2^-76-grid remainder (both exact in fp32), summed as chunked integers.
__device__ __forceinline__ void sq_add(unsigned* hi, unsigned* lo, float x) {
  const float X = x * 0x1p36f;
  const float h = rintf(X);
  red_chunks<kSqhWords, 13>(hi, (unsigned long long)__float2ll_rn(h));
  red_chunks<kSqlWords, 14>(lo, (unsigned long long)(__float2ll_rn((X - h) * 0x1p40f) + (1ll << 39)));
}

// Rounded quotient of an int64 by a positive int.
__device__ __forceinline__ long long div_round(long long a, int k) {
  long long q = a / k, rem = a - q * k;
  if (2 * (rem < 0 ? -rem : rem) >= k) q += (a < 0 ? -1 : 1);
  return q;
}

__host__ __device__ constexpr size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

// c + w a as a float pair (a, c integers below 2^24; w = wh + wl, the fp64 parameter to
// about 2^-48): TwoProduct of wh a, TwoSum with c.
__device__ __forceinline__ float2 lin_ff(int c, int a, float wh, float wl) {
  const float fa = (float)a;
  const float p = wh * fa;
  const float e = fmaf(wh, fa, -p);
  float h, t;
  two_sum((float)c, p, h, t);
  return make_float2(h, t + e + wl * fa);
}

// Eq. (combain) as a float pair: (c_own + w (C_Q - c_own)) / (t_own + w (T_Q - t_own)).
// Numerator and denominator come out of the same operations, so a class whose leaves
// share one reward gets exactly 1 (or exactly 0).
__device__ __forceinline__ float2 score_ff(int c, int t, int C, int T, float wh, float wl) {
  return ff_div(lin_ff(c, C - c, wh, wl), lin_ff(t, T - t, wh, wl));
}

// r_step = (S(v) - S(p(v))) (1 - eta) on the 2^-50 grid (|r| <= 1), from pair-valued
// scores and eta: the pair arithmetic keeps r to ~2^-46 relative, well below the grid
// of the exact group sums that follow.
__device__ __forceinline__ long long step_reward_fixed(float2 S, float2 Sp, float2 eta) {
  const float2 d = ff_add(S, make_float2(-Sp.x, -Sp.y));
  const float2 r = ff_mul(d, ff_add(make_float2(1.0f, 0.0f), make_float2(-eta.x, -eta.y)));
  return __float2ll_rn(r.x * 0x1p50f) + __float2ll_rn(r.y * 0x1p50f);
}

// Scratch arrays of group_advantages.  Class sums are indexed by the class root
// (a local state index), correctness-group sums by the key (the class of the
// parent, or n for the prompt root); the route sums reuse the class arrays.
struct GroupScratch {
  int* ccnt;            // [n]   |Q|
  int* csum;            // [n]   C_Q = sum of the members' rewards
  int* lsum;            // [n]   sum of the members' depths
  unsigned* l2;         // [n][2] sum of the squared depths, 2 x 13-bit chunks
  int* kcnt;            // [n+1] edges per correctness group
  unsigned* ksum;       // [n+1][kSumWords] sum of r (chunked, see above)
  unsigned* kqh;        // [n+1][kSqhWords] sum of (r - mean)^2, 2^-36 grid part
  unsigned* kql;        // [n+1][kSqlWords] and its 2^-76 grid remainder
  float* aeff;          // [n]   A_eff of each route end (over ccnt)
  float* E;             // [n]   routed A_eff (over lsum)
  unsigned char* cov;   // [n]   covered by a route (over l2)
  int* rootc;           // [1]   sum of the group's rewards
};

constexpr int kClassWords = 5;                                   // 4-byte words per class
constexpr int kKeyWords = 1 + kSumWords + kSqhWords + kSqlWords;  // per key

// Separate layout: class and key arrays side by side, for callers that zero
// them ahead of time (group_scratch_zero); bytes for a group of up to n states.
__host__ __device__ constexpr size_t group_scratch_sep_bytes(int n) {
  return 4 * (kClassWords * (size_t)n + kKeyWords * (size_t)(n + 1)) + 16;
}

__device__ __forceinline__ void group_scratch_carve(GroupScratch& g, unsigned char* cls, unsigned char* key, int n) {
  g.ccnt = reinterpret_cast<int*>(cls);
  g.csum = g.ccnt + n;
  g.lsum = g.csum + n;
  g.l2 = reinterpret_cast<unsigned*>(g.lsum + n);
  g.kcnt = reinterpret_cast<int*>(key);
  g.ksum = reinterpret_cast<unsigned*>(g.kcnt + (n + 1));
  g.kqh = g.ksum + kSumWords * (n + 1);
  g.kql = g.kqh + kSqhWords * (n + 1);
  g.aeff = reinterpret_cast<float*>(g.ccnt);
  g.E = reinterpret_cast<float*>(g.lsum);
  g.cov = reinterpret_cast<unsigned char*>(g.l2);
}

__device__ __forceinline__ GroupScratch group_scratch_sep(unsigned char* X, int n) {
  GroupScratch g;
  group_scratch_carve(g, X, X + 4 * kClassWords * (size_t)n, n);
  g.rootc = reinterpret_cast<int*>(X + 4 * (kClassWords * (size_t)n + kKeyWords * (size_t)(n + 1)));
  return g;
}

// Zero the sums of a separate-layout scratch (before the barrier that precedes
// group_advantages<kPer, true>).
__device__ __forceinline__ void group_scratch_zero(unsigned char* X, int n, int tid, int nt) {
  int* w = reinterpret_cast<int*>(X);
  const int nw = kClassWords * n + kKeyWords * (n + 1) + 1;
  for (int i = tid; i < nw; i += nt) w[i] = 0;
}

// Shared layout: the class, key and route arrays overlay one region (the largest
// is the key sums), for large groups; group_advantages zeroes each in turn, at the
// cost of extra barriers.
__host__ __device__ constexpr size_t group_scratch_bytes(int n) {
  return al16(4 * kKeyWords * (size_t)(n + 1) + 32);
}

__device__ __forceinline__ GroupScratch group_scratch_shared(unsigned char* X, int n, int* rootc) {
  GroupScratch g;
  group_scratch_carve(g, X, X, n);
  g.rootc = rootc;
  return g;
}

// One group, `nt` cooperating threads (thread index tid), kPer * nt >= n.
//   lab     [n] shared union-find forest on entry, class labels (local index of
//           the smallest member) on exit
//   roll    [n] rollout of each state, local to the group (0..nr-1)
//   dep     [n] depth of each state (1 = first step)
//   rstart  [nr+1] local state offsets of the rollouts
//   rew     [nr] rewards
//   sc      scratch: separate layout zeroed by the caller (kZeroed), or the
//           shared layout (!kZeroed)
//   eta(i)  eta(p(v), v) of local state i as a float pair (already clamped at 0)
//   out(i, label, S, acor, E, dual, mask) is called once per state by its owner
//   sync()  barrier over the nt threads
//
// Precision: fp32 arithmetic with exact integer class sums and an exact
// fixed-point group mean (the one quantity whose rounding the standardisation
// amplifies).  Per-class and per-group constants are recomputed by every state
// that needs them (same operands, same operations, so the same value), which
// saves a barrier per constant.  Sums go through integer atomics, so results do
// not depend on the order in which threads add.
template <int kPer, bool kZeroed, class IdxT, class Sync, class Eta, class Out>
__device__ __forceinline__ void group_advantages(int n, int nr, int* lab, const IdxT* roll, const IdxT* dep,
                                                 const int* rstart, const uint8_t* rew, const GroupScratch& sc,
                                                 const Params& p, int tid, int nt, Sync sync, Eta eta, Out out) {
  const float w = p.w_hi, eps = p.eps_f;
  const float wl = p.w_lo;  // w = w + wl to ~2^-48
  // ---- phase A: class sums C_Q (rewards), |Q|, sum l, sum l^2
  if (!kZeroed) {
    for (int i = tid; i < n; i += nt) {
      sc.ccnt[i] = sc.csum[i] = sc.lsum[i] = 0;
      sc.l2[2 * i] = sc.l2[2 * i + 1] = 0u;
    }
    if (tid == 0) *sc.rootc = 0;
    sync();
  }
  int lb[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    lb[k] = 0;
    if (i < n) {
      // writing the root over the parent keeps every concurrent find on the same root
      lb[k] = uf_find(lab, i);
      lab[i] = lb[k];
      const int d = dep[i];
      atomicAdd(&sc.ccnt[lb[k]], 1);
      atomicAdd(&sc.csum[lb[k]], (int)rew[roll[i]]);
      atomicAdd(&sc.lsum[lb[k]], d);
      red_chunks<2, 13>(&sc.l2[2 * lb[k]], (unsigned long long)d * d);  // d <= 4096: d^2 <= 2^24
    }
  }
  for (int r = tid; r < nr; r += nt) atomicAdd(sc.rootc, (int)rew[r]);
  sync();
  const float2 S_root = ff_div(make_float2((float)*sc.rootc, 0.f), make_float2((float)nr, 0.f));
  float S[kPer], aeff[kPer];
  long long rf[kPer];
  int key[kPer];
  bool route_end[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    S[k] = aeff[k] = 0.f;
    rf[k] = 0;
    key[k] = n;
    route_end[k] = false;
    if (i >= n) continue;
    const int L = lb[k], Q = sc.ccnt[L], d = dep[i], c = rew[roll[i]];
    // Eq. (combain): (c_own + w sum_{q != v} c_own(q)) / (t_own + w sum_{q != v} t_own(q)), t_own = 1,
    // as a float pair (a class whose members share one reward gets S exactly 0 or 1)
    const float2 Sv = score_ff(c, 1, sc.csum[L], Q, w, wl);
    S[k] = Sv.x;
    if (Q >= 2) {
      // Sbar_Q = mean of S over Q = C_Q / |Q| (every member has t_own = 1);
      // sum (l - mean)^2 = (Q sum l^2 - (sum l)^2) / Q with an exact integer numerator;
      // A_eff(v) = Sbar (mean l - l_v) / (sd + eps) = g (sum l - Q l_v),
      // g = C_Q / (Q^2 (sd + eps)).  Fast reciprocal square root and division here (a few
      // ulp; A_eff has no exact special value to keep).
      const long long ls = sc.lsum[L];
      const float num = (float)((long long)Q * (long long)sum_chunks<2, 13>(&sc.l2[2 * L]) - ls * ls);
      const float var = __fdividef(num, (float)Q * (float)(Q - p.ddof));
      const float sd = var > 0.f ? var * rsqrtf(var) : 0.f;
      const float g = __fdividef((float)sc.csum[L], (float)Q * (float)Q * (sd + eps));
      route_end[k] = true;
      aeff[k] = g * (float)(sc.lsum[L] - Q * d);
    }
    float2 Sp = S_root;
    if (d != 1) {
      const int Lp = lab[i - 1];  // parent: the previous state of the same rollout (same reward c)
      Sp = score_ff(c, 1, sc.csum[Lp], sc.ccnt[Lp], w, wl);
      key[k] = Lp;
    }
    rf[k] = step_reward_fixed(Sv, Sp, eta(i));
  }

  // ---- phase B: correctness groups, key = class of p(v), n = the prompt root
  if (!kZeroed) {
    sync();  // class sums no longer read
    for (int i = tid; i < (kKeyWords) * (n + 1); i += nt) reinterpret_cast<int*>(sc.kcnt)[i] = 0;
    sync();
  }
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    if (tid + k * nt < n) {
      // |r| <= 1 and a group holds at most 4096 edges: a 2^50 fixed point cannot overflow
      atomicAdd(&sc.kcnt[key[k]], 1);
      red_chunks<kSumWords, 18>(&sc.ksum[kSumWords * key[k]], (unsigned long long)(rf[k] + (1ll << 50)));
    }
  }
  sync();
  float dv[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    dv[k] = 0.f;
    if (tid + k * nt < n) {
      const int cnt = sc.kcnt[key[k]];
      // offsets removed in unsigned arithmetic (the biased sum can reach 2^63)
      const long long tot = (long long)(sum_chunks<kSumWords, 18>(&sc.ksum[kSumWords * key[k]]) - ((unsigned long long)cnt << 50));
      const long long mean = div_round(tot, cnt);  // exact mean on the 2^-50 grid
      dv[k] = (float)(rf[k] - mean) * 0x1p-50f;
      sq_add(&sc.kqh[kSqhWords * key[k]], &sc.kql[kSqlWords * key[k]], dv[k] * dv[k]);
    }
    if (kZeroed && tid + k * nt < n) {  // route arrays overlay the class sums, read last above
      sc.aeff[tid + k * nt] = aeff[k];
      sc.cov[tid + k * nt] = route_end[k] ? 1 : 0;
    }
  }
  sync();
  float acor[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    acor[k] = 0.f;
    const int K = key[k], cnt = sc.kcnt[K];
    if (tid + k * nt < n && cnt >= 2) {  // groups of one edge get no advantage
      const long long qh = (long long)sum_chunks<kSqhWords, 13>(&sc.kqh[kSqhWords * K]);
      const long long ql = (long long)(sum_chunks<kSqlWords, 14>(&sc.kql[kSqlWords * K]) - ((unsigned long long)cnt << 39));
      const float ss = (float)qh * 0x1p-36f + (float)ql * 0x1p-76f;  // sum (r - mean)^2
      const float var = __fdividef(ss, (float)(cnt - p.ddof));
      const float sd = var > 0.f ? var * rsqrtf(var) : 0.f;
      acor[k] = dv[k] * __fdividef(1.0f, sd + eps);  // a zero deviation stays exactly 0
    }
  }

  // ---- phase C: every edge on root -> v receives A_eff(v) (suffix sums per rollout)
  if (!kZeroed) {  // the route arrays overlay the key sums, read last just above
    sync();
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int i = tid + k * nt;
      if (i < n) {
        sc.aeff[i] = aeff[k];
        sc.cov[i] = route_end[k] ? 1 : 0;
      }
    }
    sync();
  }
  // suffix sums along each rollout, one warp per rollout: 32 states at a time from the
  // rollout's end, a shuffle scan within the warp plus the running total of later states
  {
    const int lane = tid & 31, nw = nt >> 5;
    for (int rr = tid >> 5; rr < nr; rr += nw) {
      const int lo = rstart[rr];
      float carry = 0.f;
      bool ccov = false;
      for (int hi = rstart[rr + 1]; hi > lo; hi -= 32) {
        const int i = hi - 1 - lane;  // lane 0 holds the last state of the chunk
        const bool in = i >= lo;
        float v = in ? sc.aeff[i] : 0.f;
        const bool c = in && sc.cov[i] != 0;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const float y = __shfl_up_sync(0xffffffffu, v, off);
          if (lane >= off) v += y;
        }
        const uint32_t cb = __ballot_sync(0xffffffffu, c);
        const float tot = __shfl_sync(0xffffffffu, v, 31);
        if (in) {
          sc.E[i] = v + carry;
          sc.cov[i] = (ccov || (cb & (0xFFFFFFFFu >> (31 - lane))) != 0) ? 1 : 0;
        }
        carry += tot;
        ccov = ccov || cb != 0;
      }
    }
  }
  sync();
  const float lam = p.lambda_f;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) out(i, lb[k], S[k], acor[k], sc.E[i], fmaf(lam, sc.E[i], acor[k]), sc.cov[i]);
  }
  sync();
}

// ---------------------------------------------------------------------------------
// Tree layout (branching rollouts, parent pointers, states in depth-first pre-order):
// the same quantities as group_advantages, with the provenance tree's own statistics
//   c_own(v) = sum of R(z) over the leaves z of v's subtree, t_own(v) = their number
//             (bottom-up along direct edges, Sec. 4.3), given by the caller;
//   S(v)      (c_own + w (C_Q - c_own)) / (t_own + w (T_Q - t_own)), class sums
//             C_Q, T_Q; S(root) = sum R / number of leaves                  (Eq. (combain))
//   r_step    (S(v) - S(p(v))) (1 - eta(p(v), v))                          (Sec. 4.3)
//   A_cor     edges grouped by the class of p(v), as in the chain layout    (Sec. 4.4)
//   A_eff     per class |Q| >= 2: Sbar_Q (mean d - d_v) / (std(d) + eps) (the z-score of
//             -l_v, l_v = d(v) - d(a_Q), does not depend on d(a_Q)); routed onto every
//             edge of a_Q -> v, a_Q the deepest state that is a strict ancestor of every
//             member.  In pre-order the lowest common ancestor of a set is that of its
//             smallest and largest index, so a_Q follows from the class's label L (its
//             smallest member) and its largest member h: walk up from L to the first
//             state whose subtree reaches h; that state is a_Q unless it is L itself
//             (then L is an ancestor of every member and a_Q = p(L)).
//             The edge entering x carries the sum of A_eff(j) over the members j of
//             its subtree whose a_Q lies strictly above x, summed in index order by one
//             warp per x (work = sum of the depths; deterministic order).
//   A_dual    A_cor + lambda_eff * routed A_eff                             (Sec. 4.5)

// Sums of the tree variant.  Class arrays are indexed by the class root, key arrays by
// the class of p(v) (n for the prompt root), both over n (+1) entries of the group.
struct TreeScratch {
  int* ccnt;        // [n]    |Q|
  int* csum;        // [n]    C_Q = sum of the members' c_own
  int* tsum;        // [n]    T_Q = sum of the members' t_own
  int* lsum;        // [n]    sum of the members' depths
  unsigned* l2;     // [n][2] sum of the squared depths, 2 x 13-bit chunks
  int* hi;          // [n]    largest member
  unsigned* ssum;   // [n][3] sum of S on the 2^-40 grid, 3 x 14-bit chunks
  int* aqd;         // [n]    depth of a_Q
  int* kcnt;        // [n+1]  edges per correctness group
  unsigned* ksum;   // [n+1][kSumWords]
  unsigned* kqh;    // [n+1][kSqhWords]
  unsigned* kql;    // [n+1][kSqlWords]
  float* aeff;      // [n]    A_eff of each state (0 unless |Q| >= 2)
  int* rdep;        // [n]    depth of a_Q of the state's class, or a large value without a route
  float* E;         // [n]    routed A_eff (over ccnt, written once the class sums are read)
  unsigned char* cov;  // [n] covered by a route (over csum)
  int* rootc;       // [1]    sum of the group's rewards
  int nzero;        // words from ccnt that start at zero (class and key sums, rootc)
};

constexpr int kTreeClassWords = 11;
constexpr int kTreeStateWords = 2;

__host__ __device__ constexpr size_t tree_scratch_words(int n) {
  return (size_t)kTreeClassWords * n + (size_t)kKeyWords * (n + 1) + 1 + (size_t)kTreeStateWords * n;
}
__host__ __device__ constexpr size_t tree_scratch_bytes(int n) { return al16(4 * tree_scratch_words(n)); }

// Carves a tree scratch of tree_scratch_bytes(n) bytes (4-byte aligned).
__device__ __forceinline__ TreeScratch tree_scratch(void* base, int n) {
  TreeScratch t;
  int* w = reinterpret_cast<int*>(base);
  t.ccnt = w;
  t.csum = w + n;
  t.tsum = w + 2 * n;
  t.lsum = w + 3 * n;
  t.l2 = reinterpret_cast<unsigned*>(w + 4 * n);
  t.hi = w + 6 * n;
  t.ssum = reinterpret_cast<unsigned*>(w + 7 * n);
  t.aqd = w + 10 * n;
  int* k = w + kTreeClassWords * n;
  t.kcnt = k;
  t.ksum = reinterpret_cast<unsigned*>(k + (n + 1));
  t.kqh = t.ksum + kSumWords * (n + 1);
  t.kql = t.kqh + kSqhWords * (n + 1);
  t.rootc = k + kKeyWords * (n + 1);
  t.aeff = reinterpret_cast<float*>(t.rootc + 1);
  t.rdep = reinterpret_cast<int*>(t.aeff + n);
  t.E = reinterpret_cast<float*>(t.ccnt);
  t.cov = reinterpret_cast<unsigned char*>(t.csum);
  t.nzero = kTreeClassWords * n + kKeyWords * (n + 1) + 1;
  return t;
}

// One group, nt cooperating threads (a multiple of 32; tid = thread index, lane = tid & 31
// must be the hardware lane), kPer * nt >= n.
//   lab    [n] union-find forest on entry (lab[x] <= x), class labels on exit
//   par    [n] local parent, -1 for the prompt root (par[x] < x)
//   dep    [n] depth (1 = child of the root);  end [n] local end of the subtree
//   cown, town [n] own terminal statistics;  nleaf = number of leaves (> 0)
//   sc     tree scratch (zeroed here), eta(i), out(...) and sync() as in group_advantages
template <int kPer, class IdxT, class Sync, class Eta, class Out>
__device__ __forceinline__ void group_advantages_tree(int n, int nleaf, int* lab, const IdxT* par, const IdxT* dep,
                                                      const IdxT* end, const IdxT* cown, const IdxT* town,
                                                      const TreeScratch& sc, const Params& p, int tid, int nt,
                                                      Sync sync, Eta eta, Out out) {
  const float w = p.w_hi, eps = p.eps_f;
  const float wl = p.w_lo;
  for (int i = tid; i < sc.nzero; i += nt) sc.ccnt[i] = 0;
  sync();
  // ---- phase A: class sums
  int lb[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    lb[k] = 0;
    if (i < n) {
      lb[k] = uf_find(lab, i);
      lab[i] = lb[k];
      const int d = dep[i];
      atomicAdd(&sc.ccnt[lb[k]], 1);
      atomicAdd(&sc.csum[lb[k]], (int)cown[i]);
      atomicAdd(&sc.tsum[lb[k]], (int)town[i]);
      atomicAdd(&sc.lsum[lb[k]], d);
      red_chunks<2, 13>(&sc.l2[2 * lb[k]], (unsigned long long)d * d);
      atomicMax(&sc.hi[lb[k]], i);
      if (par[i] < 0) atomicAdd(sc.rootc, (int)cown[i]);
    }
  }
  sync();
  // ---- phase A2: S, the parent's S, r_step; S and r into their sums; a_Q per class
  const float2 S_root = ff_div(make_float2((float)*sc.rootc, 0.f), make_float2((float)nleaf, 0.f));
  float S[kPer];
  int key[kPer];
  long long rf[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    S[k] = 0.f;
    key[k] = n;
    rf[k] = 0;
    if (i >= n) continue;
    const int L = lb[k], c = cown[i], t = town[i];
    // Eq. (combain) as a float pair: a class whose leaves share one reward gets S exactly 0 or 1
    const float2 Sv = score_ff(c, t, sc.csum[L], sc.tsum[L], w, wl);
    S[k] = Sv.x;
    const int pp = par[i];
    float2 Sp = S_root;
    if (pp >= 0) {
      const int Lp = lab[pp];  // the parent's S, recomputed alike
      Sp = score_ff(cown[pp], town[pp], sc.csum[Lp], sc.tsum[Lp], w, wl);
      key[k] = Lp;
    }
    rf[k] = step_reward_fixed(Sv, Sp, eta(i));
    red_chunks<3, 14>(&sc.ssum[3 * L],
                      (unsigned long long)(__float2ll_rn(Sv.x * 0x1p40f) + __float2ll_rn(Sv.y * 0x1p40f)));
    atomicAdd(&sc.kcnt[key[k]], 1);
    red_chunks<kSumWords, 18>(&sc.ksum[kSumWords * key[k]], (unsigned long long)(rf[k] + (1ll << 50)));
    if (i == L && sc.ccnt[L] >= 2) {
      const int h = sc.hi[L];
      int x = L;
      while (x >= 0 && end[x] <= h) x = par[x];
      sc.aqd[L] = x == L ? (int)dep[L] - 1 : (x < 0 ? 0 : (int)dep[x]);
    }
  }
  sync();
  // ---- phase B2: exact group means and squared deviations; A_eff per state
  float dv[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    dv[k] = 0.f;
    if (i >= n) continue;
    const int cnt = sc.kcnt[key[k]];
    const long long tot =
        (long long)(sum_chunks<kSumWords, 18>(&sc.ksum[kSumWords * key[k]]) - ((unsigned long long)cnt << 50));
    const long long mean = div_round(tot, cnt);
    dv[k] = (float)(rf[k] - mean) * 0x1p-50f;
    sq_add(&sc.kqh[kSqhWords * key[k]], &sc.kql[kSqlWords * key[k]], dv[k] * dv[k]);
    const int L = lb[k], Q = sc.ccnt[L], d = dep[i];
    float a = 0.f;
    int rd = 0x7fffffff;
    if (Q >= 2) {
      // Sbar_Q = sum S / Q; sum (d - mean)^2 = (Q sum d^2 - (sum d)^2) / Q (exact numerator);
      // A_eff = Sbar (mean d - d_v) / (sd + eps) = g (sum d - Q d_v), g = sum S / (Q^2 (sd + eps))
      const long long ls = sc.lsum[L];
      const float num = (float)((long long)Q * (long long)sum_chunks<2, 13>(&sc.l2[2 * L]) - ls * ls);
      const float var = __fdividef(num, (float)Q * (float)(Q - p.ddof));
      const float sd = var > 0.f ? var * rsqrtf(var) : 0.f;
      const float ssum = (float)sum_chunks<3, 14>(&sc.ssum[3 * L]) * 0x1p-40f;
      const float g = __fdividef(ssum, (float)Q * (float)Q * (sd + eps));
      a = g * (float)(ls - (long long)Q * d);
      rd = sc.aqd[L];
    }
    sc.aeff[i] = a;
    sc.rdep[i] = rd;
  }
  sync();
  // ---- phase B3: A_cor; phase C: routed A_eff (class sums are dead: E and cov overlay them)
  float acor[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    acor[k] = 0.f;
    const int K = key[k];
    if (tid + k * nt < n && sc.kcnt[K] >= 2) {
      const int cnt = sc.kcnt[K];
      const long long qh = (long long)sum_chunks<kSqhWords, 13>(&sc.kqh[kSqhWords * K]);
      const long long ql =
          (long long)(sum_chunks<kSqlWords, 14>(&sc.kql[kSqlWords * K]) - ((unsigned long long)cnt << 39));
      const float ss = (float)qh * 0x1p-36f + (float)ql * 0x1p-76f;
      const float var = __fdividef(ss, (float)(cnt - p.ddof));
      const float sd = var > 0.f ? var * rsqrtf(var) : 0.f;
      acor[k] = dv[k] * __fdividef(1.0f, sd + eps);
    }
  }
  {
    const int lane = tid & 31, nw = nt >> 5;
    for (int x = tid >> 5; x < n; x += nw) {
      const int dx = dep[x], e = end[x];
      float s = 0.f;
      bool c = false;
      for (int j = x + lane; j < e; j += 32) {
        if (sc.rdep[j] < dx) {
          s += sc.aeff[j];
          c = true;
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      c = __any_sync(0xffffffffu, c);
      if (lane == 0) {
        sc.E[x] = s;
        sc.cov[x] = c ? 1 : 0;
      }
    }
  }
  sync();
  const float lam = p.lambda_f;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) out(i, lb[k], S[k], acor[k], sc.E[i], fmaf(lam, sc.E[i], acor[k]), sc.cov[i]);
  }
  sync();
}

// ---------------------------------------------------------------------------------
// Exploration efficiency, Eq. (eq1): the share of a group's step tokens spent on
// steps from which a correct final answer can be reached.
//   tree reading   own(i): a correct leaf lies below state i (c_own > 0; in the chain
//                  layout the rollout is correct, the paper's chain case)
//   graph reading  reachable through direct edges and merged states: a class reaches a
//                  correct answer if one of its members does by the tree reading or a
//                  member's child's class does; the least fixed point, by rounds that mark
//                  the class of p(v) for every v whose class is marked (at most n + 1
//                  rounds: each round before the last marks a new class)
// lab      [n] final class labels
// mark     [n] scratch words; sums: 3 scratch 64-bit words
// par(i)   group-local parent of state i, or -1 for the prompt root
// len(i)   tokens of the edge entering state i
// any(f)   barrier over the nt threads that returns whether any thread passed true
// Writes eff_tree / eff_graph (NULL: skipped) from thread 0; results are exact token
// counts divided once.
template <class Own, class Par, class Len, class Sync, class Any>
__device__ __forceinline__ void group_efficiency(int n, const int* lab, int* mark, unsigned long long* sums, int tid,
                                                 int nt, Own own, Par par, Len len, Sync sync, Any any,
                                                 float* eff_tree, float* eff_graph) {
  const int lane = tid & 31;
  auto warp_sum = [&](unsigned long long x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
  };
  for (int i = tid; i < n; i += nt) mark[i] = 0;
  if (tid < 3) sums[tid] = 0ull;
  sync();
  unsigned long long tot = 0, good = 0;
  for (int i = tid; i < n; i += nt) {
    const unsigned long long l = (unsigned long long)(unsigned)len(i);
    tot += l;
    if (own(i)) {
      good += l;
      mark[lab[i]] = 1;  // every such class is in the fixed point (a correct leaf lies below)
    }
  }
  tot = warp_sum(tot);
  good = warp_sum(good);
  if (lane == 0) {
    atomicAdd(&sums[0], tot);
    atomicAdd(&sums[1], good);
  }
  sync();
  if (eff_graph) {
    bool changed = true;
    for (int round = 0; round <= n && changed; ++round) {
      bool ch = false;
      for (int i = tid; i < n; i += nt) {
        const int pp = par(i);
        if (pp >= 0 && mark[lab[i]] && !mark[lab[pp]]) {
          mark[lab[pp]] = 1;
          ch = true;
        }
      }
      changed = any(ch);
    }
    unsigned long long gg = 0;
    for (int i = tid; i < n; i += nt)
      if (mark[lab[i]]) gg += (unsigned long long)(unsigned)len(i);
    gg = warp_sum(gg);
    if (lane == 0) atomicAdd(&sums[2], gg);
    sync();
  }
  if (tid == 0) {
    const double t = (double)sums[0];
    if (eff_tree) *eff_tree = t > 0.0 ? (float)((double)sums[1] / t) : 0.f;
    if (eff_graph) *eff_graph = t > 0.0 ? (float)((double)sums[2] / t) : 0.f;
  }
  sync();
}

// ---------------------------------------------------------------------------------
// Next-layer budgets after layer `layer` of a branching group (Sec. 4.2: a path that
// reaches an existing equivalence class has its next-layer budget halved, keeping at
// least one continuation, and the saved budget goes to other paths; Algorithm S.1
// Stage 1 reallocates it to the active frontier states that are not redundant).
//   frontier   states of depth `layer` with active(i)
//   redundant  a frontier state whose class holds a state registered before it: one of
//              an earlier layer, or one of the same layer with a smaller index
//   budget     b_next for a non-redundant frontier state, max(1, b_next / 2) for a
//              redundant one, 0 elsewhere; the saved budget S (redundant count x
//              (b_next - max(1, b_next / 2))) is split over the k non-redundant frontier
//              states: S / k each and one more for the first S % k of them by index
// lab    [n] union-find forest of the classes (flattened here)
// first  [n] scratch; cnt: 2 scratch words; wt: one scratch word per warp of the nt threads
// out(i, label, budget) is called once per state.
template <class IdxT, class Active, class Sync, class Out>
__device__ __forceinline__ void group_budget(int n, int* lab, const IdxT* dep, int layer, int b_next, int* first,
                                             int* cnt, int* wt, int tid, int nt, Active active, Sync sync, Out out) {
  const int lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < n; i += nt) {
    lab[i] = uf_find(lab, i);  // concurrent finds only ever write roots
    first[i] = 0x7FFFFFFF;
  }
  if (tid < 2) cnt[tid] = 0;
  sync();
  // registration order: layer, then index within the layer (n <= 4096 < 2^13)
  auto key = [&](int i) { return ((int)dep[i] << 13) | i; };
  for (int i = tid; i < n; i += nt) atomicMin(&first[lab[i]], key(i));
  sync();
  auto frontier = [&](int i) { return (int)dep[i] == layer && active(i); };
  for (int base = 0; base < n; base += nt) {
    const int i = base + tid;
    const bool f = i < n && frontier(i);
    const bool red = f && first[lab[i]] != key(i);
    const uint32_t mr = __ballot_sync(0xffffffffu, red), mk = __ballot_sync(0xffffffffu, f && !red);
    if (lane == 0) {
      if (mr) atomicAdd(&cnt[0], __popc(mr));
      if (mk) atomicAdd(&cnt[1], __popc(mk));
    }
  }
  sync();
  const int halved = b_next / 2 > 1 ? b_next / 2 : 1;
  const long long saved = (long long)cnt[0] * (b_next - halved);
  const int k = cnt[1];
  const long long share = k ? saved / k : 0, extra = k ? saved % k : 0;
  int carry = 0;  // non-redundant frontier states before this chunk
  for (int base = 0; base < n; base += nt) {
    const int i = base + tid;
    const bool f = i < n && frontier(i);
    const bool red = f && first[lab[i]] != key(i);
    const uint32_t m = __ballot_sync(0xffffffffu, f && !red);
    if (lane == 0) wt[warp] = __popc(m);
    sync();
    int before = 0, total = 0;
    for (int w = 0; w < nt / 32; ++w) {
      before += w < warp ? wt[w] : 0;
      total += wt[w];
    }
    if (i < n) {
      const int rank = carry + before + __popc(m & ((1u << lane) - 1u));
      const long long bud = !f ? 0 : (red ? halved : b_next + share + (rank < extra ? 1 : 0));
      out(i, lab[i], (int)bud);
    }
    carry += total;
    sync();
  }
}

}  // namespace gpo
