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

// Exact, order-independent sum of non-negative fp32 values below 2^26: each value
// is split into a 2^-36-grid part and a 2^-76-grid remainder (both exact in
// fp32) that go into two int64 accumulators.
__device__ __forceinline__ void fx_add32(long long* hi, long long* lo, float x) {
  const float X = x * 0x1p36f;
  const float h = rintf(X);
  const long long hl = __float2ll_rn(h);
  const long long ll = __float2ll_rn((X - h) * 0x1p40f);
  atomicAdd(reinterpret_cast<unsigned long long*>(hi), (unsigned long long)hl);
  atomicAdd(reinterpret_cast<unsigned long long*>(lo), (unsigned long long)ll);
}

// Rounded quotient of an int64 by a positive int.
__device__ __forceinline__ long long div_round(long long a, int k) {
  long long q = a / k, rem = a - q * k;
  if (2 * (rem < 0 ? -rem : rem) >= k) q += (a < 0 ? -1 : 1);
  return q;
}

__host__ __device__ constexpr size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

// Scratch arrays of group_advantages.  Class sums are indexed by the class root
// (a local state index), correctness-group sums by the key (the class of the
// parent, or n for the prompt root); the route sums reuse the class arrays.
struct GroupScratch {
  int* ccnt;            // [n]   |Q|
  int* csum;            // [n]   C_Q = sum of the members' rewards
  int* lsum;            // [n]   sum of the members' depths
  long long* l2;        // [n]   sum of the squared depths
  int* kcnt;            // [n+1] edges per correctness group
  long long* ksum;      // [n+1] sum of r on the 2^-50 grid
  long long* kq_hi;     // [n+1] sum of (r - mean)^2, 2^-36 grid part
  long long* kq_lo;     // [n+1] and 2^-76 grid remainder
  float* aeff;          // [n]   A_eff of each route end (over ccnt / csum)
  float* E;             // [n]   routed A_eff (over lsum)
  unsigned char* cov;   // [n]   covered by a route (over l2)
  int* rootc;           // [1]   sum of the group's rewards
};

// Separate layout: class and key arrays side by side, for callers that zero
// them ahead of time (group_scratch_zero); bytes for a group of up to n states.
__host__ __device__ constexpr size_t group_scratch_sep_bytes(int n) {
  return al16(12 * (size_t)n) + al16(8 * (size_t)n) + al16(4 * (size_t)(n + 1)) + 3 * al16(8 * (size_t)(n + 1)) + 16;
}

__device__ __forceinline__ GroupScratch group_scratch_sep(unsigned char* X, int n) {
  GroupScratch g;
  g.ccnt = reinterpret_cast<int*>(X);
  g.csum = g.ccnt + n;
  g.lsum = g.csum + n;
  g.l2 = reinterpret_cast<long long*>(X + al16(12 * (size_t)n));
  unsigned char* k = X + al16(12 * (size_t)n) + al16(8 * (size_t)n);
  g.kcnt = reinterpret_cast<int*>(k);
  g.ksum = reinterpret_cast<long long*>(k + al16(4 * (size_t)(n + 1)));
  g.kq_hi = g.ksum + (n + 1);
  g.kq_lo = g.kq_hi + (n + 1);
  g.rootc = reinterpret_cast<int*>(k + al16(4 * (size_t)(n + 1)) + 3 * al16(8 * (size_t)(n + 1)));
  g.aeff = reinterpret_cast<float*>(g.ccnt);
  g.E = reinterpret_cast<float*>(g.lsum);
  g.cov = reinterpret_cast<unsigned char*>(g.l2);
  return g;
}

// Zero the sums of a separate-layout scratch (before the barrier that precedes
// group_advantages<kPer, true>).
__device__ __forceinline__ void group_scratch_zero(const GroupScratch& g, int n, int tid, int nt) {
  for (int i = tid; i < n; i += nt) {
    g.ccnt[i] = g.csum[i] = g.lsum[i] = 0;
    g.l2[i] = 0;
  }
  for (int i = tid; i <= n; i += nt) {
    g.kcnt[i] = 0;
    g.ksum[i] = g.kq_hi[i] = g.kq_lo[i] = 0;
  }
  if (tid == 0) *g.rootc = 0;
}

// Shared layout: the class, key and route arrays overlay one region (the
// largest is the key sums, 28 B per key), for large groups; group_advantages
// zeroes each in turn, at the cost of extra barriers.
__host__ __device__ constexpr size_t group_scratch_bytes(int n) {
  return al16(28 * (size_t)(n + 1) + 32);
}

__device__ __forceinline__ GroupScratch group_scratch_shared(unsigned char* X, int n, int* rootc) {
  GroupScratch g;
  g.ccnt = reinterpret_cast<int*>(X);
  g.csum = g.ccnt + n;
  g.lsum = g.csum + n;
  g.l2 = reinterpret_cast<long long*>(X + al16(12 * (size_t)n));
  g.kcnt = reinterpret_cast<int*>(X);
  g.ksum = reinterpret_cast<long long*>(X + al16(4 * (size_t)(n + 1)));
  g.kq_hi = g.ksum + (n + 1);
  g.kq_lo = g.kq_hi + (n + 1);
  g.aeff = reinterpret_cast<float*>(X);
  g.E = g.aeff + n;
  g.cov = reinterpret_cast<unsigned char*>(g.E + n);
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
//   eta(i)  eta(p(v), v) of local state i (fp32, already clamped at 0)
//   out(i, label, S, acor, E, dual, mask) is called once per state by its owner
//   sync()  barrier over the nt threads
//
// Precision: fp32 arithmetic with exact integer class sums and an exact
// fixed-point group mean (the one quantity whose rounding the standardisation
// amplifies).  Per-class and per-group constants are recomputed by every state
// that needs them (same operands, same operations, so the same value), which
// saves a barrier per constant.  Sums go through integer atomics, so results do
// not depend on the order in which threads add.
template <int kPer, bool kZeroed, class Sync, class Eta, class Out>
__device__ __forceinline__ void group_advantages(int n, int nr, int* lab, const int* roll, const int* dep,
                                                 const int* rstart, const uint8_t* rew, const GroupScratch& sc,
                                                 const Params& p, int tid, int nt, Sync sync, Eta eta, Out out) {
  const float w = (float)p.w, eps = (float)p.eps;
  // ---- phase A: class sums C_Q (rewards), |Q|, sum l, sum l^2
  if (!kZeroed) {
    for (int i = tid; i < n; i += nt) {
      sc.ccnt[i] = sc.csum[i] = sc.lsum[i] = 0;
      sc.l2[i] = 0;
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
      atomicAdd(reinterpret_cast<unsigned long long*>(&sc.l2[lb[k]]), (unsigned long long)((long long)d * d));
    }
  }
  for (int r = tid; r < nr; r += nt) atomicAdd(sc.rootc, (int)rew[r]);
  sync();
  const float S_root = (float)*sc.rootc / (float)nr;
  float S[kPer], aeff[kPer], r[kPer];
  int key[kPer];
  bool route_end[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    S[k] = aeff[k] = r[k] = 0.f;
    key[k] = n;
    route_end[k] = false;
    if (i >= n) continue;
    const int L = lb[k], Q = sc.ccnt[L], d = dep[i], c = rew[roll[i]];
    // Eq. (combain): (c_own + w sum_{q != v} c_own(q)) / (t_own + w sum_{q != v} t_own(q)), t_own = 1.
    // Correctly rounded, with numerator and denominator formed by the same fma, so that a
    // class whose members share one reward gets S exactly 0 or 1 (as the exact formula).
    S[k] = fmaf(w, (float)(sc.csum[L] - c), (float)c) / fmaf(w, (float)(Q - 1), 1.0f);
    if (Q >= 2) {
      // Sbar_Q = mean of S over Q = C_Q / |Q| (every member has t_own = 1);
      // sum (l - mean)^2 = (Q sum l^2 - (sum l)^2) / Q with an exact integer numerator;
      // A_eff(v) = Sbar (mean l - l_v) / (sd + eps) = g (sum l - Q l_v)
      const long long ls = sc.lsum[L];
      const float ss = (float)((long long)Q * sc.l2[L] - ls * ls) / (float)Q;
      const float sd = sqrtf(ss / (float)(Q - p.ddof));
      const float g = ((float)sc.csum[L] / (float)Q) / ((sd + eps) * (float)Q);
      route_end[k] = true;
      aeff[k] = g * (float)(sc.lsum[L] - Q * d);
    }
    float Sp;
    if (d == 1) {
      Sp = S_root;
    } else {
      const int Lp = lab[i - 1];  // parent: the previous state of the same rollout (same reward c)
      Sp = fmaf(w, (float)(sc.csum[Lp] - c), (float)c) / fmaf(w, (float)(sc.ccnt[Lp] - 1), 1.0f);
      key[k] = Lp;
    }
    r[k] = (S[k] - Sp) * (1.0f - eta(i));
  }

  // ---- phase B: correctness groups, key = class of p(v), n = the prompt root
  if (!kZeroed) {
    sync();  // class sums no longer read
    for (int i = tid; i <= n; i += nt) {
      sc.kcnt[i] = 0;
      sc.ksum[i] = sc.kq_hi[i] = sc.kq_lo[i] = 0;
    }
    sync();
  }
  long long rf[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    rf[k] = 0;
    if (tid + k * nt < n) {
      // |r| <= 1 and a group holds at most 4096 edges: a 2^50 fixed point cannot overflow
      rf[k] = __float2ll_rn(r[k] * 0x1p50f);
      atomicAdd(&sc.kcnt[key[k]], 1);
      atomicAdd(reinterpret_cast<unsigned long long*>(&sc.ksum[key[k]]), (unsigned long long)rf[k]);
    }
  }
  sync();
  float dv[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    dv[k] = 0.f;
    if (tid + k * nt < n) {
      const long long mean = div_round(sc.ksum[key[k]], sc.kcnt[key[k]]);  // exact mean on the 2^-50 grid
      dv[k] = (float)(rf[k] - mean) * 0x1p-50f;
      fx_add32(&sc.kq_hi[key[k]], &sc.kq_lo[key[k]], dv[k] * dv[k]);
    }
  }
  sync();
  float acor[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    acor[k] = 0.f;
    const int K = key[k], cnt = sc.kcnt[K];
    if (tid + k * nt < n && cnt >= 2) {  // groups of one edge get no advantage
      const float ss = (float)sc.kq_hi[K] * 0x1p-36f + (float)sc.kq_lo[K] * 0x1p-76f;  // sum (r - mean)^2
      acor[k] = dv[k] * (1.0f / (sqrtf(ss / (float)(cnt - p.ddof)) + eps));
    }
  }

  // ---- phase C: every edge on root -> v receives A_eff(v) (suffix sums per rollout)
  if (!kZeroed) sync();  // key sums no longer read (the route arrays overlay them)
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) {
      sc.aeff[i] = aeff[k];
      sc.cov[i] = route_end[k] ? 1 : 0;
    }
  }
  sync();
  for (int rr = tid; rr < nr; rr += nt) {
    float acc = 0.f;
    unsigned char cov = 0;
    for (int i = rstart[rr + 1] - 1; i >= rstart[rr]; --i) {
      acc += sc.aeff[i];
      cov |= sc.cov[i];
      sc.E[i] = acc;
      sc.cov[i] = cov;
    }
  }
  sync();
  const float lam = (float)p.lambda_eff;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) out(i, lb[k], S[k], acor[k], sc.E[i], fmaf(lam, sc.E[i], acor[k]), sc.cov[i]);
  }
  sync();
}

}  // namespace gpo
