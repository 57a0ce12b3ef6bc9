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
// in fp64.  Group sums go through exact two-word fixed-point accumulators
// (resolution 2^-76) in shared-memory int64 atomics, so the results do not
// depend on the order in which threads add.
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

// Scratch bytes group_advantages needs for a group of n states: the largest of
// its three phases (class sums 24 B/class, correctness-group sums 28 B/group,
// route sums 9 B/state).
__host__ __device__ constexpr size_t group_scratch_bytes(int n) {
  return al16(28 * (size_t)(n + 1) + 32);
}

// One group, `nt` cooperating threads (thread index tid), kPer * nt >= n.
//   lab     [n] shared union-find forest on entry, class labels (local index of
//           the smallest member) on exit
//   roll    [n] rollout of each state, local to the group (0..nr-1)
//   dep     [n] depth of each state (1 = first step)
//   rstart  [nr+1] local state offsets of the rollouts
//   rew     [nr] rewards
//   X       shared scratch of group_scratch_bytes(n), 16-byte aligned
//   eta(i)  eta(p(v), v) of local state i (fp32, already clamped at 0)
//   out(i, label, S, acor, E, dual, mask) is called once per state by its owner
//   sync()  barrier over the nt threads
//
// Precision: fp32 arithmetic with exact integer class sums and an exact
// fixed-point group mean (the one quantity whose rounding the standardisation
// amplifies).  Per-class and per-group constants are computed once by one
// thread.  Sums go through integer atomics, so results do not depend on the
// order in which threads add.
template <int kPer, class Sync, class Eta, class Out>
__device__ __forceinline__ void group_advantages(int n, int nr, int* lab, const int* roll, const int* dep,
                                                 const int* rstart, const uint8_t* rew, unsigned char* X,
                                                 const Params& p, int tid, int nt, Sync sync, Eta eta, Out out) {
  const float w = (float)p.w, eps = (float)p.eps;
  // ---- phase A: class sums C_Q (rewards), |Q|, sum l, sum l^2
  int* ccnt = reinterpret_cast<int*>(X);
  int* csum = ccnt + n;
  int* lsum = csum + n;
  long long* l2 = reinterpret_cast<long long*>(X + al16(12 * (size_t)n));
  float* cg = reinterpret_cast<float*>(l2 + n);    // efficiency factor of the class
  __shared__ int s_rootc;

  for (int i = tid; i < n; i += nt) {
    ccnt[i] = csum[i] = lsum[i] = 0;
    l2[i] = 0;
  }
  if (tid == 0) s_rootc = 0;
  int lb[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    lb[k] = i < n ? uf_find(lab, i) : 0;
  }
  sync();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) {
      lab[i] = lb[k];
      const int d = dep[i];
      atomicAdd(&ccnt[lb[k]], 1);
      atomicAdd(&csum[lb[k]], (int)rew[roll[i]]);
      atomicAdd(&lsum[lb[k]], d);
      atomicAdd(reinterpret_cast<unsigned long long*>(&l2[lb[k]]), (unsigned long long)((long long)d * d));
    }
  }
  for (int r = tid; r < nr; r += nt) atomicAdd(&s_rootc, (int)rew[r]);
  sync();
  for (int L = tid; L < n; L += nt) {  // class constants, once per class
    const int Q = ccnt[L];
    if (Q == 0) continue;
    float g = 0.f;
    if (Q >= 2) {
      // Sbar_Q = mean of S over Q = C_Q / |Q| (every member has t_own = 1);
      // sum (l - mean)^2 = (Q sum l^2 - (sum l)^2) / Q with an exact integer numerator;
      // A_eff(v) = Sbar (mean l - l_v) / (sd + eps) = g (sum l - Q l_v)
      const long long ls = lsum[L];
      const float ss = (float)((long long)Q * l2[L] - ls * ls) / (float)Q;
      const float sd = sqrtf(ss / (float)(Q - p.ddof));
      g = ((float)csum[L] / (float)Q) / ((sd + eps) * (float)Q);
    }
    cg[L] = g;
  }
  sync();
  const float S_root = (float)s_rootc / (float)nr;
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
    const int L = lb[k], Q = ccnt[L], d = dep[i], c = rew[roll[i]];
    // Eq. (combain): (c_own + w sum_{q != v} c_own(q)) / (t_own + w sum_{q != v} t_own(q)), t_own = 1.
    // Correctly rounded, with numerator and denominator formed by the same fma, so that a
    // class whose members share one reward gets S exactly 0 or 1 (as the exact formula).
    S[k] = fmaf(w, (float)(csum[L] - c), (float)c) / fmaf(w, (float)(Q - 1), 1.0f);
    if (Q >= 2) {
      route_end[k] = true;
      aeff[k] = cg[L] * (float)(lsum[L] - Q * d);
    }
    float Sp;
    if (d == 1) {
      Sp = S_root;
    } else {
      const int Lp = lab[i - 1];  // parent: the previous state of the same rollout (same reward c)
      Sp = fmaf(w, (float)(csum[Lp] - c), (float)c) / fmaf(w, (float)(ccnt[Lp] - 1), 1.0f);
      key[k] = Lp;
    }
    r[k] = (S[k] - Sp) * (1.0f - eta(i));
  }
  sync();  // phase A scratch no longer read

  // ---- phase B: correctness groups, key = class of p(v), n = the prompt root
  int* kcnt = reinterpret_cast<int*>(X);
  long long* ksum = reinterpret_cast<long long*>(X + al16(4 * (size_t)(n + 1)));  // becomes the mean
  long long* kq_hi = ksum + (n + 1);
  long long* kq_lo = kq_hi + (n + 1);
  float* kinv = reinterpret_cast<float*>(kq_hi);  // 1 / (sd + eps), written over kq_hi after use
  for (int i = tid; i <= n; i += nt) {
    kcnt[i] = 0;
    ksum[i] = kq_hi[i] = kq_lo[i] = 0;
  }
  sync();
  long long rf[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    rf[k] = 0;
    if (tid + k * nt < n) {
      // |r| <= 1 and a group holds at most 4096 edges: a 2^50 fixed point cannot overflow
      rf[k] = __float2ll_rn(r[k] * 0x1p50f);
      atomicAdd(&kcnt[key[k]], 1);
      atomicAdd(reinterpret_cast<unsigned long long*>(&ksum[key[k]]), (unsigned long long)rf[k]);
    }
  }
  sync();
  for (int K = tid; K <= n; K += nt)
    if (kcnt[K] > 0) ksum[K] = div_round(ksum[K], kcnt[K]);  // exact mean on the 2^-50 grid
  sync();
  float dv[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    dv[k] = 0.f;
    if (tid + k * nt < n) {
      dv[k] = (float)(rf[k] - ksum[key[k]]) * 0x1p-50f;
      fx_add32(&kq_hi[key[k]], &kq_lo[key[k]], dv[k] * dv[k]);
    }
  }
  sync();
  for (int K = tid; K <= n; K += nt) {
    const int cnt = kcnt[K];
    float inv = 0.f;  // groups of one edge get no advantage
    if (cnt >= 2) {
      const float ss = (float)kq_hi[K] * 0x1p-36f + (float)kq_lo[K] * 0x1p-76f;  // sum (r - mean)^2
      inv = 1.0f / (sqrtf(ss / (float)(cnt - p.ddof)) + eps);
    }
    kinv[2 * K] = inv;  // kq_hi[K]'s first word; only this thread touches kq_*[K]
  }
  sync();
  float acor[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) acor[k] = (tid + k * nt < n) ? dv[k] * kinv[2 * key[k]] : 0.f;
  sync();  // phase B scratch no longer read

  // ---- phase C: every edge on root -> v receives A_eff(v) (suffix sums per rollout)
  float* s_aeff = reinterpret_cast<float*>(X);
  float* s_E = s_aeff + n;
  unsigned char* s_cov = reinterpret_cast<unsigned char*>(s_E + n);
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) {
      s_aeff[i] = aeff[k];
      s_cov[i] = route_end[k] ? 1 : 0;
    }
  }
  sync();
  for (int rr = tid; rr < nr; rr += nt) {
    float acc = 0.f;
    unsigned char cov = 0;
    for (int i = rstart[rr + 1] - 1; i >= rstart[rr]; --i) {
      acc += s_aeff[i];
      cov |= s_cov[i];
      s_E[i] = acc;
      s_cov[i] = cov;
    }
  }
  sync();
  const float lam = (float)p.lambda_eff;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) out(i, lb[k], S[k], acor[k], s_E[i], fmaf(lam, s_E[i], acor[k]), s_cov[i]);
  }
  sync();
}

}  // namespace gpo
