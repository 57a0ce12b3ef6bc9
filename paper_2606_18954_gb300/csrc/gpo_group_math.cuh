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

// x in [-2^12, 2^12]: hi = round(x 2^36), lo = round((x 2^36 - hi) 2^40).
__device__ __forceinline__ void fx_add(long long* hi, long long* lo, double x) {
  const double X = x * 0x1p36;
  const double h = rint(X);
  const long long hl = (long long)h;
  const long long ll = llrint((X - h) * 0x1p40);
  atomicAdd(reinterpret_cast<unsigned long long*>(hi), (unsigned long long)hl);
  atomicAdd(reinterpret_cast<unsigned long long*>(lo), (unsigned long long)ll);
}

__device__ __forceinline__ double fx_get(const long long* hi, const long long* lo) {
  return (double)*((volatile const long long*)hi) * 0x1p-36 + (double)*((volatile const long long*)lo) * 0x1p-76;
}

__host__ __device__ constexpr size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

// Scratch bytes group_advantages needs for a group of n states.
__host__ __device__ constexpr size_t group_scratch_bytes(int n) {
  return al16(((al16(3 * sizeof(int) * (size_t)n) + 3 * sizeof(long long) * (size_t)n) >
               (al16(sizeof(int) * (size_t)(n + 1)) + 4 * sizeof(long long) * (size_t)(n + 1)))
                  ? ((al16(3 * sizeof(int) * (size_t)n) + 3 * sizeof(long long) * (size_t)n) >
                             (2 * sizeof(double) * (size_t)n + (size_t)n)
                         ? al16(3 * sizeof(int) * (size_t)n) + 3 * sizeof(long long) * (size_t)n
                         : 2 * sizeof(double) * (size_t)n + (size_t)n)
                  : ((al16(sizeof(int) * (size_t)(n + 1)) + 4 * sizeof(long long) * (size_t)(n + 1)) >
                             (2 * sizeof(double) * (size_t)n + (size_t)n)
                         ? al16(sizeof(int) * (size_t)(n + 1)) + 4 * sizeof(long long) * (size_t)(n + 1)
                         : 2 * sizeof(double) * (size_t)n + (size_t)n));
}

__device__ __forceinline__ double pooled_score(int c, int C, int Q, double w) {
  // (c_own + w sum_{q != v} c_own(q)) / (t_own + w sum_{q != v} t_own(q)), t_own = 1
  return ((double)c + w * (double)(C - c)) / (1.0 + w * (double)(Q - 1));
}

// One group, `nt` cooperating threads (thread index tid), kPer * nt >= n.
//   lab     [n] shared union-find forest on entry, class labels (local index of
//           the smallest member) on exit
//   roll    [n] rollout of each state, local to the group (0..nr-1)
//   dep     [n] depth of each state (1 = first step)
//   rstart  [nr+1] local state offsets of the rollouts
//   rew     [nr] rewards
//   X       shared scratch of group_scratch_bytes(n)
//   eta(i)  eta(p(v), v) of local state i (fp64, already clamped at 0)
//   out(i, label, S, acor, E, dual, mask) is called once per state by its owner
//   sync()  barrier over the nt threads
template <int kPer, class Sync, class Eta, class Out>
__device__ __forceinline__ void group_advantages(int n, int nr, int* lab, const int* roll, const int* dep,
                                                 const int* rstart, const uint8_t* rew, unsigned char* X,
                                                 const Params& p, int tid, int nt, Sync sync, Eta eta, Out out) {
  int* ccnt = reinterpret_cast<int*>(X);
  int* csum = ccnt + n;
  int* lsum = csum + n;
  long long* l2sum = reinterpret_cast<long long*>(X + al16(3 * sizeof(int) * (size_t)n));
  long long* sb_hi = l2sum + n;
  long long* sb_lo = sb_hi + n;
  __shared__ int s_rootc;

  for (int i = tid; i < n; i += nt) {
    ccnt[i] = csum[i] = lsum[i] = 0;
    l2sum[i] = sb_hi[i] = sb_lo[i] = 0;
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
    if (i < n) lab[i] = lb[k];
  }
  for (int r = tid; r < nr; r += nt) atomicAdd(&s_rootc, (int)rew[r]);
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) {
      const int d = dep[i];
      atomicAdd(&ccnt[lb[k]], 1);
      atomicAdd(&csum[lb[k]], (int)rew[roll[i]]);
      atomicAdd(&lsum[lb[k]], d);
      atomicAdd(reinterpret_cast<unsigned long long*>(&l2sum[lb[k]]), (unsigned long long)((long long)d * d));
    }
  }
  sync();
  const double S_root = (double)s_rootc / (double)nr;
  double S[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    S[k] = 0.0;
    if (i < n) {
      S[k] = pooled_score(rew[roll[i]], csum[lb[k]], ccnt[lb[k]], p.w);
      fx_add(&sb_hi[lb[k]], &sb_lo[lb[k]], S[k]);
    }
  }
  sync();
  double aeff[kPer], r[kPer];
  int key[kPer];
  bool route_end[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    aeff[k] = r[k] = 0.0;
    key[k] = n;
    route_end[k] = false;
    if (i >= n) continue;
    const int L = lb[k];
    const int Q = ccnt[L];
    const int d = dep[i];
    if (Q >= 2) {
      route_end[k] = true;
      const double sbar = fx_get(&sb_hi[L], &sb_lo[L]) / (double)Q;
      const long long ls = lsum[L], l2 = l2sum[L];
      const double mean_l = (double)ls / (double)Q;
      // sum (l - mean)^2 = (Q sum l^2 - (sum l)^2) / Q, exact integer numerator
      const double ss = (double)((long long)Q * l2 - ls * ls) / (double)Q;
      const double sd = sqrt(ss / (double)(Q - p.ddof));
      aeff[k] = sbar * (mean_l - (double)d) / (sd + p.eps);
    }
    double Sp;
    if (d == 1) {
      Sp = S_root;
    } else {
      const int Lp = lab[i - 1];
      Sp = pooled_score(rew[roll[i]], csum[Lp], ccnt[Lp], p.w);  // parent: same rollout, same reward
      key[k] = Lp;
    }
    r[k] = (S[k] - Sp) * (1.0 - eta(i));
  }
  sync();  // class accumulators no longer read: X is reused

  int* gcnt = reinterpret_cast<int*>(X);
  long long* gs_hi = reinterpret_cast<long long*>(X + al16(sizeof(int) * (size_t)(n + 1)));
  long long* gs_lo = gs_hi + (n + 1);
  long long* gq_hi = gs_lo + (n + 1);
  long long* gq_lo = gq_hi + (n + 1);
  for (int i = tid; i <= n; i += nt) {
    gcnt[i] = 0;
    gs_hi[i] = gs_lo[i] = gq_hi[i] = gq_lo[i] = 0;
  }
  sync();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    if (tid + k * nt < n) {
      atomicAdd(&gcnt[key[k]], 1);
      fx_add(&gs_hi[key[k]], &gs_lo[key[k]], r[k]);
    }
  }
  sync();
  double mean[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    mean[k] = 0.0;
    if (tid + k * nt < n) {
      mean[k] = fx_get(&gs_hi[key[k]], &gs_lo[key[k]]) / (double)gcnt[key[k]];
      const double dv = r[k] - mean[k];
      fx_add(&gq_hi[key[k]], &gq_lo[key[k]], dv * dv);
    }
  }
  sync();
  double acor[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    acor[k] = 0.0;
    if (tid + k * nt < n) {
      const int K = gcnt[key[k]];
      if (K >= 2) {
        const double sd = sqrt(fx_get(&gq_hi[key[k]], &gq_lo[key[k]]) / (double)(K - p.ddof));
        acor[k] = (r[k] - mean[k]) / (sd + p.eps);
      }
    }
  }
  sync();  // X reused again

  double* s_aeff = reinterpret_cast<double*>(X);
  double* s_E = s_aeff + n;
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
  // every edge on root -> v receives A_eff(v): suffix sums along each rollout
  for (int rr = tid; rr < nr; rr += nt) {
    double acc = 0.0;
    unsigned char cov = 0;
    for (int i = rstart[rr + 1] - 1; i >= rstart[rr]; --i) {
      acc += s_aeff[i];
      cov |= s_cov[i];
      s_E[i] = acc;
      s_cov[i] = cov;
    }
  }
  sync();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) out(i, lb[k], S[k], acor[k], s_E[i], acor[k] + p.lambda_eff * s_E[i], s_cov[i]);
  }
  sync();
}

}  // namespace gpo
