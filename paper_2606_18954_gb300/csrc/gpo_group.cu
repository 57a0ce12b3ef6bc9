// Per prompt group (one CTA): equivalence classes, graph reward and
// dual-group advantage of every generated edge.
//
//   classes   union of the similarity items' spanning forests in shared
//             memory; label = smallest state index (Sec. 4.2, Alg. S.1)
//   S(v)      Eq. (combain): chain layout gives c_own(v) = R of v's rollout and
//             t_own(v) = 1, so S(v) = (c + w (C_Q - c)) / (1 + w (|Q| - 1));
//             S(root) = sum R / R_g                                (Sec. 4.3)
//   r_step    (S(v) - S(p(v))) (1 - max(0, cos(z_p(v), z_v)))    (Sec. 4.3)
//   A_cor     edges (p(v), v) grouped by the class of p(v) (E_cor(u) is the same
//             set for every u in Q(u)); groups of one edge get 0      (Sec. 4.4)
//   A_eff     per class with |Q| >= 2: a_Q is the prompt root (members lie in
//             at least two rollouts), l_v = depth, Sbar_Q = mean S over Q,
//             A_eff(v) = Sbar_Q (-l_v - mean(-l)) / (std(-l) + eps); every edge
//             on root -> v receives A_eff(v) (sum over routes)      (Sec. 4.4)
//   A_dual    A_cor + lambda_eff * routed A_eff                      (Sec. 4.5)
//
// Arithmetic is fp64.  Group sums use an exact two-word fixed-point
// accumulator (resolution 2^-76) in shared-memory int64 atomics, so the result
// does not depend on the order in which threads add.
#include "gpo_internal.cuh"

namespace gpo {

namespace {

constexpr int kPer = 4;  // states per thread (blockDim >= n / kPer)

__device__ __forceinline__ int gfind(const int* p, int x) {
  const volatile int* vp = p;
  while (true) {
    const int y = vp[x];
    if (y == x) return x;
    x = y;
  }
}

__device__ __forceinline__ void gunion(int* p, int a, int b) {
  while (true) {
    a = gfind(p, a);
    b = gfind(p, b);
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

__host__ __device__ inline size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

// Shared memory: labels [n] int, then one region reused by three phases.
__host__ __device__ inline size_t region_bytes(int n) {
  const size_t ph1 = al16(3 * sizeof(int) * (size_t)n) + 3 * sizeof(long long) * (size_t)n;
  const size_t ph2 = al16(sizeof(int) * (size_t)(n + 1)) + 4 * sizeof(long long) * (size_t)(n + 1);
  const size_t ph3 = 2 * sizeof(double) * (size_t)n + (size_t)n;
  size_t m = ph1 > ph2 ? ph1 : ph2;
  return m > ph3 ? m : ph3;
}

__host__ __device__ inline size_t group_smem(int n) { return al16(sizeof(int) * (size_t)n) + region_bytes(n) + 64; }

__device__ __forceinline__ double pooled_score(int c, int C, int Q, double w) {
  // (c_own + w * sum_{q != v} c_own(q)) / (t_own + w * sum_{q != v} t_own(q)), t_own = 1
  return ((double)c + w * (double)(C - c)) / (1.0 + w * (double)(Q - 1));
}

__global__ void __launch_bounds__(1024) groups_kernel(gpo_batch b, gpo_outputs o, Sizes sz, Ws ws, Params p) {
  extern __shared__ __align__(16) unsigned char sm[];
  __shared__ int s_rootc;
  uint32_t* st = ws.status;
  if (aborted(st)) return;
  const int g = blockIdx.x;
  const GroupInfo gi = ws.groups[g];
  const int n = gi.n, s0 = gi.s0, nt = blockDim.x, tid = threadIdx.x;
  if (gi.nr == 0 || n == 0) return;

  int* lab = reinterpret_cast<int*>(sm);
  unsigned char* X = sm + al16(sizeof(int) * (size_t)n);
  // phase 1: class accumulators
  int* ccnt = reinterpret_cast<int*>(X);
  int* csum = ccnt + n;
  int* lsum = csum + n;
  long long* l2sum = reinterpret_cast<long long*>(X + al16(3 * sizeof(int) * (size_t)n));
  long long* sb_hi = l2sum + n;
  long long* sb_lo = sb_hi + n;

  for (int i = tid; i < n; i += nt) {
    lab[i] = i;
    ccnt[i] = csum[i] = lsum[i] = 0;
    l2sum[i] = sb_hi[i] = sb_lo[i] = 0;
  }
  if (tid == 0) s_rootc = 0;
  __syncthreads();

  // ---- equivalence classes from the items' spanning forests
  const int it0 = ws.group_items[g], it1 = ws.group_items[g + 1];
  for (int it = it0; it < it1; ++it) {
    const int ne = ws.edge_count[it];
    const int2* E = ws.edges + (size_t)it * kEdgeCap;
    for (int e = tid; e < ne; e += nt) {
      const int2 uv = E[e];
      const int u = uv.x - s0, v = uv.y - s0;
      if ((unsigned)u < (unsigned)n && (unsigned)v < (unsigned)n) gunion(lab, u, v);
    }
  }
  __syncthreads();
  int lb[kPer], rol[kPer], dep[kPer], rew[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    lb[k] = i < n ? gfind(lab, i) : 0;
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i < n) lab[i] = lb[k];
  }
  // ---- own statistics and class sums
  for (int r = tid; r < gi.nr; r += nt) atomicAdd(&s_rootc, (int)b.reward[gi.r0 + r]);
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    rol[k] = dep[k] = rew[k] = 0;
    if (i < n) {
      const int2 m = ws.state_meta[s0 + i];
      rol[k] = m.x;
      dep[k] = m.y;
      rew[k] = b.reward[m.x];
      atomicAdd(&ccnt[lb[k]], 1);
      atomicAdd(&csum[lb[k]], rew[k]);
      atomicAdd(&lsum[lb[k]], dep[k]);
      atomicAdd(reinterpret_cast<unsigned long long*>(&l2sum[lb[k]]), (unsigned long long)((long long)dep[k] * dep[k]));
    }
  }
  __syncthreads();
  const double S_root = (double)s_rootc / (double)gi.nr;
  double S[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    S[k] = 0.0;
    if (i < n) {
      S[k] = pooled_score(rew[k], csum[lb[k]], ccnt[lb[k]], p.w);
      fx_add(&sb_hi[lb[k]], &sb_lo[lb[k]], S[k]);
    }
  }
  __syncthreads();
  // ---- efficiency advantage per state, step reward per edge
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
    if (Q >= 2) {
      route_end[k] = true;
      const double sbar = fx_get(&sb_hi[L], &sb_lo[L]) / (double)Q;
      const long long ls = lsum[L], l2 = l2sum[L];
      const double mean_l = (double)ls / (double)Q;
      // sum (l - mean)^2 = (Q sum l^2 - (sum l)^2) / Q, exact integer numerator
      const double ss = (double)((long long)Q * l2 - ls * ls) / (double)Q;
      const double sd = sqrt(ss / (double)(Q - p.ddof));
      aeff[k] = sbar * (mean_l - (double)dep[k]) / (sd + p.eps);
    }
    // eta(p(v), v) from fp32 row statistics; zero rows give 0
    const int v = s0 + i;
    double Sp, eta = 0.0;
    if (dep[k] == 1) {
      Sp = S_root;
      if (b.root_emb) {
        const float n1 = ws.root_n2[g], n2 = ws.nrm2[v];
        if (n1 > 0.f && n2 > 0.f) eta = (double)ws.dotp[v] / sqrt((double)n1 * (double)n2);
      }
    } else {
      const int Lp = lab[i - 1];
      Sp = pooled_score(rew[k], csum[Lp], ccnt[Lp], p.w);  // same rollout, same reward
      const float n1 = ws.nrm2[v - 1], n2 = ws.nrm2[v];
      if (n1 > 0.f && n2 > 0.f) eta = (double)ws.dotp[v] / sqrt((double)n1 * (double)n2);
      key[k] = Lp;
    }
    eta = eta > 0.0 ? eta : 0.0;
    r[k] = (S[k] - Sp) * (1.0 - eta);
  }
  __syncthreads();  // class accumulators no longer read: region X is reused

  // ---- correctness groups: key = class of p(v), n = the prompt root
  int* gcnt = reinterpret_cast<int*>(X);
  long long* gs_hi = reinterpret_cast<long long*>(X + al16(sizeof(int) * (size_t)(n + 1)));
  long long* gs_lo = gs_hi + (n + 1);
  long long* gq_hi = gs_lo + (n + 1);
  long long* gq_lo = gq_hi + (n + 1);
  for (int i = tid; i <= n; i += nt) {
    gcnt[i] = 0;
    gs_hi[i] = gs_lo[i] = gq_hi[i] = gq_lo[i] = 0;
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    if (tid + k * nt < n) {
      atomicAdd(&gcnt[key[k]], 1);
      fx_add(&gs_hi[key[k]], &gs_lo[key[k]], r[k]);
    }
  }
  __syncthreads();
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
  __syncthreads();
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
  __syncthreads();  // region X reused again

  // ---- routes: every edge on root -> v receives A_eff(v) (suffix sums per rollout)
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
  __syncthreads();
  const int32_t* so = b.rollout_step_off;
  for (int rr = tid; rr < gi.nr; rr += nt) {
    const int R = gi.r0 + rr;
    const int a = so[R] - s0, e = so[R + 1] - s0;
    double acc = 0.0;
    unsigned char cov = 0;
    for (int i = e - 1; i >= a; --i) {
      acc += s_aeff[i];
      cov |= s_cov[i];
      s_E[i] = acc;
      s_cov[i] = cov;
    }
    int64_t t = b.rollout_token_off[R];
    for (int i = a; i < e; ++i) {
      ws.tok_start[s0 + i] = t;
      t += b.step_len[s0 + i];
    }
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int i = tid + k * nt;
    if (i >= n) continue;
    const int v = s0 + i;
    const double E = s_E[i];
    const double dual = acor[k] + p.lambda_eff * E;
    ws.e_adv[v] = (float)dual;
    ws.e_cor[v] = (float)acor[k];
    ws.e_eff[v] = (float)E;
    ws.e_mask[v] = s_cov[i];
    if (o.edge_adv) o.edge_adv[v] = (float)dual;
    if (o.class_id) o.class_id[v] = s0 + lb[k];
    if (o.node_score) o.node_score[v] = (float)S[k];
  }
}

}  // namespace

size_t groups_smem_bytes(int maxn) { return group_smem(maxn < 1 ? 1 : maxn); }

static int groups_threads(int maxn) {
  int t = (maxn + kPer - 1) / kPer;
  t = (t + 31) & ~31;
  return t < 64 ? 64 : (t > 1024 ? 1024 : t);
}

cudaError_t setup_groups() {
  return cudaFuncSetAttribute(groups_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)group_smem(GPO_MAX_GROUP_STATES));
}

cudaError_t launch_groups(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                          const Ws& ws, const Params& p) {
  if (sz.G == 0) return cudaSuccess;
  groups_kernel<<<sz.G, groups_threads(sz.maxn), groups_smem_bytes(sz.maxn), lc.stream>>>(b, o, sz, ws, p);
  return cudaGetLastError();
}

}  // namespace gpo
