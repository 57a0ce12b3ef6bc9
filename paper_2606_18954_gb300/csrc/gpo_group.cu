// Per prompt group (one CTA) of the tiled path: equivalence classes from the
// similarity items' spanning forests, then the graph reward and dual-group
// advantage of every generated edge (gpo_group_math.cuh), and the first token
// of every edge for the token scatter.
#include "gpo_group_math.cuh"

namespace gpo {

namespace {

constexpr int kPer = 4;  // states per thread (blockDim >= n / kPer)

// Shared memory: labels, rollout/depth per state (16-bit: a group holds at most
// 4096 states), rollout offsets, rewards, then the scratch of group_advantages.
__host__ __device__ inline size_t group_smem(int n) {
  return al16(sizeof(int) * (size_t)n) + 2 * al16(sizeof(int16_t) * (size_t)n) + al16(sizeof(int) * (size_t)(n + 1)) +
         al16((size_t)n) + group_scratch_bytes(n) + 64;
}

__global__ void __launch_bounds__(1024) groups_kernel(gpo_batch b, gpo_outputs o, Sizes sz, Ws ws, Params p) {
  extern __shared__ __align__(16) unsigned char sm[];
  uint32_t* st = ws.status;
  if (aborted(st)) return;
  const int g = blockIdx.x;
  const GroupInfo gi = ws.groups[g];
  const int n = gi.n, s0 = gi.s0, nr = gi.nr, nt = blockDim.x, tid = threadIdx.x;
  if (nr == 0 || n == 0 || n > sz.maxn) return;

  int* lab = reinterpret_cast<int*>(sm);
  int16_t* roll = reinterpret_cast<int16_t*>(sm + al16(sizeof(int) * (size_t)n));
  int16_t* dep = roll + al16(sizeof(int16_t) * (size_t)n) / sizeof(int16_t);
  int* rstart = reinterpret_cast<int*>(reinterpret_cast<unsigned char*>(dep) + al16(sizeof(int16_t) * (size_t)n));
  uint8_t* rew = reinterpret_cast<uint8_t*>(rstart) + al16(sizeof(int) * (size_t)(n + 1));
  unsigned char* X = rew + al16((size_t)n);

  for (int i = tid; i < n; i += nt) {
    lab[i] = i;
    const int2 m = ws.state_meta[s0 + i];
    roll[i] = (int16_t)(m.x - gi.r0);
    dep[i] = (int16_t)m.y;
  }
  for (int r = tid; r <= nr; r += nt) rstart[r] = b.rollout_step_off[gi.r0 + r] - s0;
  for (int r = tid; r < nr; r += nt) rew[r] = b.reward[gi.r0 + r];
  __syncthreads();

  // equivalence classes from the items' spanning forests
  const int it0 = ws.group_items[g], it1 = ws.group_items[g + 1];
  for (int it = it0; it < it1; ++it) {
    const int ne = ws.edge_count[it];
    const int2* E = ws.edges + (size_t)it * kEdgeCap;
    for (int e = tid; e < ne; e += nt) {
      const int2 uv = E[e];
      const int u = uv.x - s0, v = uv.y - s0;
      if ((unsigned)u < (unsigned)n && (unsigned)v < (unsigned)n) uf_union(lab, u, v);
    }
  }
  __syncthreads();

  // eta(p(v), v) from the fp32 row statistics; zero rows give 0
  auto eta = [&](int i) -> float {
    const int v = s0 + i;
    float e = 0.f, n1 = 0.f, dot = 0.f;
    if (dep[i] == 1) {
      if (b.root_emb) {
        n1 = ws.root_n2[g];
        dot = ws.dotp[v];
      }
    } else {
      n1 = ws.nrm2[v - 1];
      dot = ws.dotp[v];
    }
    const float n2 = ws.nrm2[v];
    if (n1 > 0.f && n2 > 0.f) e = dot / sqrtf(n1 * n2);
    return e > 0.f ? e : 0.f;
  };
  auto out = [&](int i, int label, float S, float acor, float E, float dual, unsigned char mask) {
    const int v = s0 + i;
    ws.e_adv[v] = dual;
    ws.e_cor[v] = acor;
    ws.e_eff[v] = E;
    ws.e_mask[v] = mask;
    if (o.edge_adv) o.edge_adv[v] = dual;
    if (o.class_id) o.class_id[v] = s0 + label;
    if (o.node_score) o.node_score[v] = S;
  };
  __shared__ int s_rootc;
  group_advantages<kPer, false, int16_t>(n, nr, lab, roll, dep, rstart, rew, group_scratch_shared(X, n, &s_rootc), p,
                                         tid, nt, [] { __syncthreads(); }, eta, out);

  // first token of every edge
  for (int rr = tid; rr < nr; rr += nt) {
    int64_t t = b.rollout_token_off[gi.r0 + rr];
    for (int i = rstart[rr]; i < rstart[rr + 1]; ++i) {
      ws.tok_start[s0 + i] = t;
      t += b.step_len[s0 + i];
    }
  }
}

int groups_threads(int maxn) {
  int t = (maxn + kPer - 1) / kPer;
  t = (t + 31) & ~31;
  return t < 64 ? 64 : (t > 1024 ? 1024 : t);
}

}  // namespace

size_t groups_smem_bytes(int maxn) { return group_smem(maxn < 1 ? 1 : maxn); }

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
