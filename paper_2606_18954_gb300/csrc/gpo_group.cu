// Per prompt group (one CTA) of the tiled path: equivalence classes from the
// similarity items' spanning forests, then the graph reward and dual-group
// advantage of every generated edge (gpo_group_math.cuh), and the first token
// of every edge for the token scatter.
#include "gpo_group_math.cuh"

namespace gpo {

namespace {

// States per thread: 2 for groups of up to 2048 states, 4 above (blockDim >= n / kPer, at
// most 1024 threads).
constexpr int kMaxRounds = 64;  // hook-and-shortcut rounds before falling back to root unions

// Shared memory: labels, rollout/depth per state (16-bit: a group holds at most
// 4096 states), rollout offsets, rewards, then the scratch of group_advantages.
// X also holds the tree's own statistics (2 al16(2n) <= 4n + 30 bytes) followed by the
// efficiency marks (4n): within group_scratch_bytes(n) >= 4 kKeyWords (n + 1) + 32
static_assert(kKeyWords >= 2, "efficiency marks after the tree's own statistics");
__host__ __device__ inline size_t group_smem(int n) {
  return al16(sizeof(int) * (size_t)n) + 2 * al16(sizeof(int16_t) * (size_t)n) + al16(sizeof(int) * (size_t)(n + 1)) +
         al16((size_t)n) + group_scratch_bytes(n) + 64;
}

template <int kPer>
__global__ void __launch_bounds__(1024) groups_kernel(gpo_batch b, gpo_outputs o, Sizes sz, Ws ws, Params p) {
  extern __shared__ __align__(16) unsigned char sm[];
  uint32_t* st = ws.status;
  if (aborted(st)) return;
  const int g = blockIdx.x;
  const GroupInfo gi = ws.groups[g];
  const int n = gi.n, s0 = gi.s0, nr = gi.nr, nt = blockDim.x, tid = threadIdx.x;
  if (nr == 0 || n == 0 || n > sz.maxn) {
    if (n == 0 && tid == 0) {  // a group without states: Eff 0 (no tokens)
      if (o.group_eff) o.group_eff[g] = 0.f;
      if (o.group_eff_graph) o.group_eff_graph[g] = 0.f;
    }
    return;
  }

  const bool tree = b.parent != nullptr;
  int* lab = reinterpret_cast<int*>(sm);
  int16_t* roll = reinterpret_cast<int16_t*>(sm + al16(sizeof(int) * (size_t)n));
  int16_t* dep = roll + al16(sizeof(int16_t) * (size_t)n) / sizeof(int16_t);
  int* rstart = reinterpret_cast<int*>(reinterpret_cast<unsigned char*>(dep) + al16(sizeof(int16_t) * (size_t)n));
  uint8_t* rew = reinterpret_cast<uint8_t*>(rstart) + al16(sizeof(int) * (size_t)(n + 1));
  unsigned char* X = rew + al16((size_t)n);
  // tree layout: parent (roll's place), subtree end and own statistics (rstart's place and
  // the scratch region), all group-local; the group-math sums live in the workspace
  int16_t* tpar = roll;
  int16_t* tend = reinterpret_cast<int16_t*>(rstart);
  int16_t* tcown = reinterpret_cast<int16_t*>(X);
  int16_t* ttown = tcown + al16(sizeof(int16_t) * (size_t)n) / sizeof(int16_t);

  for (int i = tid; i < n; i += nt) {
    lab[i] = i;
    const int2 m = ws.state_meta[s0 + i];
    dep[i] = (int16_t)m.y;
    if (tree) {
      const int pp = ws.tree_par[s0 + i];
      const int2 own = ws.tree_own[s0 + i];
      tpar[i] = (int16_t)(pp < 0 ? -1 : pp - s0);
      tend[i] = (int16_t)(ws.tree_end[s0 + i] - s0);
      tcown[i] = (int16_t)own.x;
      ttown[i] = (int16_t)own.y;
    } else {
      roll[i] = (int16_t)(m.x - gi.r0);
    }
  }
  if (!tree) {
    for (int r = tid; r <= nr; r += nt) rstart[r] = b.rollout_step_off[gi.r0 + r] - s0;
    for (int r = tid; r < nr; r += nt) rew[r] = b.reward[gi.r0 + r];
  }
  __syncthreads();

  // equivalence classes from the items' spanning forests, in the label forest lab
  // (lab[x] <= x, within x's class): rounds of hooking over every listed pair (the larger of
  // the two current labels is pointed at the smaller, an atomic min) and shortcutting
  // (lab[x] = lab[lab[x]]) until no pair has unequal labels and every label is a root: then
  // each class's label is its smallest member.  Lock-free root unions (correct from any such
  // forest) finish the job if the rounds have not settled after kMaxRounds.
  // Items are dealt to warps (one item per warp at a time, lanes over its edges); the items'
  // edge counts are read once into shared memory (X, free until the group math).
  const int nit = gi.nblk + gi.noff;  // the group's diagonal items, then its off-diagonal ones
  auto item_at = [&](int k) { return k < gi.nblk ? gi.blk0 + k : gi.off0 + (k - gi.nblk); };
  int* ecnt = reinterpret_cast<int*>(X);
  const bool cached = !tree && (size_t)nit * sizeof(int) <= group_scratch_bytes(n);
  if (cached)
    for (int k = tid; k < nit; k += nt) ecnt[k] = min(ws.edge_count[item_at(k)], kEdgeCap);
  __syncthreads();
  const int lane = tid & 31, wid = tid >> 5, nwarp = nt >> 5;
  bool settled = false;
  for (int round = 0; round < kMaxRounds && !settled; ++round) {
    int ch = 0;
    for (int k = wid; k < nit; k += nwarp) {
      const int ne = cached ? ecnt[k] : min(ws.edge_count[item_at(k)], kEdgeCap);
      const int2* E = ws.edges + (size_t)item_at(k) * kEdgeCap;
      for (int e = lane; e < ne; e += 32) {
        const int2 uv = E[e];
        const int u = uv.x - s0, v = uv.y - s0;
        if ((unsigned)u < (unsigned)n && (unsigned)v < (unsigned)n) {
          const int lu = lab[u], lv = lab[v];
          if (lu != lv) {
            atomicMin(&lab[max(lu, lv)], min(lu, lv));
            ch = 1;
          }
        }
      }
    }
    for (int x = tid; x < n; x += nt) {
      const int l = lab[x], ll = lab[l];
      if (ll != l) {
        lab[x] = ll;
        ch = 1;
      }
    }
    settled = __syncthreads_or(ch) == 0;
  }
  if (!settled) {
    for (int k = 0; k < nit; ++k) {
      const int ne = min(ws.edge_count[item_at(k)], kEdgeCap);
      const int2* E = ws.edges + (size_t)item_at(k) * kEdgeCap;
      for (int e = tid; e < ne; e += nt) {
        const int2 uv = E[e];
        const int u = uv.x - s0, v = uv.y - s0;
        if ((unsigned)u < (unsigned)n && (unsigned)v < (unsigned)n) uf_union(lab, u, v);
      }
    }
    __syncthreads();
  }

  if (p.mode == 1) {  // next-layer budgets (gpo_layer_budget; tree layout only)
    __shared__ int s_bud[2 + 32];
    auto active = [&](int i) { return p.active == nullptr || p.active[s0 + i] != 0; };
    auto put = [&](int i, int label, int bud) {
      p.budget[s0 + i] = bud;
      if (o.class_id) o.class_id[s0 + i] = s0 + label;
    };
    // the own statistics take 2 al16(2n) bytes at the start of X
    group_budget(n, lab, dep, p.layer, p.b_next, reinterpret_cast<int*>(X + 2 * al16(sizeof(int16_t) * (size_t)n)),
                 s_bud, s_bud + 2, tid, nt, active, [] { __syncthreads(); }, put);
    return;
  }

  // eta(p(v), v) from the compensated row statistics (pairs); zero rows give 0
  const float2 zero2 = make_float2(0.f, 0.f);
  auto eta = [&](int i) -> float2 {
    const int v = s0 + i;
    const float2 n1 = dep[i] == 1 ? (b.root_emb ? ws.x_root_n2[g] : zero2) : ws.x_n2[v - 1];
    return ff_eta(ws.x_dot[v], n1, ws.x_n2[v]);
  };
  auto out = [&](int i, int label, float S, float acor, float E, float dual, unsigned char mask) {
    const int v = s0 + i;
    if (!GPO_BOUNDS(st, v, sz.N, kWhereStateOut)) return;
    ws.e_adv[v] = dual;
    ws.e_cor[v] = acor;
    ws.e_eff[v] = E;
    ws.e_mask[v] = mask;
    if (o.edge_adv) o.edge_adv[v] = dual;
    if (o.class_id) o.class_id[v] = s0 + label;
    if (o.node_score) o.node_score[v] = S;
    if (o.edge_cor) o.edge_cor[v] = acor;
    if (o.edge_eff) o.edge_eff[v] = E;
    if (o.edge_eff_mask) o.edge_eff_mask[v] = mask;
  };
  // exploration efficiency, Eq. (eq1), once the classes are final; `mark` is scratch that
  // the group math no longer needs
  __shared__ unsigned long long s_eff[3];
  auto efficiency = [&](int* mark) {
    if (!o.group_eff && !o.group_eff_graph) return;
    auto own = [&](int i) { return tree ? tcown[i] > 0 : rew[roll[i]] != 0; };
    auto par = [&](int i) { return tree ? (int)tpar[i] : (dep[i] == 1 ? -1 : i - 1); };
    auto len = [&](int i) { return b.step_len[s0 + i]; };
    group_efficiency(n, lab, mark, s_eff, tid, nt, own, par, len, [] { __syncthreads(); },
                     [](bool f) { return __syncthreads_or(f) != 0; }, o.group_eff ? o.group_eff + g : nullptr,
                     o.group_eff_graph ? o.group_eff_graph + g : nullptr);
  };
  if (tree) {
    auto eta_t = [&](int i) -> float2 {
      const int v = s0 + i;
      const float2 n1 = tpar[i] < 0 ? (b.root_emb ? ws.x_root_n2[g] : zero2) : ws.x_n2[s0 + tpar[i]];
      return ff_eta(ws.x_dot[v], n1, ws.x_n2[v]);
    };
    static_assert(tree_scratch_words(1) == 23 + 11 && tree_scratch_words(2) == 2 * 23 + 11,
                  "workspace layout of the tree sums");
    group_advantages_tree<kPer, int16_t>(n, nr, lab, tpar, dep, tend, tcown, ttown,
                                         tree_scratch(ws.tree_x + (size_t)23 * s0 + (size_t)11 * g, n), p, tid, nt,
                                         [] { __syncthreads(); }, eta_t, out);
    // the own statistics take 2 al16(2n) bytes at the start of X
    efficiency(reinterpret_cast<int*>(X + 2 * al16(sizeof(int16_t) * (size_t)n)));
    return;  // the tree prep kernel wrote the first token of every edge
  }
  __shared__ int s_rootc;
  group_advantages<kPer, false, int16_t>(n, nr, lab, roll, dep, rstart, rew, group_scratch_shared(X, n, &s_rootc), p,
                                         tid, nt, [] { __syncthreads(); }, eta, out);
  efficiency(reinterpret_cast<int*>(X));

  // first token of every edge: one warp per rollout, an exclusive scan of the step lengths
  {
    const int lane = tid & 31;
    for (int rr = tid >> 5; rr < nr; rr += nt >> 5) {
      int64_t t = b.rollout_token_off[gi.r0 + rr];
      for (int i0 = rstart[rr]; i0 < rstart[rr + 1]; i0 += 32) {
        const int i = i0 + lane;
        const int64_t len = i < rstart[rr + 1] ? b.step_len[s0 + i] : 0;
        int64_t incl = len;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int64_t y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        if (i < rstart[rr + 1]) ws.tok_start[s0 + i] = t + incl - len;
        t += __shfl_sync(0xffffffffu, incl, 31);
      }
    }
  }
}

constexpr int kPerSmall = 2, kPerLarge = 4, kSmallMax = 2048;

int groups_threads(int maxn) {
  const int per = maxn <= kSmallMax ? kPerSmall : kPerLarge;
  int t = (maxn + per - 1) / per;
  t = (t + 31) & ~31;
  return t < 64 ? 64 : (t > 1024 ? 1024 : t);
}

}  // namespace

size_t groups_smem_bytes(int maxn) { return group_smem(maxn < 1 ? 1 : maxn); }

cudaError_t setup_groups() {
  const int bytes = (int)group_smem(GPO_MAX_GROUP_STATES);
  cudaError_t e = cudaFuncSetAttribute(groups_kernel<kPerSmall>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(groups_kernel<kPerLarge>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  return e;
}

cudaError_t launch_groups(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                          const Ws& ws, const Params& p) {
  if (sz.G == 0) return cudaSuccess;
  if (sz.maxn <= kSmallMax)
    groups_kernel<kPerSmall><<<sz.G, groups_threads(sz.maxn), groups_smem_bytes(sz.maxn), lc.stream>>>(b, o, sz, ws, p);
  else
    groups_kernel<kPerLarge><<<sz.G, groups_threads(sz.maxn), groups_smem_bytes(sz.maxn), lc.stream>>>(b, o, sz, ws, p);
  return cudaGetLastError();
}

}  // namespace gpo
