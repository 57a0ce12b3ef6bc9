/*
 * GraphPO advantage construction -- CPU ORACLE (test infrastructure only;
 * see oracle.h).  Plain C, fp64, one prompt group at a time, every quantity
 * computed from its definition in the paper:
 *
 *   Sec. 4.2  sim(u,v) = z_u.z_v / (|z_u||z_v|); only pairs that are not in an
 *             ancestor-descendant relation are compared; pairs with sim >= kappa
 *             are linked and the equivalence classes Q are the connected
 *             components (transitive closure, Algorithm S.1 "Union-Find").
 *   Sec. 4.3  c_own(v) = sum of R(z) over terminals z reachable from v along
 *             direct edges, t_own(v) = their number (propagated bottom-up);
 *             Eq. (combain) pooled score S(v); r_step(u,v) =
 *             (S(v) - S(u)) (1 - eta(u,v)), eta = max(0, sim).
 *   Sec. 4.4  A_cor over E_cor(u) = {(p(v),v) | v in C_g(u)},
 *             C_g(u) = union of the direct suffixes of all members of Q(u);
 *             A_eff(v) = Sbar_Q * z-score of -l_v within Q, l_v = number of
 *             direct edges from the deepest common predecessor a_Q to v, added
 *             to every generated edge on the route a_Q -> v.
 *   Sec. 4.5  A_dual(e) = A_cor(e) + lambda_eff * A_eff(e); every token of an
 *             edge carries the edge's advantage.
 *   Eq. (eq1) exploration efficiency Eff = (tokens of correct steps) / (tokens of
 *             all steps); a step (p(v), v) is correct when a correct final
 *             answer can be reached from v: along direct edges (tree reading,
 *             c_own(v) > 0; in the chain layout this is the paper's chain case,
 *             the whole trajectory counted as one step), or along direct edges
 *             and equivalences of the merged graph (graph reading).
 *
 * The same definitions serve both input layouts (oracle.h): in the chain layout
 * every rollout is a path from the root, in the tree layout the provenance
 * tree is given by parent pointers and its leaves are the terminal states.
 *
 * Readings where the paper leaves a choice open (each is a parameter or a
 * stated constant): std = sqrt(sum (x-mean)^2 / (K - ddof)) and the
 * standardisation divides by (std + eps); correctness groups of one edge and
 * classes of one state get no advantage (Algorithm S.1 only visits
 * |C_g(u)| > 1 and |Q| >= 2); a_Q is the deepest node that is a strict ancestor
 * of every member; every edge on a route receives the full A_eff(v), and an
 * edge on several routes receives their sum; the prompt root has no embedding
 * unless root_emb is given, in which case eta on root edges uses it; a state
 * with a zero embedding has similarity 0 with every state; the class label is
 * the smallest state index in the class.
 */
#include "oracle.h"

#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- inputs -- */

static double emb_value(const oracle_batch* b, const void* base, int64_t row, int k) {
  if (b->emb_is_bf16) {
    uint16_t u = ((const uint16_t*)base)[row * b->emb_row_stride + k];
    uint32_t x = (uint32_t)u << 16;
    float f;
    memcpy(&f, &x, sizeof f);
    return (double)f;
  }
  return (double)((const float*)base)[row * b->emb_row_stride + k];
}

static int validate_embeddings(const oracle_batch* b) {
  for (int64_t v = 0; v < b->num_states; ++v)
    for (int k = 0; k < b->d; ++k)
      if (!isfinite(emb_value(b, b->emb, v, k))) return ORACLE_ERR_NONFINITE;
  if (b->root_emb)
    for (int g = 0; g < b->num_groups; ++g)
      for (int k = 0; k < b->d; ++k)
        if (!isfinite(emb_value(b, b->root_emb, g, k))) return ORACLE_ERR_NONFINITE;
  return ORACLE_OK;
}

/* Tree layout: offsets, parents that precede their children, depth-first
 * pre-order (the strict descendants of u are exactly the states u+1 ..
 * u + (number of descendants of u)), one rollout per leaf, token spans. */
static int validate_tree(const oracle_batch* b) {
  const int G = b->num_groups, R = b->num_rollouts, N = b->num_states;
  const int32_t* go = b->group_rollout_off;
  const int32_t* gs = b->group_state_off;
  const int64_t* gt = b->group_token_off;
  if (!go || !gs || !gt) return ORACLE_ERR_INVALID_ARG;
  if (go[0] != 0 || go[G] != R || gs[0] != 0 || gs[G] != N || gt[0] != 0 || gt[G] != b->total_tokens)
    return ORACLE_ERR_SHAPE;
  for (int g = 0; g < G; ++g)
    if (go[g + 1] < go[g] || gs[g + 1] < gs[g] || gt[g + 1] < gt[g]) return ORACLE_ERR_SHAPE;
  for (int g = 0; g < G; ++g) {
    const int s0 = gs[g], n = gs[g + 1] - gs[g];
    for (int v = 0; v < n; ++v)
      if (b->parent[s0 + v] < -1 || b->parent[s0 + v] >= v) return ORACLE_ERR_SHAPE;
    int* desc = calloc(n > 0 ? n : 1, sizeof(int));
    int* kids = calloc(n > 0 ? n : 1, sizeof(int));
    if (!desc || !kids) return ORACLE_ERR_NOMEM;
    for (int v = 0; v < n; ++v) {
      if (b->parent[s0 + v] >= 0) kids[b->parent[s0 + v]]++;
      for (int a = b->parent[s0 + v]; a >= 0; a = b->parent[s0 + a]) desc[a]++;
    }
    int bad = 0, leaves = 0;
    for (int v = 0; v < n && !bad; ++v) {
      leaves += kids[v] == 0;
      for (int a = b->parent[s0 + v]; a >= 0; a = b->parent[s0 + a])
        if (!(a < v && v <= a + desc[a])) bad = 1;
    }
    free(desc);
    free(kids);
    if (bad || leaves != go[g + 1] - go[g]) return ORACLE_ERR_SHAPE;
    int64_t sum = 0;
    for (int v = gs[g]; v < gs[g + 1]; ++v) {
      if (b->step_len[v] < 1) return ORACLE_ERR_SHAPE;
      sum += b->step_len[v];
    }
    if (gt[g + 1] - gt[g] != sum) return ORACLE_ERR_SHAPE;
  }
  for (int r = 0; r < R; ++r)
    if (b->reward[r] > 1) return ORACLE_ERR_BAD_REWARD; /* R(z) in {0,1}, Sec. 4.3 */
  return validate_embeddings(b);
}

int oracle_validate(const oracle_batch* b) {
  if (!b) return ORACLE_ERR_INVALID_ARG;
  const int G = b->num_groups, R = b->num_rollouts, N = b->num_states;
  if (G < 0 || R < 0 || N < 0 || b->d <= 0 || b->total_tokens < 0) return ORACLE_ERR_INVALID_ARG;
  if (b->emb_row_stride < b->d) return ORACLE_ERR_INVALID_ARG;
  if (N > 0 && (!b->step_len || !b->emb)) return ORACLE_ERR_INVALID_ARG;
  if (R > 0 && !b->reward) return ORACLE_ERR_INVALID_ARG;
  if (b->parent) return validate_tree(b);
  if (!b->group_rollout_off || !b->rollout_step_off || !b->rollout_token_off) return ORACLE_ERR_INVALID_ARG;
  const int32_t* go = b->group_rollout_off;
  const int32_t* so = b->rollout_step_off;
  const int64_t* to = b->rollout_token_off;
  if (go[0] != 0 || go[G] != R) return ORACLE_ERR_SHAPE;
  for (int g = 0; g < G; ++g)
    if (go[g + 1] < go[g]) return ORACLE_ERR_SHAPE;
  if (so[0] != 0 || so[R] != N) return ORACLE_ERR_SHAPE;
  for (int r = 0; r < R; ++r)
    if (so[r + 1] <= so[r]) return ORACLE_ERR_SHAPE; /* a rollout has at least one step */
  if (to[0] != 0 || to[R] != b->total_tokens) return ORACLE_ERR_SHAPE;
  for (int r = 0; r < R; ++r) {
    int64_t sum = 0;
    for (int v = so[r]; v < so[r + 1]; ++v) {
      if (b->step_len[v] < 1) return ORACLE_ERR_SHAPE;
      sum += b->step_len[v];
    }
    if (to[r + 1] - to[r] != sum) return ORACLE_ERR_SHAPE;
  }
  for (int r = 0; r < R; ++r)
    if (b->reward[r] > 1) return ORACLE_ERR_BAD_REWARD; /* R(z) in {0,1}, Sec. 4.3 */
  return validate_embeddings(b);
}

/* ------------------------------------------------------------ one group -- */

/* Node numbering inside a group: 0 is the prompt root v0; node i >= 1 is the
 * state with global index s0 + i - 1. */
typedef struct {
  int n;            /* nodes including the root */
  int32_t s0;       /* first global state index */
  int* parent;      /* generation predecessor p(v); -1 for the root */
  int* depth;       /* d(v); 0 for the root */
  int* rollout;     /* global rollout index; -1 for the root */
  int* terminal;    /* 1 for the last state of a rollout */
  int* child_off;   /* direct successors C(u) as CSR */
  int* child_list;
  double* z;        /* n x d, row 0 is the root embedding if present */
  double* nrm;      /* |z| */
  int has_root_emb;
  unsigned char* adj; /* n x n linked pairs */
  int* label;       /* local node index of the smallest member of Q(v) */
  int* mem_off;     /* members of each class, CSR keyed by label */
  int* mem_list;
} group_t;

static int is_strict_ancestor(const group_t* G, int a, int b) {
  for (int x = G->parent[b]; x >= 0; x = G->parent[x])
    if (x == a) return 1;
  return 0;
}

static double cosine(const group_t* G, int d, int i, int j) {
  if (G->nrm[i] == 0.0 || G->nrm[j] == 0.0) return 0.0;
  double dot = 0.0;
  for (int k = 0; k < d; ++k) dot += G->z[(int64_t)i * d + k] * G->z[(int64_t)j * d + k];
  return dot / (G->nrm[i] * G->nrm[j]);
}

static double mean_of(const double* x, int n) {
  double s = 0.0;
  for (int i = 0; i < n; ++i) s += x[i];
  return s / n;
}

static double std_of(const double* x, int n, double mean, int ddof) {
  double s = 0.0;
  for (int i = 0; i < n; ++i) s += (x[i] - mean) * (x[i] - mean);
  return sqrt(s / (n - ddof));
}

static int run_group(const oracle_batch* b, const oracle_params* p, oracle_outputs* o, int g) {
  const int32_t* go = b->group_rollout_off;
  const int32_t* so = b->rollout_step_off;
  const int tree = b->parent != NULL;
  const int r0 = go[g], r1 = go[g + 1];
  const int32_t s0 = tree ? b->group_state_off[g] : so[r0];
  const int32_t s1 = tree ? b->group_state_off[g + 1] : so[r1];
  const int Ng = s1 - s0, n = Ng + 1, d = b->d;
  if (r1 == r0) return ORACLE_OK; /* empty prompt group: nothing to label */

  group_t G;
  memset(&G, 0, sizeof G);
  G.n = n;
  G.s0 = s0;
  G.parent = malloc(sizeof(int) * n);
  G.depth = malloc(sizeof(int) * n);
  G.rollout = malloc(sizeof(int) * n);
  G.terminal = malloc(sizeof(int) * n);
  G.child_off = calloc(n + 1, sizeof(int));
  G.child_list = malloc(sizeof(int) * n);
  G.z = malloc(sizeof(double) * (size_t)n * d);
  G.nrm = malloc(sizeof(double) * n);
  G.adj = calloc((size_t)n * n, 1);
  G.label = malloc(sizeof(int) * n);
  G.mem_off = calloc(n + 1, sizeof(int));
  G.mem_list = malloc(sizeof(int) * n);
  double* c_own = calloc(n, sizeof(double));
  double* t_own = calloc(n, sizeof(double));
  double* S = malloc(sizeof(double) * n);
  double* eta = calloc(n, sizeof(double));
  double* r = calloc(n, sizeof(double));
  double* a_cor = calloc(n, sizeof(double));
  int* gsize = malloc(sizeof(int) * n);
  double* a_eff = calloc(n, sizeof(double));
  double* e_eff = calloc(n, sizeof(double));
  unsigned char* emask = calloc(n, 1);
  int* queue = malloc(sizeof(int) * n);
  int* order = malloc(sizeof(int) * n);
  int* cnt = malloc(sizeof(int) * n);
  int* tmp = malloc(sizeof(int) * n);
  double* xs = malloc(sizeof(double) * n);
  unsigned char* reach = calloc(n, 1);
  if (!G.parent || !G.depth || !G.rollout || !G.terminal || !G.child_off || !G.child_list ||
      !G.z || !G.nrm || !G.adj || !G.label || !G.mem_off || !G.mem_list || !c_own || !t_own ||
      !S || !eta || !r || !a_cor || !gsize || !a_eff || !e_eff || !emask || !queue || !order ||
      !cnt || !tmp || !xs || !reach)
    return ORACLE_ERR_NOMEM; /* the process is about to fail anyway; no cleanup */

  /* --- the rollout graph: root v0 plus one node per generated step (Sec. 4.2) --- */
  G.parent[0] = -1;
  G.depth[0] = 0;
  G.rollout[0] = -1;
  G.terminal[0] = 0;
  if (!tree) {
    for (int rr = r0; rr < r1; ++rr) {
      const int nr = so[rr + 1] - so[rr];
      for (int h = 1; h <= nr; ++h) {
        const int i = so[rr] + h - 1 - s0 + 1;
        G.parent[i] = (h == 1) ? 0 : i - 1;
        G.depth[i] = h;
        G.rollout[i] = rr;
        G.terminal[i] = (h == nr);
      }
    }
  } else {
    /* explicit provenance: parents precede their children, so depths follow in order */
    for (int i = 1; i < n; ++i) {
      G.parent[i] = b->parent[s0 + i - 1] + 1;
      G.depth[i] = G.depth[G.parent[i]] + 1;
    }
  }
  for (int i = 1; i < n; ++i) G.child_off[G.parent[i] + 1]++;
  for (int i = 0; i < n; ++i) G.child_off[i + 1] += G.child_off[i];
  for (int i = 0; i < n; ++i) tmp[i] = G.child_off[i];
  for (int i = 1; i < n; ++i) G.child_list[tmp[G.parent[i]]++] = i;
  if (tree) {
    /* the terminal states are the leaves; leaf k (in state order) is rollout r0 + k */
    int k = 0;
    for (int i = 1; i < n; ++i) {
      G.terminal[i] = G.child_off[i + 1] == G.child_off[i];
      G.rollout[i] = G.terminal[i] ? r0 + k++ : -1;
    }
  }

  /* --- embeddings z_v (Sec. 4.2) --- */
  G.has_root_emb = b->root_emb != NULL;
  for (int k = 0; k < d; ++k) G.z[k] = G.has_root_emb ? emb_value(b, b->root_emb, g, k) : 0.0;
  for (int i = 1; i < n; ++i)
    for (int k = 0; k < d; ++k) G.z[(int64_t)i * d + k] = emb_value(b, b->emb, s0 + i - 1, k);
  for (int i = 0; i < n; ++i) {
    double s = 0.0;
    for (int k = 0; k < d; ++k) s += G.z[(int64_t)i * d + k] * G.z[(int64_t)i * d + k];
    G.nrm[i] = sqrt(s);
  }

  /* --- link comparable pairs with sim >= kappa (Sec. 4.2, Algorithm S.1) --- */
  for (int i = 1; i < n; ++i)
    for (int j = i + 1; j < n; ++j) {
      if (is_strict_ancestor(&G, i, j) || is_strict_ancestor(&G, j, i)) continue;
      if (p->merge_rule == 1 && G.depth[i] != G.depth[j]) continue;
      if (cosine(&G, d, i, j) >= p->kappa) G.adj[(size_t)i * n + j] = G.adj[(size_t)j * n + i] = 1;
    }

  /* --- equivalence classes = connected components; label = smallest member --- */
  for (int i = 0; i < n; ++i) G.label[i] = -1;
  G.label[0] = 0; /* the root is an ancestor of every state: never comparable */
  for (int i = 1; i < n; ++i) {
    if (G.label[i] >= 0) continue;
    int qh = 0, qt = 0;
    queue[qt++] = i;
    G.label[i] = i; /* nodes below i are all labelled already, so i is the minimum */
    while (qh < qt) {
      const int x = queue[qh++];
      for (int y = 1; y < n; ++y)
        if (G.adj[(size_t)x * n + y] && G.label[y] < 0) {
          G.label[y] = i;
          queue[qt++] = y;
        }
    }
  }
  for (int i = 0; i < n; ++i) G.mem_off[G.label[i] + 1]++;
  for (int i = 0; i < n; ++i) G.mem_off[i + 1] += G.mem_off[i];
  for (int i = 0; i < n; ++i) tmp[i] = G.mem_off[i];
  for (int i = 0; i < n; ++i) G.mem_list[tmp[G.label[i]]++] = i;

  /* --- own terminal statistics, bottom-up along direct edges (Sec. 4.3) --- */
  /* nodes by decreasing depth, so every child is finished before its parent */
  {
    int maxd = 0;
    for (int i = 0; i < n; ++i) maxd = G.depth[i] > maxd ? G.depth[i] : maxd;
    int k = 0;
    for (int dd = maxd; dd >= 0; --dd)
      for (int i = 0; i < n; ++i)
        if (G.depth[i] == dd) order[k++] = i;
  }
  for (int k = 0; k < n; ++k) {
    const int i = order[k];
    if (G.terminal[i]) {
      c_own[i] += (double)b->reward[G.rollout[i]];
      t_own[i] += 1.0;
    }
    if (G.parent[i] >= 0) {
      c_own[G.parent[i]] += c_own[i];
      t_own[G.parent[i]] += t_own[i];
    }
  }

  /* --- pooled node score, Eq. (combain) --- */
  for (int i = 0; i < n; ++i) {
    const int L = G.label[i];
    double oc = 0.0, ot = 0.0;
    for (int m = G.mem_off[L]; m < G.mem_off[L + 1]; ++m) {
      const int q = G.mem_list[m];
      if (q == i) continue;
      oc += c_own[q];
      ot += t_own[q];
    }
    const double den = t_own[i] + p->w * ot;
    S[i] = den > 0.0 ? (c_own[i] + p->w * oc) / den : 0.0; /* "when the denominator is positive" */
  }

  /* --- step reward on every direct edge (Sec. 4.3) --- */
  for (int i = 1; i < n; ++i) {
    const int u = G.parent[i];
    double sim = 0.0;
    if (u > 0 || G.has_root_emb) sim = cosine(&G, d, u, i);
    eta[i] = sim > 0.0 ? sim : 0.0;
    r[i] = (S[i] - S[u]) * (1.0 - eta[i]);
  }

  /* --- correctness advantage over E_cor(u) for every semantic state u (Sec. 4.4) --- */
  for (int i = 1; i < n; ++i) gsize[i] = 1;
  for (int u = 0; u < n; ++u) {
    const int L = G.label[u];
    int K = 0; /* C_g(u) = C(u) plus the direct suffixes of the other members of Q(u) */
    for (int m = G.mem_off[L]; m < G.mem_off[L + 1]; ++m) {
      const int q = G.mem_list[m];
      for (int c = G.child_off[q]; c < G.child_off[q + 1]; ++c) tmp[K++] = G.child_list[c];
    }
    if (K <= 1) continue;
    for (int k = 0; k < K; ++k) xs[k] = r[tmp[k]]; /* reward of the generated edge (p(v), v) */
    const double mean = mean_of(xs, K);
    const double sd = std_of(xs, K, mean, p->std_ddof);
    for (int k = 0; k < K; ++k) {
      a_cor[tmp[k]] = (xs[k] - mean) / (sd + p->std_eps);
      gsize[tmp[k]] = K;
    }
  }

  /* --- efficiency advantage per class with |Q| >= 2 (Sec. 4.4) --- */
  for (int L = 1; L < n; ++L) {
    const int q0 = G.mem_off[L], q1 = G.mem_off[L + 1], Q = q1 - q0;
    if (Q < 2) continue;
    /* deepest common strict ancestor a_Q */
    for (int i = 0; i < n; ++i) cnt[i] = 0;
    for (int m = q0; m < q1; ++m)
      for (int x = G.parent[G.mem_list[m]]; x >= 0; x = G.parent[x]) cnt[x]++;
    int aQ = -1;
    for (int i = 0; i < n; ++i)
      if (cnt[i] == Q && (aQ < 0 || G.depth[i] > G.depth[aQ])) aQ = i;
    double sbar = 0.0;
    for (int m = q0; m < q1; ++m) sbar += S[G.mem_list[m]];
    sbar /= Q;
    for (int m = q0; m < q1; ++m) xs[m - q0] = -(double)(G.depth[G.mem_list[m]] - G.depth[aQ]);
    const double mean = mean_of(xs, Q);
    const double sd = std_of(xs, Q, mean, p->std_ddof);
    for (int m = q0; m < q1; ++m) {
      const int v = G.mem_list[m];
      const double A = sbar * (xs[m - q0] - mean) / (sd + p->std_eps);
      a_eff[v] = A;
      for (int x = v; x != aQ; x = G.parent[x]) { /* every generated edge on a_Q -> v */
        e_eff[x] += A;
        emask[x] = 1;
      }
    }
  }

  /* --- exploration efficiency, Eq. (eq1) --- */
  if (o->eff_tree || o->eff_graph) {
    /* graph reading: a class reaches a correct answer if one of its members is a correct
       terminal, or a member has a child whose class reaches one; breadth-first search
       backwards over the quotient graph's edges class(child) -> class(parent) */
    int qh = 0, qt = 0;
    for (int i = 1; i < n; ++i)
      if (G.terminal[i] && b->reward[G.rollout[i]] && !reach[G.label[i]]) {
        reach[G.label[i]] = 1;
        queue[qt++] = G.label[i];
      }
    while (qh < qt) {
      const int L = queue[qh++];
      for (int i = 1; i < n; ++i) {
        const int u = G.parent[i];
        if (G.label[i] == L && u > 0 && !reach[G.label[u]]) {
          reach[G.label[u]] = 1;
          queue[qt++] = G.label[u];
        }
      }
    }
    double tok = 0.0, good_tree = 0.0, good_graph = 0.0;
    for (int i = 1; i < n; ++i) {
      const double len = (double)b->step_len[s0 + i - 1];
      tok += len;
      if (c_own[i] > 0.0) good_tree += len; /* a correct terminal lies below v */
      if (reach[G.label[i]]) good_graph += len;
    }
    if (o->eff_tree) o->eff_tree[g] = tok > 0.0 ? good_tree / tok : 0.0;
    if (o->eff_graph) o->eff_graph[g] = tok > 0.0 ? good_graph / tok : 0.0;
  }

  /* --- outputs: per state / edge, then every token of the edge (Sec. 4.5) --- */
  if (o->root_score) o->root_score[g] = S[0];
  for (int i = 1; i < n; ++i) {
    const int64_t v = s0 + i - 1;
    const double dual = a_cor[i] + p->lambda_eff * e_eff[i];
    if (o->class_id) o->class_id[v] = s0 + G.label[i] - 1;
    if (o->node_score) o->node_score[v] = S[i];
    if (o->eta) o->eta[v] = eta[i];
    if (o->step_reward) o->step_reward[v] = r[i];
    if (o->a_cor) o->a_cor[v] = a_cor[i];
    if (o->a_eff_node) o->a_eff_node[v] = a_eff[i];
    if (o->e_eff) o->e_eff[v] = e_eff[i];
    if (o->edge_adv) o->edge_adv[v] = dual;
    if (o->edge_eff_mask) o->edge_eff_mask[v] = emask[i];
    if (o->cor_group_size) o->cor_group_size[v] = gsize[i];
  }
  /* chain layout: each rollout's span holds its steps in order; tree layout: the
     group's span holds every edge once, in state order */
  for (int rr = tree ? 0 : r0; rr < (tree ? 1 : r1); ++rr) {
    int64_t t = tree ? b->group_token_off[g] : b->rollout_token_off[rr];
    const int v0 = tree ? s0 : so[rr], v1 = tree ? s1 : so[rr + 1];
    for (int v = v0; v < v1; ++v) {
      const int i = v - s0 + 1;
      const double dual = a_cor[i] + p->lambda_eff * e_eff[i];
      for (int k = 0; k < b->step_len[v]; ++k, ++t) {
        if (o->adv) o->adv[t] = dual;
        if (o->adv_cor) o->adv_cor[t] = a_cor[i];
        if (o->adv_eff) o->adv_eff[t] = e_eff[i];
        if (o->eff_mask) o->eff_mask[t] = emask[i];
      }
    }
  }

  free(G.parent); free(G.depth); free(G.rollout); free(G.terminal); free(G.child_off);
  free(G.child_list); free(G.z); free(G.nrm); free(G.adj); free(G.label); free(G.mem_off);
  free(G.mem_list); free(c_own); free(t_own); free(S); free(eta); free(r); free(a_cor);
  free(gsize); free(a_eff); free(e_eff); free(emask); free(queue); free(order); free(cnt);
  free(tmp); free(xs); free(reach);
  return ORACLE_OK;
}

/* ------------------------------------------------------------- threads -- */

typedef struct {
  const oracle_batch* b;
  const oracle_params* p;
  oracle_outputs* o;
  int tid, nthreads;
  int status;
} worker_t;

static void* worker(void* arg) {
  worker_t* w = (worker_t*)arg;
  for (int g = w->tid; g < w->b->num_groups; g += w->nthreads) {
    const int st = run_group(w->b, w->p, w->o, g);
    if (st != ORACLE_OK) {
      w->status = st;
      break;
    }
  }
  return NULL;
}

int oracle_run(const oracle_batch* b, const oracle_params* p, oracle_outputs* o, int num_threads) {
  if (!p || !o) return ORACLE_ERR_INVALID_ARG;
  const int st = oracle_validate(b);
  if (st != ORACLE_OK) return st;
  if (!(p->w >= 0.0 && p->w <= 1.0) || !(p->lambda_eff >= 0.0) || !(p->std_eps >= 0.0) ||
      p->std_ddof < 0 || p->std_ddof > 1 || p->merge_rule < 0 || p->merge_rule > 1 ||
      !isfinite(p->kappa))
    return ORACLE_ERR_INVALID_ARG;
  if (num_threads < 1) num_threads = 1;
  if (num_threads > b->num_groups) num_threads = b->num_groups > 0 ? b->num_groups : 1;
  worker_t* ws = calloc(num_threads, sizeof(worker_t));
  pthread_t* th = calloc(num_threads, sizeof(pthread_t));
  if (!ws || !th) return ORACLE_ERR_NOMEM;
  for (int t = 0; t < num_threads; ++t) {
    ws[t] = (worker_t){b, p, o, t, num_threads, ORACLE_OK};
    if (t > 0) pthread_create(&th[t], NULL, worker, &ws[t]);
  }
  worker(&ws[0]);
  int out = ORACLE_OK;
  for (int t = 0; t < num_threads; ++t) {
    if (t > 0) pthread_join(th[t], NULL);
    if (ws[t].status != ORACLE_OK) out = ws[t].status;
  }
  free(ws);
  free(th);
  return out;
}
