/*
 * GraphPO advantage construction -- CPU ORACLE (test infrastructure only).
 *
 * A plain, slow, fp64 statement of what the method computes, written from the
 * paper (GraphPO: Sec. 4.2 graph construction, Sec. 4.3 graph reward, Sec. 4.4
 * dual-group advantage, Sec. 4.5 token-level objective, Algorithm S.1).  It is
 * used only by the tests, by the smoke check and by the benchmark's CPU
 * baseline; the product path never links or calls it.  It shares no code with
 * the CUDA path.
 *
 * Input layout ("chain layout"): each rollout r of prompt group g is a chain
 * root -> s_1 -> ... -> s_{n_r}; state (r, h) is the node reached after step h
 * and that step is the direct edge entering it.  Arrays are host memory:
 *   group_rollout_off int32[G+1], rollout_step_off int32[R+1],
 *   step_len int32[N], rollout_token_off int64[R+1], reward uint8[R],
 *   emb [N x d] (bf16 bit patterns or float32, row stride emb_row_stride
 *   elements), root_emb [G x d] optional (NULL: eta on root edges is 0).
 *
 * Tree layout (branching rollouts, GraphPO Sec. 4.2 layer-by-layer expansion
 * with a branching schedule; selected by parent != NULL): group g owns states
 * [group_state_off[g], group_state_off[g+1]) in depth-first pre-order (every
 * subtree is a contiguous range starting at its top state); parent[v] is the
 * group-local index of p(v), or -1 when p(v) is the prompt root.  The
 * terminal states are the leaves; the group's rollouts [group_rollout_off[g],
 * group_rollout_off[g+1]) are its leaves in state order and reward[r] is the
 * verifier reward of leaf r.  Every direct edge's tokens appear once (the
 * objective of Sec. 4.5 sums over direct edges): group g covers tokens
 * [group_token_off[g], group_token_off[g+1]) and edge v's span follows those
 * of the group's earlier states.  rollout_step_off and rollout_token_off are
 * not read.
 *
 * All outputs are optional (NULL = not wanted); per-token arrays are packed
 * like the input tokens, per-edge arrays are indexed by the state the edge
 * enters.
 */
#ifndef GRAPHPO_ORACLE_H
#define GRAPHPO_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  ORACLE_OK = 0,
  ORACLE_ERR_INVALID_ARG = 1,
  ORACLE_ERR_SHAPE = 2,
  ORACLE_ERR_BAD_REWARD = 3,
  ORACLE_ERR_NONFINITE = 4,
  ORACLE_ERR_NOMEM = 5
};

typedef struct {
  int32_t num_groups, num_rollouts, num_states, d;
  int32_t emb_is_bf16;       /* 1: uint16 bf16 bit patterns, 0: float32 */
  int64_t emb_row_stride;    /* elements between consecutive rows */
  int64_t total_tokens;
  const int32_t* group_rollout_off;
  const int32_t* rollout_step_off;
  const int32_t* step_len;
  const int64_t* rollout_token_off;
  const void* emb;
  const uint8_t* reward;
  const void* root_emb;      /* optional, same dtype and stride as emb */
  const int32_t* parent;          /* tree layout: [N] group-local p(v), -1 = root; NULL = chain */
  const int32_t* group_state_off; /* tree layout: [G+1] */
  const int64_t* group_token_off; /* tree layout: [G+1] */
} oracle_batch;

typedef struct {
  double kappa;      /* merge threshold on cosine similarity (inclusive) */
  double w;          /* pooling coefficient, Eq. (combain) */
  double lambda_eff; /* efficiency weight in A_dual */
  double std_eps;    /* added to every standard deviation */
  int32_t std_ddof;  /* 1: sample std, 0: population std */
  int32_t merge_rule;/* 0: any non-ancestor pair (paper); 1: additionally same depth */
} oracle_params;

typedef struct {
  double* adv;            /* [T] A_dual on every token */
  double* adv_cor;        /* [T] A_cor on every token */
  double* adv_eff;        /* [T] distributed efficiency advantage (before lambda) */
  uint8_t* eff_mask;      /* [T] 1 where some efficiency route covers the edge */
  int32_t* class_id;      /* [N] smallest state index of the equivalence class */
  double* node_score;     /* [N] pooled score S(v) */
  double* root_score;     /* [G] S(root) */
  double* eta;            /* [N] eta(p(v), v) */
  double* step_reward;    /* [N] r_step(p(v), v) */
  double* a_cor;          /* [N] correctness advantage of edge (p(v), v) */
  double* a_eff_node;     /* [N] path-level A_eff(v); 0 when |Q(v)| < 2 */
  double* e_eff;          /* [N] sum of A_eff routed through edge (p(v), v) */
  double* edge_adv;       /* [N] A_dual of edge (p(v), v) */
  uint8_t* edge_eff_mask; /* [N] */
  int32_t* cor_group_size;/* [N] size of the correctness group holding the edge */
  double* eff_tree;       /* [G] exploration efficiency Eff, Eq. (eq1): a step is correct when a
                             correct terminal is reachable from it along direct edges */
  double* eff_graph;      /* [G] the same with reachability in the merged (quotient) graph */
} oracle_outputs;

/* Runs the whole path on `num_threads` host threads (groups are independent).
 * Returns ORACLE_OK or an ORACLE_ERR_* code (outputs undefined then). */
int oracle_run(const oracle_batch* b, const oracle_params* p, oracle_outputs* o,
               int num_threads);

/* Validation only (same checks as oracle_run). */
int oracle_validate(const oracle_batch* b);

#ifdef __cplusplus
}
#endif
#endif
