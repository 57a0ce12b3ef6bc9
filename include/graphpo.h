/*
 * graphpo.h -- C ABI of the GB300 (sm_103a) GraphPO advantage-construction path.
 *
 * One call turns a batch of sampled rollout groups into per-token advantages:
 *
 *   state embeddings z_v, step boundaries, step lengths, binary rewards
 *     -> cosine similarity of every comparable state pair of a prompt group
 *        (tcgen05 tensor cores for bf16 embeddings)              GraphPO Sec. 4.2
 *     -> pairs with sim >= kappa linked into equivalence classes
 *        (union-find, class label = smallest state index)       Sec. 4.2, Alg. S.1
 *     -> pooled node scores S(v), Eq. (combain); step rewards
 *        r_step = (S(v) - S(p(v))) (1 - max(0, sim(p(v), v)))   Sec. 4.3
 *     -> correctness advantages over E_cor(u), efficiency advantages
 *        A_eff on every edge of the routes a_Q -> v              Sec. 4.4
 *     -> A_dual = A_cor + lambda_eff * A_eff on every token      Sec. 4.5
 *
 * Batch layout ("chain layout"): prompt group g owns rollouts
 * [group_rollout_off[g], group_rollout_off[g+1]); rollout r owns states
 * [rollout_step_off[r], rollout_step_off[r+1]) in step order (at least one);
 * state v is the node reached after the step that enters it, and that step is
 * the generated edge (p(v), v) with step_len[v] >= 1 tokens.  Its tokens are
 * packed per rollout: rollout r covers tokens [rollout_token_off[r],
 * rollout_token_off[r+1]) and the spans of its steps follow each other in step
 * order, so rollout_token_off[r+1] - rollout_token_off[r] = sum of its
 * step_len.  rollout_step_off[0] = rollout_token_off[0] = 0.
 *
 * Tree layout (branching rollouts, selected by parent != NULL; GraphPO Sec. 4.2
 * expands every active state of layer h-1 into b_h continuations, Algorithm S.1,
 * and its branching-schedule study): group g owns states [group_state_off[g],
 * group_state_off[g+1]) listed in depth-first pre-order, so that the subtree of a
 * state is the contiguous range that starts at it; parent[v] is the group-local
 * index of the generation predecessor p(v) (always < the state's own local index)
 * or -1 when p(v) is the prompt root.  The terminal states are the leaves of that
 * tree; the group's rollouts [group_rollout_off[g], group_rollout_off[g+1]) are
 * its leaves in state order and reward[r] is the verifier reward of leaf r (so
 * num_rollouts = number of leaves).  The tokens of every direct edge appear once:
 * group g covers tokens [group_token_off[g], group_token_off[g+1]) and the span of
 * the edge entering state v follows those of the group's earlier states, so
 * group_token_off[g+1] - group_token_off[g] = the group's sum of step_len.
 * rollout_step_off and rollout_token_off are not read (they may be NULL).  A
 * chain-layout batch written this way (every rollout a path from the root) gives
 * the same results.
 *
 * Memory: every array pointer in gpo_batch and gpo_outputs is DEVICE memory of
 * the current CUDA device, owned by the caller; the library never allocates
 * on the compute path.  The caller also provides the workspace
 * (gpo_workspace_size bytes, 256-byte aligned).  A context owns only a few
 * host-side bytes and one pinned status word.
 *
 * Errors: host-checkable problems (NULL pointers, bad sizes, parameters out of
 * range, misaligned embeddings, a too small workspace, a group larger than
 * GPO_MAX_GROUP_STATES) make gpo_compute return an error before anything is
 * enqueued.  Problems that need the device arrays (non-monotone offsets, step
 * lengths that do not tile a rollout's tokens, rewards outside {0,1},
 * non-finite embeddings; in the tree layout also parents that are not earlier
 * states, an order that is not a depth-first pre-order, or a leaf count that
 * differs from the group's rollout count) are found by the kernels, which then
 * skip the rest of the work; gpo_sync_status returns them.  Outputs are
 * undefined after any error.  No C++ exception, abort or device trap crosses
 * this interface.
 *
 * Threading: a context may be used by one host thread at a time; calls on
 * one context and one stream are ordered by the stream.  Calls that share a
 * workspace must be ordered on the GPU.
 */
#ifndef GRAPHPO_H
#define GRAPHPO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GPO_MAX_GROUP_STATES 4096 /* states of one prompt group (one CTA holds a group) */

typedef enum {
  GPO_OK = 0,
  GPO_ERR_INVALID_ARG = 1, /* NULL pointer, negative size, parameter out of range */
  GPO_ERR_SHAPE = 2,       /* offsets / step lengths / token spans inconsistent */
  GPO_ERR_BAD_REWARD = 3,  /* a reward is not 0 or 1 (GraphPO Sec. 4.3: R(z) in {0,1}) */
  GPO_ERR_NONFINITE = 4,   /* an embedding row is non-finite (or its squared norm overflows fp32) */
  GPO_ERR_UNSUPPORTED = 5, /* e.g. a group above GPO_MAX_GROUP_STATES, misaligned embeddings */
  GPO_ERR_CUDA = 6,        /* a CUDA runtime call failed; see gpo_last_error */
  GPO_ERR_TIMEOUT = 7,     /* a device-side wait gave up (the kernel returned cleanly) */
  GPO_ERR_WORKSPACE = 8,   /* workspace missing or smaller than gpo_workspace_size */
  GPO_ERR_BOUNDS = 9       /* debug build only (GPO_DEBUG): an index computed inside a kernel fell
                              outside its array; the access was skipped (the kernel and index are
                              in gpo_last_error) */
} gpo_status;

typedef enum {
  GPO_MERGE_NONCAUSAL = 0, /* compare every pair not in an ancestor-descendant relation
                              (Sec. 4.2); in chain layout: states of different rollouts */
  GPO_MERGE_SAME_DEPTH = 1 /* additionally require equal step depth (layer-wise merging) */
} gpo_merge_rule;

typedef enum { GPO_EMB_BF16 = 0, GPO_EMB_F32 = 1 } gpo_emb_dtype;

typedef struct {
  double kappa;      /* merge threshold, > 0: linked when sim >= kappa (Sec. 4.2; the paper
                        takes kappa in (0,1) and uses 0.92; kappa > 1 disables merging) */
  double w;          /* pooling coefficient in [0,1], Eq. (combain) (paper uses 0.7) */
  double lambda_eff; /* >= 0, weight of A_eff in A_dual (Sec. 4.5; paper gives no value) */
  double std_eps;    /* >= 0, added to every standard deviation (GRPO convention 1e-6) */
  int32_t std_ddof;  /* 1: sample standard deviation, 0: population */
  int32_t merge_rule;/* gpo_merge_rule */
  int32_t flags;     /* GPO_FLAG_* bits, 0 by default */
} gpo_params;

/* Compute the pairwise similarities of bf16 embeddings on the CUDA cores (fp32
 * FMA) instead of the tcgen05 tensor cores; fp32 embeddings always use them. */
#define GPO_FLAG_SIMT_SIMILARITY 1
/* Use the multi-kernel tiled path even when every group fits a group-resident
 * kernel (bf16 embeddings with max_states_per_group <= 384, or fp32 embeddings in
 * the chain layout with small groups, see gpo_compute_groups); for comparisons
 * and tests. */
#define GPO_FLAG_TILED 2
/* For tests of the failure path only: in every CTA of the tensor-core kernels the MMA warp's
 * first wait runs out (it waits about a millisecond on an mbarrier that nothing arrives on),
 * as a stalled copy or MMA would make it; the kernel then reports GPO_ERR_TIMEOUT and winds
 * down as it does after any timed-out wait (copies in flight land, issued MMAs complete,
 * TMEM is released).  gpo_sync_status returns GPO_ERR_TIMEOUT; outputs are undefined; the
 * CUDA context stays usable.  Paths without tensor-core kernels (fp32 embeddings,
 * GPO_FLAG_SIMT_SIMILARITY) ignore the flag. */
#define GPO_FLAG_DEBUG_TIMEOUT 4

typedef struct {
  int32_t num_groups;     /* G >= 0 */
  int32_t num_rollouts;   /* R >= 0 */
  int32_t num_states;     /* N >= 0 */
  int32_t d;              /* embedding width >= 1 */
  int32_t emb_dtype;      /* gpo_emb_dtype */
  int32_t max_states_per_group; /* upper bound on any group's state count (sizes the workspace) */
  int64_t emb_row_stride; /* elements between rows; row bytes must be a multiple of 16 */
  int64_t total_tokens;   /* T = rollout_token_off[R] (tree layout: group_token_off[G]) */
  const int32_t* group_rollout_off; /* [G+1] */
  const int32_t* rollout_step_off;  /* [R+1] */
  const int32_t* step_len;          /* [N] */
  const int64_t* rollout_token_off; /* [R+1] */
  const void* emb;                  /* [N x emb_row_stride], 16-byte aligned */
  const uint8_t* reward;            /* [R] verifier rewards in {0,1} */
  const void* root_emb;             /* optional [G x emb_row_stride] prompt embeddings; NULL:
                                       eta on the first step of every rollout is 0 */
  /* Tree layout only (all three NULL for the chain layout): */
  const int32_t* parent;            /* [N] group-local index of p(v), -1 = the prompt root */
  const int32_t* group_state_off;   /* [G+1] states of each group, pre-order */
  const int64_t* group_token_off;   /* [G+1] packed token span of each group */
} gpo_batch;

typedef struct {
  float* adv;         /* [T] required: A_dual of the edge holding each token */
  float* adv_cor;     /* [T] optional: A_cor of the edge */
  float* adv_eff;     /* [T] optional: efficiency advantage routed through the edge (no lambda) */
  uint8_t* eff_mask;  /* [T] optional: 1 where some route a_Q -> v covers the edge */
  int32_t* class_id;  /* [N] optional: smallest state index of the state's class */
  float* node_score;  /* [N] optional: pooled score S(v) */
  float* edge_adv;    /* [N] optional: A_dual of the edge entering each state */
  /* Per-edge components, the inputs of the split loss form (gpo_token_loss): */
  float* edge_cor;       /* [N] optional: A_cor of the edge entering each state */
  float* edge_eff;       /* [N] optional: efficiency advantage routed through that edge (no lambda) */
  uint8_t* edge_eff_mask;/* [N] optional: 1 where some route a_Q -> v covers that edge */
  /* Exploration efficiency, GraphPO Eq. (eq1): tokens of the steps from which a correct
   * final answer can be reached / tokens of all steps of the group (0 for a group without
   * states).  Tree reading: a correct terminal lies below the step's state (c_own > 0; in
   * the chain layout: the rollout is correct, each trajectory counted as one step).  Graph
   * reading: reachable along direct edges and through merged states (a class reaches a
   * correct answer when a member is, or has a child whose class is, such a state). */
  float* group_eff;       /* [G] optional: tree reading */
  float* group_eff_graph; /* [G] optional: graph reading */
} gpo_outputs;

typedef struct gpo_ctx gpo_ctx;

/* Creates a context for the current CUDA device.  Returns GPO_ERR_INVALID_ARG
 * for parameters out of range, GPO_ERR_UNSUPPORTED if the device is not
 * sm_103, GPO_ERR_CUDA if the runtime fails. */
gpo_status gpo_create(gpo_ctx** ctx, const gpo_params* params);

/* Bytes of device workspace gpo_compute needs for batches of this shape.
 * Reads only the host-side sizes of `batch` and the nullness and alignment of
 * its pointers (no device access), and returns the status gpo_compute would
 * give for those checks.  `ctx` may be NULL (no device or context needed);
 * with a context, the reason for a failure is left in gpo_last_error. */
gpo_status gpo_workspace_size(const gpo_ctx* ctx, const gpo_batch* batch, size_t* bytes);

/* Enqueues the whole path on `stream` (a cudaStream_t; NULL = legacy default
 * stream).  Asynchronous: returns once the kernels are enqueued. */
gpo_status gpo_compute(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out,
                       void* workspace, size_t workspace_bytes, void* stream);

/* The path for prompt groups [first_group, first_group + num_groups) only (the
 * paper has no counterpart: it lets a caller overlap the upload of later
 * groups' embeddings with the work on earlier ones).  `batch` and `out`
 * describe the WHOLE batch, with the same layout, ownership and checks as for
 * gpo_compute; only the listed groups' embedding rows must hold their values
 * when the call runs on the GPU, and only their tokens and states are written
 * (a group's tokens are all written by the call that covers the group).
 * clear_status != 0 clears the workspace's status words first; calls for later
 * ranges add to them, so that one gpo_sync_status after the last range reports
 * the first error of any.  num_groups = 0 with clear_status = 1 only clears.
 * Calls for disjoint ranges may run concurrently on different streams once the
 * clearing call has completed; they share the workspace's status words only.
 * A range other than the whole batch needs a group-resident path -- bf16
 * embeddings with max_states_per_group <= 384, or fp32 embeddings in the chain
 * layout with max_states_per_group <= 128 and max_states_per_group x
 * (d rounded up to 32, plus 4) floats within 160 KiB; no flags -- otherwise
 * GPO_ERR_UNSUPPORTED.  A range outside [0, num_groups] gives
 * GPO_ERR_INVALID_ARG. */
gpo_status gpo_compute_groups(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out, int64_t first_group,
                              int64_t num_groups, int clear_status, void* workspace, size_t workspace_bytes,
                              void* stream);

/* End-to-end variant for a batch held in HOST memory (the paper has no counterpart: it
 * lets a caller whose rollouts and embeddings arrive in host memory overlap their upload
 * with the work, and take the per-token advantages back into host memory).
 *   host      the batch, every array in host memory: pinned (page-locked) memory for the
 *             copies to be asynchronous and overlap; pageable memory works but each copy
 *             then completes before the call goes on.  The host arrays must stay valid
 *             and unchanged until `stream` reaches the end of this call's work.
 *   dev       the same batch's device staging buffers: identical sizes, layout and row
 *             stride, every array pointer a device buffer of the same size as its host
 *             array, owned by the caller; the library copies the host arrays into them.
 *   out       device outputs as for gpo_compute (adv required; optional outputs are
 *             written on the device, not copied back).
 *   host_adv  host array of total_tokens floats that receives out->adv.
 *   chunk_bytes  about how many bytes of embeddings one pipeline stage uploads
 *             (0: the larger of 8 MiB and a tenth of the embeddings; a value above the
 *             embeddings' size: one stage).
 * Enqueues, in order of `stream`: the small arrays' uploads, then the groups in chunks of
 * about equal state counts -- chunk k's embeddings are uploaded while earlier chunks run,
 * and each chunk's advantages are copied to host_adv once they are ready -- on helper
 * streams of the context that rejoin `stream` at the end (so work enqueued later on
 * `stream`, such as gpo_sync_status, follows all of it).  The chunks are the calls of
 * gpo_compute_groups and need the group-resident path (bf16 embeddings,
 * max_states_per_group <= 384, no flags) and host offsets that partition the batch;
 * otherwise: one upload, gpo_compute and one download, all on `stream`.  The first
 * pipelined call on a context creates its helper streams and events (released by
 * gpo_destroy).  Checks and errors as for gpo_compute, plus GPO_ERR_INVALID_ARG when the
 * two batches differ in size or layout or a host array is NULL. */
gpo_status gpo_compute_host(gpo_ctx* ctx, const gpo_batch* host, const gpo_batch* dev, const gpo_outputs* out,
                            float* host_adv, int64_t chunk_bytes, void* workspace, size_t workspace_bytes,
                            void* stream);

/* Waits for `stream` and returns the first error the kernels of the last
 * gpo_compute (or of the gpo_compute_groups calls since the last clearing one)
 * on this context reported (GPO_OK if none). */
gpo_status gpo_sync_status(gpo_ctx* ctx, void* stream);

/* Static description of a status code. */
const char* gpo_status_string(gpo_status status);

/* Last error message recorded on the context (never NULL). */
const char* gpo_last_error(const gpo_ctx* ctx);

/* Per-stage device timing (instrumentation; the paper has no counterpart).
 * When enabled, gpo_compute records a CUDA event on the stream before the
 * first and after every kernel it launches.  gpo_stage_times waits for the
 * last of those events and writes, for each stage of the last gpo_compute, its
 * name and its device time in milliseconds (names stay valid for the
 * context's lifetime).  Stages not launched report 0.  Returns
 * GPO_ERR_INVALID_ARG if timing was not enabled or capacity is too small. */
gpo_status gpo_enable_timing(gpo_ctx* ctx, int enable);
gpo_status gpo_stage_times(gpo_ctx* ctx, float* ms, const char** names, int capacity, int* count);

/* Allocation-free variant of gpo_compute (the paper has no counterpart).
 * For callers that cannot allocate device memory when they need the
 * advantages -- a trainer whose device memory is all owned by a framework
 * pool, a plug-in whose host forbids allocation calls, a loop that cannot take
 * cudaMalloc's implicit synchronisation.  Same inputs and outputs as
 * gpo_compute, but the workspace is one array of GPO_NOALLOC_SCRATCH_BYTES
 * compiled into the library; it calls no cudaMalloc/cudaFree.  The array
 * belongs to a CUDA context, not to a device: it is reserved in the current
 * context when this library's device code is first loaded there (at the latest
 * by the first gpo_compute_noalloc call in that context) and stays there until
 * the context is destroyed; every context has its own.  The first call in a
 * context looks up the array's address in that context (it is cached per
 * context, so other contexts and a new primary context after a device reset
 * get their own); make that first call before any stream capture.  Batches
 * whose gpo_workspace_size exceeds GPO_NOALLOC_SCRATCH_BYTES are rejected with
 * GPO_ERR_WORKSPACE before anything is enqueued.  All calls in one context
 * share the array: calls that overlap on the GPU race and must be ordered by
 * the caller.  Errors and gpo_sync_status behave as for gpo_compute. */
#define GPO_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)
gpo_status gpo_compute_noalloc(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out, void* stream);

/* Next-layer budgets of layer-by-layer graph construction (GraphPO Sec. 4.2: a path
 * that reaches an existing equivalence class has its next-layer budget halved, keeping
 * at least one continuation, and the saved budget is reallocated; Algorithm S.1 Stage 1:
 * after layer h is sampled, every non-causal pair is linked and the saved budget goes
 * to the active frontier states that are not redundant).
 *
 * `batch`: the tree layout of the states sampled so far (depth <= layer), its leaves
 * as the rollouts (their rewards are not used but must be 0 or 1); the similarity part
 * runs as in gpo_compute (same parameters, workspace size and checks).
 * Per group:
 *   frontier   the states of depth `layer` with active[v] != 0 (active NULL: all)
 *   redundant  a frontier state whose class holds a state registered before it: one of
 *              an earlier layer, or one of the same layer with a smaller index
 *   budget[v]  b_next for a non-redundant frontier state, max(1, b_next / 2) for a
 *              redundant one, 0 for every other state; the saved budget (the redundant
 *              count times b_next - max(1, b_next / 2)) is split over the k non-redundant
 *              frontier states: saved / k each plus one for the first saved % k of them
 *              by index (with k = 0 it is not spent)
 *   class_id   optional [N]: the classes of all states sampled so far (as gpo_compute)
 * After the last layer the classes equal those of gpo_compute on the whole batch (every
 * non-causal pair has been compared once).  1 <= layer, 1 <= b_next <= 65536; the chain
 * layout gives GPO_ERR_UNSUPPORTED.  Asynchronous; device-side errors via
 * gpo_sync_status as for gpo_compute. */
gpo_status gpo_layer_budget(gpo_ctx* ctx, const gpo_batch* batch, int32_t layer, int32_t b_next,
                            const uint8_t* active, int32_t* budget, int32_t* class_id, void* workspace,
                            size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Policy loss on per-token log-probabilities (GraphPO Sec. 4.5: the objective
 * J_GraphPO, DAPO's clipped surrogate on the graph advantage averaged over each
 * edge's tokens and each prompt graph's edges; Algorithm S.1 Stage 4: the split
 * form with separate correctness and efficiency terms).  The paper has no
 * counterpart of the plan; the loss itself is what a trainer minimises after
 * gpo_compute, once per optimiser step.
 *
 *   J = 1/G' sum_g 1/|E_g| sum_{e in E_g} 1/|e| sum_{t in e} (f_t - beta k_t)
 *                                                       (GPO_LOSS_NORM_EDGE)
 *   J = 1/T sum_t (f_t - beta k_t)                      (GPO_LOSS_NORM_TOKEN: DAPO's token mean)
 *   phi(A) = min(r_t A, clip(r_t, 1 - clip_low, 1 + clip_high) A),
 *   r_t = exp(logp_t - old_logp_t)
 *   dual form:  f_t = phi(A_dual(e))                      (gpo_outputs.edge_adv)
 *   split form: f_t = phi(A_cor(e)) + lambda_eff m_eff(e) phi(A_eff(e))
 *               (gpo_outputs.edge_cor, edge_eff, edge_eff_mask)
 *   k_t = exp(x) - x - 1, x = ref_logp_t - logp_t (the k3 estimate of KL(pi_theta || pi_ref))
 *   loss = -J;  grad_logp[t] = d loss / d logp_t, taken where the min picks the
 *   unclipped term (r A <= clip(r) A) and 0 where the clipped term is smaller
 *
 * G' = groups with at least one state, |E_g| = the states of group g (one direct
 * edge enters each state), |e| = step_len of the edge's state, e the edge holding
 * token t in the batch's token layout (that of gpo_compute's per-token outputs).
 * The entropy bonus of Algorithm S.1 needs the whole vocabulary distribution and
 * is left to the caller.
 */
typedef enum { GPO_LOSS_DUAL = 0, GPO_LOSS_SPLIT = 1 } gpo_loss_form;
typedef enum { GPO_LOSS_NORM_EDGE = 0, GPO_LOSS_NORM_TOKEN = 1 } gpo_loss_norm;

typedef struct {
  double clip_low;   /* in [0, 1): lower clip bound 1 - clip_low (the paper: 0.2) */
  double clip_high;  /* >= 0: upper clip bound 1 + clip_high (the paper: 0.2; DAPO raises it) */
  double beta_kl;    /* >= 0: weight of the KL estimate (0: ref_logp is not read) */
  double lambda_eff; /* >= 0: split form's weight of the efficiency term */
  int32_t form;      /* gpo_loss_form */
  int32_t norm;      /* gpo_loss_norm */
} gpo_loss_params;

typedef struct {
  const float* logp;          /* [T] log pi_theta of every token, 16-byte aligned */
  const float* old_logp;      /* [T] log pi_theta_old (the sampling policy), 16-byte aligned */
  const float* ref_logp;      /* [T] log pi_ref, 16-byte aligned; read only when beta_kl > 0 */
  const float* edge_adv;      /* [N] dual form: A_dual of the edge entering each state */
  const float* edge_cor;      /* [N] split form: A_cor */
  const float* edge_eff;      /* [N] split form: routed A_eff (no lambda) */
  const uint8_t* edge_eff_mask; /* [N] split form: m_eff */
} gpo_loss_inputs;

#define GPO_LOSS_NSTATS 4
typedef struct {
  float* loss;       /* [1] required: -J */
  float* grad_logp;  /* [T] optional: d loss / d logp, 16-byte aligned */
  double* stats;     /* [GPO_LOSS_NSTATS] optional: the policy term sum w f, the KL term sum w k
                        (0 when beta_kl = 0), the number of tokens whose (first) surrogate took
                        the clipped branch, the token mean of r */
} gpo_loss_outputs;

/* Bytes of a loss plan for batches of this shape (reads the host-side sizes only). */
gpo_status gpo_loss_plan_size(const gpo_batch* batch, size_t* bytes);

/* Builds a loss plan (the first token and the weight of every edge, the first edge of
 * every token tile) from the batch's structure: the offsets and step_len (embeddings and
 * rewards are not read).  `plan`: device memory of gpo_loss_plan_size bytes, 256-byte
 * aligned, owned by the caller.  Asynchronous on `stream`; layout errors the kernels find
 * (as for gpo_compute) are returned by gpo_sync_status, and gpo_token_loss calls on that
 * plan then leave their outputs unwritten.  A plan serves every gpo_token_loss call on
 * the same batch structure.  It also holds those calls' reduction scratch: calls that
 * share a plan must be ordered on the GPU. */
gpo_status gpo_loss_plan(gpo_ctx* ctx, const gpo_batch* batch, void* plan, size_t plan_bytes, void* stream);

/* Enqueues the loss, its gradient and statistics on `stream` (one kernel; the token
 * tiles' reductions are combined in a fixed order, so results are deterministic).
 * Host-checked: parameters, NULL inputs for the chosen form, alignment
 * (GPO_ERR_UNSUPPORTED), plan size. */
gpo_status gpo_token_loss(gpo_ctx* ctx, const gpo_batch* batch, void* plan, const gpo_loss_params* params,
                          const gpo_loss_inputs* in, const gpo_loss_outputs* out, void* stream);

/* Library version string. */
const char* gpo_version(void);

void gpo_destroy(gpo_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* GRAPHPO_H */
