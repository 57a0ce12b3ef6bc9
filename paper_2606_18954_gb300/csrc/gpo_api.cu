// Host implementation of the C ABI declared in include/graphpo.h: argument
// checks, workspace layout, TMA descriptor encoding and the launch sequence
//   prep (validate + plan) -> row stats -> similarity merge -> per-group
//   advantages -> per-token scatter
// all on the caller's stream.  Nothing here allocates device memory.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include <algorithm>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "gpo_internal.cuh"

struct gpo_ctx {
  gpo_params params;
  int device;
  int num_sms;
  uint32_t* host_status;      // pinned copy of the workspace status words
  const uint32_t* last_status; // device status words of the last gpo_compute
  char msg[512];
  bool timing;
  int nstages;                 // stages recorded by the last gpo_compute
  cudaEvent_t ev[gpo::kMaxStages + 1];
  const char* stage_name[gpo::kMaxStages];
  // gpo_compute_host: helper streams and events (created by its first pipelined call) and
  // the per-group state and token offsets of the last host batch
  bool pipe_ready;
  cudaStream_t pipe_in, pipe_out, pipe_comp[gpo::kPipeComputeStreams];
  cudaEvent_t pipe_ev[2 * gpo::kPipeMaxChunks + 2];
  std::vector<int64_t> pipe_s, pipe_t;
};

namespace gpo {
namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

void set_msg(gpo_ctx* c, const char* fmt, ...) {
  if (!c) return;
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(c->msg, sizeof c->msg, fmt, ap);
  va_end(ap);
}

constexpr size_t kAlign = 256;
inline size_t up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

int64_t max_blocks_for(int64_t N, int64_t G) { return N / 128 + G + 8; }  // sum of ceil(n/128)

int64_t max_items_for(int64_t N, int64_t G, int64_t maxn) {
  // per group: ceil(n/128) diagonal items plus the off-diagonal chunks of 256 columns,
  // at most n^2/32768 + 3n/256 + 1
  return N * maxn / 32768 + (3 * N) / 256 + G + max_blocks_for(N, G);
}

struct Layout {
  size_t status, items, blk_ready, groups, state_meta, nrm2, rn, edge_count,
      edges, e_adv, e_cor, e_eff, e_mask, tok_start, tree_par, tree_end, tree_own, tree_x, x_n2, x_dot, x_root_n2,
      total;
  int max_items;
  bool tree;
};

// 4-byte words of the tree layout's group-math sums: tree_scratch_words(n) = 23 n + 11 per group
constexpr int64_t kTreeWordsPerState = 23, kTreeWordsPerGroup = 11;

bool layout(const gpo_batch& b, Layout& L) {
  const int64_t G = b.num_groups, R = b.num_rollouts, N = b.num_states;
  const int64_t mi = max_items_for(N, G, b.max_states_per_group);
  if (mi > (1 << 30)) return false;
  L.max_items = (int)mi;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = up(o + bytes);
    return at;
  };
  L.status = take(sizeof(uint32_t) * kStatusWords);
  L.items = take(sizeof(Item) * mi);
  L.blk_ready = take(sizeof(int) * mi);  // indexed by the diagonal items' positions
  L.groups = take(sizeof(GroupInfo) * G);
  L.state_meta = take(sizeof(int2) * N);
  L.nrm2 = take(sizeof(float) * N);
  L.rn = take(sizeof(float) * N);
  L.edge_count = take(sizeof(int) * mi);
  L.edges = take(sizeof(int2) * (size_t)kEdgeCap * mi);
  L.e_adv = take(sizeof(float) * N);
  L.e_cor = take(sizeof(float) * N);
  L.e_eff = take(sizeof(float) * N);
  L.e_mask = take(N);
  L.tok_start = take(sizeof(int64_t) * N);
  L.x_n2 = take(sizeof(float2) * N);
  L.x_dot = take(sizeof(float2) * N);
  L.x_root_n2 = take(sizeof(float2) * G);
  L.tree = b.parent != nullptr;
  if (L.tree) {
    L.tree_par = take(sizeof(int) * N);
    L.tree_end = take(sizeof(int) * N);
    L.tree_own = take(sizeof(int2) * N);
    L.tree_x = take(4 * (size_t)(kTreeWordsPerState * N + kTreeWordsPerGroup * G));
  }
  L.total = o;
  return true;
}

Ws workspace_views(void* base, const Layout& L) {
  unsigned char* p = static_cast<unsigned char*>(base);
  Ws w;
  w.status = reinterpret_cast<uint32_t*>(p + L.status);
  w.items = reinterpret_cast<Item*>(p + L.items);
  w.blk_ready = reinterpret_cast<int*>(p + L.blk_ready);
  w.groups = reinterpret_cast<GroupInfo*>(p + L.groups);
  w.state_meta = reinterpret_cast<int2*>(p + L.state_meta);
  w.nrm2 = reinterpret_cast<float*>(p + L.nrm2);
  w.rn = reinterpret_cast<float*>(p + L.rn);
  w.edge_count = reinterpret_cast<int*>(p + L.edge_count);
  w.edges = reinterpret_cast<int2*>(p + L.edges);
  w.e_adv = reinterpret_cast<float*>(p + L.e_adv);
  w.e_cor = reinterpret_cast<float*>(p + L.e_cor);
  w.e_eff = reinterpret_cast<float*>(p + L.e_eff);
  w.e_mask = p + L.e_mask;
  w.tok_start = reinterpret_cast<int64_t*>(p + L.tok_start);
  w.tree_par = L.tree ? reinterpret_cast<int*>(p + L.tree_par) : nullptr;
  w.tree_end = L.tree ? reinterpret_cast<int*>(p + L.tree_end) : nullptr;
  w.tree_own = L.tree ? reinterpret_cast<int2*>(p + L.tree_own) : nullptr;
  w.tree_x = L.tree ? reinterpret_cast<int*>(p + L.tree_x) : nullptr;
  w.x_n2 = reinterpret_cast<float2*>(p + L.x_n2);
  w.x_dot = reinterpret_cast<float2*>(p + L.x_dot);
  w.x_root_n2 = reinterpret_cast<float2*>(p + L.x_root_n2);
  w.max_items = L.max_items;
  return w;
}

gpo_status check_params(const gpo_params& p) {
  if (!std::isfinite(p.kappa) || !(p.kappa > 0.0) || !(p.w >= 0.0 && p.w <= 1.0) || !(p.lambda_eff >= 0.0) ||
      !std::isfinite(p.lambda_eff) || !(p.std_eps >= 0.0) || !std::isfinite(p.std_eps) || p.std_ddof < 0 ||
      p.std_ddof > 1 || p.merge_rule < 0 || p.merge_rule > 1 || (p.flags & ~(GPO_FLAG_SIMT_SIMILARITY | GPO_FLAG_TILED | GPO_FLAG_DEBUG_TIMEOUT)))
    return GPO_ERR_INVALID_ARG;
  return GPO_OK;
}

inline bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

gpo_status check_batch(gpo_ctx* c, const gpo_batch* b) {
  if (!b) return set_msg(c, "batch is NULL"), GPO_ERR_INVALID_ARG;
  if (b->num_groups < 0 || b->num_rollouts < 0 || b->num_states < 0 || b->total_tokens < 0 || b->d < 1 ||
      b->max_states_per_group < 0)
    return set_msg(c, "negative size or d < 1"), GPO_ERR_INVALID_ARG;
  if (b->emb_dtype != GPO_EMB_BF16 && b->emb_dtype != GPO_EMB_F32)
    return set_msg(c, "unknown emb_dtype %d", b->emb_dtype), GPO_ERR_INVALID_ARG;
  if (b->max_states_per_group > GPO_MAX_GROUP_STATES)
    return set_msg(c, "max_states_per_group %d above %d", b->max_states_per_group, GPO_MAX_GROUP_STATES),
           GPO_ERR_UNSUPPORTED;
  if (b->num_states > 0 && b->max_states_per_group < 1)
    return set_msg(c, "max_states_per_group must be >= 1"), GPO_ERR_INVALID_ARG;
  if (b->num_rollouts > b->num_states) return set_msg(c, "more rollouts than states"), GPO_ERR_SHAPE;
  if (b->emb_row_stride < b->d) return set_msg(c, "emb_row_stride < d"), GPO_ERR_INVALID_ARG;
  const int64_t esz = b->emb_dtype == GPO_EMB_BF16 ? 2 : 4;
  if ((b->emb_row_stride * esz) % 16 != 0)
    return set_msg(c, "embedding row bytes must be a multiple of 16"), GPO_ERR_UNSUPPORTED;
  if (b->parent) {
    if (!b->group_rollout_off || !b->group_state_off || !b->group_token_off)
      return set_msg(c, "tree layout: an offset array is NULL"), GPO_ERR_INVALID_ARG;
  } else if (b->group_state_off || b->group_token_off) {
    return set_msg(c, "group_state_off / group_token_off given without parent"), GPO_ERR_INVALID_ARG;
  } else if (!b->group_rollout_off || !b->rollout_step_off || !b->rollout_token_off) {
    return set_msg(c, "offset array is NULL"), GPO_ERR_INVALID_ARG;
  }
  if (b->num_states > 0 && (!b->step_len || !b->emb)) return set_msg(c, "step_len/emb NULL"), GPO_ERR_INVALID_ARG;
  if (b->num_rollouts > 0 && !b->reward) return set_msg(c, "reward NULL"), GPO_ERR_INVALID_ARG;
  if ((b->emb && !aligned(b->emb, 16)) || (b->root_emb && !aligned(b->root_emb, 16)))
    return set_msg(c, "embeddings must be 16-byte aligned"), GPO_ERR_UNSUPPORTED;
  if (b->emb_row_stride >= (int64_t)1 << 40 || (int64_t)b->num_states * b->emb_row_stride >= (int64_t)1 << 40)
    return set_msg(c, "embedding matrix too large"), GPO_ERR_UNSUPPORTED;
  return GPO_OK;
}

gpo_status check_outputs(gpo_ctx* c, const gpo_batch* b, const gpo_outputs* o) {
  if (!o) return set_msg(c, "outputs is NULL"), GPO_ERR_INVALID_ARG;
  if (b->total_tokens > 0 && !o->adv) return set_msg(c, "adv output is NULL"), GPO_ERR_INVALID_ARG;
  if (!aligned(o->adv, 16) || !aligned(o->adv_cor, 16) || !aligned(o->adv_eff, 16) || !aligned(o->eff_mask, 4))
    return set_msg(c, "token outputs must be 16-byte (eff_mask 4-byte) aligned"), GPO_ERR_UNSUPPORTED;
  return GPO_OK;
}

}  // namespace

void note_error(gpo_ctx* ctx, const char* msg) { set_msg(ctx, "%s", msg); }

}  // namespace gpo

using namespace gpo;

extern "C" {

#ifdef GPO_DEBUG
const char* gpo_version(void) { return "graphpo-gb300 0.1 (sm_103a, GPO_DEBUG bounds checks)"; }
#else
const char* gpo_version(void) { return "graphpo-gb300 0.1 (sm_103a)"; }
#endif

const char* gpo_status_string(gpo_status s) {
  switch (s) {
    case GPO_OK: return "ok";
    case GPO_ERR_INVALID_ARG: return "invalid argument";
    case GPO_ERR_SHAPE: return "inconsistent offsets, step lengths or token spans";
    case GPO_ERR_BAD_REWARD: return "reward outside {0,1}";
    case GPO_ERR_NONFINITE: return "non-finite embedding";
    case GPO_ERR_UNSUPPORTED: return "unsupported input or device";
    case GPO_ERR_CUDA: return "CUDA runtime error";
    case GPO_ERR_TIMEOUT: return "device-side wait timed out";
    case GPO_ERR_WORKSPACE: return "workspace missing or too small";
    case GPO_ERR_BOUNDS: return "index out of bounds inside a kernel (debug build)";
  }
  return "unknown status";
}

const char* gpo_last_error(const gpo_ctx* ctx) { return ctx ? ctx->msg : "no context"; }

gpo_status gpo_create(gpo_ctx** out, const gpo_params* params) {
  if (!out || !params) return GPO_ERR_INVALID_ARG;
  *out = nullptr;
  if (check_params(*params) != GPO_OK) return GPO_ERR_INVALID_ARG;
  gpo_ctx* c = new (std::nothrow) gpo_ctx();
  if (!c) return GPO_ERR_CUDA;
  c->params = *params;
  c->last_status = nullptr;
  c->msg[0] = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&c->device) != cudaSuccess || cudaGetDeviceProperties(&prop, c->device) != cudaSuccess) {
    delete c;
    return GPO_ERR_CUDA;
  }
  if (!(prop.major == 10 && prop.minor == 3)) {
    delete c;
    return GPO_ERR_UNSUPPORTED;
  }
  c->num_sms = prop.multiProcessorCount;
  c->timing = false;
  c->pipe_ready = false;
  c->nstages = 0;
  for (int i = 0; i <= kMaxStages; ++i) {
    if (cudaEventCreate(&c->ev[i]) != cudaSuccess) {
      cudaGetLastError();
      delete c;
      return GPO_ERR_CUDA;
    }
  }
  if (setup_sim_tc() != cudaSuccess || setup_groups() != cudaSuccess || setup_fused() != cudaSuccess ||
      setup_fused_f32() != cudaSuccess ||
      setup_tree_prep() != cudaSuccess || setup_loss() != cudaSuccess ||
      cudaMallocHost(&c->host_status, sizeof(uint32_t) * kStatusWords) != cudaSuccess) {
    cudaGetLastError();
    delete c;
    return GPO_ERR_CUDA;
  }
  *out = c;
  return GPO_OK;
}

void gpo_destroy(gpo_ctx* ctx) {
  if (!ctx) return;
  if (ctx->pipe_ready) {
    cudaStreamDestroy(ctx->pipe_in);
    cudaStreamDestroy(ctx->pipe_out);
    for (cudaStream_t cs : ctx->pipe_comp) cudaStreamDestroy(cs);
    for (cudaEvent_t ev : ctx->pipe_ev) cudaEventDestroy(ev);
  }
  if (ctx->host_status) cudaFreeHost(ctx->host_status);
  for (int i = 0; i <= kMaxStages; ++i)
    if (ctx->ev[i]) cudaEventDestroy(ctx->ev[i]);
  delete ctx;
}

gpo_status gpo_workspace_size(const gpo_ctx* ctx, const gpo_batch* batch, size_t* bytes) {
  if (!bytes) return GPO_ERR_INVALID_ARG;
  gpo_status s = check_batch(const_cast<gpo_ctx*>(ctx), batch);
  if (s != GPO_OK) return s;
  Layout L;
  if (!layout(*batch, L)) return GPO_ERR_UNSUPPORTED;
  *bytes = L.total;
  return GPO_OK;
}

}  // extern "C"

namespace {

// Next-layer budget request of gpo_layer_budget (mode 1 of the kernels).
struct BudgetReq {
  int layer, b_next;
  const uint8_t* active;
  int32_t* budget;
};

// The path for groups [g0, g1) of the batch; clears the status words first if `clear`.
// With `bud`, the classes and the next-layer budgets instead of the advantages.
gpo_status compute_impl(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out, void* workspace,
                        size_t workspace_bytes, int64_t g0, int64_t g1, bool clear, void* stream,
                        const BudgetReq* bud = nullptr) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  ctx->msg[0] = 0;
  gpo_status s = check_batch(ctx, batch);
  if (s != GPO_OK) return s;
  s = bud ? GPO_OK : check_outputs(ctx, batch, out);
  if (s != GPO_OK) return s;
  Layout L;
  if (!layout(*batch, L)) return set_msg(ctx, "batch too large"), GPO_ERR_UNSUPPORTED;
  if (!workspace || !aligned(workspace, kAlign) || workspace_bytes < L.total)
    return set_msg(ctx, "workspace needs %zu bytes, 256-byte aligned", L.total), GPO_ERR_WORKSPACE;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev != ctx->device)
    return set_msg(ctx, "current device differs from the context's"), GPO_ERR_INVALID_ARG;

  const gpo_batch& b = *batch;
  const gpo_params& p = ctx->params;
  Sizes sz;
  sz.G = b.num_groups;
  sz.R = b.num_rollouts;
  sz.N = b.num_states;
  sz.d = b.d;
  sz.T = b.total_tokens;
  sz.stride = b.emb_row_stride;
  sz.maxn = b.max_states_per_group;
  sz.g0 = (int)g0;
  sz.g1 = (int)g1;
  Params pp;
  pp.kappa = p.kappa;
  pp.w = p.w;
  pp.lambda_eff = p.lambda_eff;
  pp.eps = p.std_eps;
  pp.kappa_f = (float)pp.kappa;
  pp.w_hi = (float)pp.w;
  pp.w_lo = (float)(pp.w - (double)pp.w_hi);
  pp.lambda_f = (float)pp.lambda_eff;
  pp.eps_f = (float)pp.eps;
  pp.ddof = p.std_ddof;
  pp.rule = p.merge_rule;
  pp.mode = bud ? 1 : 0;
  pp.layer = bud ? bud->layer : 0;
  pp.b_next = bud ? bud->b_next : 0;
  pp.active = bud ? bud->active : nullptr;
  pp.budget = bud ? bud->budget : nullptr;
  pp.stats_in_kernel = 0;
  pp.debug_timeout = (p.flags & GPO_FLAG_DEBUG_TIMEOUT) != 0;
  const Ws ws = workspace_views(workspace, L);
  LaunchCtx lc;
  lc.stream = static_cast<cudaStream_t>(stream);
  lc.num_sms = ctx->num_sms;

  const bool use_tc = b.emb_dtype == GPO_EMB_BF16 && !(p.flags & GPO_FLAG_SIMT_SIMILARITY) && sz.N > 0;
  const bool fused = use_tc && !(p.flags & GPO_FLAG_TILED) && sz.G > 0 && sz.maxn <= kFusedMaxStates;
  // fp32 embeddings, chain layout, small groups: the one-launch CUDA-core path
  const bool fused32 = b.emb_dtype == GPO_EMB_F32 && !b.parent && !bud && !(p.flags & GPO_FLAG_TILED) && sz.G > 0 &&
                       sz.N > 0 && fused_f32_fits(sz.d, sz.maxn);
  const bool whole = g0 == 0 && g1 == sz.G;
  if (!whole && !fused && !fused32 && g1 > g0) {
    return set_msg(ctx, "a group range needs a group-resident path (bf16 with at most %d states per group, or fp32 "
                        "chain layout with small groups; no flags)", kFusedMaxStates), GPO_ERR_UNSUPPORTED;
  }
  // embedding tensor maps: boxes of 64 elements x 128 rows and x 32 rows, 128B swizzle
  CUtensorMap map, map32;
  memset(&map, 0, sizeof map);
  memset(&map32, 0, sizeof map32);
  if (use_tc) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return set_msg(ctx, "cuTensorMapEncodeTiled unavailable"), GPO_ERR_CUDA;
    const cuuint64_t dims[2] = {(cuuint64_t)sz.d, (cuuint64_t)sz.N};
    const cuuint64_t strides[1] = {(cuuint64_t)(sz.stride * 2)};
    const cuuint32_t estr[2] = {1, 1};
    CUtensorMap* maps[2] = {&map, &map32};
    const cuuint32_t rows[2] = {(cuuint32_t)kTileM, 32};
    for (int m = 0; m < 2; ++m) {
      const cuuint32_t box[2] = {(cuuint32_t)kTileK, rows[m]};
      const CUresult r = enc(maps[m], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(b.emb), dims, strides, box,
                             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS) return set_msg(ctx, "cuTensorMapEncodeTiled failed (%d)", (int)r), GPO_ERR_UNSUPPORTED;
    }
  }

  int ns = 0;
  // one kernel launch of the path: an NVTX range around its enqueue (host-side trace) and,
  // with timing on, a CUDA event after it
  auto stage = [&](const char* name, auto launch) {
    nvtxRangePushA(name);
    cudaError_t e = launch();
    nvtxRangePop();
    if (ctx->timing && e == cudaSuccess && ns < kMaxStages) {
      ctx->stage_name[ns] = name;
      e = cudaEventRecord(ctx->ev[++ns], lc.stream);
    }
    return e;
  };
  cudaError_t e = cudaSuccess;
  if (ctx->timing) e = cudaEventRecord(ctx->ev[0], lc.stream);
  if (e == cudaSuccess && clear) e = cudaMemsetAsync(ws.status, 0, sizeof(uint32_t) * kStatusWords, lc.stream);
  if (g1 <= g0) {
    // nothing to compute (a call that only clears the status words)
  } else if (fused32) {
    if (e == cudaSuccess) e = stage("fused_f32", [&] { return launch_fused_f32(lc, b, *out, sz, ws, pp); });
  } else if (fused) {
    // one group per CTA at a time: the group warps compute the compensated statistics of
    // each CTA's first group while it streams in; the groups after those (more groups than
    // CTAs) get theirs from a launch of its own first, on the whole GPU, so that the group
    // warps keep pace with the stream
    pp.stats_in_kernel = !bud;
    const int grid = fused_grid(lc, sz);
    if (e == cudaSuccess && !bud && (int64_t)(g1 - g0) > (int64_t)grid) {
      Sizes rest = sz;
      rest.g0 = sz.g0 + grid;
      e = stage("exact_stats", [&] { return launch_exact_stats(lc, b, rest, ws); });
    }
    if (e == cudaSuccess) e = stage("fused", [&] { return launch_fused(lc, map, map32, b, *out, sz, ws, pp); });
  } else {
    if (e == cudaSuccess && b.parent) e = stage("tree_prep", [&] { return launch_tree_prep(lc, b, sz, ws); });
    if (e == cudaSuccess) e = stage("prep", [&] { return launch_prep(lc, b, sz, ws); });
    if (e == cudaSuccess && sz.N > 0) {
      // the fp32 norms of the threshold test come from the Gram tiles (tcgen05) or from
      // row_stats (CUDA cores); eta takes compensated norms and parent dots (exact_stats),
      // after the similarity stage so that the fp32 norms give the sums' biases
      if (e == cudaSuccess && !use_tc) e = stage("row_stats", [&] { return launch_row_stats(lc, b, sz, ws); });
      if (e == cudaSuccess)
        e = stage("similarity", [&] {
          return use_tc ? launch_sim_tc(lc, map, b, sz, ws, pp) : launch_sim_simt(lc, b, sz, ws, pp);
        });
      if (e == cudaSuccess && !bud) e = stage("exact_stats", [&] { return launch_exact_stats(lc, b, sz, ws, true); });
      if (e == cudaSuccess) e = stage("groups", [&] { return launch_groups(lc, b, *out, sz, ws, pp); });
      if (e == cudaSuccess && !bud) e = stage("tokens", [&] { return launch_tokens(lc, b, *out, sz, ws); });
    }
  }
  ctx->nstages = ns;
  ctx->last_status = ws.status;
  if (e != cudaSuccess) return set_msg(ctx, "launch failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  return GPO_OK;
}

}  // namespace

extern "C" {

gpo_status gpo_compute(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out, void* workspace,
                       size_t workspace_bytes, void* stream) {
  if (!ctx || !batch) return GPO_ERR_INVALID_ARG;
  return compute_impl(ctx, batch, out, workspace, workspace_bytes, 0, batch->num_groups, true, stream);
}

gpo_status gpo_layer_budget(gpo_ctx* ctx, const gpo_batch* batch, int32_t layer, int32_t b_next, const uint8_t* active,
                            int32_t* budget, int32_t* class_id, void* workspace, size_t workspace_bytes, void* stream) {
  if (!ctx || !batch) return GPO_ERR_INVALID_ARG;
  ctx->msg[0] = 0;
  if (!batch->parent) return set_msg(ctx, "next-layer budgets need the tree layout"), GPO_ERR_UNSUPPORTED;
  if (layer < 1 || b_next < 1 || b_next > (1 << 16))
    return set_msg(ctx, "layer must be >= 1 and b_next in [1, 65536]"), GPO_ERR_INVALID_ARG;
  if (batch->num_states > 0 && !budget) return set_msg(ctx, "budget output is NULL"), GPO_ERR_INVALID_ARG;
  gpo_outputs o;
  memset(&o, 0, sizeof o);
  o.class_id = class_id;
  const BudgetReq req = {layer, b_next, active, budget};
  return compute_impl(ctx, batch, &o, workspace, workspace_bytes, 0, batch->num_groups, true, stream, &req);
}

gpo_status gpo_compute_groups(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out, int64_t first_group,
                              int64_t num_groups, int clear_status, void* workspace, size_t workspace_bytes,
                              void* stream) {
  if (!ctx || !batch) return GPO_ERR_INVALID_ARG;
  if (first_group < 0 || num_groups < 0 || first_group > batch->num_groups ||
      num_groups > batch->num_groups - first_group)
    return set_msg(ctx, "group range [%lld, %lld) outside the batch's %lld groups", (long long)first_group,
                   (long long)(first_group + num_groups), (long long)batch->num_groups), GPO_ERR_INVALID_ARG;
  return compute_impl(ctx, batch, out, workspace, workspace_bytes, first_group, first_group + num_groups,
                      clear_status != 0, stream);
}

gpo_status gpo_compute_host(gpo_ctx* ctx, const gpo_batch* host, const gpo_batch* dev, const gpo_outputs* out,
                            float* host_adv, int64_t chunk_bytes, void* workspace, size_t workspace_bytes,
                            void* stream) {
  if (!ctx || !host || !dev) return GPO_ERR_INVALID_ARG;
  ctx->msg[0] = 0;
  gpo_status s = check_batch(ctx, dev);
  if (s == GPO_OK) s = check_outputs(ctx, dev, out);
  if (s != GPO_OK) return s;
  const gpo_batch& h = *host;
  const gpo_batch& d = *dev;
  const bool tree = d.parent != nullptr;
  if (h.num_groups != d.num_groups || h.num_rollouts != d.num_rollouts || h.num_states != d.num_states ||
      h.d != d.d || h.emb_dtype != d.emb_dtype || h.emb_row_stride != d.emb_row_stride ||
      h.total_tokens != d.total_tokens || (h.parent != nullptr) != tree || (h.root_emb != nullptr) != (d.root_emb != nullptr))
    return set_msg(ctx, "host and device batches differ in size or layout"), GPO_ERR_INVALID_ARG;
  const int64_t G = d.num_groups, R = d.num_rollouts, N = d.num_states, T = d.total_tokens;
  if (!h.group_rollout_off || (N > 0 && (!h.step_len || !h.emb)) || (R > 0 && !h.reward) ||
      (tree ? (!h.group_state_off || !h.group_token_off) : (!h.rollout_step_off || !h.rollout_token_off)) ||
      (T > 0 && !host_adv))
    return set_msg(ctx, "a host array is NULL"), GPO_ERR_INVALID_ARG;
  if (chunk_bytes < 0) return set_msg(ctx, "chunk_bytes < 0"), GPO_ERR_INVALID_ARG;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t esz = d.emb_dtype == GPO_EMB_BF16 ? 2 : 4;
  const size_t row = (size_t)d.emb_row_stride * esz;
  cudaError_t e = cudaSuccess;
  auto up = [&](const void* dst, const void* src, size_t bytes, cudaStream_t s) {
    if (e == cudaSuccess && bytes > 0) e = cudaMemcpyAsync(const_cast<void*>(dst), src, bytes, cudaMemcpyHostToDevice, s);
  };
  // the small arrays first, on the caller's stream
  up(d.group_rollout_off, h.group_rollout_off, 4 * (G + 1), st);
  if (tree) {
    up(d.parent, h.parent, 4 * N, st);
    up(d.group_state_off, h.group_state_off, 4 * (G + 1), st);
    up(d.group_token_off, h.group_token_off, 8 * (G + 1), st);
  }
  if (d.rollout_step_off && h.rollout_step_off) up(d.rollout_step_off, h.rollout_step_off, 4 * (R + 1), st);
  if (d.rollout_token_off && h.rollout_token_off) up(d.rollout_token_off, h.rollout_token_off, 8 * (R + 1), st);
  up(d.step_len, h.step_len, 4 * N, st);
  up(d.reward, h.reward, R, st);
  if (d.root_emb) up(d.root_emb, h.root_emb, row * G, st);
  if (e != cudaSuccess) return set_msg(ctx, "upload failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;

  // chunks of groups with about equal numbers of states, from the host offsets (checked here;
  // offsets that do not partition the batch leave it to one launch, whose kernels report them)
  const int64_t emb_bytes = N * (int64_t)row;
  // default: stages of at least 8 MiB, at most ten of them
  if (chunk_bytes == 0) chunk_bytes = std::max<int64_t>(kPipeMinChunkBytes, emb_bytes / 10);
  int64_t nchunk = emb_bytes / chunk_bytes;
  nchunk = std::min<int64_t>(std::min<int64_t>(nchunk, G), kPipeMaxChunks);
  bool piped = nchunk >= 2 && d.emb_dtype == GPO_EMB_BF16 && ctx->params.flags == 0 &&
               d.max_states_per_group <= kFusedMaxStates;
  if (piped) {
    ctx->pipe_s.resize(G + 1);
    ctx->pipe_t.resize(G + 1);
    for (int64_t g = 0; g <= G && piped; ++g) {
      int64_t sv, tv;
      if (tree) {
        sv = h.group_state_off[g];
        tv = h.group_token_off[g];
      } else {
        const int32_t r = h.group_rollout_off[g];
        piped = r >= 0 && r <= R;
        sv = piped ? h.rollout_step_off[r] : 0;
        tv = piped ? h.rollout_token_off[r] : 0;
      }
      piped = piped && sv >= 0 && sv <= N && tv >= 0 && tv <= T &&
              (g == 0 ? sv == 0 && tv == 0 : sv >= ctx->pipe_s[g - 1] && tv >= ctx->pipe_t[g - 1]) &&
              (g < G || (sv == N && tv == T));
      ctx->pipe_s[g] = sv;
      ctx->pipe_t[g] = tv;
    }
  }
  if (piped && !ctx->pipe_ready) {
    bool ok = cudaStreamCreateWithFlags(&ctx->pipe_in, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&ctx->pipe_out, cudaStreamNonBlocking) == cudaSuccess;
    for (cudaStream_t& cs : ctx->pipe_comp) ok = ok && cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) == cudaSuccess;
    for (cudaEvent_t& ev : ctx->pipe_ev) ok = ok && cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      cudaGetLastError();
      return set_msg(ctx, "could not create the pipeline's streams and events"), GPO_ERR_CUDA;
    }
    ctx->pipe_ready = true;
  }
  if (!piped) {  // one upload, the whole path, one download
    up(d.emb, h.emb, (size_t)emb_bytes, st);
    if (e != cudaSuccess) return set_msg(ctx, "upload failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
    s = compute_impl(ctx, dev, out, workspace, workspace_bytes, 0, G, true, stream);
    if (s != GPO_OK) return s;
    if (T > 0 && (e = cudaMemcpyAsync(host_adv, out->adv, 4 * T, cudaMemcpyDeviceToHost, st)) != cudaSuccess)
      return set_msg(ctx, "download failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
    return GPO_OK;
  }
  nvtxRangePushA("gpo_compute_host pipeline");
  const bool timing = ctx->timing;  // per-stage events would interleave across the streams
  ctx->timing = false;
  s = compute_impl(ctx, dev, out, workspace, workspace_bytes, 0, 0, true, stream);  // clears the status words
  cudaEvent_t* ev = ctx->pipe_ev;
  const cudaEvent_t ready = ev[2 * kPipeMaxChunks], done = ev[2 * kPipeMaxChunks + 1];
  if (s == GPO_OK) {
    e = cudaEventRecord(ready, st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->pipe_in, ready, 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->pipe_out, ready, 0);
    for (cudaStream_t cs : ctx->pipe_comp)
      if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ready, 0);
    // chunk k: its embeddings in on pipe_in, its groups on a compute stream
    int64_t bounds[kPipeMaxChunks + 1];
    int64_t nb = 0, ga = 0;
    bounds[0] = 0;
    for (int64_t k = 0; k < nchunk && e == cudaSuccess && s == GPO_OK; ++k) {
      int64_t gb = ga;
      const int64_t target = k + 1 == nchunk ? N : N * (k + 1) / nchunk;
      while (gb < G && (ctx->pipe_s[gb] < target || gb == ga)) ++gb;
      if (k + 1 == nchunk) gb = G;
      if (gb <= ga) continue;
      const int64_t sa = ctx->pipe_s[ga], sb = ctx->pipe_s[gb];
      up(static_cast<const char*>(d.emb) + sa * row, static_cast<const char*>(h.emb) + sa * row, (size_t)(sb - sa) * row,
         ctx->pipe_in);
      if (e == cudaSuccess) e = cudaEventRecord(ev[2 * nb], ctx->pipe_in);
      const cudaStream_t cs = ctx->pipe_comp[nb % kPipeComputeStreams];
      if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ev[2 * nb], 0);
      if (e == cudaSuccess) s = compute_impl(ctx, dev, out, workspace, workspace_bytes, ga, gb, false, cs);
      if (e == cudaSuccess && s == GPO_OK) e = cudaEventRecord(ev[2 * nb + 1], cs);
      bounds[++nb] = gb;
      ga = gb;
    }
    // the chunks' tokens out on pipe_out, each as soon as its groups are done: downloads
    // share the host link with the later chunks' uploads, which moves more bytes per second
    // than uploads first and downloads after
    for (int64_t k = 0; k < nb && e == cudaSuccess && s == GPO_OK; ++k) {
      const int64_t ta = ctx->pipe_t[bounds[k]], tb = ctx->pipe_t[bounds[k + 1]];
      e = cudaStreamWaitEvent(ctx->pipe_out, ev[2 * k + 1], 0);
      if (e == cudaSuccess && tb > ta)
        e = cudaMemcpyAsync(host_adv + ta, out->adv + ta, 4 * (tb - ta), cudaMemcpyDeviceToHost, ctx->pipe_out);
    }
    // the caller's stream continues after the last download (which follows every chunk)
    if (e == cudaSuccess) e = cudaEventRecord(done, ctx->pipe_out);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, done, 0);
  }
  ctx->timing = timing;
  nvtxRangePop();
  if (s != GPO_OK) return s;
  if (e != cudaSuccess) return set_msg(ctx, "pipeline enqueue failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  return GPO_OK;
}

}  // extern "C"

namespace {

struct LossLayout {
  size_t head, start, w, tile_edge, partial, total;
  int64_t ntiles;
};

bool loss_layout(const gpo_batch& b, LossLayout& L) {
  const int64_t N = b.num_states, T = b.total_tokens;
  L.ntiles = (T + kLossTile - 1) / kLossTile;
  if (N >= ((int64_t)1 << 31) - 1) return false;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = up(o + bytes);
    return at;
  };
  L.head = take(kLossPlanHead);
  L.start = take(sizeof(int64_t) * (size_t)(N + 1));
  L.w = take(sizeof(float) * (size_t)(N > 0 ? N : 1));
  L.tile_edge = take(sizeof(int32_t) * (size_t)(L.ntiles + 1));
  L.partial = take(sizeof(double) * 4 * (size_t)kLossMaxBlocks);
  L.total = o;
  return true;
}

LossPlan loss_views(void* base, const LossLayout& L) {
  unsigned char* p = static_cast<unsigned char*>(base);
  LossPlan lp;
  lp.status = reinterpret_cast<uint32_t*>(p + L.head);
  lp.dims = reinterpret_cast<int64_t*>(p + L.head + 128);
  lp.start = reinterpret_cast<int64_t*>(p + L.start);
  lp.w = reinterpret_cast<float*>(p + L.w);
  lp.tile_edge = reinterpret_cast<int32_t*>(p + L.tile_edge);
  lp.partial = reinterpret_cast<double*>(p + L.partial);
  lp.ntiles = L.ntiles;
  return lp;
}

Sizes loss_sizes(const gpo_batch& b) {
  Sizes sz;
  sz.G = b.num_groups;
  sz.R = b.num_rollouts;
  sz.N = b.num_states;
  sz.d = b.d;
  sz.T = b.total_tokens;
  sz.stride = b.emb_row_stride;
  sz.maxn = b.max_states_per_group;
  sz.g0 = 0;
  sz.g1 = b.num_groups;
  return sz;
}

// The structure the loss reads: sizes and offsets (embeddings and rewards are not needed).
gpo_status check_loss_batch(gpo_ctx* c, const gpo_batch* b) {
  if (!b) return set_msg(c, "batch is NULL"), GPO_ERR_INVALID_ARG;
  if (b->num_groups < 0 || b->num_rollouts < 0 || b->num_states < 0 || b->total_tokens < 0)
    return set_msg(c, "negative size"), GPO_ERR_INVALID_ARG;
  if (b->num_states == 0 && b->total_tokens != 0) return set_msg(c, "tokens without states"), GPO_ERR_SHAPE;
  if (b->num_groups == 0 && (b->num_states != 0 || b->num_rollouts != 0))
    return set_msg(c, "states without groups"), GPO_ERR_SHAPE;
  if (b->parent) {
    if (!b->group_rollout_off || !b->group_state_off || !b->group_token_off)
      return set_msg(c, "tree layout: an offset array is NULL"), GPO_ERR_INVALID_ARG;
  } else if (b->group_state_off || b->group_token_off) {
    return set_msg(c, "group_state_off / group_token_off given without parent"), GPO_ERR_INVALID_ARG;
  } else if (!b->group_rollout_off || !b->rollout_step_off || !b->rollout_token_off) {
    return set_msg(c, "offset array is NULL"), GPO_ERR_INVALID_ARG;
  }
  if (b->num_states > 0 && !b->step_len) return set_msg(c, "step_len is NULL"), GPO_ERR_INVALID_ARG;
  return GPO_OK;
}

}  // namespace

extern "C" {

gpo_status gpo_loss_plan_size(const gpo_batch* batch, size_t* bytes) {
  if (!batch || !bytes) return GPO_ERR_INVALID_ARG;
  LossLayout L;
  if (batch->num_states < 0 || batch->total_tokens < 0 || !loss_layout(*batch, L)) return GPO_ERR_INVALID_ARG;
  *bytes = L.total;
  return GPO_OK;
}

gpo_status gpo_loss_plan(gpo_ctx* ctx, const gpo_batch* batch, void* plan, size_t plan_bytes, void* stream) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  ctx->msg[0] = 0;
  gpo_status s = check_loss_batch(ctx, batch);
  if (s != GPO_OK) return s;
  LossLayout L;
  if (!loss_layout(*batch, L)) return set_msg(ctx, "batch too large"), GPO_ERR_UNSUPPORTED;
  if (!plan || !aligned(plan, kAlign) || plan_bytes < L.total)
    return set_msg(ctx, "the plan needs %zu bytes, 256-byte aligned", L.total), GPO_ERR_WORKSPACE;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev != ctx->device)
    return set_msg(ctx, "current device differs from the context's"), GPO_ERR_INVALID_ARG;
  const LossPlan lp = loss_views(plan, L);
  LaunchCtx lc;
  lc.stream = static_cast<cudaStream_t>(stream);
  lc.num_sms = ctx->num_sms;
  cudaError_t e = cudaMemsetAsync(lp.status, 0, kLossPlanHead, lc.stream);
  if (e == cudaSuccess) e = launch_loss_plan(lc, *batch, loss_sizes(*batch), lp);
  ctx->nstages = 0;
  ctx->last_status = lp.status;
  if (e != cudaSuccess) return set_msg(ctx, "launch failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  return GPO_OK;
}

gpo_status gpo_token_loss(gpo_ctx* ctx, const gpo_batch* batch, void* plan, const gpo_loss_params* params,
                          const gpo_loss_inputs* in, const gpo_loss_outputs* out, void* stream) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  ctx->msg[0] = 0;
  gpo_status s = check_loss_batch(ctx, batch);
  if (s != GPO_OK) return s;
  if (!params || !in || !out) return set_msg(ctx, "params, inputs or outputs NULL"), GPO_ERR_INVALID_ARG;
  const gpo_loss_params& p = *params;
  if (!(p.clip_low >= 0.0 && p.clip_low < 1.0) || !(p.clip_high >= 0.0) || !std::isfinite(p.clip_high) ||
      !(p.beta_kl >= 0.0) || !std::isfinite(p.beta_kl) || !(p.lambda_eff >= 0.0) || !std::isfinite(p.lambda_eff) ||
      (p.form != GPO_LOSS_DUAL && p.form != GPO_LOSS_SPLIT) || (p.norm != GPO_LOSS_NORM_EDGE && p.norm != GPO_LOSS_NORM_TOKEN))
    return set_msg(ctx, "loss parameters out of range"), GPO_ERR_INVALID_ARG;
  const bool split = p.form == GPO_LOSS_SPLIT, kl = p.beta_kl > 0.0;
  const int64_t T = batch->total_tokens, N = batch->num_states;
  if (!out->loss) return set_msg(ctx, "loss output is NULL"), GPO_ERR_INVALID_ARG;
  if (T > 0 && (!in->logp || !in->old_logp || (kl && !in->ref_logp)))
    return set_msg(ctx, "log-probabilities NULL"), GPO_ERR_INVALID_ARG;
  if (N > 0 && (split ? (!in->edge_cor || !in->edge_eff || !in->edge_eff_mask) : !in->edge_adv))
    return set_msg(ctx, "per-edge advantages of the %s form NULL", split ? "split" : "dual"), GPO_ERR_INVALID_ARG;
  if (!aligned(in->logp, 16) || !aligned(in->old_logp, 16) || (kl && !aligned(in->ref_logp, 16)) ||
      !aligned(out->grad_logp, 16))
    return set_msg(ctx, "per-token arrays must be 16-byte aligned"), GPO_ERR_UNSUPPORTED;
  LossLayout L;
  if (!loss_layout(*batch, L)) return set_msg(ctx, "batch too large"), GPO_ERR_UNSUPPORTED;
  if (!plan || !aligned(plan, kAlign)) return set_msg(ctx, "plan NULL or misaligned"), GPO_ERR_WORKSPACE;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev != ctx->device)
    return set_msg(ctx, "current device differs from the context's"), GPO_ERR_INVALID_ARG;
  const LossPlan lp = loss_views(plan, L);
  LossArgs a;
  a.logp = in->logp;
  a.old_logp = in->old_logp;
  a.ref_logp = kl ? in->ref_logp : nullptr;
  a.adv = split ? in->edge_cor : in->edge_adv;
  a.eff = split ? in->edge_eff : nullptr;
  a.mask = split ? in->edge_eff_mask : nullptr;
  a.loss = out->loss;
  a.grad = out->grad_logp;
  a.stats = out->stats;
  a.lo = (float)(1.0 - p.clip_low);
  a.hi = (float)(1.0 + p.clip_high);
  a.beta = (float)p.beta_kl;
  a.lambda = (float)p.lambda_eff;
  a.inv_t = T > 0 ? (float)(1.0 / (double)T) : 0.f;
  a.norm_token = p.norm == GPO_LOSS_NORM_TOKEN;
  a.split = split;
  a.kl = kl;
  a.N = (int)N;
  a.T = T;
  LaunchCtx lc;
  lc.stream = static_cast<cudaStream_t>(stream);
  lc.num_sms = ctx->num_sms;
  int ns = 0;
  cudaError_t e = cudaSuccess;
  if (ctx->timing) e = cudaEventRecord(ctx->ev[0], lc.stream);
  if (e == cudaSuccess) e = launch_token_loss(lc, lp, a);
  if (e == cudaSuccess && ctx->timing) {
    ctx->stage_name[ns] = "token_loss";
    e = cudaEventRecord(ctx->ev[++ns], lc.stream);
  }
  ctx->nstages = ns;
  ctx->last_status = lp.status;
  if (e != cudaSuccess) return set_msg(ctx, "launch failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  return GPO_OK;
}

gpo_status gpo_enable_timing(gpo_ctx* ctx, int enable) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  ctx->timing = enable != 0;
  ctx->nstages = 0;
  return GPO_OK;
}

gpo_status gpo_stage_times(gpo_ctx* ctx, float* ms, const char** names, int capacity, int* count) {
  if (!ctx || !ctx->timing || !count) return GPO_ERR_INVALID_ARG;
  *count = ctx->nstages;
  if (capacity < ctx->nstages) return GPO_ERR_INVALID_ARG;
  if (ctx->nstages == 0) return GPO_OK;
  cudaError_t e = cudaEventSynchronize(ctx->ev[ctx->nstages]);
  for (int i = 0; i < ctx->nstages && e == cudaSuccess; ++i) {
    float t = 0.f;
    e = cudaEventElapsedTime(&t, ctx->ev[i], ctx->ev[i + 1]);
    if (ms) ms[i] = t;
    if (names) names[i] = ctx->stage_name[i];
  }
  if (e != cudaSuccess) return set_msg(ctx, "event timing failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  return GPO_OK;
}

gpo_status gpo_sync_status(gpo_ctx* ctx, void* stream) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return set_msg(ctx, "stream error: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  if (!ctx->last_status) return GPO_OK;
  e = cudaMemcpy(ctx->host_status, ctx->last_status, sizeof(uint32_t) * kStatusWords, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return set_msg(ctx, "status read failed: %s", cudaGetErrorString(e)), GPO_ERR_CUDA;
  const uint32_t code = ctx->host_status[kStError];
  if (code != 0)
    set_msg(ctx, "%s (kernel %u, index %u)", gpo_status_string((gpo_status)code), ctx->host_status[kStWhere],
            ctx->host_status[kStDetail]);
  return (gpo_status)code;
}

}  // extern "C"
