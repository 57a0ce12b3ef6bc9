// Internal declarations shared by the translation units of libgraphpo.
// Device-side workspace layout, error reporting, and the inline-PTX wrappers
// for mbarrier, TMA (cp.async.bulk.tensor) and tcgen05 used by the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/graphpo.h"

namespace gpo {

// ------------------------------------------------------------------ sizes

constexpr int kTileM = 128;          // rows of one similarity tile (tcgen05 M)
constexpr int kTileN = 256;          // max columns of one work item (tcgen05 N)
constexpr int kTileK = 64;           // bf16 elements per 128-byte swizzle row
constexpr int kEdgeCap = 384;        // spanning-forest edges one item can emit (< rows+cols)
constexpr int kStatusWords = 16;
constexpr int kMaxStages = 8;        // timed stages of one gpo_compute
constexpr int kFusedMaxStates = 384; // largest group of the fused group-resident kernel
constexpr int kPipeMaxChunks = 64;   // gpo_compute_host: pipeline stages at most
constexpr int kPipeComputeStreams = 3;
constexpr int64_t kPipeMinChunkBytes = (int64_t)8 << 20;

// status words (uint32) at the head of the workspace
enum : int {
  kStError = 0,     // first gpo_status reported by any kernel
  kStAbort = 1,     // nonzero: kernels stop early
  kStItems = 2,     // number of similarity work items planned
  kStTicket = 3,    // last-block ticket of the prep kernel
  kStDetail = 4,    // first failing index (debug aid)
  kStWhere = 5,     // kernel that reported the error (debug aid)
};

// A similarity work item: rows [row0, row0+128) of one prompt group against
// columns [col0, col0+ncols) of the same group (col0 >= row0).
struct Item {
  int row0, col0, ncols, group;
};

struct GroupInfo {
  int s0, n;        // states [s0, s0+n)
  int r0, nr;       // rollouts [r0, r0+nr)
  int blk0, nblk;   // its 128-row blocks: diagonal items [blk0, blk0+nblk)
  int off0, noff;   // then its off-diagonal items [off0, off0+noff), off0 = blk0 + nblk
};

// Device pointers into the caller's workspace (computed on the host).
struct Ws {
  uint32_t* status;      // [kStatusWords]
  Item* items;           // [max_items]: per group, its diagonal items, then its off-diagonal ones
  int* blk_ready;        // [max_items]: at a diagonal item's position, set once it has written its norms
  GroupInfo* groups;     // [G]
  int2* state_meta;      // [N] {rollout, depth}
  float* nrm2;           // [N] squared norm (fp32 accumulation; the threshold test)
  float* rn;             // [N] 1/|z| (0 for a zero row)
  int* edge_count;       // [max_items]
  int2* edges;           // [max_items * kEdgeCap]
  float* e_adv;          // [N] A_dual per edge
  float* e_cor;          // [N] A_cor per edge
  float* e_eff;          // [N] routed efficiency advantage per edge
  uint8_t* e_mask;       // [N]
  int64_t* tok_start;    // [N] first token of each edge
  // tree layout only (null otherwise)
  int* tree_par;         // [N] parent (global index, -1 = the prompt root)
  int* tree_end;         // [N] end of the state's subtree (global, exclusive)
  int2* tree_own;        // [N] {c_own, t_own}: rewards and number of the leaves of the subtree
  int* tree_x;           // [23 N + 11 G] group-math sums, tree_scratch of group g at 23 s0 + 11 g
  // accurate row statistics (unevaluated float pairs hi + lo, see exact_stats_kernel)
  float2* x_n2;          // [N] |z_v|^2
  float2* x_dot;         // [N] <z_{p(v)}, z_v> (prompt embedding for a root child, 0 without one)
  float2* x_root_n2;     // [G] |prompt embedding|^2
  int max_items;
};

struct Sizes {
  int G, R, N, d;
  int64_t T;
  int64_t stride;        // embedding row stride in elements
  int maxn;              // max states per group (host bound)
  int g0, g1;            // groups processed by this call: [g0, g1) (the whole batch but for
                         // gpo_compute_groups, which only the group-resident path serves)
};

struct Params {
  double kappa, w, lambda_eff, eps;
  // the same in fp32, rounded once on the host: w = w_hi + w_lo to ~2^-48
  float kappa_f, w_hi, w_lo, lambda_f, eps_f;
  int ddof, rule;
  // mode 1: next-layer budgets after layer `layer` instead of advantages (gpo_layer_budget)
  int mode, layer, b_next;
  int stats_in_kernel;    // fused path: the group warps compute the compensated row statistics
                          // of each CTA's first group (the other groups' come from exact_stats)
  int debug_timeout;      // GPO_FLAG_DEBUG_TIMEOUT: the MMA warp's first wait runs out
  const uint8_t* active;  // [N] frontier states to expand (NULL: all of depth `layer`)
  int32_t* budget;        // [N] output of mode 1
};

// ------------------------------------------------------------------ errors

__device__ __forceinline__ void report(uint32_t* st, int code, int where, int detail) {
  if (atomicCAS(&st[kStError], 0u, (uint32_t)code) == 0u) {
    st[kStWhere] = (uint32_t)where;
    st[kStDetail] = (uint32_t)detail;
  }
  atomicExch(&st[kStAbort], 1u);
}

// Bounds checks of the debug build (-DGPO_DEBUG, a stand-in for a device memory checker):
// GPO_BOUNDS(st, i, n, where) is true when 0 <= i < n; otherwise it reports GPO_ERR_BOUNDS
// with the index and the check's number (kWhere*), and the caller skips the access.  In the
// release build it is the constant true and costs nothing.
#ifdef GPO_DEBUG
__device__ __forceinline__ bool bounds_ok(uint32_t* st, int64_t i, int64_t n, int where) {
  if (i >= 0 && i < n) return true;
  if (atomicCAS(&st[kStError], 0u, (uint32_t)GPO_ERR_BOUNDS) == 0u) {
    st[kStWhere] = (uint32_t)where;
    st[kStDetail] = (uint32_t)i;
  }
  atomicExch(&st[kStAbort], 1u);
  return false;
}
#define GPO_BOUNDS(st, i, n, where) ::gpo::bounds_ok((st), (int64_t)(i), (int64_t)(n), (where))
#else
#define GPO_BOUNDS(st, i, n, where) true
#endif
// check numbers (the `where` of GPO_ERR_BOUNDS)
enum : int {
  kWhereTokens = 100,      // a token output (index of the 16-byte chunk or of the token)
  kWhereStateOut = 101,    // a per-state output
  kWhereStats = 102,       // a row of the compensated statistics (read or written)
  kWhereEdges = 103,       // an item's spanning-forest edge
  kWhereNorms = 104,       // an fp32 norm of the similarity stage
  kWhereSmemRow = 105,     // a row of the fp32 group-resident kernel's shared-memory copy
};

__device__ __forceinline__ bool aborted(const uint32_t* st) {
  return *((volatile const uint32_t*)&st[kStAbort]) != 0u;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------------ PTX: smem / mbarrier

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase with the given parity.  Gives up after `limit_ns` of
// wall time or when another thread raised the abort flag: then it reports
// GPO_ERR_TIMEOUT (first time) and returns false so that the caller can wind
// down cleanly instead of hanging the GPU.
// Wind-down waits (copies or MMAs still in flight before the CTA exits) pass
// honor_abort = false so that they only stop at their time limit.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t* st, int where,
                                          uint64_t limit_ns = 2000000000ull, bool honor_abort = true) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0u) {
      if (honor_abort && aborted(st)) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        report(st, GPO_ERR_TIMEOUT, where, 0);
        return false;
      }
    }
  }
}

// GPO_FLAG_DEBUG_TIMEOUT: a wait that runs out on purpose, on an mbarrier that has no arrival
// before the caller's own later commit (about a millisecond, then GPO_ERR_TIMEOUT as any
// timed-out wait reports it).
constexpr uint64_t kDebugTimeoutNs = 1000000ull;

// ------------------------------------------------------------------ flags between CTAs

__device__ __forceinline__ int ld_acquire_gpu(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_gpu(int* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Waits until *flag != 0 (acquire).  Gives up after `limit_ns` or when the abort flag
// is raised, reporting GPO_ERR_TIMEOUT on a timeout; returns whether the flag was seen.
__device__ __forceinline__ bool wait_flag(const int* flag, uint32_t* st, int where,
                                          uint64_t limit_ns = 2000000000ull) {
  if (ld_acquire_gpu(flag)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(64);
    if (ld_acquire_gpu(flag)) return true;
    if ((it & 63u) == 0u) {
      if (aborted(st)) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        report(st, GPO_ERR_TIMEOUT, where, 0);
        return false;
      }
    }
  }
}

// ------------------------------------------------------------------ PTX: TMA

__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// 2-D tiled bulk tensor load into shared memory; completion is signalled as
// transaction bytes on `bar`.  x is the innermost (element) coordinate.
__device__ __forceinline__ void tma_load_2d(void* smem_dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], "
      "[%2];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

// The same with an L2 cache policy (createpolicy) for the bytes it reads.
__device__ __forceinline__ void tma_load_2d_hint(void* smem_dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                                 uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%3, "
      "%4}], [%2], %5;" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

// L2 cache policies: keep (evict_last) or drop first (evict_first) the lines they cover.
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ------------------------------------------------------------------ PTX: tcgen05

__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulation, one CTA.
__device__ __forceinline__ void mma_bf16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives once on `bar` when every tcgen05 operation issued so far by this
// thread has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// 32 lanes x 32 consecutive fp32 columns: thread t of the warp receives TMEM
// lane (base lane + t), columns [col, col+32).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor for a K-major operand stored as rows of 128
// bytes with the 128-byte swizzle (8-row atoms of 1024 bytes, stacked densely):
// start address, leading offset (unused for this layout, encoded 1), stride
// offset 1024 bytes between 8-row groups, descriptor version 1, swizzle mode 2.
__device__ __forceinline__ uint64_t smem_desc_k128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1u << 16;             // leading byte offset >> 4
  d |= (uint64_t)(1024u >> 4) << 32;   // stride byte offset >> 4
  d |= (uint64_t)1u << 46;             // descriptor version
  d |= (uint64_t)2u << 61;             // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, shape M x N.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ------------------------------------------------------------------ float-float arithmetic
// Unevaluated pairs hi + lo of fp32 numbers carry about 48 significant bits.  The
// error-free transformations are Knuth's TwoSum and the fma-based TwoProduct (Ogita,
// Rump and Oishi, "Accurate sum and dot product", SIAM J. Sci. Comput. 2005); the
// pair operations follow Dekker's double-length arithmetic.  They are used where the
// standardisation of Sec. 4.4 amplifies rounding: the cosine eta(p(v), v) and the
// step reward r_step of nearly equal edges.

// s + e = a + b exactly.
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = a + b;
  const float bb = s - a;
  e = (a - (s - bb)) + (b - bb);
}

// Adds x to the pair (hi, lo) (compensated summation: the rounding error of every
// addition is collected in lo).
__device__ __forceinline__ void ff_acc(float& hi, float& lo, float x) {
  float s, e;
  two_sum(hi, x, s, e);
  hi = s;
  lo += e;
}

// Pair sum (a.x + a.y) + (b.x + b.y).
__device__ __forceinline__ float2 ff_add(float2 a, float2 b) {
  float s, e;
  two_sum(a.x, b.x, s, e);
  e += a.y + b.y;
  float h, l;
  two_sum(s, e, h, l);
  return make_float2(h, l);
}

// Pair product a * b.
__device__ __forceinline__ float2 ff_mul(float2 a, float2 b) {
  const float p = a.x * b.x;
  const float e = fmaf(a.x, b.x, -p) + (a.x * b.y + a.y * b.x);
  float h, l;
  two_sum(p, e, h, l);
  return make_float2(h, l);
}

// Pair quotient a / b (b.x > 0): one correction step of the fp32 quotient.
__device__ __forceinline__ float2 ff_div(float2 a, float2 b) {
  const float q = a.x / b.x;
  const float r = fmaf(-q, b.x, a.x) + a.y - q * b.y;
  float h, l;
  two_sum(q, r / b.x, h, l);
  return make_float2(h, l);
}

// Pair square root (a.x > 0): one correction step of the fp32 root.
__device__ __forceinline__ float2 ff_sqrt(float2 a) {
  const float s = sqrtf(a.x);
  const float e = fmaf(-s, s, a.x) + a.y;
  float h, l;
  two_sum(s, e / (2.0f * s), h, l);
  return make_float2(h, l);
}

// eta = max(0, dot / sqrt(np nv)) as a pair, from pair-valued dot and squared norms;
// 0 when a norm is zero (a zero embedding has similarity 0 with every state).
__device__ __forceinline__ float2 ff_eta(float2 dot, float2 np, float2 nv) {
  if (!(np.x > 0.f) || !(nv.x > 0.f)) return make_float2(0.f, 0.f);
  if (dot.x + dot.y <= 0.f) return make_float2(0.f, 0.f);
  return ff_div(dot, ff_sqrt(ff_mul(np, nv)));
}

// Two fp32 lanes per instruction (sm_100 and later): a pair (lo, hi) in one 64-bit
// register.  Used where compensated sums must keep pace with the tile stream.
__device__ __forceinline__ uint64_t f2add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2sub(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// The two bf16 of a 32-bit word as fp32 lanes (low half first).
// Packing and unpacking go through mov.b64 {lo, hi}, a register pair, rather than 64-bit
// shifts and ors.
__device__ __forceinline__ uint64_t pack_f2(uint32_t lo, uint32_t hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
__device__ __forceinline__ void unpack_f2(uint64_t a, uint32_t& lo, uint32_t& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=r"(lo), "=r"(hi) : "l"(a));
}
__device__ __forceinline__ uint64_t bf16x2_f32x2(uint32_t w) { return pack_f2(w << 16, w & 0xFFFF0000u); }
// Compensated accumulation (TwoSum per lane) of x into (s, e).
__device__ __forceinline__ void f2_acc(uint64_t& s, uint64_t& e, uint64_t x) {
  const uint64_t t = f2add(s, x);
  const uint64_t bb = f2sub(t, s);
  e = f2add(e, f2add(f2sub(s, f2sub(t, bb)), f2sub(x, bb)));
  s = t;
}
// The float pair of a two-lane compensated sum.
__device__ __forceinline__ float2 f2_finish(uint64_t s, uint64_t e) {
  const float s0 = __uint_as_float((uint32_t)s), s1 = __uint_as_float((uint32_t)(s >> 32));
  const float e0 = __uint_as_float((uint32_t)e), e1 = __uint_as_float((uint32_t)(e >> 32));
  float h, t;
  two_sum(s0, s1, h, t);
  float hh, ll;
  two_sum(h, t + e0 + e1, hh, ll);
  return make_float2(hh, ll);
}

// ------------------------------------------------------------------ biased error-free sums
// Sums of exact products (bf16 x bf16 is exact in fp32) with four fp32 operations per
// product instead of TwoSum's seven, at the same accuracy.  The running sum carries a bias
// sigma, a power of two >= 2 B where B bounds the sum of |products| added so far: then the
// running sum s stays in [sigma/2, 3 sigma/2], every product p has |p| <= sigma/2 <= |s|,
// so t = fl(s + p) is Dekker's Fast2Sum case (Dekker 1971; Muller et al., Handbook of
// Floating-Point Arithmetic, Sec. 4.3): s - t and p + (s - t) are exact, and
//   t = fma(x, y, s),  z = s - t,  err = fma(x, y, z) = p - (t - s)
// gives the rounding error of every addition exactly (collected, rounded, in e).  s - sigma
// is exact (Sterbenz), so the sum is (s - sigma) + e.  B comes from a plain fp32 pass over
// the next segment of the operands (sum of x^2, and (x^2 + y^2) / 2 >= |x y| for a dot),
// with a relative margin that covers that pass's rounding; when 2 B would pass sigma, the
// current epoch is closed into a float pair by TwoSum and a new one starts with
// sigma = 2^ceil(log2 4 B).  Two fp32 lanes per instruction, as in f2_acc.

__device__ __forceinline__ uint64_t f2fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2splat(float x) { return pack_f2(__float_as_uint(x), __float_as_uint(x)); }
// The sum of a pair's two fp32 lanes (rounded once).
__device__ __forceinline__ float f2_lanes_sum(uint64_t a) {
  uint32_t lo, hi;
  unpack_f2(a, lo, hi);
  return __uint_as_float(lo) + __uint_as_float(hi);
}
// Smallest power of two >= x, for finite x >= 0 (0 for 0; +inf beyond the fp32 range).
__device__ __forceinline__ float pow2_ceil(float x) {
  return __uint_as_float((__float_as_uint(x) + 0x007FFFFFu) & 0xFF800000u);
}

struct BiasedSum {
  uint64_t s, e;  // biased running sums and their rounding errors (two lanes)
  uint64_t h, l;  // float pairs (two lanes) of the epochs closed so far
  float sigma;    // bias of the current epoch (both lanes)
  float bound;    // bound of the sum of |products| added so far (plus the reserved segment)
};

__device__ __forceinline__ void bs_init(BiasedSum& a) {
  a.s = a.e = a.h = a.l = 0ull;
  a.sigma = 0.f;
  a.bound = 0.f;
}
// Closes the current epoch: (s - sigma) + e joins the pair (h, l).
__device__ __forceinline__ void bs_close(BiasedSum& a) {
  f2_acc(a.h, a.l, f2sub(a.s, f2splat(a.sigma)));  // s - sigma is exact in each lane
  a.l = f2add(a.l, a.e);
}
// Reserves room for a segment whose sum of |products| is at most `add` (a plain fp32
// estimate; the relative margin 2^-12 covers its rounding and that of the bound itself).
__device__ __forceinline__ void bs_reserve(BiasedSum& a, float add) {
  a.bound = fmaf(add, 1.000244140625f, a.bound);
  if (2.f * a.bound > a.sigma) {
    bs_close(a);
    a.sigma = pow2_ceil(4.f * a.bound);
    a.s = f2splat(a.sigma);
    a.e = 0ull;
  }
}
// One Fast2Sum step of a biased running sum s (error collected in e): the exact products
// x y (two lanes), |x y| <= |s| with s - t exact (the caller's bias guarantees both).
__device__ __forceinline__ void biased_add(uint64_t& s, uint64_t& e, uint64_t x, uint64_t y) {
  const uint64_t t = f2fma(x, y, s);
  e = f2add(e, f2fma(x, y, f2sub(s, t)));
  s = t;
}
// Adds the exact products x y (two lanes).
__device__ __forceinline__ void bs_add(BiasedSum& a, uint64_t x, uint64_t y) {
  const uint64_t t = f2fma(x, y, a.s);
  const uint64_t z = f2sub(a.s, t);
  a.e = f2add(a.e, f2fma(x, y, z));
  a.s = t;
}
// The two lanes' pairs of the finished sum, to be combined by f2_finish.
__device__ __forceinline__ void bs_finish(BiasedSum& a, uint64_t& s, uint64_t& e) {
  bs_close(a);
  s = a.h;
  e = a.l;
}

// One warp: |z|^2 of the row at element offset zrow of `base` and, if has_p, its dot with
// the row at poff of `pbase`, as float pairs.  bf16 products are exact in fp32, fp32
// products are split by TwoProduct, sums are compensated (Sum2) per lane and the lanes'
// pairs combined in a fixed butterfly (deterministic).  Rows start on 16-byte boundaries.
template <bool kBf16>
__device__ __forceinline__ void exact_pair_sums(const void* base, int64_t zrow, const void* pbase, int64_t prow,
                                                bool has_p, int d, int lane, float2& n2, float2& dot) {
  float nh = 0.f, nl = 0.f, dh = 0.f, dl = 0.f;
  constexpr int kVec = kBf16 ? 8 : 4;  // elements per 16-byte chunk
  const int nvec = d / kVec;
  for (int c = lane; c < nvec; c += 32) {
    float x[kVec], y[kVec];
    if (kBf16) {
      const uint4 u = *reinterpret_cast<const uint4*>(reinterpret_cast<const uint16_t*>(base) + zrow + 8 * c);
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
      }
      if (has_p) {
        const uint4 v = *reinterpret_cast<const uint4*>(reinterpret_cast<const uint16_t*>(pbase) + prow + 8 * c);
        const uint32_t q[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          y[2 * i] = __uint_as_float(q[i] << 16);
          y[2 * i + 1] = __uint_as_float(q[i] & 0xFFFF0000u);
        }
      }
    } else {
      const float4 u = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(base) + zrow + 4 * c);
      x[0] = u.x; x[1] = u.y; x[2] = u.z; x[3] = u.w;
      if (has_p) {
        const float4 v = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(pbase) + prow + 4 * c);
        y[0] = v.x; y[1] = v.y; y[2] = v.z; y[3] = v.w;
      }
    }
#pragma unroll
    for (int i = 0; i < kVec; ++i) {
      const float sq = x[i] * x[i];
      ff_acc(nh, nl, sq);
      if (!kBf16) nl += fmaf(x[i], x[i], -sq);  // TwoProduct error (bf16 squares are exact)
      if (has_p) {
        const float pr = x[i] * y[i];
        ff_acc(dh, dl, pr);
        if (!kBf16) dl += fmaf(x[i], y[i], -pr);
      }
    }
  }
  for (int k = nvec * kVec + lane; k < d; k += 32) {  // ragged tail of the row
    const float x = kBf16 ? __uint_as_float((uint32_t)(reinterpret_cast<const uint16_t*>(base)[zrow + k]) << 16)
                          : reinterpret_cast<const float*>(base)[zrow + k];
    const float sq = x * x;
    ff_acc(nh, nl, sq);
    nl += fmaf(x, x, -sq);
    if (has_p) {
      const float y = kBf16 ? __uint_as_float((uint32_t)(reinterpret_cast<const uint16_t*>(pbase)[prow + k]) << 16)
                            : reinterpret_cast<const float*>(pbase)[prow + k];
      const float pr = x * y;
      ff_acc(dh, dl, pr);
      dl += fmaf(x, y, -pr);
    }
  }
  // combine the lanes' pairs (fixed butterfly order: deterministic)
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float a = __shfl_xor_sync(0xffffffffu, nh, o), b = __shfl_xor_sync(0xffffffffu, nl, o);
    const float c = __shfl_xor_sync(0xffffffffu, dh, o), e = __shfl_xor_sync(0xffffffffu, dl, o);
    float s, t;
    two_sum(nh, a, s, t);
    nh = s;
    nl = nl + b + t;
    two_sum(dh, c, s, t);
    dh = s;
    dl = dl + e + t;
  }
  float h, l;
  two_sum(nh, nl, h, l);
  n2 = make_float2(h, l);
  two_sum(dh, dl, h, l);
  dot = make_float2(h, l);
}

// ------------------------------------------------------------------ token spans

// One warp writes value v to dst[ts, te): 16-byte stores in the aligned middle,
// scalar stores for the unaligned ends (dst must be 16-byte aligned).
__device__ __forceinline__ void write_span(float* dst, int64_t ts, int64_t te, float v, int lane) {
  const int64_t a = min(te, (ts + 3) & ~int64_t(3));
  const int64_t z = max(a, te & ~int64_t(3));
  if (lane < a - ts) dst[ts + lane] = v;
  const float4 v4 = make_float4(v, v, v, v);
  for (int64_t q = (a >> 2) + lane; q < (z >> 2); q += 32) reinterpret_cast<float4*>(dst)[q] = v4;
  if (lane < te - z) dst[z + lane] = v;
}

__device__ __forceinline__ void write_span_u8(uint8_t* dst, int64_t ts, int64_t te, uint8_t v, int lane) {
  const int64_t a = min(te, (ts + 3) & ~int64_t(3));
  const int64_t z = max(a, te & ~int64_t(3));
  if (lane < a - ts) dst[ts + lane] = v;
  const uint32_t v4 = 0x01010101u * v;
  for (int64_t q = (a >> 2) + lane; q < (z >> 2); q += 32) reinterpret_cast<uint32_t*>(dst)[q] = v4;
  if (lane < te - z) dst[z + lane] = v;
}

// ------------------------------------------------------------------ launchers (host)

struct LaunchCtx {
  cudaStream_t stream;
  int num_sms;
};

cudaError_t launch_prep(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws);
// with_norms: ws.nrm2 holds every row's fp32 squared norm (the similarity stage ran first)
cudaError_t launch_exact_stats(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws,
                               bool with_norms = false);
cudaError_t launch_tree_prep(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws);
cudaError_t setup_tree_prep();
cudaError_t launch_row_stats(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws);
cudaError_t launch_sim_tc(const LaunchCtx& lc, const CUtensorMap& map, const gpo_batch& b, const Sizes& sz,
                          const Ws& ws, const Params& p);
cudaError_t launch_sim_simt(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const Ws& ws,
                            const Params& p);
cudaError_t launch_groups(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                          const Ws& ws, const Params& p);
cudaError_t launch_tokens(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                          const Ws& ws);

// Records a message on the context (gpo_last_error).
void note_error(gpo_ctx* ctx, const char* msg);

// CTAs the fused kernel runs with for groups [g0, g1) (one group each when ng <= this).
int fused_grid(const LaunchCtx& lc, const Sizes& sz);
cudaError_t launch_fused(const LaunchCtx& lc, const CUtensorMap& map, const CUtensorMap& map32, const gpo_batch& b,
                         const gpo_outputs& o, const Sizes& sz, const Ws& ws, const Params& p);
cudaError_t setup_fused();
// fp32 group-resident path (chain layout, small groups whose rows fit in shared memory)
bool fused_f32_fits(int d, int maxn);
cudaError_t setup_fused_f32();
cudaError_t launch_fused_f32(const LaunchCtx& lc, const gpo_batch& b, const gpo_outputs& o, const Sizes& sz,
                             const Ws& ws, const Params& p);
cudaError_t setup_sim_tc();
cudaError_t setup_groups();
size_t sim_tc_smem_bytes();
size_t groups_smem_bytes(int maxn);

// ------------------------------------------------------------------ policy loss

constexpr int kLossTile = 4096;        // tokens per tile of the loss kernel
constexpr int kLossMaxBlocks = 1024;   // CTAs of one loss launch at most (reduction scratch)
constexpr int kLossPlanHead = 256;     // bytes: status words, then the group count and the ticket
constexpr int kLossWordGroups = kStatusWords, kLossWordTicket = kStatusWords + 1;

// Device views of a loss plan (gpo_loss_plan), laid out on the host.
struct LossPlan {
  uint32_t* status;      // [kStatusWords], then [kLossWordGroups] groups with states, [kLossWordTicket]
  int64_t* dims;         // [2] N and T of the batch the plan was built for (in the head, at byte 128)
  int64_t* start;        // [N+1] first token of every edge, start[N] = T
  float* w;              // [N] 1 / (G' |E_g| |e|) of the edge's tokens (first the group's |E_g|)
  int32_t* tile_edge;    // [ntiles+1] edge holding each tile's first token; [ntiles] = N - 1
  double* partial;       // [kLossMaxBlocks * 4] per-CTA sums of one loss launch
  int64_t ntiles;
};

struct LossArgs {
  const float* logp;
  const float* old_logp;
  const float* ref_logp;
  const float* adv;      // dual: A_dual; split: A_cor
  const float* eff;      // split: routed A_eff
  const uint8_t* mask;   // split: m_eff
  float* loss;
  float* grad;
  double* stats;
  float lo, hi, beta, lambda;
  float inv_t;           // (float)(1 / T) rounded once on the host (0 for T = 0)
  int norm_token;        // 1: weights 1/T
  int split, kl;
  int N;
  int64_t T;
};

cudaError_t launch_loss_plan(const LaunchCtx& lc, const gpo_batch& b, const Sizes& sz, const LossPlan& lp);
cudaError_t launch_token_loss(const LaunchCtx& lc, const LossPlan& lp, const LossArgs& a);
cudaError_t setup_loss();

}  // namespace gpo
