// Fused group-resident path: the whole advantage construction for bf16
// prompt groups of at most 384 states, persistent CTAs working through their
// groups.  Two instances of the kernel body (gpo_fused_body.cuh): one for groups
// of up to 384 states (512 threads, one CTA per SM, 160 KB tile ring, 512 TMEM
// columns) and one for groups of up to 128 states (256 threads, two CTAs per SM,
// 76 KB ring, 128 TMEM columns), chosen by the batch's largest group.
//
// Per group g (states [s0, s0+n), rollouts [r0, r0+nr)):
//   producer warp   TMA: per k-slice of 64 embedding elements, the group's
//                   rows as ceil(n/128) boxes of 128 rows x 128 B (128B swizzle)
//   MMA warp        tcgen05.mma kind::f16 (bf16 -> fp32 in TMEM) of the upper
//                   triangle in 128-row blocks: block b against columns
//                   [128 b, n), at most 512 accumulator columns per pass;
//                   if a group needs more, blocks >= 1 go first, block 0 second
//                   (Sec. 4.2: sim of every comparable pair)
//   warps 4..       TMEM drain of each pass (three (large) or one (small) warps per
//                   accumulator lane quarter, splitting the 32-column chunks): the diagonal
//                   entries give |z_i|^2 (the norms of the threshold test); then every
//                   comparable pair (not ancestor-related; optionally same depth) with
//                   cos = acc / (|z_i||z_j|) >= kappa goes to an edge list; the
//                   accumulator is released and the listed pairs are united in a
//                   shared-memory union-find forest (Alg. S.1)
//   warps 2..       per-group validation; the compensated row statistics of the group
//                   (eta(p(v), v) needs them) while the producer streams it, when every
//                   CTA has one group (else exact_stats runs as a launch of its own just
//                   before, on the whole GPU); graph reward and dual-group advantage
//                   (gpo_group_math.cuh) and the token scatter (Sec. 4.5), overlapping
//                   the next group's loads and MMAs
// Group ranges are assigned round-robin to CTAs.  Every wait is bounded.
#include "gpo_group_math.cuh"

namespace gpo {

namespace fused_large {
constexpr int kMaxN = kFusedMaxStates;  // 384
constexpr int kThreads = 512;
constexpr int kMinBlocks = 1;
constexpr int kRingBytes = 160 * 1024;
constexpr int kTmemCols = 512;
#include "gpo_fused_body.cuh"
}  // namespace fused_large

namespace fused_small {
constexpr int kMaxN = 128;
constexpr int kThreads = 256;
constexpr int kMinBlocks = 2;
constexpr int kRingBytes = 76 * 1024;
constexpr int kTmemCols = 128;
#include "gpo_fused_body.cuh"
}  // namespace fused_small

cudaError_t setup_fused() {
  cudaError_t e = cudaFuncSetAttribute(fused_large::fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)fused_large::fused_smem());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(fused_small::fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)fused_small::fused_smem());
  return e;
}

int fused_grid(const LaunchCtx& lc, const Sizes& sz) {
  const int ng = sz.g1 - sz.g0;
  const int cap = lc.num_sms * (sz.maxn <= fused_small::kMaxN ? fused_small::kMinBlocks : fused_large::kMinBlocks);
  return ng < cap ? ng : cap;
}

cudaError_t launch_fused(const LaunchCtx& lc, const CUtensorMap& map, const CUtensorMap& map32, const gpo_batch& b,
                         const gpo_outputs& o, const Sizes& sz, const Ws& ws, const Params& p) {
  const int ng = sz.g1 - sz.g0;
  if (ng <= 0) return cudaSuccess;
  const int grid = fused_grid(lc, sz);
  if (sz.maxn <= fused_small::kMaxN)
    fused_small::fused_kernel<<<grid, fused_small::kThreads, fused_small::fused_smem(), lc.stream>>>(map, map32, b, o,
                                                                                                   sz, ws, p);
  else
    fused_large::fused_kernel<<<grid, fused_large::kThreads, fused_large::fused_smem(), lc.stream>>>(map, map32, b, o,
                                                                                                   sz, ws, p);
  return cudaGetLastError();
}

}  // namespace gpo
