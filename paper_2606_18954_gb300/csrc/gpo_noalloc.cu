// gpo_compute_noalloc: the whole advantage path without any device allocation
// by the caller or by the library.
//
// Some callers cannot allocate device memory at the moment they need the
// advantages: a trainer whose device memory is entirely owned by a
// framework's pool with no head-room left, a plug-in hosted by an application
// that forbids allocation calls from its extensions, or a latency-critical
// loop that cannot afford cudaMalloc's implicit device-wide synchronisation.
// For them the workspace comes from one fixed array compiled into this
// library (GPO_NOALLOC_SCRATCH_BYTES).  Every GPU that loads the library
// holds that array until the process exits.
//
// The first call on a device looks up the array's device address
// (cudaGetSymbolAddress, with that device current) and caches it; make that
// first call before any stream capture.  Every later call on the device reuses
// the same array, which keeps whatever the previous call left in it: the
// status words at its head are cleared by each call, and every other part of
// the workspace is written before it is read.  Calls whose work overlaps on the
// GPU (other streams, other contexts, other host threads) share the array and
// race; the caller must order them.
#include <cstdio>
#include <mutex>

#include "gpo_internal.cuh"

namespace {

constexpr size_t kScratchBytes = GPO_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices];  // device address of g_scratch, per device (null until set up)

}  // namespace

extern "C" gpo_status gpo_compute_noalloc(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out,
                                          void* stream) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  size_t need = 0;
  const gpo_status s = gpo_workspace_size(ctx, batch, &need);
  if (s != GPO_OK) return s;
  if (need > kScratchBytes) {
    char msg[160];
    snprintf(msg, sizeof msg, "batch needs %zu bytes of workspace; the built-in scratch holds %zu", need,
             kScratchBytes);
    gpo::note_error(ctx, msg);
    return GPO_ERR_WORKSPACE;
  }
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    gpo::note_error(ctx, "no usable current device for the built-in scratch");
    return GPO_ERR_CUDA;
  }
  void* p = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    p = g_scratch_addr[dev];
    if (!p) {
      const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        gpo::note_error(ctx, "cudaGetSymbolAddress of the built-in scratch failed");
        return GPO_ERR_CUDA;
      }
      g_scratch_addr[dev] = p;
    }
  }
  return gpo_compute(ctx, batch, out, p, kScratchBytes, stream);
}
