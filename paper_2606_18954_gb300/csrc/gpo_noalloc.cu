// gpo_compute_noalloc: the whole advantage path without any device allocation
// by the caller or by the library.
//
// Some callers cannot allocate device memory at the moment they need the
// advantages: a trainer whose device memory is entirely owned by a
// framework's pool with no head-room left, a plug-in hosted by an application
// that forbids allocation calls from its extensions, or a latency-critical
// loop that cannot afford cudaMalloc's implicit device-wide synchronisation.
// For them the workspace comes from one fixed array compiled into this
// library (GPO_NOALLOC_SCRATCH_BYTES).
//
// A file-scope __device__ array exists once per CUDA context: each context
// loads its own copy of this module (with lazy module loading, when the module
// is first used there) and keeps it until the context is destroyed.  In host
// code the array's name is only a host-side stand-in, so the first call in a
// context looks up the array's device address in that context
// (cudaGetSymbolAddress, which also loads the module) and caches it under the
// context's unique id (cuCtxGetId), so that a call from another context, or
// from a new primary context after cudaDeviceReset, never receives an address
// that belongs to a different context.  Make the first call in each context
// before any stream capture.  Every later call in the same context reuses the
// same array, which keeps whatever the previous call left in it: the status
// words at its head are cleared by each call, and every other part of the
// workspace is written before it is read.  Calls in one context whose work
// overlaps on the GPU (other streams, other host threads) share the array and
// race; the caller must order them.
#include <cstdio>
#include <mutex>

#include "gpo_internal.cuh"

namespace {

constexpr size_t kScratchBytes = GPO_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxContexts = 64;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

struct Cached {
  unsigned long long ctx_id;
  void* addr;
};

std::mutex g_mu;
CtxGetCurrentFn g_get_current = nullptr;
CtxGetIdFn g_get_id = nullptr;
bool g_fns_looked_up = false;
Cached g_cache[kMaxContexts];
int g_ncached = 0;

void* driver_fn(const char* name) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}

// Unique id of the calling thread's current context; false if there is none.
bool current_ctx_id(unsigned long long* id) {
  CUcontext c = nullptr;
  return g_get_current && g_get_id && g_get_current(&c) == CUDA_SUCCESS && c && g_get_id(c, id) == CUDA_SUCCESS;
}

}  // namespace

extern "C" gpo_status gpo_compute_noalloc(gpo_ctx* ctx, const gpo_batch* batch, const gpo_outputs* out,
                                          void* stream) {
  if (!ctx) return GPO_ERR_INVALID_ARG;
  gpo::note_error(ctx, "");
  size_t need = 0;
  const gpo_status s = gpo_workspace_size(ctx, batch, &need);
  if (s != GPO_OK) {
    if (gpo_last_error(ctx)[0] == 0) gpo::note_error(ctx, "batch too large for a workspace layout");
    return s;
  }
  if (need > kScratchBytes) {
    char msg[160];
    snprintf(msg, sizeof msg, "batch needs %zu bytes of workspace; the built-in scratch holds %zu", need,
             kScratchBytes);
    gpo::note_error(ctx, msg);
    return GPO_ERR_WORKSPACE;
  }
  void* p = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_fns_looked_up) {
      g_get_current = reinterpret_cast<CtxGetCurrentFn>(driver_fn("cuCtxGetCurrent"));
      g_get_id = reinterpret_cast<CtxGetIdFn>(driver_fn("cuCtxGetId"));
      g_fns_looked_up = true;
    }
    unsigned long long id = 0;
    bool have_id = current_ctx_id(&id);
    for (int i = 0; have_id && i < g_ncached && !p; ++i)
      if (g_cache[i].ctx_id == id) p = g_cache[i].addr;
    if (!p) {
      // the address in the current context (makes the device's primary context current
      // first if the thread has none, and loads the module there if needed)
      const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        gpo::note_error(ctx, "cudaGetSymbolAddress of the built-in scratch failed");
        return GPO_ERR_CUDA;
      }
      if (!have_id) have_id = current_ctx_id(&id);
      if (have_id && g_ncached < kMaxContexts) g_cache[g_ncached++] = Cached{id, p};
    }
  }
  return gpo_compute(ctx, batch, out, p, kScratchBytes, stream);
}
