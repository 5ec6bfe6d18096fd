// vp_router_noalloc: the router (vp_router) for callers that cannot allocate device memory.
//
// Some callers cannot hand the library a workspace: they run where device allocation is
// not available to them at call time, for example a plug-in inside a host framework whose
// memory pool already reserves the GPU's memory and forbids raw cudaMalloc, or a service
// that must not allocate once it is running.  This entry point takes the router's scratch
// (split partials, counters, pooled queries, bins, error word) from a fixed buffer that lives
// in the library's own device memory instead of a caller workspace.  It checks its arguments
// with the same functions as vp_router and runs exactly the kernels of vp_router.
//
// The buffer is a file-scope __device__ array of kStaticScratchBytes, the router scratch for
// up to kMaxHeads = 32 heads (about 1.56 MiB).  Every GPU that loads the library holds it until
// the process exits.  The CUDA runtime places it in device memory when it loads this file's
// device code, which by default (lazy module loading) happens at the first call on a device.
// All calls on a device share it and it keeps the last call's contents; the counters that
// must start at zero are cleared at the start of every call (launch_router), while the error
// word accumulates until vp_router_noalloc_error reads and clears it.  Calls whose kernels
// overlap on the GPU (different streams, or different host threads, without ordering between
// them) race on the buffer and must be serialised by the caller.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "internal.h"
#include "vp.h"

namespace vp {
namespace {

constexpr size_t kStaticScratchBytes = 1634304;
static_assert(router_scratch_bytes(kMaxHeads) <= kStaticScratchBytes,
              "the fixed router scratch no longer holds the router scratch of kMaxHeads heads");

static __device__ __align__(256) unsigned char g_router_scratch[kStaticScratchBytes];

// Device address of g_router_scratch per device, with the context it was looked up in.  In
// host code the array's name is only a host-side stand-in, never a device address, so the
// address comes from cudaGetSymbolAddress with the device current.  A device reset or the
// teardown of the primary context gives the device a new context, in which the module (and
// the buffer) is loaded again: the address is looked up again whenever the current context
// is not the one it was found in.
struct ScratchSlot {
  CUcontext ctx = nullptr;
  void* addr = nullptr;
};
ScratchSlot g_slot[64];
std::mutex g_slot_mu;

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
CtxGetCurrentFn g_ctx_get_current = nullptr;
std::once_flag g_ctx_once;

CUcontext current_context() {
  std::call_once(g_ctx_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_ctx_get_current = reinterpret_cast<CtxGetCurrentFn>(fn);
  });
  CUcontext c = nullptr;
  if (!g_ctx_get_current || g_ctx_get_current(&c) != CUDA_SUCCESS) return nullptr;
  return c;
}

// Set-up, once per device and context, with that device current.
vp_status static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return VP_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_slot_mu);
  ScratchSlot& s = g_slot[dev];
  CUcontext ctx = current_context();
  if (!s.addr || !ctx || ctx != s.ctx) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_router_scratch) != cudaSuccess || !p) return VP_ERR_CUDA;
    s.addr = p;
    s.ctx = current_context();  // the runtime made the device's primary context current
  }
  *out = s.addr;
  return VP_OK;
}

}  // namespace
}  // namespace vp

using namespace vp;

extern "C" vp_status vp_router_noalloc(const vp_dims* dims, const vp_bf16* qkv,
                                       const vp_router_weights* rw, const int32_t* force_modes,
                                       float* s, int32_t* modes, float* q_pool, float* ctx,
                                       float* mean_v, float* r, void* stream) {
  vp_status st = check_dims(dims);  // shape (1 <= H <= 32), taus, variant bits, as vp_router
  if (st != VP_OK) return st;
  if (router_scratch_bytes(dims->H) > kStaticScratchBytes) return VP_ERR_STATIC_SCRATCH;
  if (!qkv || !s || !modes) return VP_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(qkv) & 15u) return VP_ERR_ALIGNMENT;
  if ((st = check_router_weights(rw)) != VP_OK) return st;
  if (!device_is_sm103()) return VP_ERR_UNSUPPORTED_DEVICE;
  void* ws = nullptr;
  if ((st = static_scratch(&ws)) != VP_OK) return st;
  RouterScratch sc = carve_router_scratch(ws, dims->H);
  RouterArgs a = make_router_args(dims, qkv, rw, force_modes);
  a.s_out = s;
  a.modes_out = modes;
  a.q_pool_out = q_pool;
  a.ctx_out = ctx;
  a.mean_v_out = mean_v;
  a.r_out = r;
  return launch_router(a, sc, device_sm_count(), static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? VP_OK
             : VP_ERR_CUDA;
}

extern "C" vp_status vp_router_noalloc_error(uint32_t* host_bits, void* stream) {
  if (!host_bits) return VP_ERR_INVALID_ARG;
  void* ws = nullptr;
  vp_status st = static_scratch(&ws);
  if (st != VP_OK) return st;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  uint32_t bits = 0;
  if (cudaMemcpyAsync(&bits, ws, 4, cudaMemcpyDeviceToHost, cs) != cudaSuccess) return VP_ERR_CUDA;
  if (cudaStreamSynchronize(cs) != cudaSuccess) return VP_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, 4, cs) != cudaSuccess) return VP_ERR_CUDA;
  *host_bits = bits;
  return (bits & VP_DEVERR_WAIT_TIMEOUT) ? VP_ERR_DEVICE_TIMEOUT : VP_OK;
}
