// vp_router_noalloc: the router (vp_router) for callers that cannot allocate device memory.
//
// Some callers cannot hand the library a workspace: they run where device allocation is
// not available to them at call time, for example a plug-in inside a host framework whose
// memory pool already reserves the GPU's memory and forbids raw cudaMalloc, or a service
// that must not allocate once it is running.  This entry point takes the router's scratch
// (split partials, counters, pooled queries, bins) from a fixed buffer that lives in the
// library's own device memory instead of a caller workspace.  It runs exactly the kernels
// of vp_router.
//
// The buffer is a file-scope __device__ array of kStaticScratchBytes, the router scratch for
// up to 32 heads (about 1.56 MiB).  Every GPU that loads the library holds it until the
// process exits.  All calls on a device share it and it keeps the last call's contents; the
// counters that must start at zero, and the error word, are cleared at the start of every
// call.  Calls whose kernels overlap on the GPU (different streams, or different host
// threads, without ordering between them) race on the buffer and must be serialised by the
// caller.
#include <cuda_runtime.h>

#include <mutex>

#include "internal.h"
#include "vp.h"

namespace vp {
namespace {

constexpr size_t kStaticScratchBytes = 1634304;  // router_scratch_bytes() for H <= 32

static __device__ __align__(256) unsigned char g_router_scratch[kStaticScratchBytes];

// Device address of g_router_scratch, looked up once per device with that device current.
// In host code the array's name is only a host-side stand-in, never a device address.
void* g_scratch_addr[64];
std::mutex g_scratch_mu;

vp_status static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return VP_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_router_scratch) != cudaSuccess || !p) return VP_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return VP_OK;
}

}  // namespace
}  // namespace vp

using namespace vp;

extern "C" vp_status vp_router_noalloc(const vp_dims* dims, const vp_bf16* qkv,
                                       const vp_router_weights* rw, const int32_t* force_modes,
                                       float* s, int32_t* modes, float* q_pool, float* ctx,
                                       float* mean_v, float* r, void* stream) {
  if (!dims) return VP_ERR_INVALID_ARG;
  if (dims->d != kHeadDim || dims->L != kHidden || dims->H < 1 || dims->N < 1)
    return VP_ERR_UNSUPPORTED_SHAPE;
  if (dims->H > kMaxHeads || router_scratch_bytes(dims->H) > kStaticScratchBytes)
    return VP_ERR_STATIC_SCRATCH;  // more scratch than the fixed buffer holds
  if (!(dims->tau_low == dims->tau_low) || !(dims->tau_high == dims->tau_high))
    return VP_ERR_INVALID_ARG;
  if (!qkv || !s || !modes || !rw || !rw->W || !rw->U || !rw->w) return VP_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(qkv) & 15u) || (reinterpret_cast<uintptr_t>(rw->W) & 15u) ||
      (reinterpret_cast<uintptr_t>(rw->U) & 15u))
    return VP_ERR_ALIGNMENT;
  if (!device_is_sm103()) return VP_ERR_UNSUPPORTED_DEVICE;
  void* ws = nullptr;
  vp_status st = static_scratch(&ws);
  if (st != VP_OK) return st;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  RouterScratch sc = carve_router_scratch(ws, dims->H);
  if (cudaMemsetAsync(sc.err, 0, sizeof(unsigned int), cs) != cudaSuccess) return VP_ERR_CUDA;
  RouterArgs a{};
  a.N = dims->N;
  a.H = dims->H;
  a.tau_low = dims->tau_low;
  a.tau_high = dims->tau_high;
  a.qkv = reinterpret_cast<const __nv_bfloat16*>(qkv);
  a.W = reinterpret_cast<const __nv_bfloat16*>(rw->W);
  a.U = reinterpret_cast<const __nv_bfloat16*>(rw->U);
  a.w = reinterpret_cast<const __nv_bfloat16*>(rw->w);
  a.bW = rw->bW;
  a.bU = rw->bU;
  a.beta = rw->beta;
  a.force_modes = force_modes;
  a.s_out = s;
  a.modes_out = modes;
  a.q_pool_out = q_pool;
  a.ctx_out = ctx;
  a.mean_v_out = mean_v;
  a.r_out = r;
  return launch_router(a, sc, device_sm_count(), cs) == cudaSuccess ? VP_OK : VP_ERR_CUDA;
}
