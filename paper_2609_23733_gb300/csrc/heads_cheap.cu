// The routed head outputs Y of one layer (Algorithm 1, step 2): full-mode heads in
// attn_full_kernel, then the surrogate (§4.3) and mean heads queued behind it with
// programmatic dependent launch (heads_cheap_tc.cu).  The full-attention CTAs signal their
// dependents as soon as they start, so cheap-head CTAs take each SM as soon as a
// full-attention CTA retires.  The cheap kernels read only router outputs (bins, C_h, mean of
// V), which were complete before the full-attention kernel started; they wait for the
// full-attention grid (griddepcontrol.wait) before they exit, so work queued after them sees
// every head's Y.
//
// Two §5 ablations change the cheap heads.  Linear attention replaces the surrogate: its two
// tcgen05 kernels (linear_attn_tc.cu) run before the full-attention kernel.  Without the
// token-wise correction a surrogate head is y_i = C_h, a broadcast like a mean head.  In both
// variants broadcast_heads_kernel writes the broadcast rows (the no-residual surrogate heads and
// the mean heads) behind the full-attention kernel.
#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kThreads = 256;
constexpr int kRows = 256;  // rows per work item

// Y[r0 .. min(N, r0 + kRows))[h][:] = Broadcast(vec[0..63]): 8 threads per row, 16-byte stores.
__device__ __forceinline__ void broadcast_rows(const HeadAttnArgs& a, const float* vec, int h,
                                               int r0, int tid) {
  const int part = tid & 7, rg = tid >> 3;
  const float* mv = vec + 8 * part;
  uint4 val;
  val.x = pack_bf16x2(__ldg(mv + 0), __ldg(mv + 1));
  val.y = pack_bf16x2(__ldg(mv + 2), __ldg(mv + 3));
  val.z = pack_bf16x2(__ldg(mv + 4), __ldg(mv + 5));
  val.w = pack_bf16x2(__ldg(mv + 6), __ldg(mv + 7));
  const int r1 = min(a.N, r0 + kRows);
  for (int row = r0 + rg; row < r1; row += kThreads / 8)
    *reinterpret_cast<uint4*>(a.y + ((size_t)row * a.H + h) * 64 + 8 * part) = val;
}

__global__ void __launch_bounds__(kThreads, 3) broadcast_heads_kernel(HeadAttnArgs a) {
  __shared__ int s_item;
  const int tid = threadIdx.x;
  const int s_first = __ldg(a.offsets + 1), m_first = __ldg(a.offsets + 0);
  const int n_surr = __ldg(a.offsets + 2) - s_first;
  const int n_mean = s_first - m_first;
  const int chunks = (a.N + kRows - 1) / kRows;
  // Surrogate heads are broadcast rows only without the token-wise correction.
  const int s_items = (a.variant & VP_VARIANT_NO_RESIDUAL) ? n_surr * chunks : 0;
  const int items = s_items + (a.skip_mean_y ? 0 : n_mean * chunks);
  // Items (surrogate rows head-major, then mean rows) from a counter, so that CTAs started
  // early (on SMs freed early) do more of them.
  for (;;) {
    __syncthreads();  // s_item is free
    if (tid == 0) s_item = (int)atomicAdd(a.cheap_counter, 1u);
    __syncthreads();
    const int it = s_item;
    if (it >= items) break;
    if (it < s_items) {
      const int slot = it / chunks, chunk = it - slot * chunks;
      const int h = __ldg(a.head_ids + s_first + slot);
      broadcast_rows(a, a.ctx + h * 64, h, chunk * kRows, tid);
    } else {
      const int it2 = it - s_items;
      const int slot = it2 / chunks, chunk = it2 - slot * chunks;
      const int h = __ldg(a.head_ids + m_first + slot);
      broadcast_rows(a, a.mean_v + h * 64, h, chunk * kRows, tid);
    }
  }
  // Do not complete before the full-attention grid: later work in the stream reads all of Y.
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

}  // namespace

cudaError_t launch_heads(const HeadAttnArgs& a, int num_sms, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(a.cheap_counter, 0, sizeof(unsigned int), st);
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(a.fa_count, 0, sizeof(unsigned int) * kFaCountWords, st);
  if (e != cudaSuccess) return e;
  if (a.s_attn) {  // 0 for the heads that are not in full mode; full heads max into it
    e = cudaMemsetAsync(a.s_attn, 0, sizeof(float) * a.H, st);
    if (e != cudaSuccess) return e;
  }
  if (a.variant & VP_VARIANT_LINEAR_ATTENTION) {
    // The surrogate heads in linear-attention form, state then apply, before the
    // full-attention kernel; the mean heads stay in the cheap-heads kernel behind it.
    e = cudaMemsetAsync(a.lin_state, 0, sizeof(float) * kLinState * a.H, st);
    if (e != cudaSuccess) return e;
    prof_before(VP_KERNEL_SURROGATE, st);
    e = launch_linear_state_tc(a, num_sms, st);
    if (e == cudaSuccess) e = launch_linear_apply_tc(a, num_sms, st);
    prof_extra_launch();
    prof_after(st);
    if (e != cudaSuccess) return e;
  }
  prof_before(VP_KERNEL_ATTN_FULL, st);  // both kernels: no event may separate them
  e = launch_full_heads(a, num_sms, st);
  if (e != cudaSuccess) return e;
  if (!(a.variant & (VP_VARIANT_NO_RESIDUAL | VP_VARIANT_LINEAR_ATTENTION))) {
    e = launch_cheap_heads_tc(a, num_sms, st);
    prof_extra_launch();
    prof_after(st);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(3 * num_sms);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, broadcast_heads_kernel, a);
  prof_extra_launch();
  prof_after(st);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace vp
