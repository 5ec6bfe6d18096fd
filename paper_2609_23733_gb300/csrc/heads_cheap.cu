// The routed head outputs Y of one layer (Algorithm 1, step 2): full-mode heads in
// attn_full_kernel, then surrogate (§4.3) and mean heads in cheap_heads_kernel, queued
// behind it with programmatic dependent launch.  The full-attention CTAs signal their
// dependents as soon as they start, so cheap-head CTAs take each SM as soon as a
// full-attention CTA retires: the cheap heads fill the SMs that the last round of
// full-attention items leaves idle.  The cheap kernel reads only router outputs (bins, C_h,
// mean of V), which were complete before the full-attention kernel started; it waits for
// the full-attention grid (griddepcontrol.wait) before it exits, so work queued after it
// sees every head's Y.
#include "cheap_modes.cuh"
#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads, 3) cheap_heads_kernel(HeadAttnArgs a) {
  __shared__ __align__(16) cheap::SurrSmem surr;
  __shared__ int s_item;
  const int tid = threadIdx.x, lane = tid & 31;
  const int s_first = __ldg(a.offsets + 1), m_first = __ldg(a.offsets + 0);
  const int n_surr = __ldg(a.offsets + 2) - s_first;
  const int n_mean = s_first - m_first;
  const int s_chunks = (a.N + cheap::kSurrRows - 1) / cheap::kSurrRows;
  const int m_chunks = (a.N + cheap::kMeanRows - 1) / cheap::kMeanRows;
  // The linear-attention form of the surrogate heads runs in its own kernels, before this one.
  const int s_items = (a.variant & VP_VARIANT_LINEAR_ATTENTION) ? 0 : n_surr * s_chunks;
  const int items = s_items + n_mean * m_chunks;
  int cur_h = -1;
  // Items in order: surrogate rows (head-major), then mean rows; taken from a counter so
  // that CTAs started early (on SMs freed early) do more of them.
  for (;;) {
    __syncthreads();  // s_item is free, and the previous item's weights are no longer read
    if (tid == 0) s_item = (int)atomicAdd(a.cheap_counter, 1u);
    __syncthreads();
    const int it = s_item;
    if (it >= items) break;
    if (it < s_items) {
      const int slot = it / s_chunks, chunk = it - slot * s_chunks;
      const int h = __ldg(a.head_ids + s_first + slot);
      if (a.variant & VP_VARIANT_NO_RESIDUAL) {  // §5: y_i = C_h, no token-wise correction
        cheap::broadcast_rows(a, a.ctx + h * 64, h, chunk * cheap::kSurrRows, cheap::kSurrRows, tid);
        continue;
      }
      if (h != cur_h) {
        cheap::surrogate_stage(a, surr, h, tid);
        __syncthreads();
        cheap::surrogate_fold(a, surr, h, tid);
        __syncthreads();
        cur_h = h;
      }
      cheap::surrogate_rows(a, surr, h, chunk, tid >> 5, lane);
    } else {
      const int it2 = it - s_items;
      const int slot = it2 / m_chunks, chunk = it2 - slot * m_chunks;
      cheap::mean_item(a, __ldg(a.head_ids + m_first + slot), chunk, tid);
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
  e = cudaLaunchKernelEx(&cfg, cheap_heads_kernel, a);
  prof_extra_launch();
  prof_after(st);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace vp
