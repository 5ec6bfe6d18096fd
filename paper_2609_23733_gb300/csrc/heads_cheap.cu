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
constexpr int kLinTile = 64;  // tokens per shared-memory tile of the linear-attention state

// §5 compute-mode ablation: the state of linear attention for every surrogate head,
// S_h[c][e] = sum_j phi(k_j)[c] v_j[e] and z_h[c] = sum_j phi(k_j)[c] (fp32 CUDA cores:
// 4,096 FMA per token).  Grid (splits, H): blockIdx.y is the slot in the surrogate bin (CTAs
// past the bin's end return); each CTA sums a token range and adds its partial state to
// lin_state (zeroed by the launcher) with atomics.  Thread t owns the 4 x 4 block
// S[4 (t / 16) ..+4][4 (t % 16) ..+4]: two 16-byte shared loads per token for 16 FMA.
__global__ void __launch_bounds__(kThreads) linear_state_kernel(HeadAttnArgs a, int n_split) {
  __shared__ __align__(16) float s_fk[kLinTile][64];
  __shared__ __align__(16) float s_v[kLinTile][64];
  const int s_first = __ldg(a.offsets + 1), n_surr = __ldg(a.offsets + 2) - s_first;
  if ((int)blockIdx.y >= n_surr) return;
  const int h = __ldg(a.head_ids + s_first + blockIdx.y);
  const int tid = threadIdx.x, c0 = (tid >> 4) * 4, e0 = (tid & 15) * 4;
  const int per = (a.N + n_split - 1) / n_split;
  const int t0 = blockIdx.x * per, t1 = min(a.N, t0 + per);
  const size_t row_pitch = (size_t)3 * a.H * kHeadDim;
  float acc[4][4], zc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int k = 0; k < 4; ++k) acc[i][k] = 0.f;
  for (int base = t0; base < t1; base += kLinTile) {
    __syncthreads();  // the previous tile is no longer read
    // Stage phi(K) and V for kLinTile tokens (zeros past t1): 8 channels per thread and matrix.
    for (int i = tid; i < kLinTile * 8; i += kThreads) {
      const int r = i >> 3, ch = (i & 7) * 8, t = base + r;
      float fk[8], vv[8];
      if (t < t1) {
        const __nv_bfloat16* row = a.qkv + (size_t)t * row_pitch;
        const uint4 ku = __ldg(reinterpret_cast<const uint4*>(row + (size_t)(a.H + h) * kHeadDim + ch));
        const uint4 vu = __ldg(reinterpret_cast<const uint4*>(row + (size_t)(2 * a.H + h) * kHeadDim + ch));
        const uint32_t kw[4] = {ku.x, ku.y, ku.z, ku.w}, vw[4] = {vu.x, vu.y, vu.z, vu.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          fk[2 * k] = cheap::elu1(bf16_lo(kw[k]));
          fk[2 * k + 1] = cheap::elu1(bf16_hi(kw[k]));
          vv[2 * k] = bf16_lo(vw[k]);
          vv[2 * k + 1] = bf16_hi(vw[k]);
        }
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) fk[k] = vv[k] = 0.f;
      }
      float4* dk = reinterpret_cast<float4*>(&s_fk[r][ch]);
      float4* dv = reinterpret_cast<float4*>(&s_v[r][ch]);
      dk[0] = make_float4(fk[0], fk[1], fk[2], fk[3]);
      dk[1] = make_float4(fk[4], fk[5], fk[6], fk[7]);
      dv[0] = make_float4(vv[0], vv[1], vv[2], vv[3]);
      dv[1] = make_float4(vv[4], vv[5], vv[6], vv[7]);
    }
    __syncthreads();
    const int rows = min(kLinTile, t1 - base);
    for (int r = 0; r < rows; ++r) {
      const float4 f4 = *reinterpret_cast<const float4*>(&s_fk[r][c0]);
      const float4 v4 = *reinterpret_cast<const float4*>(&s_v[r][e0]);
      const float f[4] = {f4.x, f4.y, f4.z, f4.w}, v[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        zc[i] += f[i];
#pragma unroll
        for (int k = 0; k < 4; ++k) acc[i][k] = fmaf(f[i], v[k], acc[i][k]);
      }
    }
  }
  float* st = a.lin_state + (size_t)h * kLinState;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int k = 0; k < 4; ++k) atomicAdd(st + (c0 + i) * 64 + e0 + k, acc[i][k]);
  if ((tid & 15) == 0)
#pragma unroll
    for (int i = 0; i < 4; ++i) atomicAdd(st + 64 * 64 + c0 + i, zc[i]);
}

__global__ void __launch_bounds__(kThreads, 3) cheap_heads_kernel(HeadAttnArgs a) {
  __shared__ __align__(16) union {
    cheap::SurrSmem surr;
    cheap::LinSmem lin;
  } sm;
  cheap::SurrSmem& surr = sm.surr;
  __shared__ int s_item;
  const int tid = threadIdx.x, lane = tid & 31;
  const int s_first = __ldg(a.offsets + 1), m_first = __ldg(a.offsets + 0);
  const int n_surr = __ldg(a.offsets + 2) - s_first;
  const int n_mean = s_first - m_first;
  const int s_chunks = (a.N + cheap::kSurrRows - 1) / cheap::kSurrRows;
  const int m_chunks = (a.N + cheap::kMeanRows - 1) / cheap::kMeanRows;
  const int items = n_surr * s_chunks + n_mean * m_chunks;
  int cur_h = -1;
  // Items in order: surrogate rows (head-major), then mean rows; taken from a counter so
  // that CTAs started early (on SMs freed early) do more of them.
  for (;;) {
    __syncthreads();  // s_item is free, and the previous item's weights are no longer read
    if (tid == 0) s_item = (int)atomicAdd(a.cheap_counter, 1u);
    __syncthreads();
    const int it = s_item;
    if (it >= items) break;
    if (it < n_surr * s_chunks) {
      const int slot = it / s_chunks, chunk = it - slot * s_chunks;
      const int h = __ldg(a.head_ids + s_first + slot);
      if (a.variant & VP_VARIANT_NO_RESIDUAL) {  // §5: y_i = C_h, no token-wise correction
        cheap::broadcast_rows(a, a.ctx + h * 64, h, chunk * cheap::kSurrRows, cheap::kSurrRows, tid);
        continue;
      }
      if (a.variant & VP_VARIANT_LINEAR_ATTENTION) {  // §5: linear attention instead
        if (h != cur_h) {
          cheap::linear_stage(a, sm.lin, h, tid);
          __syncthreads();
          cur_h = h;
        }
        cheap::linear_rows(a, sm.lin, h, chunk, tid >> 5, lane);
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
      const int it2 = it - n_surr * s_chunks;
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
    // The state is complete before the full-attention kernel starts, hence before the
    // cheap-heads kernel (which follows that one) reads it.
    e = cudaMemsetAsync(a.lin_state, 0, sizeof(float) * kLinState * a.H, st);
    if (e != cudaSuccess) return e;
    const int n_split = max(1, min((a.N + 1023) / 1024, (4 * num_sms + a.H - 1) / a.H));
    prof_before(VP_KERNEL_SURROGATE, st);
    linear_state_kernel<<<dim3(n_split, a.H), kThreads, 0, st>>>(a, n_split);
    prof_after(st);
    e = cudaGetLastError();
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
