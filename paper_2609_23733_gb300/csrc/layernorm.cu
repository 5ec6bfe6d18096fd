// LayerNorm of Algorithm 1 (steps 1 and 4): out = (x - mean) / sqrt(var + eps) * gamma + beta
// over rows of D channels (biased variance), bf16 in and out, fp32 statistics.
// One warp per row; each lane holds D/32 values in registers (two passes over registers,
// one pass over HBM).
#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

template <int C>  // 16-byte chunks per lane: D = 256 C
__global__ void __launch_bounds__(256) layernorm_kernel(int M, const __nv_bfloat16* x,
                                                        const float* g, const float* b,
                                                        float eps, __nv_bfloat16* out) {
  constexpr int D = 256 * C;
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const __nv_bfloat16* xr = x + (size_t)row * D;
  float v[8 * C];
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(xr + (c * 32 + lane) * 8));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[8 * c + 2 * e] = bf16_lo(w[e]);
      v[8 * c + 2 * e + 1] = bf16_hi(w[e]);
    }
  }
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 8 * C; ++i) s += v[i];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  const float mean = s * (1.f / D);
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < 8 * C; ++i) {
    const float t = v[i] - mean;
    q += t * t;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  const float rstd = rsqrtf(q * (1.f / D) + eps);
  __nv_bfloat16* orow = out + (size_t)row * D;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int col = (c * 32 + lane) * 8;
    float y[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) y[e] = (v[8 * c + e] - mean) * rstd * __ldg(g + col + e) + __ldg(b + col + e);
    uint4 u;
    u.x = pack_bf16x2(y[0], y[1]);
    u.y = pack_bf16x2(y[2], y[3]);
    u.z = pack_bf16x2(y[4], y[5]);
    u.w = pack_bf16x2(y[6], y[7]);
    *reinterpret_cast<uint4*>(orow + col) = u;
  }
}

}  // namespace

cudaError_t launch_layer_norm(int M, int D, const __nv_bfloat16* x, const float* g,
                              const float* b, float eps, __nv_bfloat16* out, cudaStream_t st) {
  const int blocks = (M + 7) / 8;
  prof_before(VP_KERNEL_LAYER_NORM, st);
  switch (D / 256) {
    case 1: layernorm_kernel<1><<<blocks, 256, 0, st>>>(M, x, g, b, eps, out); break;
    case 2: layernorm_kernel<2><<<blocks, 256, 0, st>>>(M, x, g, b, eps, out); break;
    case 3: layernorm_kernel<3><<<blocks, 256, 0, st>>>(M, x, g, b, eps, out); break;
    case 4: layernorm_kernel<4><<<blocks, 256, 0, st>>>(M, x, g, b, eps, out); break;
    case 8: layernorm_kernel<8><<<blocks, 256, 0, st>>>(M, x, g, b, eps, out); break;
    case 16: layernorm_kernel<16><<<blocks, 256, 0, st>>>(M, x, g, b, eps, out); break;
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

}  // namespace vp
