// LayerNorm of Algorithm 1 (steps 1 and 4): out = (x - mean) / sqrt(var + eps) * gamma + beta
// over rows of D channels (biased variance), bf16 in and out, fp32 statistics.
// Persistent warps, two rows per iteration; each lane holds D/32 values of a row and its
// channels' gamma / beta in registers (two passes over registers, one pass over HBM).
#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

template <int C>  // 16-byte chunks per lane: D = 256 C
__global__ void __launch_bounds__(256) layernorm_kernel(int M, const __nv_bfloat16* x,
                                                        const float* g, const float* b,
                                                        float eps, __nv_bfloat16* out) {
  constexpr int D = 256 * C;
  // Up to D = 1024 a lane keeps its channels' gamma / beta in registers and has two rows
  // in flight; wider rows read gamma / beta per row (from L1) and go one row at a time.
  constexpr bool kKeep = C <= 4;
  constexpr int kRows = kKeep ? 2 : 1;
  const int lane = threadIdx.x & 31;
  const int warp_global = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int n_warps = gridDim.x * 8;
  float gr[kKeep ? 8 * C : 1], br[kKeep ? 8 * C : 1];
#pragma unroll
  for (int c = 0; c < (kKeep ? C : 0); ++c) {
    const int col = (c * 32 + lane) * 8;
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(g + col));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(g + col) + 1);
    const float4 b0 = __ldg(reinterpret_cast<const float4*>(b + col));
    const float4 b1 = __ldg(reinterpret_cast<const float4*>(b + col) + 1);
    gr[8 * c + 0] = g0.x; gr[8 * c + 1] = g0.y; gr[8 * c + 2] = g0.z; gr[8 * c + 3] = g0.w;
    gr[8 * c + 4] = g1.x; gr[8 * c + 5] = g1.y; gr[8 * c + 6] = g1.z; gr[8 * c + 7] = g1.w;
    br[8 * c + 0] = b0.x; br[8 * c + 1] = b0.y; br[8 * c + 2] = b0.z; br[8 * c + 3] = b0.w;
    br[8 * c + 4] = b1.x; br[8 * c + 5] = b1.y; br[8 * c + 6] = b1.z; br[8 * c + 7] = b1.w;
  }
  // kRows rows per iteration: all of their loads are issued before any arithmetic.
  for (int r0 = kRows * warp_global; r0 < M; r0 += kRows * n_warps) {
    uint4 u[kRows][C];
#pragma unroll
    for (int k = 0; k < kRows; ++k) {
      const int row = min(r0 + k, M - 1);
#pragma unroll
      for (int c = 0; c < C; ++c)
        u[k][c] = __ldg(reinterpret_cast<const uint4*>(x + (size_t)row * D + (c * 32 + lane) * 8));
    }
#pragma unroll
    for (int k = 0; k < kRows; ++k) {
      const int row = r0 + k;
      float v[8 * C];
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t w[4] = {u[k][c].x, u[k][c].y, u[k][c].z, u[k][c].w};
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
      if (row < M) {
        __nv_bfloat16* orow = out + (size_t)row * D;
#pragma unroll
        for (int c = 0; c < C; ++c) {
          float y[8];
          if constexpr (kKeep) {
#pragma unroll
            for (int e = 0; e < 8; ++e) y[e] = (v[8 * c + e] - mean) * rstd * gr[8 * c + e] + br[8 * c + e];
          } else {
            const int col = (c * 32 + lane) * 8;
            const float4 g0 = __ldg(reinterpret_cast<const float4*>(g + col));
            const float4 g1 = __ldg(reinterpret_cast<const float4*>(g + col) + 1);
            const float4 b0 = __ldg(reinterpret_cast<const float4*>(b + col));
            const float4 b1 = __ldg(reinterpret_cast<const float4*>(b + col) + 1);
            const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
            const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) y[e] = (v[8 * c + e] - mean) * rstd * gg[e] + bb[e];
          }
          uint4 o4;
          o4.x = pack_bf16x2(y[0], y[1]);
          o4.y = pack_bf16x2(y[2], y[3]);
          o4.z = pack_bf16x2(y[4], y[5]);
          o4.w = pack_bf16x2(y[6], y[7]);
          *reinterpret_cast<uint4*>(orow + (c * 32 + lane) * 8) = o4;
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_layer_norm(int M, int D, const __nv_bfloat16* x, const float* g,
                              const float* b, float eps, __nv_bfloat16* out, cudaStream_t st) {
  // Persistent warps (one row pair at a time); grid sized to fill every SM.
  int sms = 0, dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int blocks = max(1, min((M + 15) / 16, sms * 4));
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
