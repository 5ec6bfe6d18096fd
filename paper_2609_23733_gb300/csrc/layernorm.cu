// LayerNorm of Algorithm 1 (steps 1 and 4): out = (x - mean) / sqrt(var + eps) * gamma + beta
// over rows of D channels (biased variance), bf16 in and out, fp32 statistics; and the two
// pieces of the LayerNorm that the block stack folds into its projections instead (row
// statistics per 128-column block, and the weights W diag(gamma), W 1, b + W beta).
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

// Row statistics for a LayerNorm folded into the next projection: per 128-column block of
// a row, (mean, M2 = sum (x - mean)^2).  One warp per row; lane l holds 16-byte chunks
// c 32 + l (coalesced), i.e. chunk c of lanes 0-15 is block 2c and of lanes 16-31 block
// 2c + 1; the 16 lanes of a block combine their (mean, M2) pairwise (equal counts n:
// mean = (a + b) / 2, M2 = M2_a + M2_b + (a - b)^2 n / 2).
template <int C>
__global__ void __launch_bounds__(256) ln_partials_kernel(int M, const __nv_bfloat16* x,
                                                          float2* part) {
  constexpr int D = 256 * C;
  const int lane = threadIdx.x & 31;
  const int n_warps = gridDim.x * 8;
  for (int row = blockIdx.x * 8 + (threadIdx.x >> 5); row < M; row += n_warps) {
    uint4 u[C];
#pragma unroll
    for (int c = 0; c < C; ++c)
      u[c] = __ldg(reinterpret_cast<const uint4*>(x + (size_t)row * D + (c * 32 + lane) * 8));
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t w[4] = {u[c].x, u[c].y, u[c].z, u[c].w};
      float v[8];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[2 * e] = bf16_lo(w[e]);
        v[2 * e + 1] = bf16_hi(w[e]);
      }
      float mean = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) mean += v[e];
      mean *= 0.125f;
      float m2 = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) m2 += (v[e] - mean) * (v[e] - mean);
      float n = 8.f;
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) {
        const float mo = __shfl_xor_sync(0xffffffffu, mean, o);
        const float qo = __shfl_xor_sync(0xffffffffu, m2, o);
        m2 += qo + (mean - mo) * (mean - mo) * (0.5f * n);
        mean = 0.5f * (mean + mo);
        n *= 2.f;
      }
      if ((lane & 15) == 0) part[(size_t)row * (D / 128) + 2 * c + (lane >> 4)] = make_float2(mean, m2);
    }
  }
}

// Folded LayerNorm weights: one warp per output row o of W [Nout][K]; lane l holds the
// 16-byte chunks c 32 + l of the row.
template <int C>
__global__ void __launch_bounds__(256) ln_fold_kernel(int Nout, const __nv_bfloat16* W,
                                                      const float* g, const float* beta,
                                                      const float* b, __nv_bfloat16* Wp,
                                                      float* cs, float* bp) {
  constexpr int K = 256 * C;
  const int lane = threadIdx.x & 31;
  const int o = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (o >= Nout) return;
  float csum = 0.f, bsum = 0.f;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int k0 = (c * 32 + lane) * 8;
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(W + (size_t)o * K + k0));
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(g + k0));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(g + k0) + 1);
    const float4 e0 = __ldg(reinterpret_cast<const float4*>(beta + k0));
    const float4 e1 = __ldg(reinterpret_cast<const float4*>(beta + k0) + 1);
    const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
    const float ee[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    uint32_t pw[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float w0 = bf16_lo(w[e]), w1 = bf16_hi(w[e]);
      pw[e] = pack_bf16x2(w0 * gg[2 * e], w1 * gg[2 * e + 1]);
      csum += bf16_lo(pw[e]) + bf16_hi(pw[e]);
      bsum = fmaf(w0, ee[2 * e], bsum);
      bsum = fmaf(w1, ee[2 * e + 1], bsum);
    }
    *reinterpret_cast<uint4*>(Wp + (size_t)o * K + k0) = make_uint4(pw[0], pw[1], pw[2], pw[3]);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    csum += __shfl_xor_sync(0xffffffffu, csum, off);
    bsum += __shfl_xor_sync(0xffffffffu, bsum, off);
  }
  if (lane == 0) {
    cs[o] = csum;
    bp[o] = (b ? b[o] : 0.f) + bsum;
  }
}

}  // namespace

cudaError_t launch_ln_partials(int M, int D, const __nv_bfloat16* x, float2* part,
                               cudaStream_t st) {
  int sms = 0, dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int blocks = max(1, min((M + 7) / 8, sms * 8));
  prof_before(VP_KERNEL_LAYER_NORM, st);
  switch (D / 256) {
    case 1: ln_partials_kernel<1><<<blocks, 256, 0, st>>>(M, x, part); break;
    case 2: ln_partials_kernel<2><<<blocks, 256, 0, st>>>(M, x, part); break;
    case 3: ln_partials_kernel<3><<<blocks, 256, 0, st>>>(M, x, part); break;
    case 4: ln_partials_kernel<4><<<blocks, 256, 0, st>>>(M, x, part); break;
    case 8: ln_partials_kernel<8><<<blocks, 256, 0, st>>>(M, x, part); break;
    case 16: ln_partials_kernel<16><<<blocks, 256, 0, st>>>(M, x, part); break;
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

cudaError_t launch_ln_fold_weights(int Nout, int K, const __nv_bfloat16* W, const float* g,
                                   const float* beta, const float* b, __nv_bfloat16* Wp,
                                   float* c, float* bp, cudaStream_t st) {
  const int blocks = (Nout + 7) / 8;
  prof_before(VP_KERNEL_LAYER_NORM, st);
  switch (K / 256) {
    case 1: ln_fold_kernel<1><<<blocks, 256, 0, st>>>(Nout, W, g, beta, b, Wp, c, bp); break;
    case 2: ln_fold_kernel<2><<<blocks, 256, 0, st>>>(Nout, W, g, beta, b, Wp, c, bp); break;
    case 3: ln_fold_kernel<3><<<blocks, 256, 0, st>>>(Nout, W, g, beta, b, Wp, c, bp); break;
    case 4: ln_fold_kernel<4><<<blocks, 256, 0, st>>>(Nout, W, g, beta, b, Wp, c, bp); break;
    case 8: ln_fold_kernel<8><<<blocks, 256, 0, st>>>(Nout, W, g, beta, b, Wp, c, bp); break;
    case 16: ln_fold_kernel<16><<<blocks, 256, 0, st>>>(Nout, W, g, beta, b, Wp, c, bp); break;
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

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
