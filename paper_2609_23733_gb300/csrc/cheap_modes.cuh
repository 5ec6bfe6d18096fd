// Device code of the two cheap computation modes of a routed head, run inside the
// full-attention kernel by CTAs that have finished their full-attention work:
//   mean mode (Algorithm 1, step 2, s_h <= tau_low):  Y_h = Broadcast((1/N) sum_i V_{h,i})
//   surrogate mode (§4.3, tau_low < s_h < tau_high):
//       C_h = r_h V_h (computed by the router's key sweep),
//       z_i = [v_i, C_h], y_i = C_h + sigma(MLP_gamma(z_i)) (.) MLP_delta(z_i),
//       MLP = Linear(2d -> 64) -> GELU -> Linear(64 -> d).
// The surrogate's first layer splits as W1 z = W1[:, :d] v_i + (W1[:, d:] C_h + b1); the
// second term is one vector per head, computed once per head change.  The per-token
// products ([16 x 64] x [64 x 128], then two [16 x 64] x [64 x 64]) run on the tensor cores
// (mma.sync, fp32 accumulation); V is read once and Y written once.  A group of eight warps
// (256 threads) processes one work item at a time: 128 rows of one surrogate head, or 256
// rows of one mean head.
#pragma once

#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {
namespace cheap {

constexpr int kBStride = 72;  // padded smem rows (bf16): 144 bytes, conflict-free fragment loads
constexpr int kSurrRows = 128;
constexpr int kMeanRows = 256;

__device__ __forceinline__ void mma_bf16_16816(float* d, const uint32_t* a, uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// sigma(x) = 1 / (1 + e^{-x}) for a packed pair (MUFU ex2 and approximate reciprocal; an
// overflowing e^{-x} gives 0).
__device__ __forceinline__ float2 sigmoid2(float2 x) {
  const float kLog2e = 1.4426950408889634f;
  const float2 a = fmul2(x, make_float2(-kLog2e, -kLog2e));
  const float2 d = make_float2(1.f + fast_exp2(a.x), 1.f + fast_exp2(a.y));
  float2 r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r.x) : "f"(d.x));
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r.y) : "f"(d.y));
  return r;
}

struct SurrSmem {
  __nv_bfloat16 w1[128 * kBStride];  // rows 0..63: MLP_gamma layer 1 (value half), 64..127: MLP_delta
  __nv_bfloat16 w2[128 * kBStride];  // rows 0..63: MLP_gamma layer 2, 64..127: MLP_delta layer 2
  float c1[128];                     // W1[:, d:] C_h + b1 (gamma | delta)
  float b2[128];                     // b2 (gamma | delta)
  float ctx[64];
};

// Y[r0 .. min(N, r0 + rows))[h][:] = Broadcast(vec[0..63]): 8 threads per row, 16-byte stores.
__device__ __forceinline__ void broadcast_rows(const HeadAttnArgs& a, const float* vec, int h,
                                               int r0, int rows, int tid) {
  const int part = tid & 7, rg = tid >> 3;
  const float* mv = vec + 8 * part;
  uint4 val;
  val.x = pack_bf16x2(__ldg(mv + 0), __ldg(mv + 1));
  val.y = pack_bf16x2(__ldg(mv + 2), __ldg(mv + 3));
  val.z = pack_bf16x2(__ldg(mv + 4), __ldg(mv + 5));
  val.w = pack_bf16x2(__ldg(mv + 6), __ldg(mv + 7));
  const int r1 = min(a.N, r0 + rows);
  for (int row = r0 + rg; row < r1; row += 32)
    *reinterpret_cast<uint4*>(a.y + ((size_t)row * a.H + h) * 64 + 8 * part) = val;
}

// Mean head h, rows [chunk * 256, +256).
__device__ __forceinline__ void mean_item(const HeadAttnArgs& a, int h, int chunk, int tid) {
  broadcast_rows(a, a.mean_v + h * 64, h, chunk * kMeanRows, kMeanRows, tid);
}

// Stages head h's surrogate weights (both MLPs' value halves of layer 1, both layer 2s,
// biases and C_h).  The context half of layer 1 is folded into c1 by surrogate_fold after
// the group has synchronised.
__device__ __forceinline__ void surrogate_stage(const HeadAttnArgs& a, SurrSmem& sm, int h, int tid) {
  for (int i = tid; i < 128 * 8; i += 256) {
    const int row = i >> 3, ch = i & 7;
    const bool g = row < 64;
    const __nv_bfloat16* w1 = (g ? a.sw.g1_w : a.sw.d1_w) + ((size_t)h * 64 + (row & 63)) * 128 + ch * 8;
    const __nv_bfloat16* w2 = (g ? a.sw.g2_w : a.sw.d2_w) + ((size_t)h * 64 + (row & 63)) * 64 + ch * 8;
    *reinterpret_cast<uint4*>(&sm.w1[row * kBStride + ch * 8]) = __ldg(reinterpret_cast<const uint4*>(w1));
    *reinterpret_cast<uint4*>(&sm.w2[row * kBStride + ch * 8]) = __ldg(reinterpret_cast<const uint4*>(w2));
  }
  if (tid < 64) sm.ctx[tid] = __ldg(a.ctx + h * 64 + tid);
  if (tid < 128) {
    const bool g = tid < 64;
    sm.b2[tid] = __ldg((g ? a.sw.g2_b : a.sw.d2_b) + h * 64 + (tid & 63));
  }
}

// c1[t] = b1[t] + sum_k W1[t][64 + k] C[k]  (context half of the first layer).
__device__ __forceinline__ void surrogate_fold(const HeadAttnArgs& a, SurrSmem& sm, int h, int tid) {
  if (tid < 128) {
    const bool g = tid < 64;
    const int l = tid & 63;
    const __nv_bfloat16* wr = (g ? a.sw.g1_w : a.sw.d1_w) + ((size_t)h * 64 + l) * 128 + 64;
    float acc = __ldg((g ? a.sw.g1_b : a.sw.d1_b) + h * 64 + l);
    for (int k = 0; k < 64; k += 8) {
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(wr + k));
      const uint32_t uw[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
        acc += bf16_lo(uw[i]) * sm.ctx[k + 2 * i] + bf16_hi(uw[i]) * sm.ctx[k + 2 * i + 1];
    }
    sm.c1[tid] = acc;
  }
}

// Surrogate head h, 16 rows [chunk * 128 + 16 w, +16) for group warp w (0..7).
__device__ __forceinline__ void surrogate_rows(const HeadAttnArgs& a, const SurrSmem& sm, int h,
                                               int chunk, int w, int lane) {
  const int N = a.N, H = a.H;
  const size_t row_pitch = (size_t)3 * H * kHeadDim;
  const int r = lane >> 2, c = lane & 3;
  const int base = chunk * kSurrRows + w * 16;
  if (base >= N) return;
  const int ra = base + r, rb = base + r + 8;
  const bool va = ra < N, vb = rb < N;
  // V rows, channels 16c..16c+15 (the first layer's reduction index is permuted: logical
  // pair (kk, 2c) <-> channels 16c+4kk+{0,1}, (kk, 2c+8) <-> +{2,3}, in A and B alike).
  uint32_t qa[8], qb[8];
  {
    const __nv_bfloat16* vbase = a.qkv + (size_t)(2 * H + h) * kHeadDim + 16 * c;
    const uint4* pa = reinterpret_cast<const uint4*>(vbase + (size_t)(va ? ra : base) * row_pitch);
    const uint4* pb = reinterpret_cast<const uint4*>(vbase + (size_t)(vb ? rb : base) * row_pitch);
    const uint4 x0 = __ldg(pa), x1 = __ldg(pa + 1), y0 = __ldg(pb), y1 = __ldg(pb + 1);
    qa[0] = x0.x; qa[1] = x0.y; qa[2] = x0.z; qa[3] = x0.w;
    qa[4] = x1.x; qa[5] = x1.y; qa[6] = x1.z; qa[7] = x1.w;
    qb[0] = y0.x; qb[1] = y0.y; qb[2] = y0.z; qb[3] = y0.w;
    qb[4] = y1.x; qb[5] = y1.y; qb[6] = y1.z; qb[7] = y1.w;
  }
  // Layer 1 for both MLPs: 128 hidden units (gamma 0..63, delta 64..127).
  uint32_t hid[16][2];  // bf16x2: [n-tile][row ra / row rb]
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    const uint4* pw = reinterpret_cast<const uint4*>(&sm.w1[(8 * j + r) * kBStride + 16 * c]);
    const uint4 w0 = pw[0], w1 = pw[1];
    const uint32_t bw[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const uint32_t af[4] = {qa[2 * kk], qb[2 * kk], qa[2 * kk + 1], qb[2 * kk + 1]};
      mma_bf16_16816(acc, af, bw[2 * kk], bw[2 * kk + 1]);
    }
    const int col = 8 * j + 2 * c;
    const float c0 = sm.c1[col], c1v = sm.c1[col + 1];
    const float2 ga = gelu_as2(fadd2(make_float2(acc[0], acc[1]), make_float2(c0, c1v)));
    const float2 gb = gelu_as2(fadd2(make_float2(acc[2], acc[3]), make_float2(c0, c1v)));
    hid[j][0] = pack_bf16x2(ga.x, ga.y);
    hid[j][1] = pack_bf16x2(gb.x, gb.y);
  }
  // Layer 2: the accumulator layout of two adjacent n-tiles is the A-fragment layout of one
  // 16-wide k-step.  Output n-tile j of both MLPs is finished and stored before the next.
  __nv_bfloat16* ya = a.y + ((size_t)ra * H + h) * 64;
  __nv_bfloat16* yb = a.y + ((size_t)rb * H + h) * 64;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    float og[4] = {0.f, 0.f, 0.f, 0.f}, od[4] = {0.f, 0.f, 0.f, 0.f};
    const __nv_bfloat16* rowg = &sm.w2[(8 * j + r) * kBStride];
    const __nv_bfloat16* rowd = &sm.w2[(64 + 8 * j + r) * kBStride];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const uint32_t ag[4] = {hid[2 * kk][0], hid[2 * kk][1], hid[2 * kk + 1][0], hid[2 * kk + 1][1]};
      const uint32_t ad[4] = {hid[8 + 2 * kk][0], hid[8 + 2 * kk][1], hid[9 + 2 * kk][0], hid[9 + 2 * kk][1]};
      const uint32_t g0 = *reinterpret_cast<const uint32_t*>(rowg + 16 * kk + 2 * c);
      const uint32_t g1 = *reinterpret_cast<const uint32_t*>(rowg + 16 * kk + 8 + 2 * c);
      const uint32_t d0 = *reinterpret_cast<const uint32_t*>(rowd + 16 * kk + 2 * c);
      const uint32_t d1 = *reinterpret_cast<const uint32_t*>(rowd + 16 * kk + 8 + 2 * c);
      mma_bf16_16816(og, ag, g0, g1);
      mma_bf16_16816(od, ad, d0, d1);
    }
    // y = C + sigma(gamma) (.) delta, stored as bf16 in Y[row][h][:].
    const int col = 8 * j + 2 * c;
    const float2 C = *reinterpret_cast<const float2*>(&sm.ctx[col]);
    const float2 bg = *reinterpret_cast<const float2*>(&sm.b2[col]);
    const float2 bd = *reinterpret_cast<const float2*>(&sm.b2[64 + col]);
    const float2 ya2 = ffma2(sigmoid2(fadd2(make_float2(og[0], og[1]), bg)),
                             fadd2(make_float2(od[0], od[1]), bd), C);
    const float2 yb2 = ffma2(sigmoid2(fadd2(make_float2(og[2], og[3]), bg)),
                             fadd2(make_float2(od[2], od[3]), bd), C);
    if (va) *reinterpret_cast<uint32_t*>(ya + col) = pack_bf16x2(ya2.x, ya2.y);
    if (vb) *reinterpret_cast<uint32_t*>(yb + col) = pack_bf16x2(yb2.x, yb2.y);
  }
}

}  // namespace cheap
}  // namespace vp
