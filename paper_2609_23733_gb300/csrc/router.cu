// Router of VGGT-Prime (§4.1) and routing (§4.2) on sm_103a.
//
// Two sweeps over the token axis, both split across CTAs with online-softmax partials:
//   router_pool_kernel  (§4.1, pooling): e_i = w_h^T (tanh(W_h q_i + bW) (.) sigma(U_h q_i + bU))
//       The [16 tokens x 64] x [64 x 128] projection onto [W_h; U_h] runs on the tensor
//       cores (mma.sync m16n8k16, fp32 accumulation); each warp keeps a running
//       (max, sum, sum p q) of alpha's softmax, the last CTA of a head combines the
//       partials into q_pool = sum_i alpha_i q_i.
//   router_keys_kernel  (§4.1 routing attention + §4.3 context + mean of V):
//       l_j = beta_h / sqrt(d) * q_pool . k_j; running (max, sum 2^(l-max), sum p v, sum v)
//       per CTA; the last CTA of a head derives s_h = max_j r_h(j) = 1 / sum_j e^(l_j - max),
//       C_h = r_h V_h and mean_v, applies the routing equation (§4.2), and the last head
//       to finish groups the heads by mode (bins) for the mode kernels.
// HBM traffic: Q once (pool sweep), K and V once (key sweep); no N-sized intermediate.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kPoolThreads = 128;
constexpr int kKeyThreads = 256;
constexpr int kBStride = 72;  // padded smem row (bf16 elements): 144 bytes, conflict-free

__device__ __forceinline__ void mma_bf16_16816(float* d, const uint32_t* a, uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// tanh(x) * sigma(y) for the pooling logits of §4.1, two at a time on packed f32x2 pairs, in a
// form that needs no clamps:
// tanh(x) = sign(x) (1 - e^{-2|x|}) / (1 + e^{-2|x|}) with e^{-2|x|} <= 1, and
// sigma(y) = 1 / (1 + e^{-y}), whose e^{-y} may overflow to +inf, giving 0 as it should.
__device__ __forceinline__ float2 tanh_times_sigmoid2(float2 x, float2 y) {
  const float kLog2e = 1.4426950408889634f;
  const float2 a = fmul2(make_float2(fabsf(x.x), fabsf(x.y)), make_float2(-2.f * kLog2e, -2.f * kLog2e));
  const float2 b = fmul2(y, make_float2(-kLog2e, -kLog2e));
  const float2 ea = make_float2(fast_exp2(a.x), fast_exp2(a.y));
  const float2 eb = make_float2(fast_exp2(b.x), fast_exp2(b.y));
  const float2 num = ffma2(ea, make_float2(-1.f, -1.f), make_float2(1.f, 1.f));
  const float2 den = fmul2(fadd2(ea, make_float2(1.f, 1.f)), fadd2(eb, make_float2(1.f, 1.f)));
  float2 r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r.x) : "f"(den.x));
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r.y) : "f"(den.y));
  const float2 t = fmul2(num, r);
  return make_float2(copysignf(t.x, x.x), copysignf(t.y, x.y));
}

__device__ __forceinline__ void token_range(int N, int n_split, int split, int align, int& t0,
                                            int& t1) {
  int per = (N + n_split - 1) / n_split;
  per = (per + align - 1) / align * align;
  t0 = split * per;
  t1 = min(N, t0 + per);
}

// ------------------------------------------------------------------ pooling sweep
__global__ void __launch_bounds__(kPoolThreads) router_pool_kernel(RouterArgs a, RouterScratch sc,
                                                                    int n_split) {
  const int h = blockIdx.y, split = blockIdx.x;
  const int N = a.N, H = a.H;
  const size_t row_pitch = (size_t)3 * H * kHeadDim;  // elements between consecutive tokens
  const bool mean_pool = (a.variant & VP_VARIANT_MEAN_QPOOL) != 0;  // §5 component ablation

  __shared__ __align__(16) __nv_bfloat16 sB[128 * kBStride];  // rows 0..63 W_h, 64..127 U_h
  __shared__ __align__(16) float s_bias[128];                // bW | bU
  __shared__ __align__(16) float s_w[64];
  __shared__ float s_part[4][kPoolPartial];

  const int tid = threadIdx.x;
  // Stage [W_h; U_h] (128 rows x 128 bytes) in padded rows.
  for (int i = tid; i < 128 * 8; i += kPoolThreads) {
    const int row = i >> 3, ch = i & 7;
    const __nv_bfloat16* src = (row < 64 ? a.W : a.U) + ((size_t)h * 64 + (row & 63)) * 64 + ch * 8;
    *reinterpret_cast<uint4*>(&sB[row * kBStride + ch * 8]) = *reinterpret_cast<const uint4*>(src);
  }
  if (tid < 64) {
    s_bias[tid] = a.bW ? a.bW[h * 64 + tid] : 0.f;
    s_bias[64 + tid] = a.bU ? a.bU[h * 64 + tid] : 0.f;
    s_w[tid] = __bfloat162float(a.w[h * 64 + tid]);
  }
  __syncthreads();

  int t0, t1;
  token_range(N, n_split, split, 16, t0, t1);
  const int warp = tid >> 5, lane = tid & 31;
  const int r = lane >> 2, c = lane & 3;
  const __nv_bfloat16* qbase = a.qkv + (size_t)h * kHeadDim + 16 * c;

  float M = -INFINITY, lsum = 0.f;
  float accq[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) accq[i] = 0.f;

  // Each thread holds channels 16c..16c+15 of rows ra and rb.  The MMA's reduction index k
  // is permuted consistently in A and B (logical k pair (kk, 2c) <-> channels 16c + 4kk +
  // {0,1}, pair (kk, 2c + 8) <-> 16c + 4kk + {2,3}), so that every thread reads 32 contiguous
  // bytes of its rows and of the weight rows.  The next tile's rows are loaded while the
  // current tile is computed.
  auto load_rows = [&](int base, uint4& x0, uint4& x1, uint4& y0, uint4& y1) {
    const int ra = base + r, rb = base + r + 8;
    const uint4* pa = reinterpret_cast<const uint4*>(qbase + (size_t)(ra < t1 ? ra : t0) * row_pitch);
    const uint4* pb = reinterpret_cast<const uint4*>(qbase + (size_t)(rb < t1 ? rb : t0) * row_pitch);
    x0 = __ldg(pa);
    x1 = __ldg(pa + 1);
    y0 = __ldg(pb);
    y1 = __ldg(pb + 1);
  };
  uint4 nx0, nx1, ny0, ny1;
  if (t0 + 16 * warp < t1) load_rows(t0 + 16 * warp, nx0, nx1, ny0, ny1);
  for (int base = t0 + 16 * warp; base < t1; base += 64) {
    const int ra = base + r, rb = base + r + 8;
    const bool va = ra < t1, vb = rb < t1;
    uint32_t qa[8], qb[8];
    {
      const uint4 x0 = nx0, x1 = nx1, y0 = ny0, y1 = ny1;
      if (base + 64 < t1) load_rows(base + 64, nx0, nx1, ny0, ny1);
      qa[0] = x0.x; qa[1] = x0.y; qa[2] = x0.z; qa[3] = x0.w;
      qa[4] = x1.x; qa[5] = x1.y; qa[6] = x1.z; qa[7] = x1.w;
      qb[0] = y0.x; qb[1] = y0.y; qb[2] = y0.z; qb[3] = y0.w;
      qb[4] = y1.x; qb[5] = y1.y; qb[6] = y1.z; qb[7] = y1.w;
    }
    // Pooling logits (both 0 under the mean-pooling ablation: alpha = 1/N exactly).
    float ea = 0.f, eb = 0.f;
    if (!mean_pool) {
    float acc[16][4];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
      const uint4* pw = reinterpret_cast<const uint4*>(&sB[(8 * j + r) * kBStride + 16 * c]);
      const uint4 w0 = pw[0], w1 = pw[1];
      const uint32_t bw[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint32_t af[4] = {qa[2 * kk], qb[2 * kk], qa[2 * kk + 1], qb[2 * kk + 1]};
        mma_bf16_16816(acc[j], af, bw[2 * kk], bw[2 * kk + 1]);
      }
    }
    // Pooling logits: columns 8j + 2c + e of the W half (j < 8) pair with the same
    // columns of the U half (j + 8) in the same thread; the two columns e = 0, 1 of a row
    // form one packed pair.
    float2 pa = make_float2(0.f, 0.f), pb = make_float2(0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int l = 8 * j + 2 * c;
      const float2 bw = *reinterpret_cast<const float2*>(&s_bias[l]);
      const float2 bu = *reinterpret_cast<const float2*>(&s_bias[64 + l]);
      const float2 wl = *reinterpret_cast<const float2*>(&s_w[l]);
      pa = ffma2(wl, tanh_times_sigmoid2(fadd2(make_float2(acc[j][0], acc[j][1]), bw),
                                         fadd2(make_float2(acc[j + 8][0], acc[j + 8][1]), bu)), pa);
      pb = ffma2(wl, tanh_times_sigmoid2(fadd2(make_float2(acc[j][2], acc[j][3]), bw),
                                         fadd2(make_float2(acc[j + 8][2], acc[j + 8][3]), bu)), pb);
    }
    ea = pa.x + pa.y;
    eb = pb.x + pb.y;
    ea += __shfl_xor_sync(0xffffffffu, ea, 1);
    ea += __shfl_xor_sync(0xffffffffu, ea, 2);
    eb += __shfl_xor_sync(0xffffffffu, eb, 1);
    eb += __shfl_xor_sync(0xffffffffu, eb, 2);
    }
    if (!va) ea = -INFINITY;
    if (!vb) eb = -INFINITY;
    float mc = fmaxf(ea, eb);
    mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, 4));
    mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, 8));
    mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, 16));
    if (mc == -INFINITY) continue;  // warp-uniform
    const float Mn = fmaxf(M, mc);
    const float scale = __expf(M - Mn);  // 0 when M = -inf
    const float pa = __expf(ea - Mn), pb = __expf(eb - Mn);
    lsum = lsum * scale + (pa + pb);
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      accq[2 * m] = accq[2 * m] * scale + pa * bf16_lo(qa[m]) + pb * bf16_lo(qb[m]);
      accq[2 * m + 1] = accq[2 * m + 1] * scale + pa * bf16_hi(qa[m]) + pb * bf16_hi(qb[m]);
    }
    M = Mn;
  }
  // Reduce over the 8 row groups (lane bits 2..4); M is warp-uniform.
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
#pragma unroll
    for (int i = 0; i < 16; ++i) accq[i] += __shfl_xor_sync(0xffffffffu, accq[i], o);
  }
  if (lane < 4) {
#pragma unroll
    for (int i = 0; i < 16; ++i) s_part[warp][2 + 16 * c + i] = accq[i];
    if (lane == 0) {
      s_part[warp][0] = M;
      s_part[warp][1] = lsum;
    }
  }
  __syncthreads();
  float* part = sc.pool_part + ((size_t)h * kPoolSplitMax + split) * kPoolPartial;
  if (tid < 64) {
    float Mx = -INFINITY;
    for (int w = 0; w < 4; ++w) Mx = fmaxf(Mx, s_part[w][0]);
    float acc = 0.f, l = 0.f;
    if (Mx != -INFINITY) {
      for (int w = 0; w < 4; ++w) {
        const float f = __expf(s_part[w][0] - Mx);
        acc += f * s_part[w][2 + tid];
        l += f * s_part[w][1];
      }
    }
    part[2 + tid] = acc;
    if (tid == 0) {
      part[0] = Mx;
      part[1] = l;
    }
  }
  // Last CTA of this head combines the partials into q_pool.
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(&sc.counters[h], 1u) == (unsigned)(n_split - 1));
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid < 64) {
    const float* pp = sc.pool_part + (size_t)h * kPoolSplitMax * kPoolPartial;
    float Mx = -INFINITY;
    for (int s = 0; s < n_split; ++s) Mx = fmaxf(Mx, __ldcg(pp + s * kPoolPartial));
    float acc = 0.f, l = 0.f;
    for (int s = 0; s < n_split; ++s) {
      const float ms = __ldcg(pp + s * kPoolPartial);
      if (ms == -INFINITY) continue;
      const float f = __expf(ms - Mx);
      l += f * __ldcg(pp + s * kPoolPartial + 1);
      acc += f * __ldcg(pp + s * kPoolPartial + 2 + tid);
    }
    const float q = acc / l;
    sc.q_pool[h * 64 + tid] = q;
    if (a.q_pool_out) a.q_pool_out[h * 64 + tid] = q;
  }
}

// ------------------------------------------------------------------ key sweep
__device__ __forceinline__ int select_mode(float s, float tau_low, float tau_high, bool& nan) {
  nan = isnan(s);
  if (nan || s >= tau_high) return VP_MODE_FULL;
  if (s <= tau_low) return VP_MODE_MEAN;
  return VP_MODE_SURROGATE;
}

__device__ void bin_heads_warp(int H, const int32_t* modes, int32_t* head_ids, int32_t* offsets) {
  const int lane = threadIdx.x & 31;
  const int m = lane < H ? __ldcg(modes + lane) : -1;
  int base = 0;
#pragma unroll
  for (int mode = 0; mode < 3; ++mode) {
    const unsigned mask = __ballot_sync(0xffffffffu, m == mode);
    if (m == mode) head_ids[base + __popc(mask & ((1u << lane) - 1u))] = lane;
    if (lane == 0) offsets[mode] = base;
    base += __popc(mask);
  }
  if (lane == 0) offsets[3] = base;
}

__global__ void __launch_bounds__(kKeyThreads) router_keys_kernel(RouterArgs a, RouterScratch sc,
                                                                   int n_split) {
  const int h = blockIdx.y, split = blockIdx.x;
  const int N = a.N, H = a.H;
  const size_t row_pitch = (size_t)3 * H * kHeadDim;
  const int tid = threadIdx.x;
  const int g = tid >> 3, part = tid & 7;  // 32 row groups x 8 channel groups of 8

  const float kLog2e = 1.4426950408889634f;
  const float beta = a.beta ? a.beta[h] : 1.f;
  const float cscale = beta * 0.125f * kLog2e;  // beta / sqrt(64), in log2 units
  float q[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) q[i] = __ldcg(sc.q_pool + h * 64 + 8 * part + i) * cscale;

  int t0, t1;
  token_range(N, n_split, split, 128, t0, t1);
  const __nv_bfloat16* kb = a.qkv + (size_t)(H + h) * kHeadDim + 8 * part;
  const __nv_bfloat16* vb = a.qkv + (size_t)(2 * H + h) * kHeadDim + 8 * part;

  float m = -INFINITY, l = 0.f, accv[8], sumv[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) accv[i] = sumv[i] = 0.f;

  // The loop bound is uniform across the CTA so that the 8-lane shuffles below always
  // run with the whole warp; rows past t1 are loaded from row t0 and masked.  Four rows per
  // row group are in flight (eight 16-byte loads per thread) before any arithmetic.
  // The next batch of rows is loaded while the current one is computed.
  uint4 nk[4], nv[4];
  auto load_batch = [&](int base) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int row = base + g + 32 * u;
      const size_t o = (size_t)(row < t1 ? row : t0) * row_pitch;
      nk[u] = __ldg(reinterpret_cast<const uint4*>(kb + o));
      nv[u] = __ldg(reinterpret_cast<const uint4*>(vb + o));
    }
  };
  if (t0 < t1) load_batch(t0);
  for (int base = t0; base < t1; base += 128) {
    uint4 kr[4], vr[4];
    bool valid[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      kr[u] = nk[u];
      vr[u] = nv[u];
      valid[u] = base + g + 32 * u < t1;
    }
    if (base + 128 < t1) load_batch(base + 128);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const uint32_t kw[4] = {kr[u].x, kr[u].y, kr[u].z, kr[u].w};
      const uint32_t vw[4] = {vr[u].x, vr[u].y, vr[u].z, vr[u].w};
      float dot = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) dot += q[2 * i] * bf16_lo(kw[i]) + q[2 * i + 1] * bf16_hi(kw[i]);
      dot += __shfl_xor_sync(0xffffffffu, dot, 1);
      dot += __shfl_xor_sync(0xffffffffu, dot, 2);
      dot += __shfl_xor_sync(0xffffffffu, dot, 4);
      if (!valid[u]) continue;  // no shuffles below
      if (dot > m) {
        const float f = fast_exp2(m - dot);  // 0 when m = -inf
        l *= f;
#pragma unroll
        for (int i = 0; i < 8; ++i) accv[i] *= f;
        m = dot;
      }
      const float p = fast_exp2(dot - m);
      l += p;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float v0 = bf16_lo(vw[i]), v1f = bf16_hi(vw[i]);
        accv[2 * i] += p * v0;
        accv[2 * i + 1] += p * v1f;
        sumv[2 * i] += v0;
        sumv[2 * i + 1] += v1f;
      }
    }
  }
  // Combine the 32 row groups of the CTA.
  __shared__ float s_m[32], s_l[32];
  __shared__ float s_acc[32][64], s_sum[32][64];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    s_acc[g][8 * part + i] = accv[i];
    s_sum[g][8 * part + i] = sumv[i];
  }
  if (part == 0) {
    s_m[g] = m;
    s_l[g] = l;
  }
  __syncthreads();
  float* kp = sc.key_part + ((size_t)h * kKeySplitMax + split) * kKeyPartial;
  if (tid < 64) {
    float Mx = -INFINITY;
    for (int i = 0; i < 32; ++i) Mx = fmaxf(Mx, s_m[i]);
    float acc = 0.f, sum = 0.f, ll = 0.f;
    for (int i = 0; i < 32; ++i) {
      sum += s_sum[i][tid];
      if (s_m[i] == -INFINITY) continue;
      const float f = fast_exp2(s_m[i] - Mx);
      acc += f * s_acc[i][tid];
      ll += f * s_l[i];
    }
    kp[2 + tid] = acc;
    kp[2 + 64 + tid] = sum;
    if (tid == 0) {
      kp[0] = Mx;
      kp[1] = ll;
    }
  }
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(&sc.counters[kMaxHeads + h], 1u) == (unsigned)(n_split - 1));
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // Last CTA of head h: saliency, context, mean of V, mode.
  if (tid < 64) {
    const float* pp = sc.key_part + (size_t)h * kKeySplitMax * kKeyPartial;
    float Mx = -INFINITY;
    for (int s = 0; s < n_split; ++s) Mx = fmaxf(Mx, __ldcg(pp + s * kKeyPartial));
    float acc = 0.f, sum = 0.f, ll = 0.f;
    for (int s = 0; s < n_split; ++s) {
      const float* q2 = pp + s * kKeyPartial;
      sum += __ldcg(q2 + 2 + 64 + tid);
      const float ms = __ldcg(q2);
      if (ms == -INFINITY) continue;
      const float f = fast_exp2(ms - Mx);
      ll += f * __ldcg(q2 + 1);
      acc += f * __ldcg(q2 + 2 + tid);
    }
    const float ctx = acc / ll;
    const float mv = sum / (float)N;
    sc.ctx[h * 64 + tid] = ctx;
    sc.mean_v[h * 64 + tid] = mv;
    if (a.ctx_out) a.ctx_out[h * 64 + tid] = ctx;
    if (a.mean_v_out) a.mean_v_out[h * 64 + tid] = mv;
    if (tid == 0) {
      // s_h = max_j r_h(j) = 2^(max - max) / sum_j 2^(l_j - max).
      const float s = 1.f / ll;
      bool nan;
      int mode = select_mode(s, a.tau_low, a.tau_high, nan);
      if (nan) atomicOr(sc.err, VP_DEVERR_NAN_SALIENCY);
      if (a.force_modes) mode = a.force_modes[h];
      sc.s[h] = s;
      sc.modes[h] = mode;
      sc.key_stats[2 * h] = Mx;
      sc.key_stats[2 * h + 1] = ll;
      if (a.s_out) a.s_out[h] = s;
      if (a.modes_out) a.modes_out[h] = mode;
    }
  }
  // The last head to finish groups all heads by mode.
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(&sc.counters[2 * kMaxHeads], 1u) == (unsigned)(H - 1));
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid < 32) bin_heads_warp(H, sc.modes, sc.head_ids, sc.offsets);
}

// r_h(j) = 2^(l_j - max) / sum, one more pass over K (only when the caller asks for r).
__global__ void __launch_bounds__(256) router_r_kernel(RouterArgs a, RouterScratch sc) {
  const int h = blockIdx.y;
  const int N = a.N, H = a.H;
  const size_t row_pitch = (size_t)3 * H * kHeadDim;
  const int tid = threadIdx.x, g = tid >> 3, part = tid & 7;
  const float kLog2e = 1.4426950408889634f;
  const float beta = a.beta ? a.beta[h] : 1.f;
  const float cscale = beta * 0.125f * kLog2e;
  float q[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) q[i] = __ldcg(sc.q_pool + h * 64 + 8 * part + i) * cscale;
  const float Mx = __ldcg(sc.key_stats + 2 * h), inv = 1.f / __ldcg(sc.key_stats + 2 * h + 1);
  const __nv_bfloat16* kb = a.qkv + (size_t)(H + h) * kHeadDim + 8 * part;
  for (int base = blockIdx.x * 32; base < N; base += gridDim.x * 32) {  // uniform bound
    const int row = base + g;
    const bool valid = row < N;
    const uint4 kk = __ldg(reinterpret_cast<const uint4*>(kb + (size_t)(valid ? row : 0) * row_pitch));
    const uint32_t kw[4] = {kk.x, kk.y, kk.z, kk.w};
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) dot += q[2 * i] * bf16_lo(kw[i]) + q[2 * i + 1] * bf16_hi(kw[i]);
    dot += __shfl_xor_sync(0xffffffffu, dot, 1);
    dot += __shfl_xor_sync(0xffffffffu, dot, 2);
    dot += __shfl_xor_sync(0xffffffffu, dot, 4);
    if (valid && part == 0) a.r_out[(size_t)h * N + row] = fast_exp2(dot - Mx) * inv;
  }
}

__global__ void bin_heads_kernel(int H, int N, const int32_t* modes, int32_t* head_ids,
                                 int32_t* offsets, int32_t* work, int32_t* n_work) {
  __shared__ int32_t s_ids[32], s_off[4];
  if (threadIdx.x < 32) bin_heads_warp(H, modes, s_ids, s_off);
  __syncthreads();
  if (threadIdx.x < H) head_ids[threadIdx.x] = s_ids[threadIdx.x];
  if (threadIdx.x < 4) offsets[threadIdx.x] = s_off[threadIdx.x];
  const int n_tiles = (N + kQTile - 1) / kQTile;
  const int n_full = s_off[3] - s_off[2];
  if (n_work && threadIdx.x == 0) *n_work = n_full * n_tiles;
  if (work) {
    for (int i = threadIdx.x; i < n_full * n_tiles; i += blockDim.x) {
      work[2 * i] = s_ids[s_off[2] + i / n_tiles];
      work[2 * i + 1] = i % n_tiles;
    }
  }
}

// Self-test of the bounded waits (failure handling, not the method): one warp waits on an
// mbarrier that nothing ever arrives on, so the wait must give up after limit_ns, record
// VP_DEVERR_WAIT_TIMEOUT and return.
__global__ void wait_selftest_kernel(unsigned int* err, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbarrier_init();
  }
  __syncthreads();
  mbar_wait_warp(&bar, 0, err, &abort_flag, limit_ns);
}

}  // namespace

cudaError_t launch_wait_selftest(unsigned int* err, unsigned long long limit_ns,
                                 cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(err, limit_ns);
  return cudaGetLastError();
}

size_t router_scratch_bytes(int H) {
  (void)H;
  size_t b = 256;                                                    // error word
  b += 512;                                                          // counters
  b += (size_t)kMaxHeads * kPoolSplitMax * kPoolPartial * 4;
  b += (size_t)kMaxHeads * kKeySplitMax * kKeyPartial * 4;
  b += (size_t)kMaxHeads * 64 * 4 * 3;                               // q_pool, ctx, mean_v
  b += (size_t)kMaxHeads * 4 * 4;                                    // key_stats, s, modes
  b += 256;                                                          // head_ids, offsets
  return (b + 4095) & ~(size_t)4095;
}

size_t heads_scratch_bytes(int H) {
  return router_scratch_bytes(H) + (size_t)kMaxHeads * kLinState * 4 +
         (kFaPartFloats + kFaStatsFloats + kFaCountWords) * 4;
}

RouterScratch carve_router_scratch(void* ws, int H) {
  (void)H;
  char* p = static_cast<char*>(ws);
  RouterScratch sc;
  sc.err = reinterpret_cast<unsigned int*>(p);
  p += 256;
  sc.counters = reinterpret_cast<unsigned int*>(p);
  p += 512;
  sc.pool_part = reinterpret_cast<float*>(p);
  p += (size_t)kMaxHeads * kPoolSplitMax * kPoolPartial * 4;
  sc.key_part = reinterpret_cast<float*>(p);
  p += (size_t)kMaxHeads * kKeySplitMax * kKeyPartial * 4;
  sc.q_pool = reinterpret_cast<float*>(p);
  p += kMaxHeads * 64 * 4;
  sc.ctx = reinterpret_cast<float*>(p);
  p += kMaxHeads * 64 * 4;
  sc.mean_v = reinterpret_cast<float*>(p);
  p += kMaxHeads * 64 * 4;
  sc.key_stats = reinterpret_cast<float*>(p);
  p += kMaxHeads * 2 * 4;
  sc.s = reinterpret_cast<float*>(p);
  p += kMaxHeads * 4;
  sc.modes = reinterpret_cast<int32_t*>(p);
  p += kMaxHeads * 4;
  sc.head_ids = reinterpret_cast<int32_t*>(p);
  sc.offsets = sc.head_ids + kMaxHeads;
  sc.cheap_counter = sc.counters + 96;  // counters[0 .. 2 * kMaxHeads] serve the router
  sc.lin_state = reinterpret_cast<float*>(static_cast<char*>(ws) + router_scratch_bytes(H));
  sc.fa_part = sc.lin_state + (size_t)kMaxHeads * kLinState;
  sc.fa_stats = sc.fa_part + kFaPartFloats;
  sc.fa_count = reinterpret_cast<unsigned int*>(sc.fa_stats + kFaStatsFloats);
  return sc;
}

cudaError_t launch_router(const RouterArgs& a, const RouterScratch& sc, int num_sms,
                          cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(sc.counters, 0, 512, st);
  if (e != cudaSuccess) return e;
  // Enough CTAs to cover every SM a few times; at least 64 tokens per CTA.
  int pool_split = (4 * num_sms + a.H - 1) / a.H;
  pool_split = max(1, min(min(pool_split, kPoolSplitMax), (a.N + 63) / 64));
  prof_before(VP_KERNEL_ROUTER_POOL, st);
  router_pool_kernel<<<dim3(pool_split, a.H), kPoolThreads, 0, st>>>(a, sc, pool_split);
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int key_split = (4 * num_sms + a.H - 1) / a.H;
  key_split = max(1, min(min(key_split, kKeySplitMax), (a.N + 255) / 256));
  prof_before(VP_KERNEL_ROUTER_KEYS, st);
  router_keys_kernel<<<dim3(key_split, a.H), kKeyThreads, 0, st>>>(a, sc, key_split);
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (a.r_out) {
    int blocks = max(1, min((a.N + 31) / 32, (2 * num_sms + a.H - 1) / a.H));
    prof_before(VP_KERNEL_ROUTER_R, st);
    router_r_kernel<<<dim3(blocks, a.H), 256, 0, st>>>(a, sc);
    prof_after(st);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t launch_bin_heads(int H, int N, const int32_t* modes, int32_t* head_ids,
                             int32_t* offsets, int32_t* work, int32_t* n_work, cudaStream_t st) {
  prof_before(VP_KERNEL_BIN_HEADS, st);
  bin_heads_kernel<<<1, 256, 0, st>>>(H, N, modes, head_ids, offsets, work, n_work);
  prof_after(st);
  return cudaGetLastError();
}

}  // namespace vp
