// Router of VGGT-Prime (§4.1) and routing (§4.2) on sm_103a.
//
// Two sweeps over the token axis, both split across CTAs with online-softmax partials:
//   router_pool_tc_kernel  (§4.1, pooling): e_i = w_h^T (tanh(W_h q_i + bW) (.) sigma(U_h q_i + bU))
//       The [128 tokens x 64] x [64 x 128] projection onto [W_h; U_h] runs on the
//       tcgen05 tensor cores (TMA-fed shared-memory operands, fp32 accumulators in TMEM);
//       each token thread keeps a running (max, sum, sum p q) of alpha's softmax, the CTA
//       merges them, and the last CTA of a head combines the partials into
//       q_pool = sum_i alpha_i q_i.
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

constexpr int kKeyThreads = 256;

// max(a, b) that returns NaN when either is NaN (fmaxf would return the other operand).
__device__ __forceinline__ float max_nan(float a, float b) {
  float d;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}

// tanh(x) * sigma(y) for the pooling logits of §4.1, two at a time on packed f32x2 pairs:
// tanh(x) sigma(y) = (1 - E) / ((1 + E)(1 + F)) with E = e^{-2x}, F = e^{-y}.  x is floored at
// -40 so that E stays finite (tanh(-40) is -1 in float); a huge F (y << 0) makes the
// denominator infinite and the product 0, as sigma(y) -> 0 requires.  NaNs propagate.
__device__ __forceinline__ float2 tanh_times_sigmoid2(float2 x, float2 y) {
  const float kLog2e = 1.4426950408889634f;
  const float2 xc = make_float2(max_nan(x.x, -40.f), max_nan(x.y, -40.f));
  const float2 a = fmul2(xc, make_float2(-2.f * kLog2e, -2.f * kLog2e));
  const float2 b = fmul2(y, make_float2(-kLog2e, -kLog2e));
  const float2 ea = make_float2(fast_exp2(a.x), fast_exp2(a.y));
  const float2 eb = make_float2(fast_exp2(b.x), fast_exp2(b.y));
  const float2 num = ffma2(ea, make_float2(-1.f, -1.f), make_float2(1.f, 1.f));
  const float2 den = fmul2(fadd2(ea, make_float2(1.f, 1.f)), fadd2(eb, make_float2(1.f, 1.f)));
  float2 r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r.x) : "f"(den.x));
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r.y) : "f"(den.y));
  return fmul2(num, r);
}

__device__ __forceinline__ void token_range(int N, int n_split, int split, int align, int& t0,
                                            int& t1) {
  int per = (N + n_split - 1) / n_split;
  per = (per + align - 1) / align * align;
  t0 = split * per;
  t1 = min(N, t0 + per);
}

// The last CTA of head h to publish its partial (max, sum, sum p q) combines the n_split
// partials into q_pool.  Called by every thread of the CTA.
__device__ __forceinline__ void pool_finish(const RouterArgs& a, const RouterScratch& sc, int h,
                                            int n_split) {
  __shared__ int s_last;
  const int tid = threadIdx.x;
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

// ------------------------------------------------------------------ pooling sweep (tcgen05)
// The same sweep with the [W_h; U_h] projection on the 5th-generation tensor cores: a CTA
// takes a run of 128-token tiles of one head.
//   warp 4   TMA: [W_h; U_h] once (two 64 x 64 boxes into one 128-row, 128-byte-swizzled
//            operand), then the tiles' Q rows (128 x 64, 16 KB) through a kPoolTcStages ring;
//   warp 5   TMEM owner and MMA issue: four tcgen05.mma M128 N128 K16 per tile into one of
//            two 128-column fp32 accumulators (columns 0-63: W_h q, 64-127: U_h q);
//   warps 0-3  one token per thread (TMEM lane): the logit e = w_h . (tanh(W_h q + bW) (.)
//            sigma(U_h q + bU)) from two halves of 32 + 32 accumulator columns, then a running
//            softmax of its own tokens (max M, sum, sum p q over the 64 channels of its Q row,
//            read from the shared-memory tile; rescaled only when M grows), released tile by
//            tile; at the end the 128 threads' partials merge into the CTA's (max, sum,
//            sum p q), which pool_finish combines over the CTAs of the head.
constexpr int kPoolTcStages = 4;
constexpr int kPoolTcThreads = 192;
constexpr int kPoolAccBufs = 2;    // 128-column fp32 accumulators per CTA
constexpr int kPoolCtasPerSm = 2;  // TMEM: kPoolCtasPerSm x kPoolAccBufs x 128 <= 512 columns
constexpr uint32_t kPoolTcTmemCols = 128 * kPoolAccBufs;
static_assert(kPoolCtasPerSm * kPoolTcTmemCols <= 512, "TMEM columns");

struct PoolTcSmem {
  __nv_bfloat16 q[kPoolTcStages][128 * 64];
  __nv_bfloat16 wu[128 * 64];
  float bias[128];  // bW | bU
  float wv[64];     // w_h
  float red_m[4], red_l[4];
  float red_acc[4][64];
  uint64_t q_full[kPoolTcStages], q_empty[kPoolTcStages];
  uint64_t wu_full, acc_full[kPoolAccBufs], acc_empty[kPoolAccBufs], drain;
  uint32_t tmem_base;
  int abort_flag;
};

// kBias: the optional biases inside tanh and sigma (bW, bU) are given; without them (the
// paper's form) their adds and loads are left out of the per-unit loop.
template <bool kBias>
__global__ void __launch_bounds__(kPoolTcThreads, kPoolCtasPerSm)
    router_pool_tc_kernel(const __grid_constant__ CUtensorMap tmap_q,
                          const __grid_constant__ CUtensorMap tmap_w,
                          const __grid_constant__ CUtensorMap tmap_u, RouterArgs a,
                          RouterScratch sc, int n_split) {
  extern __shared__ unsigned char smem_raw[];
  PoolTcSmem& sm = *reinterpret_cast<PoolTcSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int h = blockIdx.y, split = blockIdx.x;
  const int N = a.N;
  const int n_tiles_all = (N + 127) / 128;
  const int tile0 = (int)((long long)split * n_tiles_all / n_split);
  const int tile1 = (int)((long long)(split + 1) * n_tiles_all / n_split);
  const int n_tiles = tile1 - tile0;  // >= 1 (n_split <= n_tiles_all)
  const int tok_end = min(N, tile1 * 128);
  const int tid = threadIdx.x;
  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  unsigned int* err = sc.err;

  if (tid == 0) {
    for (int s = 0; s < kPoolTcStages; ++s) {
      mbar_init(&sm.q_full[s], 1);
      mbar_init(&sm.q_empty[s], 128);
    }
    mbar_init(&sm.wu_full, 1);
    for (int b = 0; b < kPoolAccBufs; ++b) {
      mbar_init(&sm.acc_full[b], 1);
      mbar_init(&sm.acc_empty[b], 128);
    }
    mbar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&tmap_q);
  }
  if (tid < 64) {
    sm.bias[tid] = a.bW ? a.bW[h * 64 + tid] : 0.f;
    sm.bias[64 + tid] = a.bU ? a.bU[h * 64 + tid] : 0.f;
    sm.wv[tid] = __bfloat162float(a.w[h * 64 + tid]);
  }
  if (warp == 5) {
    tmem_alloc(&sm.tmem_base, kPoolTcTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);

  float Mx = -INFINITY, lsum = 0.f;  // epilogue threads: this thread's tokens
  float acc[64];
#pragma unroll
  for (int c = 0; c < 64; ++c) acc[c] = 0.f;

  if (warp == 4) {
    // ------------------------------------------------------------ TMA producer
    bool ok = true;
    if (elect_one()) {
      mbar_arrive_expect_tx(&sm.wu_full, 128 * 64 * 2);
      tma_load_2d(sm.wu, &tmap_w, &sm.wu_full, 0, h * 64);
      tma_load_2d(sm.wu + 64 * 64, &tmap_u, &sm.wu_full, 0, h * 64);
    }
    __syncwarp();
    int i = 0;
    for (; i < n_tiles && ok; ++i) {
      const int st = i % kPoolTcStages;
      ok = mbar_wait_warp(&sm.q_empty[st], ((i / kPoolTcStages) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&sm.q_full[st], 128 * 64 * 2);
        tma_load_2d(sm.q[st], &tmap_q, &sm.q_full[st], h * 64, (tile0 + i) * 128);
      }
      __syncwarp();
    }
    if (!ok && lane == 0) {  // let issued copies land before the CTA releases its smem
      for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.wu_full, 0); ++k) {}
      for (int s = 0; s < kPoolTcStages; ++s) {
        if (i > s) {
          const int last = (i - 1 - s) / kPoolTcStages * kPoolTcStages + s;
          for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.q_full[s], (last / kPoolTcStages) & 1); ++k) {}
        }
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issue
    const uint32_t idesc = idesc_bf16(128, 128, 0, 0);
    const uint64_t db = sdesc_sw128(smem_u32(sm.wu));
    bool ok = mbar_wait_warp(&sm.wu_full, 0, err, abort_flag);
    for (int i = 0; i < n_tiles && ok; ++i) {
      const int st = i % kPoolTcStages, ab = i % kPoolAccBufs;
      ok = mbar_wait_warp(&sm.q_full[st], (i / kPoolTcStages) & 1, err, abort_flag) &&
           mbar_wait_warp(&sm.acc_empty[ab], ((i / kPoolAccBufs) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint64_t da = sdesc_sw128(smem_u32(sm.q[st]));
      if (elect_one()) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // K = 64 channels: 4 x K16, +32 bytes per step
          tc_mma_ss(tmem + ab * 128, da + 2 * kk, db + 2 * kk, idesc, kk > 0 ? 1u : 0u);
        tc_commit(&sm.acc_full[ab]);
      }
      __syncwarp();
    }
    if (!ok) {
      if (elect_one()) {
        tc_commit(&sm.drain);
        for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.drain, 0); ++k) {}
      }
      __syncwarp();
    }
  } else {
    // ------------------------------------------------------------ logits + running softmax
    const int row = warp * 32 + lane;  // TMEM lane of this thread's token
    const uint32_t t_lane = tmem + ((uint32_t)(warp * 32) << 16);
    bool ok = true;
    for (int i = 0; i < n_tiles && ok; ++i) {
      const int st = i % kPoolTcStages, ab = i % kPoolAccBufs;
      // The tile's accumulator, and its Q rows in shared memory (read below by these threads:
      // they wait on the TMA's barrier themselves rather than rely on the MMA's).
      ok = mbar_wait_warp(&sm.acc_full[ab], (i / kPoolAccBufs) & 1, err, abort_flag) &&
           mbar_wait_warp(&sm.q_full[st], (i / kPoolTcStages) & 1, err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      float e2x = 0.f, e2y = 0.f;
#pragma unroll
      for (int qtr = 0; qtr < 4; ++qtr) {  // 16 + 16 accumulator columns at a time
        float zw[16], zu[16];
        tmem_ld16(t_lane + ab * 128 + 16 * qtr, zw);
        tmem_ld16(t_lane + ab * 128 + 64 + 16 * qtr, zu);
        tmem_wait_ld();
        if (qtr == 3) {  // the accumulator is in registers: back to the MMA warp
          tc_fence_before();
          mbar_arrive(&sm.acc_empty[ab]);
        }
        float2 pe = make_float2(0.f, 0.f);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int l = 16 * qtr + 2 * k;
          const float2 wl = *reinterpret_cast<const float2*>(&sm.wv[l]);
          float2 xw = make_float2(zw[2 * k], zw[2 * k + 1]);
          float2 xu = make_float2(zu[2 * k], zu[2 * k + 1]);
          if (kBias) {
            xw = fadd2(xw, *reinterpret_cast<const float2*>(&sm.bias[l]));
            xu = fadd2(xu, *reinterpret_cast<const float2*>(&sm.bias[64 + l]));
          }
          pe = ffma2(wl, tanh_times_sigmoid2(xw, xu), pe);
        }
        e2x += pe.x;
        e2y += pe.y;
      }
      const float e = (a.variant & VP_VARIANT_MEAN_QPOOL) ? 0.f : e2x + e2y;
      const int tok = (tile0 + i) * 128 + row;
      if (tok < tok_end) {
        if (e > Mx) {  // the running maximum grows: rescale (exp(-inf) = 0 on the first token)
          const float sc_ = __expf(Mx - e);
          lsum *= sc_;
#pragma unroll
          for (int c = 0; c < 64; ++c) acc[c] *= sc_;
          Mx = e;
        }
        const float p = __expf(e - Mx);
        lsum += p;
        const unsigned char* qrow = reinterpret_cast<const unsigned char*>(sm.q[st]) + row * 128;
#pragma unroll
        for (int j = 0; j < 8; ++j) {  // 16-byte chunk j of the row sits at chunk j ^ (row & 7)
          const uint4 u = *reinterpret_cast<const uint4*>(qrow + ((j ^ (row & 7)) << 4));
          const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            acc[8 * j + 2 * k] = fmaf(p, bf16_lo(w4[k]), acc[8 * j + 2 * k]);
            acc[8 * j + 2 * k + 1] = fmaf(p, bf16_hi(w4[k]), acc[8 * j + 2 * k + 1]);
          }
        }
      }
      // The stage goes back to the TMA producer: the generic-proxy reads of the Q row above
      // are ordered before the async-proxy writes that refill it.  Without the fence the release
      // can overtake loads still in flight: a version with a two-stage ring gave q_pool values
      // up to 3 % off in repeated runs.
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(&sm.q_empty[st]);
    }
  }
  // Merge the 128 token threads' partials: the CTA maximum, then scaled sums of l and sum p q.
  if (warp < 4) {
    float m = Mx;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if (lane == 0) sm.red_m[warp] = m;
  }
  __syncthreads();
  const float M_cta = fmaxf(fmaxf(sm.red_m[0], sm.red_m[1]), fmaxf(sm.red_m[2], sm.red_m[3]));
  if (warp < 4) {
    const float f = Mx == -INFINITY ? 0.f : __expf(Mx - M_cta);
    float l = lsum * f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
#pragma unroll
    for (int c = 0; c < 64; ++c) {
      float v = acc[c] * f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      acc[c] = v;
    }
    if (lane == 0) {
      sm.red_l[warp] = l;
#pragma unroll
      for (int c = 0; c < 64; ++c) sm.red_acc[warp][c] = acc[c];
    }
  }
  __syncthreads();
  float* part = sc.pool_part + ((size_t)h * kPoolSplitMax + split) * kPoolPartial;
  if (tid < 64) {
    part[2 + tid] = sm.red_acc[0][tid] + sm.red_acc[1][tid] + sm.red_acc[2][tid] + sm.red_acc[3][tid];
    if (tid == 0) {
      part[0] = M_cta;
      part[1] = sm.red_l[0] + sm.red_l[1] + sm.red_l[2] + sm.red_l[3];
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, kPoolTcTmemCols);
  }
  pool_finish(a, sc, h, n_split);
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
      // s_h = max_j r_h(j) = 2^(max - max) / sum_j 2^(l_j - max).  No finite logit at all
      // (a NaN pooled query makes every logit NaN, and NaN never raises the running maximum)
      // means r_h is NaN, and so is s_h.
      const float s = Mx == -INFINITY ? __int_as_float(0x7fc00000) : 1.f / ll;
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

size_t heads_scratch_bytes(int H) {
  return router_scratch_bytes(H) + (size_t)kMaxHeads * kLinState * 4 +
         (kFaPartFloats + kFaStatsFloats + kFaCountWords) * 4 + (size_t)kMaxHeads * 64 * 4;
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
  sc.wo_bias = reinterpret_cast<float*>(sc.fa_count + kFaCountWords);
  return sc;
}

cudaError_t launch_router(const RouterArgs& a, const RouterScratch& sc, int num_sms,
                          cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(sc.counters, 0, 512, st);
  if (e != cudaSuccess) return e;
  // Pooling sweep on the tensor cores: two CTAs per SM (TMEM 2 x 256 columns), runs of
  // 128-token tiles.
  const int n_tiles = (a.N + 127) / 128;
  int pool_split = (kPoolCtasPerSm * num_sms + a.H - 1) / a.H;
  pool_split = max(1, min(min(pool_split, kPoolSplitMax), n_tiles));
  CUtensorMap tq, tw, tu;  // Q rows of all heads, W and U as [H 64][64]; 128-byte swizzle
  if ((e = make_tmap_bf16_2d(&tq, a.qkv, (uint64_t)3 * a.H * 64, (uint64_t)a.N,
                             (uint64_t)3 * a.H * 64, 64, 128)) != cudaSuccess)
    return e;
  if ((e = make_tmap_bf16_2d(&tw, a.W, 64, (uint64_t)a.H * 64, 64, 64, 64)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16_2d(&tu, a.U, 64, (uint64_t)a.H * 64, 64, 64, 64)) != cudaSuccess) return e;
  const int smem = (int)sizeof(PoolTcSmem) + 1024;
  const bool bias = a.bW || a.bU;
  if ((e = cudaFuncSetAttribute(bias ? router_pool_tc_kernel<true> : router_pool_tc_kernel<false>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
    return e;
  prof_before(VP_KERNEL_ROUTER_POOL, st);
  if (bias)
    router_pool_tc_kernel<true><<<dim3(pool_split, a.H), kPoolTcThreads, smem, st>>>(tq, tw, tu, a, sc,
                                                                                    pool_split);
  else
    router_pool_tc_kernel<false><<<dim3(pool_split, a.H), kPoolTcThreads, smem, st>>>(tq, tw, tu, a, sc,
                                                                                     pool_split);
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
