// Full-mode heads (Algorithm 1, step 2, s_h >= tau_high): Y_h = softmax(Q_h K_h^T / sqrt d) V_h
// as a flash-attention kernel on the sm_103a tensor cores.
//
// Persistent CTAs (one per SM) walk the work list of (full head, 128-query tile) pairs
// read from the device bins.  Warp roles:
//   warp 0     TMA producer: Q tile once per item, K/V tiles through a 3-stage ring.
//   warp 1     owns TMEM; one lane issues tcgen05.mma: S = Q K^T into one of two TMEM
//              S buffers (128 x 128 fp32 each), O += P V into a TMEM O buffer (128 x 64).
//   warps 2-5  softmax: each thread owns one query row (its TMEM lane), reads its S row,
//              keeps the running max / sum (online softmax, max rescaled lazily: O and the
//              sum are rescaled only when the max grows by more than 2^8), writes P as
//              bf16 into one of two 128-byte-swizzled smem buffers, and at the end
//              normalises O and stores Y rows.
// The S MMA of tile j+1 is issued before the P V MMA of tile j, so the tensor core works
// on the next scores while the softmax warps process the current ones.  Keys past N are
// zero-filled by TMA and masked to -inf; query rows past N are not stored.
// Every mbarrier wait is bounded (see mbar_wait); on timeout the CTA records the error,
// stops issuing work, waits for its own outstanding copies and MMAs, frees TMEM and exits.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kBM = 128;      // query rows per tile
constexpr int kBN = 128;      // keys per tile
constexpr int kStages = 3;    // K/V ring depth
constexpr int kTileBytes = 128 * 64 * 2;   // one 128 x 64 bf16 tile (16 KB)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemO = 256;          // O accumulator column offset
constexpr float kRescaleThreshold = 8.f;  // log2 units

struct FullSmem {
  __nv_bfloat16 q[128 * 64];
  __nv_bfloat16 k[kStages][128 * 64];
  __nv_bfloat16 v[kStages][128 * 64];
  __nv_bfloat16 p[2][2][128 * 64];  // [buffer][key half] 128 rows x 64 keys, swizzled
  uint64_t q_full, q_empty;
  uint64_t k_full[kStages], v_full[kStages], kv_empty[kStages];
  uint64_t s_full[2], s_empty[2], p_full[2], o_bar[2];
  uint64_t o_empty, drain;
  uint32_t tmem_base;
  int abort_flag;
};

struct FullParams {
  int N, H;
  const int32_t* head_ids;
  const int32_t* offsets;
  __nv_bfloat16* y;
  unsigned int* err;
};

__global__ void __launch_bounds__(192, 1)
    attn_full_kernel(const __grid_constant__ CUtensorMap tmap_qkv, FullParams prm) {
  extern __shared__ unsigned char smem_raw[];
  FullSmem& sm = *reinterpret_cast<FullSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);

  const int first = __ldg(prm.offsets + 2);
  const int n_heads = __ldg(prm.offsets + 3) - first;
  const int N = prm.N, H = prm.H;
  const int n_qt = (N + kBM - 1) / kBM;
  const int n_kv = (N + kBN - 1) / kBN;
  const int items = n_heads * n_qt;
  if ((int)blockIdx.x >= items) return;  // uniform across the CTA

  const int warp = warp_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;

  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    mbar_init(&sm.q_empty, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.v_full[s], 1);
      mbar_init(&sm.kv_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.s_full[b], 1);
      mbar_init(&sm.s_empty[b], 128);
      mbar_init(&sm.p_full[b], 128);
      mbar_init(&sm.o_bar[b], 1);
    }
    mbar_init(&sm.o_empty, 128);
    mbar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&tmap_qkv);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t lc = 0, ic = 0, q_issued = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++ic) {
        const int h = __ldg(prm.head_ids + first + item / n_qt);
        const int qt = item % n_qt;
        ok = mbar_wait(&sm.q_empty, (ic & 1) ^ 1, prm.err, abort_flag);
        if (!ok) break;
        ++q_issued;
        mbar_arrive_expect_tx(&sm.q_full, kTileBytes);
        tma_load_2d(sm.q, &tmap_qkv, &sm.q_full, h * 64, qt * kBM);
        for (int j = 0; j < n_kv; ++j, ++lc) {
          const int st = lc % kStages;
          const uint32_t rnd = lc / kStages;
          ok = mbar_wait(&sm.kv_empty[st], (rnd & 1) ^ 1, prm.err, abort_flag);
          if (!ok) break;
          mbar_arrive_expect_tx(&sm.k_full[st], kTileBytes);
          tma_load_2d(sm.k[st], &tmap_qkv, &sm.k_full[st], (H + h) * 64, j * kBN);
          mbar_arrive_expect_tx(&sm.v_full[st], kTileBytes);
          tma_load_2d(sm.v[st], &tmap_qkv, &sm.v_full[st], (2 * H + h) * 64, j * kBN);
        }
      }
      if (!ok) {
        // Let the copies this thread issued land before the CTA releases its smem.
        if (q_issued > 0)
          for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.q_full, (q_issued - 1) & 1); ++t) {}
        for (int s = 0; s < kStages; ++s) {
          if (lc > (uint32_t)s) {
            const uint32_t last = (lc - 1 - s) / kStages * kStages + s;  // last use of stage s
            const uint32_t par = (last / kStages) & 1;
            for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.k_full[s], par); ++t) {}
            for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.v_full[s], par); ++t) {}
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(kBM, kBN, 0, 0);   // Q (K-major) x K^T (K-major)
      const uint32_t id_o = idesc_bf16(kBM, 64, 0, 1);    // P (K-major) x V (MN-major)
      const uint64_t dq = sdesc_sw128(smem_u32(sm.q));
      uint32_t lc = 0, ic = 0, g = 0;  // g: global tile counter (S / P / O buffers)
      bool ok = true;
      for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++ic) {
        ok = mbar_wait(&sm.q_full, ic & 1, prm.err, abort_flag);
        if (!ok) break;
        tc_fence_after();
        const uint32_t lc0 = lc, g0 = g;
        // S_j = Q K_j^T into S buffer (g0 + j) & 1.
        auto issue_s = [&](int j) -> bool {
          const uint32_t l = lc0 + j, gg = g0 + j;
          const int st = l % kStages;
          if (!mbar_wait(&sm.k_full[st], (l / kStages) & 1, prm.err, abort_flag)) return false;
          if (!mbar_wait(&sm.s_empty[gg & 1], ((gg >> 1) & 1) ^ 1, prm.err, abort_flag)) return false;
          tc_fence_after();
          const uint64_t dk = sdesc_sw128(smem_u32(sm.k[st]));
          const uint32_t d_s = tmem + (gg & 1) * kBN;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // 4 x K=16 covers d = 64; +32 bytes per step
            tc_mma_ss(d_s, dq + 2 * kk, dk + 2 * kk, id_s, kk > 0);
          tc_commit(&sm.s_full[gg & 1]);
          if (j == n_kv - 1) tc_commit(&sm.q_empty);
          return true;
        };
        ok = issue_s(0);
        for (int j = 0; j < n_kv && ok; ++j) {
          if (j + 1 < n_kv) {
            ok = issue_s(j + 1);
            if (!ok) break;
          }
          // O (+)= P_j V_j
          const uint32_t l = lc0 + j, gg = g0 + j;
          const int st = l % kStages;
          ok = mbar_wait(&sm.p_full[gg & 1], (gg >> 1) & 1, prm.err, abort_flag) &&
               mbar_wait(&sm.v_full[st], (l / kStages) & 1, prm.err, abort_flag) &&
               (j > 0 || mbar_wait(&sm.o_empty, (ic & 1) ^ 1, prm.err, abort_flag));
          if (!ok) break;
          tc_fence_after();
          const uint32_t pb0 = smem_u32(sm.p[gg & 1][0]);
          const uint64_t dv = sdesc_sw128(smem_u32(sm.v[st]));
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {  // 8 x K=16 covers 128 keys
            const uint64_t da = sdesc_sw128(pb0 + (kk >> 2) * kTileBytes) + 2 * (kk & 3);
            const uint64_t db = dv + (uint64_t)(kk * 16 * 128 / 16);  // 16 keys = 2048 bytes
            tc_mma_ss(tmem + kTmemO, da, db, id_o, (j > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(&sm.o_bar[gg & 1]);
          tc_commit(&sm.kv_empty[st]);
        }
        lc = lc0 + n_kv;
        g = g0 + n_kv;
      }
      if (!ok) {
        // Wait (bounded) for every MMA this thread issued before TMEM is released.
        tc_commit(&sm.drain);
        for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.drain, 0); ++t) {}
      }
    }
  } else {
    // ------------------------------------------------------------ softmax / epilogue
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int row_in_tile = quarter * 32 + lane;
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16);
    const float c = 1.4426950408889634f * 0.125f;  // log2(e) / sqrt(64)
    const int n_tail = N - (n_kv - 1) * kBN;       // valid keys in the last tile
    uint32_t g = 0, ic = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++ic) {
      const int h = __ldg(prm.head_ids + first + item / n_qt);
      const int qt = item % n_qt;
      float m = 0.f, lsum = 0.f;
      for (int j = 0; j < n_kv; ++j, ++g) {
        const int b = g & 1;
        ok = mbar_wait(&sm.s_full[b], (g >> 1) & 1, prm.err, abort_flag);
        ok = __all_sync(0xffffffffu, ok);  // TMEM loads below need the whole warp
        if (!ok) break;
        tc_fence_after();
        float s[128];
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) tmem_ld32(t_lane + b * kBN + 32 * cc, s + 32 * cc);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(&sm.s_empty[b]);
        if (j == n_kv - 1 && n_tail < kBN) {
#pragma unroll
          for (int i = 0; i < 128; ++i)
            if (i >= n_tail) s[i] = -INFINITY;
        }
        float mx = s[0];
#pragma unroll
        for (int i = 1; i < 128; ++i) mx = fmaxf(mx, s[i]);
        const float mx2 = mx * c;
        if (j == 0) {
          m = mx2;
        } else {
          const bool need = mx2 > m + kRescaleThreshold;
          if (__any_sync(0xffffffffu, need)) {
            // Rescale O (and the sum) after P_{j-1} V_{j-1} has landed in TMEM.
            const uint32_t gp = g - 1;
            ok = mbar_wait(&sm.o_bar[gp & 1], (gp >> 1) & 1, prm.err, abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc_fence_after();
            const float alpha = need ? fast_exp2(m - mx2) : 1.f;
            float o[64];
            tmem_ld32(t_lane + kTmemO, o);
            tmem_ld32(t_lane + kTmemO + 32, o + 32);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 64; ++i) o[i] *= alpha;
            tmem_st32(t_lane + kTmemO, o);
            tmem_st32(t_lane + kTmemO + 32, o + 32);
            tmem_wait_st();
            if (need) {
              lsum *= alpha;
              m = mx2;
            }
          }
        }
        float part = 0.f;
#pragma unroll
        for (int i = 0; i < 128; ++i) {
          s[i] = fast_exp2(fmaf(s[i], c, -m));
          part += s[i];
        }
        lsum += part;
        // P buffer b is free once P_{g-2} V_{g-2} has completed.
        if (g >= 2) {
          ok = mbar_wait(&sm.o_bar[b], ((g - 2) >> 1) & 1, prm.err, abort_flag);
          ok = __all_sync(0xffffffffu, ok);
          if (!ok) break;
        }
        {
          unsigned char* pb = reinterpret_cast<unsigned char*>(sm.p[b][0]);
          const int rsw = row_in_tile & 7;
          const uint32_t row_off = (row_in_tile >> 3) * 1024 + rsw * 128;
#pragma unroll
          for (int half = 0; half < 2; ++half) {
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) {
              const float* src = s + 64 * half + 8 * ch;
              uint4 v;
              v.x = pack_bf16x2(src[0], src[1]);
              v.y = pack_bf16x2(src[2], src[3]);
              v.z = pack_bf16x2(src[4], src[5]);
              v.w = pack_bf16x2(src[6], src[7]);
              *reinterpret_cast<uint4*>(pb + half * kTileBytes + row_off + ((ch ^ rsw) << 4)) = v;
            }
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&sm.p_full[b]);
      }
      if (!ok) break;
      // Epilogue: O / sum -> bf16 -> Y[row][h][:]
      const uint32_t gl = g - 1;
      ok = mbar_wait(&sm.o_bar[gl & 1], (gl >> 1) & 1, prm.err, abort_flag);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      float o[64];
      tmem_ld32(t_lane + kTmemO, o);
      tmem_ld32(t_lane + kTmemO + 32, o + 32);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&sm.o_empty);
      const int row = qt * kBM + row_in_tile;
      if (row < N) {
        const float inv = 1.f / lsum;
        uint4* dst = reinterpret_cast<uint4*>(prm.y + ((size_t)row * H + h) * 64);
#pragma unroll
        for (int ch = 0; ch < 8; ++ch) {
          uint4 v;
          v.x = pack_bf16x2(o[8 * ch + 0] * inv, o[8 * ch + 1] * inv);
          v.y = pack_bf16x2(o[8 * ch + 2] * inv, o[8 * ch + 3] * inv);
          v.z = pack_bf16x2(o[8 * ch + 4] * inv, o[8 * ch + 5] * inv);
          v.w = pack_bf16x2(o[8 * ch + 6] * inv, o[8 * ch + 7] * inv);
          dst[ch] = v;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

cudaError_t launch_full_heads(const HeadAttnArgs& a, int num_sms, cudaStream_t st) {
  CUtensorMap tmap;
  cudaError_t e = make_tmap_bf16_2d(&tmap, a.qkv, (uint64_t)3 * a.H * 64, (uint64_t)a.N,
                                    (uint64_t)3 * a.H * 64, 64, 128);
  if (e != cudaSuccess) return e;
  const int smem = (int)sizeof(FullSmem) + 1024;
  e = cudaFuncSetAttribute(attn_full_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  FullParams prm{a.N, a.H, a.head_ids, a.offsets, a.y, a.err};
  prof_before(VP_KERNEL_ATTN_FULL, st);
  attn_full_kernel<<<num_sms, 192, smem, st>>>(tmap, prm);
  prof_after(st);
  return cudaGetLastError();
}

}  // namespace vp
