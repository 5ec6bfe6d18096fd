// Dense projections of Algorithm 1 (QKV, W_O, FFN) on the sm_103a tensor cores:
//   out[M][N] = residual + scale (.) act(A[M][K] W[N][K]^T + bias)
// optionally with a LayerNorm of A's rows folded in (A W^T -> rstd (A W^T - mu c^T), see
// LinearArgs) and with the output rows' LayerNorm statistics as (mean, M2) per 128 columns.
// Persistent CTAs (one per SM), 128 x 256 output tiles, 64-wide K blocks through a 4-stage
// TMA ring (128-byte swizzle), tcgen05.mma (M=128, N=256, K=16, bf16 -> fp32) into one of
// two TMEM accumulators, so the epilogue of tile i overlaps the main loop of tile i+1.
// Warp roles: warp 0 TMA, warp 1 TMEM owner + MMA issue, warps 2-9 epilogue: each owns a
// (32-row TMEM lane quarter, 128-column half) of the tile, one row per thread; per 32-column
// chunk it loads TMEM (the next chunk's load in flight while this one is processed), applies
// bias / GELU / LayerScale / residual, packs bf16 into a 64-byte-swizzled 32 x 32 staging
// block in shared memory and writes it with a TMA tensor store (clipped at the tensor edge).
// Tiles are visited N-fastest so the CTAs in flight share A rows and all of W in L2.
// A second instance (kSkip) leaves chosen 64-column K-blocks out: W_O with the mean heads
// folded into its bias (wo_mean_fold_kernel) skips their copies and MMAs, and with every block
// left out it is its epilogue alone.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kABytes = kBM * kBK * 2;  // 16 KB
constexpr int kBBytes = kBN * kBK * 2;  // 32 KB
constexpr uint32_t kTmemCols = 512;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;

struct GemmSmem {
  __nv_bfloat16 a[kStages][kBM * kBK];
  __nv_bfloat16 b[kStages][kBN * kBK];
  __nv_bfloat16 stage[kEpiWarps][2][32 * 32];  // per epilogue warp: two 32 x 32 output blocks
  uint64_t full[kStages], empty[kStages];
  uint64_t acc_full[2], acc_empty[2], drain;
  uint32_t tmem_base;
  uint32_t skip_mask;  // K-blocks left out (LinearArgs::skip_ids)
  int abort_flag;
};

struct GemmParams {
  int M, N, K;
  const float* bias;
  int act;
  const float* scale;
  const __nv_bfloat16* residual;
  __nv_bfloat16* out;
  unsigned int* err;
  const float2* ln_part;
  const float* ln_c;
  float ln_eps;
  float2* part_out;
  int qk_cols;  // > 0: the first qk_cols columns are Q | K of a QKV projection (see LinearArgs)
  const float* qn_g;
  const float* qn_b;
  const float* kn_g;
  const float* kn_b;
  float qk_eps;
  const float2* rope_cs;
  int tok_per_view, patch_start, grid_w;
  const int32_t* tok_index;
  const int32_t* skip_ids;
  const int32_t* skip_off;
};

// kSkip: the instance that leaves K-blocks out (GemmParams::skip_ids); the other instance has
// none of that bookkeeping.
template <bool kSkip>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_a,
                const __grid_constant__ CUtensorMap tmap_b,
                const __grid_constant__ CUtensorMap tmap_out, GemmParams prm) {
  extern __shared__ unsigned char smem_raw[];
  GemmSmem& sm = *reinterpret_cast<GemmSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int M = prm.M, N = prm.N, K = prm.K;
  const int m_tiles = (M + kBM - 1) / kBM, n_tiles = (N + kBN - 1) / kBN;
  const int tiles = m_tiles * n_tiles;
  const int k_blocks = (K + kBK - 1) / kBK;
  if ((int)blockIdx.x >= tiles) return;
  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.acc_full[b], 1);
      mbar_init(&sm.acc_empty[b], 32 * kEpiWarps);
    }
    mbar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    uint32_t skip = 0;
    if (kSkip) {
      const int s0 = __ldg(prm.skip_off), s1 = __ldg(prm.skip_off + 1);
      for (int i = s0; i < s1; ++i) skip |= 1u << (__ldg(prm.skip_ids + i) & 31);
    }
    sm.skip_mask = skip;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&tmap_a);
    tma_prefetch_desc(&tmap_b);
    tma_prefetch_desc(&tmap_out);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);
  // K-blocks left out, and whether that is all of them (A W^T is then 0).
  const uint32_t skip = kSkip ? sm.skip_mask : 0u;
  const bool acc_zero = kSkip && skip != 0 && __popc(skip & (k_blocks >= 32 ? 0xffffffffu : (1u << k_blocks) - 1u)) == k_blocks;

  if (warp == 0) {
    // TMA producer: converged warp (warp-uniform coordinates), one elected lane issues.
    uint32_t lc = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
      const int mt = t / n_tiles, nt = t - mt * n_tiles;
      for (int kb = 0; kb < k_blocks; ++kb) {
        if (kSkip && ((skip >> kb) & 1u)) continue;
        const int st = lc % kStages;
        ok = mbar_wait_warp(&sm.empty[st], ((lc / kStages) & 1) ^ 1, prm.err, abort_flag);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(&sm.full[st], kABytes + kBBytes);
          tma_load_2d(sm.a[st], &tmap_a, &sm.full[st], kb * kBK, mt * kBM);
          tma_load_2d(sm.b[st], &tmap_b, &sm.full[st], kb * kBK, nt * kBN);
        }
        __syncwarp();
        ++lc;
      }
    }
    if (!ok && lane == 0) {
      for (int s = 0; s < kStages; ++s) {
        if (lc > (uint32_t)s) {
          const uint32_t last = (lc - 1 - s) / kStages * kStages + s;
          for (int i = 0; i < 1000000 && !mbar_try_wait(&sm.full[s], (last / kStages) & 1); ++i) {}
        }
      }
    }
  } else if (warp == 1) {
    // MMA issuer: converged warp; the elected lane (always the lowest, so the same one)
    // issues the MMAs and the commits that track them.
    const uint32_t idesc = idesc_bf16(kBM, kBN, 0, 0);
    uint32_t lc = 0, i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++i) {
      const uint32_t ab = i & 1;
      ok = mbar_wait_warp(&sm.acc_empty[ab], ((i >> 1) & 1) ^ 1, prm.err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint32_t d = tmem + ab * kBN;
      bool first = true;  // the tile's first MMA overwrites the accumulator
      for (int kb = 0; kb < k_blocks; ++kb) {
        if (kSkip && ((skip >> kb) & 1u)) continue;
        const int st = lc % kStages;
        ok = mbar_wait_warp(&sm.full[st], (lc / kStages) & 1, prm.err, abort_flag);
        if (!ok) break;
        tc_fence_after();
        const uint64_t da = sdesc_sw128(smem_u32(sm.a[st]));
        const uint64_t db = sdesc_sw128(smem_u32(sm.b[st]));
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_ss(d, da + 2 * kk, db + 2 * kk, idesc, ((kSkip ? !first : kb > 0) || kk > 0) ? 1u : 0u);
          tc_commit(&sm.empty[st]);
        }
        __syncwarp();
        first = false;
        ++lc;
      }
      if (!ok) break;
      if (elect_one()) tc_commit(&sm.acc_full[ab]);
      __syncwarp();
    }
    if (!ok) {
      if (elect_one()) {
        tc_commit(&sm.drain);
        for (int it = 0; it < 1000000 && !mbar_try_wait(&sm.drain, 0); ++it) {}
      }
      __syncwarp();
    }
  } else {
    const int e = warp - 2;                 // epilogue warp 0..7
    const int quarter = warp & 3;           // TMEM lane quarter
    const int half = e >> 2;                // column half of the tile
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16);
    unsigned char* stg = reinterpret_cast<unsigned char*>(&sm.stage[e][0][0]);
    if (acc_zero) {
      // Every K-block is left out, so no MMA writes the accumulators: zero this thread's
      // columns of both once, and every tile then reads A W^T = 0.
      float z[32];
#pragma unroll
      for (int k = 0; k < 32; ++k) z[k] = 0.f;
#pragma unroll
      for (int ab = 0; ab < 2; ++ab)
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_st32(t_lane + ab * kBN + half * 128 + 32 * q, z);
      tmem_wait_st();
    }
    uint32_t i = 0, nst = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++i) {
      const int mt = t / n_tiles, nt = t - mt * n_tiles;
      const uint32_t ab = i & 1;
      if (prm.residual) {
        // Pull this thread's residual row segment (128 columns, 256 bytes) into L2 while the
        // tile's MMAs still run: read later from HBM, it would hold up the epilogue.
        const int prow = mt * kBM + quarter * 32 + lane, pcol = nt * kBN + half * 128;
        if (prow < M && pcol < N) {
          const __nv_bfloat16* pp = prm.residual + (size_t)prow * N + pcol;
          asm volatile("prefetch.global.L2 [%0];" ::"l"(pp));
          if (pcol + 64 < N) asm volatile("prefetch.global.L2 [%0];" ::"l"(pp + 64));
        }
      }
      const int row0 = mt * kBM + quarter * 32;
      const int row = row0 + lane;
      const bool row_ok = row < M;
      // Folded LayerNorm: this row's mean and 1 / sqrt(var + eps) from the (mean, M2) of its
      // 128-column blocks (equal counts: M2 = sum M2_b + 128 sum (mean_b - mean)^2).  The
      // first eight blocks (K = 1,024) are loaded before the accumulator wait.
      float ln_mu = 0.f, ln_rstd = 1.f;
      float4 lnp[4];
      const int nb = K >> 7;  // even (K % 256 == 0)
      const float4* lpp = reinterpret_cast<const float4*>(prm.ln_part + (size_t)row * nb);
      if (prm.ln_part && row_ok) {
#pragma unroll
        for (int b = 0; b < 4; ++b)
          if (2 * b < nb) lnp[b] = __ldg(lpp + b);
      }
      const bool ok = mbar_wait_warp(&sm.acc_full[ab], (i >> 1) & 1, prm.err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      if (prm.ln_part && row_ok) {
        float sm_ = 0.f;
#pragma unroll
        for (int b = 0; b < 4; ++b)
          if (2 * b < nb) sm_ += lnp[b].x + lnp[b].z;
        for (int b = 4; 2 * b < nb; ++b) {
          const float4 p4 = __ldg(lpp + b);
          sm_ += p4.x + p4.z;
        }
        ln_mu = sm_ / (float)nb;
        float m2 = 0.f;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          if (2 * b < nb) {
            const float d0 = lnp[b].x - ln_mu, d1 = lnp[b].z - ln_mu;
            m2 += lnp[b].y + lnp[b].w + 128.f * (d0 * d0 + d1 * d1);
          }
        }
        for (int b = 4; 2 * b < nb; ++b) {
          const float4 p4 = __ldg(lpp + b);
          const float d0 = p4.x - ln_mu, d1 = p4.z - ln_mu;
          m2 += p4.y + p4.w + 128.f * (d0 * d0 + d1 * d1);
        }
        ln_rstd = rsqrtf(m2 / (float)K + prm.ln_eps);
      }
      float cmean[4], cm2[4];  // output statistics per 32-column chunk (part_out)
      const uint32_t tcol = t_lane + ab * kBN + half * 128;
      // Bias, or the folded LayerNorm rstd (acc - mu c) + bias', on one 32-column chunk.
      auto bias_fold = [&](float* x, int col0) {
        if (prm.ln_part) {  // rstd (acc - mu c) + bias'
          const float2 nmu = make_float2(-ln_mu, -ln_mu), rs = make_float2(ln_rstd, ln_rstd);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const bool in = col0 + 4 * q + 3 < N;
            const float4 c4 = in ? __ldg(reinterpret_cast<const float4*>(prm.ln_c + col0) + q)
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
            const float4 b4 = in ? __ldg(reinterpret_cast<const float4*>(prm.bias + col0) + q)
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
            const float2 a0 = ffma2(rs, ffma2(nmu, make_float2(c4.x, c4.y),
                                              make_float2(x[4 * q], x[4 * q + 1])),
                                    make_float2(b4.x, b4.y));
            const float2 a1 = ffma2(rs, ffma2(nmu, make_float2(c4.z, c4.w),
                                              make_float2(x[4 * q + 2], x[4 * q + 3])),
                                    make_float2(b4.z, b4.w));
            x[4 * q] = a0.x;
            x[4 * q + 1] = a0.y;
            x[4 * q + 2] = a1.x;
            x[4 * q + 3] = a1.y;
          }
        } else if (prm.bias) {
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float4 b4 = col0 + 4 * q + 3 < N
                                  ? __ldg(reinterpret_cast<const float4*>(prm.bias + col0) + q)
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
            const float2 a0 = fadd2(make_float2(x[4 * q], x[4 * q + 1]), make_float2(b4.x, b4.y));
            const float2 a1 = fadd2(make_float2(x[4 * q + 2], x[4 * q + 3]), make_float2(b4.z, b4.w));
            x[4 * q] = a0.x;
            x[4 * q + 1] = a0.y;
            x[4 * q + 2] = a1.x;
            x[4 * q + 3] = a1.y;
          }
        }
      };
      // Stage a 32 x 32 block (row = lane, 64 bytes) and write it with a TMA tensor store.
      auto store_chunk = [&](const float* x, int col0) {
        // Stage the 32 x 32 block (row = lane, 64 bytes) in the 64-byte swizzle the
        // output tensor map uses: 16-byte chunk q of row r sits at chunk q ^ ((r >> 1) & 3).
        unsigned char* buf = stg + (nst & 1) * 2048;
        // The elected lane (lane 0, the lowest) owns this warp's bulk stores and their groups.
        if (nst >= 2 && elect_one()) tma_store_wait_read<1>();  // this buffer's last store read it
        __syncwarp();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 u;
          u.x = pack_bf16x2(x[8 * q + 0], x[8 * q + 1]);
          u.y = pack_bf16x2(x[8 * q + 2], x[8 * q + 3]);
          u.z = pack_bf16x2(x[8 * q + 4], x[8 * q + 5]);
          u.w = pack_bf16x2(x[8 * q + 6], x[8 * q + 7]);
          *reinterpret_cast<uint4*>(buf + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4)) = u;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (elect_one()) {
          tma_store_2d(&tmap_out, buf, col0, row0);
          tma_store_commit();
        }
        ++nst;
      };
      const int pcol0 = nt * kBN + half * 128;  // this thread's 128 columns: two heads
      if (prm.qk_cols > 0 && pcol0 < prm.qk_cols) {
        // Q or K columns of a QKV projection with qk-norm and / or 2-D RoPE: whole heads
        // (64 columns, two chunks) at a time.
        const bool is_q = pcol0 < (prm.qk_cols >> 1);
        const float* ng = is_q ? prm.qn_g : prm.kn_g;
        const float* nbv = is_q ? prm.qn_b : prm.kn_b;
        int py = 0, px = 0;  // the row's position inside its view
        if (prm.rope_cs) {
          const int tok = prm.tok_index && row_ok ? __ldg(prm.tok_index + row) : row;
          const int t = tok % prm.tok_per_view - prm.patch_start;
          if (t >= 0) {
            py = t / prm.grid_w + 1;
            px = t - (py - 1) * prm.grid_w + 1;
          }
        }
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
          float x[64];
          tmem_ld32(tcol + 64 * hh, x);
          tmem_ld32(tcol + 64 * hh + 32, x + 32);
          tmem_wait_ld();
          if (hh == 1) {
            tc_fence_before();
            mbar_arrive(&sm.acc_empty[ab]);
          }
          const int col0 = pcol0 + 64 * hh;
          bias_fold(x, col0);
          bias_fold(x + 32, col0 + 32);
          if (ng) {  // LayerNorm over the head's 64 channels
            float2 s2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int k = 0; k < 32; ++k) s2 = fadd2(s2, make_float2(x[2 * k], x[2 * k + 1]));
            const float mean = (s2.x + s2.y) * (1.f / 64.f);
            float2 q2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              const float2 dd = fadd2(make_float2(x[2 * k], x[2 * k + 1]), make_float2(-mean, -mean));
              q2 = ffma2(dd, dd, q2);
            }
            const float rstd = rsqrtf((q2.x + q2.y) * (1.f / 64.f) + prm.qk_eps);
            const float2 nm = make_float2(-mean * rstd, -mean * rstd), rs = make_float2(rstd, rstd);
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const float4 g4 = __ldg(reinterpret_cast<const float4*>(ng) + q);
              const float4 b4 = __ldg(reinterpret_cast<const float4*>(nbv) + q);
              const float2 a0 = ffma2(ffma2(make_float2(x[4 * q], x[4 * q + 1]), rs, nm),
                                      make_float2(g4.x, g4.y), make_float2(b4.x, b4.y));
              const float2 a1 = ffma2(ffma2(make_float2(x[4 * q + 2], x[4 * q + 3]), rs, nm),
                                      make_float2(g4.z, g4.w), make_float2(b4.z, b4.w));
              x[4 * q] = a0.x;
              x[4 * q + 1] = a0.y;
              x[4 * q + 2] = a1.x;
              x[4 * q + 3] = a1.y;
            }
          }
          if (prm.rope_cs) {  // channels [0, 32) turn with the row, [32, 64) with the column
#pragma unroll
            for (int ax = 0; ax < 2; ++ax) {
              const float4* cs = reinterpret_cast<const float4*>(prm.rope_cs + (size_t)(ax ? px : py) * 16);
#pragma unroll
              for (int q = 0; q < 8; ++q) {  // frequencies 2q, 2q + 1: (cos, sin) pairs
                const float4 t4 = __ldg(cs + q);
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                  const int i = 32 * ax + 2 * q + e;
                  const float c = e ? t4.z : t4.x, sn = e ? t4.w : t4.y;
                  const float a = x[i], b = x[i + 16];
                  x[i] = fmaf(a, c, -b * sn);
                  x[i + 16] = fmaf(b, c, a * sn);
                }
              }
            }
          }
          if (col0 < N) store_chunk(x, col0);
          if (col0 + 32 < N) store_chunk(x + 32, col0 + 32);
        }
        continue;
      }
      float v[2][32];
      tmem_ld32(tcol, v[0]);
      tmem_wait_ld();
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        if (cc + 1 < 4) tmem_ld32(tcol + 32 * (cc + 1), v[(cc + 1) & 1]);  // in flight meanwhile
        float* x = v[cc & 1];
        const int col0 = nt * kBN + half * 128 + cc * 32;
        if (col0 < N) {
          // Bias, GELU, LayerScale and residual on column pairs (packed f32x2 arithmetic).
          bias_fold(x, col0);
          if (prm.act == VP_ACT_GELU) {
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const float2 gk = gelu_as2(make_float2(x[2 * k], x[2 * k + 1]));
              x[2 * k] = gk.x;
              x[2 * k + 1] = gk.y;
            }
          }
          if (prm.scale) {
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float4 s4 = col0 + 4 * q + 3 < N
                                    ? __ldg(reinterpret_cast<const float4*>(prm.scale + col0) + q)
                                    : make_float4(0.f, 0.f, 0.f, 0.f);
              const float2 a0 = fmul2(make_float2(x[4 * q], x[4 * q + 1]), make_float2(s4.x, s4.y));
              const float2 a1 = fmul2(make_float2(x[4 * q + 2], x[4 * q + 3]), make_float2(s4.z, s4.w));
              x[4 * q] = a0.x;
              x[4 * q + 1] = a0.y;
              x[4 * q + 2] = a1.x;
              x[4 * q + 3] = a1.y;
            }
          }
          if (prm.residual && row_ok) {
            const __nv_bfloat16* rp = prm.residual + (size_t)row * N + col0;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              if (col0 + 8 * q + 7 < N) {
                const uint4 u = *reinterpret_cast<const uint4*>(rp + 8 * q);
                const uint32_t uw[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const float2 a = fadd2(make_float2(x[8 * q + 2 * k], x[8 * q + 2 * k + 1]),
                                         make_float2(bf16_lo(uw[k]), bf16_hi(uw[k])));
                  x[8 * q + 2 * k] = a.x;
                  x[8 * q + 2 * k + 1] = a.y;
                }
              }
            }
          }
          if (prm.part_out) {  // chunk mean and M2 (two passes over registers)
            float2 s2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int k = 0; k < 16; ++k) s2 = fadd2(s2, make_float2(x[2 * k], x[2 * k + 1]));
            const float cm = (s2.x + s2.y) * (1.f / 32.f);
            float2 q2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const float2 dd = fadd2(make_float2(x[2 * k], x[2 * k + 1]), make_float2(-cm, -cm));
              q2 = ffma2(dd, dd, q2);
            }
            cmean[cc] = cm;
            cm2[cc] = q2.x + q2.y;
          }
          store_chunk(x, col0);
        }
        tmem_wait_ld();
        if (cc == 3) {
          tc_fence_before();
          mbar_arrive(&sm.acc_empty[ab]);
        }
      }
      const int pcol = nt * kBN + half * 128;  // this thread's 128-column block
      if (prm.part_out && row_ok && pcol < N) {
        const float mb = 0.25f * (cmean[0] + cmean[1] + cmean[2] + cmean[3]);
        float m2 = cm2[0] + cm2[1] + cm2[2] + cm2[3];
#pragma unroll
        for (int k = 0; k < 4; ++k) m2 += 32.f * (cmean[k] - mb) * (cmean[k] - mb);
        prm.part_out[(size_t)row * (N >> 7) + (pcol >> 7)] = make_float2(mb, m2);
      }
    }
    if (elect_one()) tma_store_wait_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// RoPE angles in double precision: table[p][i] = (cos, sin)(p base^(-i / 16)).
__global__ void rope_table_kernel(int max_pos, double base, float2* table) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= (max_pos + 1) * 16) return;
  const int p = k >> 4, i = k & 15;
  double sn, cs;
  sincos((double)p * pow(base, -(double)i / 16.0), &sn, &cs);
  table[k] = make_float2((float)cs, (float)sn);
}

}  // namespace

namespace {

// A warp per output column n of W_O: lane l takes channels 2 l, 2 l + 1 of every mean head.
__global__ void wo_mean_fold_kernel(int D, int H, const __nv_bfloat16* w_o, const float* b_o,
                                    const float* mean_v, const int32_t* head_ids,
                                    const int32_t* offsets, float* bias_out) {
  const int n = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (n >= D) return;  // whole warps
  const int m0 = __ldg(offsets), m1 = __ldg(offsets + 1);
  const __nv_bfloat16* wrow = w_o + (size_t)n * H * 64 + 2 * lane;
  float acc = 0.f;
  for (int i = m0; i < m1; ++i) {
    const int h = __ldg(head_ids + i);
    const uint32_t w2 = __ldg(reinterpret_cast<const unsigned int*>(wrow + h * 64));
    // the mean head's row of Y as stored: bf16(mean_v), round to nearest even
    const float2 mv = __ldg(reinterpret_cast<const float2*>(mean_v + h * 64) + lane);
    const uint32_t mu = pack_bf16x2(mv.x, mv.y);
    acc = fmaf(bf16_lo(mu), bf16_lo(w2), fmaf(bf16_hi(mu), bf16_hi(w2), acc));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) bias_out[n] = (b_o ? __ldg(b_o + n) : 0.f) + acc;
}

}  // namespace

cudaError_t launch_rope_table(int max_pos, float base, float2* table, cudaStream_t st) {
  const int n = (max_pos + 1) * 16;
  rope_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(max_pos, (double)base, table);
  return cudaGetLastError();
}

cudaError_t launch_wo_mean_fold(int D, int H, const __nv_bfloat16* w_o, const float* b_o,
                                const float* mean_v, const int32_t* head_ids,
                                const int32_t* offsets, float* bias_out, cudaStream_t st) {
  const int threads = 256, blocks = (D * 32 + threads - 1) / threads;
  wo_mean_fold_kernel<<<blocks, threads, 0, st>>>(D, H, w_o, b_o, mean_v, head_ids, offsets,
                                                  bias_out);
  return cudaGetLastError();
}

cudaError_t launch_linear(const LinearArgs& a, int num_sms, cudaStream_t st) {
  CUtensorMap ta, tb, to;
  cudaError_t e = make_tmap_bf16_2d(&ta, a.A, (uint64_t)a.K, (uint64_t)a.M, (uint64_t)a.K, kBK, kBM);
  if (e != cudaSuccess) return e;
  e = make_tmap_bf16_2d(&tb, a.W, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K, kBK, kBN);
  if (e != cudaSuccess) return e;
  e = make_tmap_bf16_2d(&to, a.out, (uint64_t)a.N, (uint64_t)a.M, (uint64_t)a.N, 32, 32, 64);
  if (e != cudaSuccess) return e;
  const int smem = (int)sizeof(GemmSmem) + 1024;
  const bool skip = a.skip_ids != nullptr;
  e = cudaFuncSetAttribute(skip ? gemm_kernel<true> : gemm_kernel<false>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int tiles = ((a.M + kBM - 1) / kBM) * ((a.N + kBN - 1) / kBN);
  if ((a.ln_part && (a.K % 256 != 0 || !a.ln_c || !a.bias)) ||
      (a.part_out && a.N % 128 != 0))
    return cudaErrorInvalidValue;
  const bool qk = a.qk_cols > 0;
  if (a.skip_ids && (!a.skip_off || a.ln_part || qk || a.K % kBK != 0 || a.K > 32 * kBK))
    return cudaErrorInvalidValue;
  if (qk && (a.qk_cols % 256 != 0 || a.qk_cols > a.N || a.act != VP_ACT_NONE || a.scale ||
             a.residual || a.part_out || (!a.qn_g != !a.qn_b) || (!a.kn_g != !a.kn_b) ||
             (a.rope_cs && (a.tok_per_view < 1 || a.grid_w < 1 || a.patch_start < 0))))
    return cudaErrorInvalidValue;
  GemmParams prm{a.M,     a.N,   a.K,   a.bias,      a.act,  a.scale,   a.residual,
                 a.out,   a.err, a.ln_part, a.ln_c, a.ln_eps, a.part_out,
                 qk ? a.qk_cols : 0, a.qn_g, a.qn_b, a.kn_g, a.kn_b, a.qk_eps, a.rope_cs,
                 a.tok_per_view, a.patch_start, a.grid_w, a.tok_index, a.skip_ids, a.skip_off};
  prof_before(VP_KERNEL_GEMM, st);
  if (skip)
    gemm_kernel<true><<<min(num_sms, tiles), kThreads, smem, st>>>(ta, tb, to, prm);
  else
    gemm_kernel<false><<<min(num_sms, tiles), kThreads, smem, st>>>(ta, tb, to, prm);
  prof_after(st);
  return cudaGetLastError();
}

}  // namespace vp
