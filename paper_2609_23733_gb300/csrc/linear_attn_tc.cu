// §5 compute-mode ablation (linear attention in place of the surrogate): the state of every
// surrogate head, S_h[c][e] = sum_j phi(k_j)[c] v_j[e] and z_h[c] = sum_j phi(k_j)[c] with
// phi = elu + 1, on the tcgen05 tensor cores.
//
// As a matrix product over the tokens, S = Phi^T V.  Phi is split into bf16 parts (hi =
// bf16(phi), lo = bf16(phi - hi), 16 significant bits together), so that one M128 N64 MMA per
// 16 tokens computes both parts: A = [Phi_hi^T; Phi_lo^T] (128 rows: channel c of the hi part
// in row c, of the lo part in row 64 + c; the tokens along K), B = V (the tokens along K, the
// 64 value channels along N, MN-major as the TMA loads it), and S[c][e] = D[c][e] + D[64 + c][e]
// in fp32.  V is exact in bf16, so the only rounding beyond fp32 accumulation is phi's split.
//   warp 0       TMA: 64-token tiles of K_h and V_h (8 KB each, 128-byte swizzle) through a
//                kStages ring;
//   warp 1       TMEM owner and MMA issue: four tcgen05.mma M128 N64 K16 per tile into one
//                64-column fp32 accumulator kept over the CTA's whole token range;
//   warps 2-9    phi: thread (c, q) reads channel c of tokens 16 q .. 16 q + 15 from the K tile,
//                writes their hi and lo parts into rows c and 64 + c of the Phi^T tile (K-major,
//                128-byte swizzle, two buffers), and sums z_c; tokens past the CTA's range get
//                phi = 0.  At the end warps 2-5 read the accumulator, the CTA adds S and z to
//                lin_state with atomics.
// Grid (splits, H): blockIdx.y is the slot in the surrogate bin (CTAs past the bin's end
// return); each CTA takes a range of whole 64-token tiles.  Every wait is bounded; on a timeout
// the CTA records the error, stops, lets its copies and MMAs land, frees TMEM and adds nothing.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kLsTile = 64;                     // tokens per tile
constexpr int kLsStages = 4;                    // K / V ring depth
constexpr int kLsPhiThreads = 256;              // warps 2-9
constexpr int kLsThreads = 64 + kLsPhiThreads;  // + the TMA and MMA warps
constexpr uint32_t kLsTmemCols = 64;
constexpr uint32_t kLsTileBytes = kLsTile * 64 * 2;  // one K or V tile

struct LsSmem {
  __nv_bfloat16 k[kLsStages][kLsTile * 64];
  __nv_bfloat16 v[kLsStages][kLsTile * 64];
  __nv_bfloat16 phi[2][128 * kLsTile];  // [Phi_hi^T; Phi_lo^T], rows of 64 tokens
  uint64_t kv_full[kLsStages], kv_empty[kLsStages];
  uint64_t phi_full[2], phi_empty[2], d_full, drain;
  float z[4][64];
  uint32_t tmem_base;
  int abort_flag;
};
constexpr int kRedPitch = 68;  // floats per accumulator row staged at the end (padded)
static_assert(sizeof(float) * 128 * kRedPitch <= sizeof(__nv_bfloat16) * 2 * kLsStages * kLsTile * 64,
              "the K and V ring holds the accumulator's 128 padded rows at the end");

__device__ __forceinline__ float elu1(float x) { return x > 0.f ? x + 1.f : __expf(x); }

__global__ void __launch_bounds__(kLsThreads, 2)
    linear_state_tc_kernel(const __grid_constant__ CUtensorMap tmap_qkv, HeadAttnArgs a,
                           int n_split) {
  extern __shared__ unsigned char smem_raw[];
  LsSmem& sm = *reinterpret_cast<LsSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int s_first = __ldg(a.offsets + 1), n_surr = __ldg(a.offsets + 2) - s_first;
  if ((int)blockIdx.y >= n_surr) return;  // uniform across the CTA
  const int h = __ldg(a.head_ids + s_first + blockIdx.y);
  const int N = a.N, H = a.H;
  const int n_tiles_all = (N + kLsTile - 1) / kLsTile;
  const int tile0 = (int)((long long)blockIdx.x * n_tiles_all / n_split);
  const int tile1 = (int)((long long)(blockIdx.x + 1) * n_tiles_all / n_split);
  const int n_tiles = tile1 - tile0;
  if (n_tiles <= 0) return;  // uniform
  const int tok_end = min(N, tile1 * kLsTile);
  const int tid = threadIdx.x;
  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  unsigned int* err = a.err;

  if (tid == 0) {
    for (int s = 0; s < kLsStages; ++s) {
      mbar_init(&sm.kv_full[s], 1);
      mbar_init(&sm.kv_empty[s], kLsPhiThreads + 1);  // the phi threads' K reads + the MMA's V
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.phi_full[b], kLsPhiThreads);
      mbar_init(&sm.phi_empty[b], 1);
    }
    mbar_init(&sm.d_full, 1);
    mbar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&tmap_qkv);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kLsTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);
  bool ok = true;
  int issued = 0;  // K / V tiles whose copies warp 0 started

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    for (; issued < n_tiles && ok; ++issued) {
      const int j = issued, st = j % kLsStages;
      ok = mbar_wait_warp(&sm.kv_empty[st], ((j / kLsStages) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&sm.kv_full[st], 2 * kLsTileBytes);
        tma_load_2d(sm.k[st], &tmap_qkv, &sm.kv_full[st], (H + h) * 64, (tile0 + j) * kLsTile);
        tma_load_2d(sm.v[st], &tmap_qkv, &sm.kv_full[st], (2 * H + h) * 64, (tile0 + j) * kLsTile);
      }
      __syncwarp();
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    const uint32_t idesc = idesc_bf16(128, 64, 0, 1);  // Phi^T (K-major) x V (MN-major)
    for (int j = 0; j < n_tiles && ok; ++j) {
      const int st = j % kLsStages, pb = j & 1;
      ok = mbar_wait_warp(&sm.phi_full[pb], (j >> 1) & 1, err, abort_flag) &&
           mbar_wait_warp(&sm.kv_full[st], (j / kLsStages) & 1, err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint64_t da = sdesc_sw128(smem_u32(sm.phi[pb]));
      const uint64_t db = sdesc_sw128(smem_u32(sm.v[st]));
      if (elect_one()) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // 16 tokens per step: +32 bytes of A, +2 KB of V
          tc_mma_ss(tmem, da + 2 * kk, db + (uint64_t)(kk * 128), idesc, (j > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&sm.phi_empty[pb]);
        tc_commit(&sm.kv_empty[st]);
        if (j == n_tiles - 1) tc_commit(&sm.d_full);
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
    // ------------------------------------------------------------ phi = elu + 1, split
    const int pt = tid - 64, c = pt & 63, q = pt >> 6;  // channel, token quarter of a tile
    float zc = 0.f;
    for (int j = 0; j < n_tiles && ok; ++j) {
      const int st = j % kLsStages, pb = j & 1;
      ok = mbar_wait_warp(&sm.kv_full[st], (j / kLsStages) & 1, err, abort_flag) &&
           mbar_wait_warp(&sm.phi_empty[pb], ((j >> 1) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      const unsigned char* kt = reinterpret_cast<const unsigned char*>(sm.k[st]);
      const int tbase = (tile0 + j) * kLsTile;
      uint32_t hi[8], lo[8];  // tokens 16 q .. 16 q + 15 of channel c, bf16 pairs
#pragma unroll
      for (int u = 0; u < 16; u += 2) {
        float f[2];
#pragma unroll
        for (int w = 0; w < 2; ++w) {
          const int t = 16 * q + u + w;  // row of the K tile: 16-byte chunk (c / 8) ^ (t % 8)
          const uint32_t kb =
              *reinterpret_cast<const uint16_t*>(kt + t * 128 + ((((c >> 3) ^ (t & 7))) << 4) + (c & 7) * 2);
          f[w] = tbase + t < tok_end ? elu1(__uint_as_float(kb << 16)) : 0.f;
          zc += f[w];
        }
        const uint32_t hw = pack_bf16x2(f[0], f[1]);
        hi[u >> 1] = hw;
        lo[u >> 1] = pack_bf16x2(f[0] - bf16_lo(hw), f[1] - bf16_hi(hw));
      }
      // Rows c (hi) and 64 + c (lo) of Phi^T: 16-byte chunks 2 q, 2 q + 1 at chunk ^ (row % 8).
      unsigned char* ph = reinterpret_cast<unsigned char*>(sm.phi[pb]) + c * 128;
      unsigned char* pl = reinterpret_cast<unsigned char*>(sm.phi[pb]) + (64 + c) * 128;
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        const int jc = ((2 * q + m) ^ (c & 7)) << 4;
        *reinterpret_cast<uint4*>(ph + jc) = make_uint4(hi[4 * m], hi[4 * m + 1], hi[4 * m + 2], hi[4 * m + 3]);
        *reinterpret_cast<uint4*>(pl + jc) = make_uint4(lo[4 * m], lo[4 * m + 1], lo[4 * m + 2], lo[4 * m + 3]);
      }
      // The Phi^T writes and the K reads are ordered before the async proxy's use of them (the
      // MMA reads Phi^T, the TMA refills the K stage).
      fence_proxy_async_smem();
      mbar_arrive(&sm.phi_full[pb]);
      mbar_arrive(&sm.kv_empty[st]);
    }
    sm.z[q][c] = zc;
  }
  __syncthreads();  // the roles are done; z written
  if (warp == 0 && lane == 0 && *abort_flag) {  // after a timeout: let issued copies land
    for (int s = 0; s < kLsStages; ++s) {
      if (issued > s) {
        const int last = (issued - 1 - s) / kLsStages * kLsStages + s;
        for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.kv_full[s], (last / kLsStages) & 1); ++k) {}
      }
    }
  }
  __syncthreads();  // the K / V ring is free
  // The accumulator D (128 lanes x 64 columns) into shared memory (rows padded to 68 floats),
  // then S[c][e] = D[c][e] + D[64 + c][e] and z into lin_state.
  float* red = reinterpret_cast<float*>(sm.k[0]);  // k then v: one 64 KB region
  const bool alive = !*abort_flag;
  if (warp >= 2 && warp < 6 && alive) {
    const bool got = mbar_wait_warp(&sm.d_full, 0, err, abort_flag);
    if (got) {
      tc_fence_after();
      const int row = (warp & 3) * 32 + lane;
      float d[64];
      tmem_ld32(tmem + ((uint32_t)((warp & 3) * 32) << 16), d);
      tmem_ld32(tmem + ((uint32_t)((warp & 3) * 32) << 16) + 32, d + 32);
      tmem_wait_ld();
      float4* dst = reinterpret_cast<float4*>(red + row * kRedPitch);
#pragma unroll
      for (int i = 0; i < 16; ++i) dst[i] = make_float4(d[4 * i], d[4 * i + 1], d[4 * i + 2], d[4 * i + 3]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid >= 64 && !*abort_flag) {
    float* st = a.lin_state + (size_t)h * kLinState;
    for (int idx = tid - 64; idx < 64 * 64; idx += kLsPhiThreads) {
      const int cc = idx >> 6, e = idx & 63;
      atomicAdd(st + idx, red[cc * kRedPitch + e] + red[(64 + cc) * kRedPitch + e]);
    }
    if (tid - 64 < 64) {
      const int cc = tid - 64;
      atomicAdd(st + 64 * 64 + cc, sm.z[0][cc] + sm.z[1][cc] + sm.z[2][cc] + sm.z[3][cc]);
    }
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kLsTmemCols);
  }
}

}  // namespace

cudaError_t launch_linear_state_tc(const HeadAttnArgs& a, int num_sms, cudaStream_t st) {
  CUtensorMap tmap;  // [N][3 H 64] bf16: boxes of 64 tokens x 64 channels
  cudaError_t e = make_tmap_bf16_2d(&tmap, a.qkv, (uint64_t)3 * a.H * 64, (uint64_t)a.N,
                                    (uint64_t)3 * a.H * 64, 64, kLsTile);
  if (e != cudaSuccess) return e;
  const int smem = (int)sizeof(LsSmem) + 1024;
  e = cudaFuncSetAttribute(linear_state_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_tiles = (a.N + kLsTile - 1) / kLsTile;
  const int n_split = max(1, min(n_tiles, (2 * num_sms + a.H - 1) / a.H));  // two CTAs per SM
  linear_state_tc_kernel<<<dim3(n_split, a.H), kLsThreads, smem, st>>>(tmap, a, n_split);
  return cudaGetLastError();
}

namespace {

// The apply of linear attention for every surrogate head, y_i = phi(q_i)^T S / (phi(q_i)^T z),
// on the tcgen05 tensor cores, after linear_state_tc_kernel.  A CTA takes a range of 128-token
// tiles of one head; per tile one M128 N64 product with K = 64 channels for each of S's bf16
// parts (hi + lo, 16 significant bits together): D = Phi(Q) S_hi + Phi(Q) S_lo.
//   warp 0       TMA: the tiles' Q rows (128 x 64, 16 KB, 128-byte swizzle), two buffers;
//   warp 1       TMEM owner and MMA issue, two 64-column fp32 accumulators;
//   warps 2-5    one token row each (the row's TMEM lane): phi = elu + 1 of the row in place in
//                the Q tile (bf16, the A operand as it stands: tokens as rows, channels along
//                K), the denominator phi^T z in fp32 from the unrounded phi, and after the MMAs
//                y = D / den as bf16; the next tile's phi is written before this tile's output.
// S^T's parts (rows e, channels c along K) and z are staged once per CTA from lin_state.
constexpr int kLaRows = 128;
constexpr int kLaThreads = 192;
constexpr uint32_t kLaTmemCols = 128;
constexpr uint32_t kLaTileBytes = kLaRows * 64 * 2;

struct LaSmem {
  __nv_bfloat16 q[2][kLaRows * 64];
  __nv_bfloat16 bhi[64 * 64];  // S^T parts: row e, 16-byte chunk c / 8 at chunk ^ (e % 8)
  __nv_bfloat16 blo[64 * 64];
  __align__(16) float z[64];
  uint64_t q_full[2], q_empty[2], phi_full[2], d_full[2], d_empty[2], drain;
  uint32_t tmem_base;
  int abort_flag;
};

// Four floats of shared memory, read anew on every call (z is not kept in 64 registers
// across the tile loop).
__device__ __forceinline__ float4 lds_f4_volatile(const float* p) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(smem_u32(p)));
  return v;
}

__global__ void __launch_bounds__(kLaThreads, 4)
    linear_apply_tc_kernel(const __grid_constant__ CUtensorMap tmap_qkv, HeadAttnArgs a,
                           int n_split) {
  extern __shared__ unsigned char smem_raw[];
  LaSmem& sm = *reinterpret_cast<LaSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int s_first = __ldg(a.offsets + 1), n_surr = __ldg(a.offsets + 2) - s_first;
  if ((int)blockIdx.y >= n_surr) return;  // uniform across the CTA
  const int h = __ldg(a.head_ids + s_first + blockIdx.y);
  const int N = a.N, H = a.H;
  const int n_tiles_all = (N + kLaRows - 1) / kLaRows;
  const int tile0 = (int)((long long)blockIdx.x * n_tiles_all / n_split);
  const int tile1 = (int)((long long)(blockIdx.x + 1) * n_tiles_all / n_split);
  const int n_tiles = tile1 - tile0;
  if (n_tiles <= 0) return;  // uniform
  const int tid = threadIdx.x;
  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  unsigned int* err = a.err;

  if (tid == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.q_full[b], 1);
      mbar_init(&sm.q_empty[b], 1);
      mbar_init(&sm.phi_full[b], 128);
      mbar_init(&sm.d_full[b], 1);
      mbar_init(&sm.d_empty[b], 128);
    }
    mbar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    fence_mbarrier_init();
    tma_prefetch_desc(&tmap_qkv);
  }
  // S^T's hi and lo parts and z from the state.
  const float* state = a.lin_state + (size_t)h * kLinState;
  for (int i = tid; i < 64 * 8; i += kLaThreads) {
    const int e = i >> 3, jc = i & 7;
    uint32_t wh[4], wl[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float s0 = __ldcg(state + (8 * jc + 2 * k) * 64 + e);
      const float s1 = __ldcg(state + (8 * jc + 2 * k + 1) * 64 + e);
      wh[k] = pack_bf16x2(s0, s1);
      wl[k] = pack_bf16x2(s0 - bf16_lo(wh[k]), s1 - bf16_hi(wh[k]));
    }
    const int off = e * 64 + ((jc ^ (e & 7)) << 3);  // in elements
    *reinterpret_cast<uint4*>(&sm.bhi[off]) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
    *reinterpret_cast<uint4*>(&sm.blo[off]) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
  }
  if (tid < 64) sm.z[tid] = __ldcg(state + 64 * 64 + tid);
  fence_proxy_async_smem();  // the staged B operands, before the MMAs read them
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kLaTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);
  bool ok = true;
  int issued = 0;  // Q tiles whose copy warp 0 started

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    for (; issued < n_tiles && ok; ++issued) {
      const int j = issued, s = j & 1;
      ok = mbar_wait_warp(&sm.q_empty[s], ((j >> 1) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&sm.q_full[s], kLaTileBytes);
        tma_load_2d(sm.q[s], &tmap_qkv, &sm.q_full[s], h * 64, (tile0 + j) * kLaRows);
      }
      __syncwarp();
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    const uint32_t idesc = idesc_bf16(128, 64, 0, 0);  // Phi(Q) (K-major) x S^T part (K-major)
    const uint64_t dbh = sdesc_sw128(smem_u32(sm.bhi)), dbl = sdesc_sw128(smem_u32(sm.blo));
    for (int j = 0; j < n_tiles && ok; ++j) {
      const int s = j & 1;
      ok = mbar_wait_warp(&sm.phi_full[s], (j >> 1) & 1, err, abort_flag) &&
           mbar_wait_warp(&sm.d_empty[s], ((j >> 1) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint64_t da = sdesc_sw128(smem_u32(sm.q[s]));
      if (elect_one()) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // K = 64 channels: 4 x K16, +32 bytes per step
          tc_mma_ss(tmem + s * 64, da + 2 * kk, dbh + 2 * kk, idesc, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) tc_mma_ss(tmem + s * 64, da + 2 * kk, dbl + 2 * kk, idesc, 1u);
        tc_commit(&sm.q_empty[s]);
        tc_commit(&sm.d_full[s]);
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
    // ------------------------------------------------------------ phi, denominator, output
    const int row = (warp & 3) * 32 + lane;  // this thread's token row and TMEM lane
    const uint32_t t_lane = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    // phi of the rows of tile j in place; returns the denominator, or -1 after a timeout
    auto phi_rows = [&](int j) -> float {
      const int s = j & 1;
      if (!mbar_wait_warp(&sm.q_full[s], (j >> 1) & 1, err, abort_flag)) return -1.f;
      unsigned char* qr = reinterpret_cast<unsigned char*>(sm.q[s]) + row * 128;
      float d = 0.f;
#pragma unroll 2
      for (int jc = 0; jc < 8; ++jc) {  // channels 8 jc .. 8 jc + 7 at chunk jc ^ (row % 8)
        uint4* p = reinterpret_cast<uint4*>(qr + ((jc ^ (row & 7)) << 4));
        const uint4 u = *p;
        const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
        const float4 za = lds_f4_volatile(sm.z + 8 * jc), zb = lds_f4_volatile(sm.z + 8 * jc + 4);
        const float z8[8] = {za.x, za.y, za.z, za.w, zb.x, zb.y, zb.z, zb.w};
        uint32_t o4[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float f0 = elu1(bf16_lo(w4[k])), f1 = elu1(bf16_hi(w4[k]));
          d = fmaf(f0, z8[2 * k], fmaf(f1, z8[2 * k + 1], d));
          o4[k] = pack_bf16x2(f0, f1);
        }
        *p = make_uint4(o4[0], o4[1], o4[2], o4[3]);
      }
      fence_proxy_async_smem();  // the A operand written, before the MMA reads it
      mbar_arrive(&sm.phi_full[s]);
      return d;
    };
    float den_cur = phi_rows(0), den_next = 0.f;
    ok = den_cur != -1.f;
    for (int j = 0; j < n_tiles && ok; ++j) {
      if (j + 1 < n_tiles) {
        den_next = phi_rows(j + 1);
        ok = den_next != -1.f;
        if (!ok) break;
      }
      const int s = j & 1;
      ok = mbar_wait_warp(&sm.d_full[s], (j >> 1) & 1, err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const int tok = (tile0 + j) * kLaRows + row;
      const float inv = 1.f / den_cur;
      uint4* dst = reinterpret_cast<uint4*>(a.y + ((size_t)tok * H + h) * 64);
#pragma unroll
      for (int half = 0; half < 2; ++half) {  // 32 columns at a time
        float d[32];
        tmem_ld32(t_lane + s * 64 + 32 * half, d);
        tmem_wait_ld();
        if (half == 1) {
          tc_fence_before();
          mbar_arrive(&sm.d_empty[s]);
        }
        if (tok < N) {
#pragma unroll
          for (int ch = 0; ch < 4; ++ch)
            dst[4 * half + ch] = make_uint4(pack_bf16x2(d[8 * ch] * inv, d[8 * ch + 1] * inv),
                                            pack_bf16x2(d[8 * ch + 2] * inv, d[8 * ch + 3] * inv),
                                            pack_bf16x2(d[8 * ch + 4] * inv, d[8 * ch + 5] * inv),
                                            pack_bf16x2(d[8 * ch + 6] * inv, d[8 * ch + 7] * inv));
        }
      }
      den_cur = den_next;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && *abort_flag) {  // after a timeout: let issued copies land
    for (int s = 0; s < 2; ++s) {
      if (issued > s) {
        const int last = (issued - 1 - s) / 2 * 2 + s;
        for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.q_full[s], (last >> 1) & 1); ++k) {}
      }
    }
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kLaTmemCols);
  }
}

}  // namespace

cudaError_t launch_linear_apply_tc(const HeadAttnArgs& a, int num_sms, cudaStream_t st) {
  CUtensorMap tmap;  // [N][3 H 64] bf16: boxes of 128 tokens x 64 channels
  cudaError_t e = make_tmap_bf16_2d(&tmap, a.qkv, (uint64_t)3 * a.H * 64, (uint64_t)a.N,
                                    (uint64_t)3 * a.H * 64, 64, kLaRows);
  if (e != cudaSuccess) return e;
  const int smem = (int)sizeof(LaSmem) + 1024;
  e = cudaFuncSetAttribute(linear_apply_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int n_tiles = (a.N + kLaRows - 1) / kLaRows;
  const int n_split = max(1, min(n_tiles, (4 * num_sms + a.H - 1) / a.H));  // four CTAs per SM
  linear_apply_tc_kernel<<<dim3(n_split, a.H), kLaThreads, smem, st>>>(tmap, a, n_split);
  return cudaGetLastError();
}

}  // namespace vp
