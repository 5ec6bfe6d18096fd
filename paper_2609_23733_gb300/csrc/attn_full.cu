// Full-mode heads (Algorithm 1, step 2, s_h >= tau_high): Y_h = softmax(Q_h K_h^T / sqrt d) V_h
// as a flash-attention kernel on the sm_103a tensor cores.
//
// Persistent CTAs (one per SM) walk the work items (full head, group of kChains 128-query
// tiles) read from the device bins.  The query tiles of an item run as independent chains
// c = 0 .. kChains-1 that share the K/V pipeline (kBN keys per tile):
//   warp 0        TMA producer: the item's Q tiles once, K/V tiles through a kStages ring.
//   warp 1        TMEM owner.  Warps 1 .. kChains: one elected lane each issues chain c's
//                 tcgen05.mma: S_c = Q_c K^T (SS form, 128 x kBN fp32 in TMEM) and
//                 O_c += P_c V (TS form: P_c read from TMEM as bf16, V from shared memory,
//                 MN-major).
//   warps 4 ..    four softmax warps per chain: one query row per thread (its TMEM lane).
//                 The thread loads its S row together with its maximum (the load's own
//                 max reduction, tcgen05.ld.red: 6 % faster than a 3-input max tree), computes
//                 2^(s c - m) (packed f32x2 FMA + MUFU ex2), sums with packed adds, and
//                 writes P as bf16 pairs back to TMEM.  The running max is rescaled lazily:
//                 O and the sum are rescaled only when the max grows by more than 2^8;
//                 otherwise the stale max is kept (exact either way).
// S_c(j+1) is issued as soon as chain c has read S_c(j), so the tensor core works on the
// other chains while one chain's softmax runs.  The configuration (VP_ATTN_CHAINS,
// VP_ATTN_BN) is 3 chains of 64-key tiles: every SM sub-partition then holds three softmax
// warps, whose exponentials, maxima and TMEM traffic overlap (measured on GB300: 3 % faster
// than 2 chains of 128-key tiles with 16 heads, 9 % with 2 heads).  Optionally
// (VP_ATTN_MUFU_TURNS) the chains' warps on one sub-partition take turns at the exponentials
// through an mbarrier token; that helps 2 chains, which otherwise fall into step, and hurts 3.
// TMEM: S_c at [c kBN, +kBN), O_c at [kChains kBN + 64 c, +64), P_c after the O columns.
// Keys past N are zero-filled by TMA and masked to -inf; query rows past N are not stored.
// Optionally the epilogue also yields the head's MaxAttn saliency max_ij A_ij (§3).
// Every CTA signals its dependents at once (griddepcontrol.launch_dependents), so the
// cheap-heads kernel queued behind this one (heads_cheap.cu) can take the SMs that the last
// full-attention round leaves idle.
// Every mbarrier wait is bounded (mbar_wait); on timeout the CTA records the error, stops
// issuing work, waits (bounded) for its own outstanding copies and MMAs, frees TMEM, exits.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

#ifndef VP_ATTN_CHAINS
#define VP_ATTN_CHAINS 3
#endif
#ifndef VP_ATTN_BN
#define VP_ATTN_BN 64
#endif
constexpr int kChains = VP_ATTN_CHAINS;  // query tiles (chains) per work item
constexpr int kBM = 128;                 // query rows per tile
constexpr int kBN = VP_ATTN_BN;          // keys per tile
constexpr int kStages = 512 / kBN;       // K/V ring depth: 64 KB of K and 64 KB of V
constexpr int kQTileBytes = kBM * 64 * 2;
constexpr int kKVTileBytes = kBN * 64 * 2;
constexpr uint32_t kTmemCols = 512;
// TMEM: S_c (fp32, kBN columns), O_c (fp32, 64), P_c (bf16 pairs, kBN / 2) for every chain.
constexpr uint32_t kColS = 0, kColO = kChains * kBN, kColP = kColO + kChains * 64;
static_assert(kColP + kChains * kBN / 2 <= kTmemCols, "TMEM columns");
constexpr float kRescaleThreshold = 8.f;  // log2 units
#ifndef VP_ATTN_MUFU_TURNS
#define VP_ATTN_MUFU_TURNS 0
#endif
constexpr bool kMufuTurns = VP_ATTN_MUFU_TURNS != 0;
constexpr int kThreads = 128 + 128 * kChains;
// Register split (setmaxnreg): control warps drop, softmax warps rise, within the launch's
// 65,536 registers: 128 x kCtrlRegs + 128 kChains x kSoftRegs <= 65,536.
constexpr int kCtrlRegs = kChains == 3 ? 56 : 80;
constexpr int kSoftRegs = kChains == 3 ? 152 : 208;
static_assert(128 * kCtrlRegs + 128 * kChains * kSoftRegs <= 65536, "register split");

struct FullSmem {
  __nv_bfloat16 q[kChains][kBM * 64];
  __nv_bfloat16 k[kStages][kBN * 64];
  __nv_bfloat16 v[kStages][kBN * 64];
  uint64_t q_full, q_empty;
  uint64_t k_full[kStages], v_full[kStages], kv_empty[kStages];
  uint64_t s_full[kChains], s_empty[kChains], p_full[kChains], o_bar[kChains], o_empty[kChains];
  uint64_t drain[kChains];
  uint64_t mufu[kChains][4];  // [chain][SM sub-partition]: that warp finished its exponentials
  uint32_t tmem_base;
  int abort_flag;
};

struct FullParams {
  int N, H;
  const int32_t* head_ids;
  const int32_t* offsets;
  __nv_bfloat16* y;
  float* s_attn;  // [H] MaxAttn saliency (zeroed by the launcher), or NULL
  float* part;    // split-tail partial O, (m, l, xmax) and arrival counters (zeroed)
  float* stats;
  unsigned int* count;
  unsigned int* err;
};

// The work of one launch: G groups (head, kChains query tiles) over P persistent CTAs.  The
// first R = floor(G / P) rounds take whole groups; the T = G - R P groups of the last round
// are split along the keys into S parts each (at most the number of key tiles), T S part
// units that the P CTAs take round-robin, so the last round lasts ceil(T S / P) parts of a
// group instead of one whole group on T CTAs.  S minimises ceil(T S / P) (1 / S + c) with c
// the cost of a part beyond its share of the keys (its Q load, pipeline fill and drain, and
// the combine), taken as 3 % of a group (0, 1, 3 and 6 % measured within 1 ms of each
// other on the S = 100 stack, 0 the slowest).  Unit u < R P is group u; unit R P + S t + s is part
// s of group R P + t.
struct Plan {
  int R, T, S, units, whole;  // whole: units that are whole groups (they come first)
};

constexpr int kMaxParts = 64;
constexpr float kPartCost = 0.03f;

__device__ __forceinline__ Plan make_plan(int G, int P, int n_kv) {
  Plan pl;
  pl.R = G / P;
  pl.T = G - pl.R * P;
  pl.S = 1;
  if (pl.T > 0) {
    float best = 1.f;  // S = 1: the T groups whole, one round
    for (int S = 2; S <= kMaxParts && S <= n_kv && pl.T * S <= kFaTailUnits; ++S) {
      const float cost = (float)((pl.T * S + P - 1) / P) * (1.f / (float)S + kPartCost);
      if (cost < best - 1e-6f) {
        best = cost;
        pl.S = S;
      }
    }
  }
  pl.units = pl.S == 1 ? G : pl.R * P + pl.T * pl.S;
  pl.whole = pl.S == 1 ? G : pl.R * P;
  return pl;
}

struct Unit {
  int group;       // head slot * n_groups + query-tile group
  int j0, nk;      // key tiles [j0, j0 + nk)
  int slot;        // split-tail slot (t S + s), -1 for a whole group
  int tail;        // t
};

__device__ __forceinline__ Unit whole_unit(int u, int n_kv) {
  Unit w;
  w.group = u;
  w.j0 = 0;
  w.nk = n_kv;
  w.slot = -1;
  w.tail = -1;
  return w;
}

__device__ __forceinline__ Unit unit_of(const Plan& pl, int u, int P, int n_kv) {
  Unit w;
  if (pl.S == 1 || u < pl.R * P) {
    w.group = u;
    w.j0 = 0;
    w.nk = n_kv;
    w.slot = -1;
    w.tail = -1;
  } else {
    const int v = u - pl.R * P, t = v / pl.S, sp = v - t * pl.S;
    w.group = pl.R * P + t;
    w.j0 = sp * n_kv / pl.S;
    w.nk = (sp + 1) * n_kv / pl.S - w.j0;
    w.slot = v;
    w.tail = t;
  }
  return w;
}

// Split-tail epilogue of one warp (32 rows of chain c, TMEM lanes at t_o): reads the part's
// unnormalised O rows, releases O_c (o_empty), and publishes them with (m, l, xmax); the last
// part of this (group, chain, lane quarter) to arrive combines all parts, M = max m_s,
// O = sum 2^(m_s - M) O_s, l = sum 2^(m_s - M) l_s, and stores Y and the saliency.  Not
// inlined, and given only values: the attention loop's code and registers stay as they are
// without it.
__device__ __noinline__ void split_part(FullParams prm, Plan plan, Unit w, int c, int quarter,
                                        int lane, int row_in_tile, int row, int h, uint32_t t_o,
                                        uint64_t* o_empty, float m, float lsum, float xmax) {
  float o[64];
  tmem_ld32(t_o, o);
  tmem_ld32(t_o + 32, o + 32);
  tmem_wait_ld();
  tc_fence_before();
  mbar_arrive(o_empty);
  const size_t prow = (size_t)(w.slot * 4 + c) * kBM + row_in_tile;
  float4* po = reinterpret_cast<float4*>(prm.part + prow * 64);
#pragma unroll
  for (int q = 0; q < 16; ++q) po[q] = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
  reinterpret_cast<float4*>(prm.stats)[prow] = make_float4(m, lsum, xmax, 0.f);
  __threadfence();
  __syncwarp();
  unsigned int last = 0;
  if (lane == 0)
    last = atomicAdd(prm.count + (w.tail * 4 + c) * 4 + quarter, 1u) == (unsigned)(plan.S - 1);
  if (!__shfl_sync(0xffffffffu, last, 0)) return;
  __threadfence();
  const int slot0 = w.tail * plan.S;
  float M = -INFINITY, X = -INFINITY;
  for (int sp = 0; sp < plan.S; ++sp) {
    const float4 st4 = __ldcg(reinterpret_cast<const float4*>(prm.stats) +
                              (size_t)((slot0 + sp) * 4 + c) * kBM + row_in_tile);
    M = fmaxf(M, st4.x);
    X = fmaxf(X, st4.z);
  }
  float L = 0.f;
#pragma unroll
  for (int i = 0; i < 64; ++i) o[i] = 0.f;
  for (int sp = 0; sp < plan.S; ++sp) {
    const size_t qrow = (size_t)((slot0 + sp) * 4 + c) * kBM + row_in_tile;
    const float4 st4 = __ldcg(reinterpret_cast<const float4*>(prm.stats) + qrow);
    const float wgt = fast_exp2(st4.x - M);
    L = fmaf(wgt, st4.y, L);
    const float4* pq = reinterpret_cast<const float4*>(prm.part + qrow * 64);
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const float4 f = __ldcg(pq + q);
      o[4 * q] = fmaf(wgt, f.x, o[4 * q]);
      o[4 * q + 1] = fmaf(wgt, f.y, o[4 * q + 1]);
      o[4 * q + 2] = fmaf(wgt, f.z, o[4 * q + 2]);
      o[4 * q + 3] = fmaf(wgt, f.w, o[4 * q + 3]);
    }
  }
  const float inv = 1.f / L;
  if (row < prm.N) {
    uint4* dst = reinterpret_cast<uint4*>(prm.y + ((size_t)row * prm.H + h) * 64);
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
  if (prm.s_attn) {
    float a = row < prm.N ? fast_exp2(X - M) * inv : 0.f;
#pragma unroll
    for (int k = 16; k > 0; k >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, k));
    if (lane == 0) atomicMax(reinterpret_cast<int*>(prm.s_attn + h), __float_as_int(a));
  }
}

// kParts = false: the whole groups (all of them when nothing is split); kParts = true: the
// split parts, one per CTA, launched right behind (programmatic dependent launch) so that
// they take the SMs the whole groups leave.  Two instantiations keep runtime key ranges out
// of the main one's attention loop, which they would slow down by about a tenth.
template <bool kParts>
__global__ void __launch_bounds__(kThreads, 1)
    attn_full_kernel(const __grid_constant__ CUtensorMap tmap_q,
                     const __grid_constant__ CUtensorMap tmap_kv, FullParams prm) {
  extern __shared__ unsigned char smem_raw[];
  FullSmem& sm = *reinterpret_cast<FullSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);

  const int first = __ldg(prm.offsets + 2);
  const int n_heads = __ldg(prm.offsets + 3) - first;
  const int N = prm.N, H = prm.H;
  const int n_groups = (N + kChains * kBM - 1) / (kChains * kBM);  // query-tile groups per head
  const int n_kv = (N + kBN - 1) / kBN;
  const int P = gridDim.x;
  const Plan plan = make_plan(n_heads * n_groups, P, n_kv);
  // Units of this CTA: [u_begin, u_end) in steps of P.
  const int u_begin = kParts ? plan.whole + (int)blockIdx.x : (int)blockIdx.x;
  const int u_end = kParts ? plan.units : plan.whole;
  if (u_begin >= u_end) {  // uniform across the CTA
    // The parts grid completes only after the whole-group grid (its prerequisite): work
    // queued behind it then sees every row of Y.
    if (kParts && blockIdx.x == 0) {
      asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
      asm volatile("griddepcontrol.wait;" ::: "memory");
    }
    return;
  }

  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    mbar_init(&sm.q_empty, kChains);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.v_full[s], 1);
      mbar_init(&sm.kv_empty[s], kChains);
    }
    for (int c = 0; c < kChains; ++c) {
      mbar_init(&sm.s_full[c], 1);
      mbar_init(&sm.s_empty[c], 128);
      mbar_init(&sm.p_full[c], 128);
      mbar_init(&sm.o_bar[c], 1);
      mbar_init(&sm.o_empty[c], 128);
      mbar_init(&sm.drain[c], 1);
      for (int q = 0; q < 4; ++q) mbar_init(&sm.mufu[c][q], 1);
    }
    sm.abort_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&tmap_q);
    tma_prefetch_desc(&tmap_kv);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);

  if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kCtrlRegs));
  }
  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    // The whole warp walks the loop (so that coordinates and addresses stay warp-uniform);
    // one elected lane issues the copies.
    uint32_t lc = 0, ic = 0;
    bool ok = true;
    for (int u = u_begin; u < u_end && ok; u += P, ++ic) {
      const Unit w = kParts ? unit_of(plan, u, P, n_kv) : whole_unit(u, n_kv);
      const int h = __shfl_sync(0xffffffffu, __ldg(prm.head_ids + first + w.group / n_groups), 0);
      const int qg = w.group % n_groups;
      ok = mbar_wait_warp(&sm.q_empty, (ic & 1) ^ 1, prm.err, abort_flag);
      if (!ok) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&sm.q_full, kChains * kQTileBytes);
#pragma unroll
        for (int c = 0; c < kChains; ++c)
          tma_load_2d(sm.q[c], &tmap_q, &sm.q_full, h * 64, (qg * kChains + c) * kBM);
      }
      __syncwarp();
      for (int jj = 0; jj < w.nk; ++jj, ++lc) {
        const int j = w.j0 + jj, st = lc % kStages;
        ok = mbar_wait_warp(&sm.kv_empty[st], ((lc / kStages) & 1) ^ 1, prm.err, abort_flag);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(&sm.k_full[st], kKVTileBytes);
          tma_load_2d(sm.k[st], &tmap_kv, &sm.k_full[st], (H + h) * 64, j * kBN);
          mbar_arrive_expect_tx(&sm.v_full[st], kKVTileBytes);
          tma_load_2d(sm.v[st], &tmap_kv, &sm.v_full[st], (2 * H + h) * 64, j * kBN);
        }
        __syncwarp();
      }
    }
    if (!ok && lane == 0) {
      // Let the copies this warp issued land before the CTA releases its smem.
      // ic counts items whose Q load was issued when the loop broke inside the K/V loop,
      // and items + 1 when it broke at the Q wait; waiting on the last issued phase is
      // bounded either way.
      if (ic > 0)
        for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.q_full, (ic - 1) & 1); ++t) {}
      for (int s = 0; s < kStages; ++s) {
        if (lc > (uint32_t)s) {
          const uint32_t last = (lc - 1 - s) / kStages * kStages + s;  // last use of stage s
          const uint32_t par = (last / kStages) & 1;
          for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.k_full[s], par); ++t) {}
          for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.v_full[s], par); ++t) {}
        }
      }
    }
  } else if (warp <= kChains) {
    // ------------------------------------------------------------ MMA issuers (chain c)
    // Converged warp; the elected lane (the same lane every time: elect.sync picks the
    // lowest active lane) issues the MMAs and the commits that track them.
    const int c = warp - 1;
    const uint32_t id_s = idesc_bf16(kBM, kBN, 0, 0);  // Q (K-major) x K^T (K-major)
    const uint32_t id_o = idesc_bf16(kBM, 64, 0, 1);   // P (TMEM) x V (MN-major)
    const uint64_t dq = sdesc_sw128(smem_u32(sm.q[c]));
    const uint32_t t_s = tmem + kColS + c * kBN;
    const uint32_t t_o = tmem + kColO + c * 64;
    const uint32_t t_p = tmem + kColP + c * (kBN / 2);
    uint32_t lc = 0, ic = 0, g = 0;  // K/V tiles seen, units, S/P/O tiles of this chain
    bool ok = true;
    const int n_kv_all = n_kv;
    for (int u = u_begin; u < u_end && ok; u += P, ++ic) {
      const int n_kv = kParts ? unit_of(plan, u, P, n_kv_all).nk : n_kv_all;  // tiles of this unit
      ok = mbar_wait_warp(&sm.q_full, ic & 1, prm.err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint32_t lc0 = lc, g0 = g;
      auto issue_s = [&](int j) -> bool {
        const uint32_t l = lc0 + j, gg = g0 + j;
        const int st = l % kStages;
        if constexpr (kParts) {  // K landed (lanes 0-15 poll) and S_c read (lanes 16-31), at once
          const bool hi = lane_id() >= 16;
          if (!__all_sync(0xffffffffu, mbar_wait(hi ? &sm.s_empty[c] : &sm.k_full[st],
                                                 hi ? ((gg & 1) ^ 1) : ((l / kStages) & 1),
                                                 prm.err, abort_flag)))
            return false;
        } else {
          if (!mbar_wait_warp(&sm.k_full[st], (l / kStages) & 1, prm.err, abort_flag)) return false;
          if (!mbar_wait_warp(&sm.s_empty[c], (gg & 1) ^ 1, prm.err, abort_flag)) return false;
        }
        tc_fence_after();
        const uint64_t dk = sdesc_sw128(smem_u32(sm.k[st]));
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // 4 x K=16 covers d = 64 (+32 bytes per step)
            tc_mma_ss(t_s, dq + 2 * kk, dk + 2 * kk, id_s, kk > 0);
          tc_commit(&sm.s_full[c]);
          if (j == n_kv - 1) tc_commit(&sm.q_empty);
        }
        __syncwarp();
        return true;
      };
      ok = issue_s(0);
      for (int j = 0; j < n_kv && ok; ++j) {
        if (j + 1 < n_kv) {
          ok = issue_s(j + 1);  // as soon as the softmax has read S_c(j)
          if (!ok) break;
        }
        const uint32_t l = lc0 + j, gg = g0 + j;
        const int st = l % kStages;
        // P_c written, V landed and, on a unit's first tile, O_c free.  The split parts (short
        // units) poll the three at once in lane groups (0-10, 11-21, 22-31), so that the round
        // trips overlap; the whole-group instance waits one after another, which measured
        // 2.6 % faster there (the same parallel polls in both: stack unchanged, all-full layer
        // slower).
        if constexpr (kParts) {
          const int grp = lane_id() / 11;
          uint64_t* bar = grp == 0 ? &sm.p_full[c]
                        : grp == 1 ? &sm.v_full[st]
                                   : (j == 0 ? &sm.o_empty[c] : &sm.p_full[c]);
          const uint32_t par = grp == 0 ? (gg & 1)
                             : grp == 1 ? ((l / kStages) & 1)
                                        : (j == 0 ? ((ic & 1) ^ 1) : (gg & 1));
          ok = __all_sync(0xffffffffu, mbar_wait(bar, par, prm.err, abort_flag));
        } else {
          ok = mbar_wait_warp(&sm.p_full[c], gg & 1, prm.err, abort_flag) &&
               mbar_wait_warp(&sm.v_full[st], (l / kStages) & 1, prm.err, abort_flag) &&
               (j > 0 || mbar_wait_warp(&sm.o_empty[c], (ic & 1) ^ 1, prm.err, abort_flag));
        }
        if (!ok) break;
        tc_fence_after();
        const uint64_t dv = sdesc_sw128(smem_u32(sm.v[st]));
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk)  // K=16 keys per step: 8 TMEM columns, 2 KB of V
            tc_mma_ts(t_o, t_p + 8 * kk, dv + (uint64_t)(kk * 128), id_o,
                      (j > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&sm.o_bar[c]);
          tc_commit(&sm.kv_empty[st]);
        }
        __syncwarp();
      }
      lc = lc0 + n_kv;
      g = g0 + n_kv;
    }
    if (!ok) {
      if (elect_one()) {
        tc_commit(&sm.drain[c]);
        for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.drain[c], 0); ++t) {}
      }
      __syncwarp();
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ softmax / epilogue
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kSoftRegs));
    const int c = (warp - 4) >> 2;  // chain
    const int quarter = warp & 3;   // TMEM lane quarter this warp may access
    const int row_in_tile = quarter * 32 + lane;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t t_s = tmem + lane_off + kColS + c * kBN;
    const uint32_t t_o = tmem + lane_off + kColO + c * 64;
    const uint32_t t_p = tmem + lane_off + kColP + c * (kBN / 2);
    const float cs = 1.4426950408889634f * 0.125f;  // log2(e) / sqrt(64)
    const int n_tail = N - (n_kv - 1) * kBN;        // valid keys in the last tile
    uint32_t g = 0;
    bool ok = true;
    for (int u = u_begin; u < u_end && ok; u += P) {
      const Unit w = kParts ? unit_of(plan, u, P, n_kv) : whole_unit(u, n_kv);
      const int h = __ldg(prm.head_ids + first + w.group / n_groups);
      const int qg = w.group % n_groups;
      // m: the (lazily updated) reference the exponentials are taken against; xmax: the
      // true running maximum of the row's scaled scores, for the MaxAttn saliency.
      float m = 0.f, lsum = 0.f, xmax = 0.f;
      for (int jj = 0; jj < w.nk; ++jj, ++g) {
        const int j = w.j0 + jj;  // key tile
        ok = mbar_wait_warp(&sm.s_full[c], g & 1, prm.err, abort_flag);
        if (!ok) break;
        tc_fence_after();
        // The S row with the maximum of every 32 columns from the load itself (tcgen05.ld.red).
        float s[kBN], pmx[kBN / 32];
#pragma unroll
        for (int cc = 0; cc < kBN / 32; ++cc) tmem_ld32_max(t_s + 32 * cc, s + 32 * cc, pmx[cc]);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(&sm.s_empty[c]);  // the MMA warp may overwrite S_c now
        const bool tail = j == n_kv - 1 && n_tail < kBN;
        if (tail) {
#pragma unroll
          for (int i = 0; i < kBN; ++i)
            if (i >= n_tail) s[i] = -INFINITY;
        }
        float mx = pmx[0];
#pragma unroll
        for (int cc = 1; cc < kBN / 32; ++cc) mx = fmaxf(mx, pmx[cc]);
        // On the last, partial key tile the loads' maxima also saw the masked columns: the row
        // max there by eight independent 3-input max chains, then a short tree.
        if (tail) {
          // Chain k covers s[k + 8 i], i = 0..15: one 2-input max, then seven 3-input ones.
          float t[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) t[k] = fmaxf(s[k], s[8 + k]);
#pragma unroll
          for (int i = 16; i < kBN; i += 16) {
#pragma unroll
            for (int k = 0; k < 8; ++k) t[k] = fmax3(t[k], s[i + k], s[i + 8 + k]);
          }
          mx = fmaxf(fmax3(t[0], t[1], t[2]), fmax3(t[3], t[4], fmax3(t[5], t[6], t[7])));
        }
        const float mx2 = mx * cs;
        xmax = jj == 0 ? mx2 : fmaxf(xmax, mx2);
        float alpha = 1.f;
        bool need = false;
        if (jj == 0) {
          m = mx2;
        } else if (mx2 > m + kRescaleThreshold) {
          need = true;
          alpha = fast_exp2(m - mx2);
          m = mx2;
        }
        // Optional turns at the exponentials (MUFU) for the chains' warps on this SM
        // sub-partition, in chain order: chain c > 0 waits for chain c - 1's tile g, chain 0
        // for the last chain's tile g - 1.
        if (kMufuTurns && (c > 0 || g > 0)) {
          ok = mbar_wait_warp(&sm.mufu[c > 0 ? c - 1 : kChains - 1][quarter],
                              c > 0 ? (g & 1) : ((g - 1) & 1), prm.err, abort_flag);
          if (!ok) break;
        }
        // p = 2^(s cs - m), summed in packed pairs and packed to bf16 pairs for P (before the
        // wait for P_c(g-1) V below, so that only the TMEM stores follow it).
        const float2 c2 = make_float2(cs, cs), nm = make_float2(-m, -m);
        float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
        uint32_t pk[kBN / 2];
#pragma unroll
        for (int i = 0; i < kBN / 2; ++i) {
          float2 x = ffma2(make_float2(s[2 * i], s[2 * i + 1]), c2, nm);
          x.x = fast_exp2(x.x);
          x.y = fast_exp2(x.y);
          pk[i] = pack_bf16x2(x.x, x.y);
          if (i & 1)
            acc1 = fadd2(acc1, x);
          else
            acc0 = fadd2(acc0, x);
        }
        if (kMufuTurns) {
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.mufu[c][quarter]);
        }
        const float2 at = fadd2(acc0, acc1);
        lsum = lsum * alpha + (at.x + at.y);
        // P_c and O_c are free once P_c(g-1) V has completed.
        if (g > 0) {
          ok = mbar_wait_warp(&sm.o_bar[c], (g - 1) & 1, prm.err, abort_flag);
          if (!ok) break;
          tc_fence_after();
        }
#pragma unroll
        for (int cc = 0; cc < kBN / 32; ++cc) tmem_st16(t_p + 16 * cc, pk + 16 * cc);
        if (__any_sync(0xffffffffu, need)) {
          float o[64];
          tmem_ld32(t_o, o);
          tmem_ld32(t_o + 32, o + 32);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 64; ++i) o[i] *= alpha;
          tmem_st32(t_o, o);
          tmem_st32(t_o + 32, o + 32);
        }
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&sm.p_full[c]);
      }
      if (!ok) break;
      // Epilogue: O / sum -> bf16 -> Y[row][h][:]
      ok = mbar_wait_warp(&sm.o_bar[c], (g - 1) & 1, prm.err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const int row = (qg * kChains + c) * kBM + row_in_tile;
      if (kParts) {  // a part of a split group (the last round's groups)
        split_part(prm, plan, w, c, quarter, lane, row_in_tile, row, h, t_o, &sm.o_empty[c], m,
                   lsum, xmax);
        __syncwarp();
        continue;
      }
      float o[64];
      tmem_ld32(t_o, o);
      tmem_ld32(t_o + 32, o + 32);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&sm.o_empty[c]);
      const float inv = 1.f / lsum;
      if (row < N) {
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
      if (prm.s_attn) {
        // MaxAttn saliency (§3): the largest entry of row i of A is 2^(xmax - m) / lsum (the
        // row's maximum over its softmax denominator); the head's value is the maximum over
        // rows, folded in with an integer atomic max (the values are positive floats).
        float a = row < N ? fast_exp2(xmax - m) * inv : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
        if (lane == 0) atomicMax(reinterpret_cast<int*>(prm.s_attn + h), __float_as_int(a));
      }
      __syncwarp();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (kParts && blockIdx.x == 0 && threadIdx.x == 0) asm volatile("griddepcontrol.wait;" ::: "memory");
}

}  // namespace

cudaError_t launch_full_heads(const HeadAttnArgs& a, int num_sms, cudaStream_t st) {
  CUtensorMap tmap_q, tmap_kv;  // boxes of 128 query rows / kBN key rows, 64 channels
  cudaError_t e = make_tmap_bf16_2d(&tmap_q, a.qkv, (uint64_t)3 * a.H * 64, (uint64_t)a.N,
                                    (uint64_t)3 * a.H * 64, 64, kBM);
  if (e != cudaSuccess) return e;
  e = make_tmap_bf16_2d(&tmap_kv, a.qkv, (uint64_t)3 * a.H * 64, (uint64_t)a.N,
                        (uint64_t)3 * a.H * 64, 64, kBN);
  if (e != cudaSuccess) return e;
  const int smem = (int)sizeof(FullSmem) + 1024;
  e = cudaFuncSetAttribute(attn_full_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(attn_full_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  FullParams prm{a.N, a.H, a.head_ids, a.offsets, a.y, a.s_attn, a.fa_part, a.fa_stats,
                 a.fa_count, a.err};
  attn_full_kernel<false><<<num_sms, kThreads, smem, st>>>(tmap_q, tmap_kv, prm);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // The split parts of the last round (if the bins give one), on the SMs the whole groups free.
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(num_sms);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, attn_full_kernel<true>, tmap_q, tmap_kv, prm);
  prof_extra_launch();
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace vp
