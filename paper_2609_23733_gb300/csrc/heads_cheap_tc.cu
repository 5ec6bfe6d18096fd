// Surrogate heads (§4.3) and mean heads (Algorithm 1, step 2, s_h <= tau_low) of a layer on
// the sm_103a tensor cores, queued behind the full-attention kernel with programmatic
// dependent launch (its CTAs take the SMs that full attention's last round frees).
//
// Surrogate head h, per token i:  z_i = [v_i, C_h],
//   y_i = C_h + sigma(MLP_gamma(z_i)) (.) MLP_delta(z_i),  MLP = Linear(2d -> 64) -> GELU ->
//   Linear(64 -> d).
// The first layer splits as W1 z = W1[:, :d] v_i + (W1[:, d:] C_h + b1): the second term (c1)
// is one vector per head.  Per 128-token tile, with both MLPs side by side:
//   D1 = V W1v^T      [128 x 128] = tcgen05.mma M128 N128 K16 x 4 (V and [W1v_gamma; W1v_delta]
//                     from shared memory, 128-byte swizzle), fp32 in TMEM;
//   H = 2 GELU(D1 + c1) as bf16 pairs in 64 TMEM columns of their own (x2 exact in bf16);
//   D2g = H[:, :64] W2g^T, D2d = H[:, 64:] W2d^T  [128 x 64] each = tcgen05.mma M128 N64 K16
//                     x 4 each, A read from TMEM (TS form), W2 from shared memory, into D1's
//                     columns (D1 has been read by then);
//   y = C + sigma(D2g + b2g) (.) (D2d + b2d), bf16, staged in shared memory (128-byte swizzle)
//                     and written by a TMA tensor store into Y[:, h, :].
// A mean item writes Broadcast(mean of V_h) over 1,024 tokens with coalesced 16-byte stores.
//
// Roles (576 threads, one CTA per SM, persistent over items taken kBatch at a time from a
// device counter: surrogate tiles of 128 tokens head-major, then mean items of 1,024 tokens):
//   all        at the start, every surrogate head's per-head vectors into shared memory
//              (c1 = W1[:, d:] C_h + b1, the second layer's biases, C_h);
//   warp 0     producer: items, TMA loads of the V tiles (kStages ring) and of each head's
//              weights into one of two weight slots (a slot is reloaded once the MMAs of the
//              head before the previous one have completed);
//   warp 1     TMEM owner (512 columns) and MMA issue: the first layer of the next tile and
//              the second layer of a tile whose H is written, each as soon as it is ready;
//   warps 2-9, 10-17  two epilogue groups of eight warps, each with 256 TMEM columns; group
//              g takes tiles t = g (mod 2).  Its j-th tile keeps D1, then D2g | D2d, in the
//              128-column half j & 1 and H in the first 64 columns of the other half, so the
//              first layer of its next tile (the other half) runs while it reads D2.  The
//              two warps of a TMEM lane quarter split a token row's columns (kTcParts).
// The register file is split between the four SM sub-partitions: 18 warps put 5 on some of
// them, which caps a thread at 96 registers (16,384 / (5 x 32), in steps of 8).  Three warps
// per lane quarter (26 warps, 72 registers) measured slower: 0.301 vs 0.269 ms for 16 heads
// at 137,400 tokens.
// Every wait is bounded (mbar_wait); on timeout the CTA records VP_DEVERR_WAIT_TIMEOUT, stops,
// waits (bounded) for its own copies and MMAs, frees TMEM and exits.  The groups agree on
// stopping through reduction barriers, so that no thread is left at a named barrier.
#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

constexpr int kTcTile = 128;      // tokens per surrogate item
constexpr int kMeanRows = 1024;   // tokens per mean item (a pure write, handed over less often)
constexpr int kTcStages = 4;      // V tiles in flight
constexpr int kTcGroups = 2;      // epilogue groups (= TMEM accumulators)
constexpr int kTcBatch = 4;       // items taken from the counter at a time
constexpr int kTcParts = 2;       // epilogue warps per TMEM lane quarter in a group
constexpr int kGroupThreads = 128 * kTcParts;
constexpr int kTcThreads = 64 + kGroupThreads * kTcGroups;
// A row's work split over the kTcParts warps of its lane quarter: part p takes the chunk
// range [begin(p), begin(p + 1)) of the n chunks, as even as possible.  The first layer's
// 8 chunks go in part order and the second layer's 4 in reverse, so that a part short of
// first-layer chunks takes more second-layer ones.
__host__ __device__ constexpr int part_begin(int p, int n) { return (p * n + kTcParts - 1) / kTcParts; }
constexpr int kMaxGChunks = (8 + kTcParts - 1) / kTcParts;
constexpr int kMaxFChunks = (4 + kTcParts - 1) / kTcParts;
constexpr uint32_t kTcTmemCols = 512;
constexpr uint32_t kVTileBytes = kTcTile * 64 * 2;
constexpr uint32_t kW1Bytes = 128 * 64 * 2;  // [W1v_gamma; W1v_delta]: 128 hidden x 64 inputs
constexpr uint32_t kW2Bytes = 128 * 64 * 2;  // [W2_gamma; W2_delta]: 2 x (64 outputs x 64 hidden)

struct TcSmem {
  __nv_bfloat16 v[kTcStages][kTcTile * 64];
  __nv_bfloat16 w1[2][128 * 64];
  __nv_bfloat16 w2[2][128 * 64];
  __nv_bfloat16 ys[kTcGroups][kTcTile * 64];  // output staging, 128-byte swizzle
  // Every surrogate head's vectors, by slot in the surrogate bin, computed at kernel start:
  // W1[:, d:] C_h + b1 (gamma | delta), -log2(e) b2_gamma | b2_delta, and C_h.
  float c1[kMaxHeads][128];
  float b2[kMaxHeads][128];
  float cx[kMaxHeads][64];
  int stage_item[kTcStages];                  // item, or -1: no more items
  int stage_fill[kTcStages];                  // weight fill of a surrogate item (slot = fill & 1), -1
  int stage_head[kTcStages];
  int acc_item[kTcGroups], acc_head[kTcGroups];
  uint64_t full[kTcStages], empty[kTcStages];
  uint64_t w_full[2], w_empty[2];
  uint64_t d1_full[kTcGroups], h_full[kTcGroups], d2_full[kTcGroups], taken[kTcGroups];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
};

// Barrier over the threads of an epilogue group (named barrier 1 + g) that also returns
// whether p held on every one of them.
__device__ __forceinline__ bool group_all(bool p, int g) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.and.pred po, %2, %3, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)p), "r"(1 + g), "n"(kGroupThreads)
      : "memory");
  return r != 0;
}

struct TcMaps {
  CUtensorMap v, y, g1, d1, g2, d2;
};

__global__ void __launch_bounds__(kTcThreads, 1) cheap_heads_tc_kernel(const __grid_constant__ TcMaps maps, HeadAttnArgs a) {
  extern __shared__ unsigned char smem_raw[];
  TcSmem& sm = *reinterpret_cast<TcSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int tid = threadIdx.x;
  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  unsigned int* err = a.err;
  const int H = a.H;
  const int m_first = __ldg(a.offsets + 0), s_first = __ldg(a.offsets + 1);
  const int n_surr = __ldg(a.offsets + 2) - s_first, n_mean = s_first - m_first;
  const int T = (a.N + kTcTile - 1) / kTcTile;
  const int surr_items = n_surr * T;
  const int Tm = (a.N + kMeanRows - 1) / kMeanRows;  // mean items per head
  // Mean heads folded into W_O's bias (skip_mean_y) need no rows of Y.
  const int items = surr_items + (a.skip_mean_y ? 0 : n_mean * Tm);

  if (tid == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.w_full[s], 1);
      mbar_init(&sm.w_empty[s], 1);
    }
    for (int g = 0; g < kTcGroups; ++g) {
      mbar_init(&sm.d1_full[g], 2);  // the MMA commit (or a stand-in) + the item hand-over
      mbar_init(&sm.h_full[g], kGroupThreads);
      mbar_init(&sm.d2_full[g], 1);
      mbar_init(&sm.taken[g], 1);      // the group has read a tile's item and left its last one
    }
    mbar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&maps.v);
    tma_prefetch_desc(&maps.y);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTcTmemCols);
    tmem_relinquish();
  }
  // The surrogate heads' per-head vectors: the first layer's context half folded into c1 (one
  // 64-term dot product per hidden unit), the second layer's biases, C_h.
  for (int i = tid; i < n_surr * 128; i += kTcThreads) {
    const int slot = i >> 7, u = i & 127, uu = u & 63;
    const int h = __ldg(a.head_ids + s_first + slot);
    const float4* ctx = reinterpret_cast<const float4*>(a.ctx + h * 64);
    const __nv_bfloat16* w = (u < 64 ? a.sw.g1_w : a.sw.d1_w) + ((size_t)h * 64 + uu) * 128 + 64;
    float acc = __ldg((u < 64 ? a.sw.g1_b : a.sw.d1_b) + h * 64 + uu);
#pragma unroll
    for (int kq = 0; kq < 8; ++kq) {
      const uint4 wv = __ldg(reinterpret_cast<const uint4*>(w) + kq);
      const float4 c0 = __ldg(ctx + 2 * kq), c1 = __ldg(ctx + 2 * kq + 1);
      acc = fmaf(bf16_lo(wv.x), c0.x, fmaf(bf16_hi(wv.x), c0.y, acc));
      acc = fmaf(bf16_lo(wv.y), c0.z, fmaf(bf16_hi(wv.y), c0.w, acc));
      acc = fmaf(bf16_lo(wv.z), c1.x, fmaf(bf16_hi(wv.z), c1.y, acc));
      acc = fmaf(bf16_lo(wv.w), c1.z, fmaf(bf16_hi(wv.w), c1.w, acc));
    }
    sm.c1[slot][u] = acc;
    const float b = __ldg((u < 64 ? a.sw.g2_b : a.sw.d2_b) + h * 64 + uu);
    sm.b2[slot][u] = u < 64 ? -1.4426950408889634f * b : b;  // gamma's enters sigma's exponent
    if (u < 64) sm.cx[slot][u] = __ldg(a.ctx + h * 64 + u);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    int fill = -1, cur_h = -1, next = 0, left = 0;
    int tma_k[kTcStages];  // last item index k whose V tile went to stage s (-1: none)
#pragma unroll
    for (int s = 0; s < kTcStages; ++s) tma_k[s] = -1;
    bool ok = true;
    for (int k = 0;; ++k) {
      if (left == 0) {
        int b = 0;
        if (lane == 0) b = (int)atomicAdd(a.cheap_counter, (unsigned)kTcBatch);
        next = __shfl_sync(0xffffffffu, b, 0);
        left = kTcBatch;
      }
      const int it = next++;
      --left;
      const int st = k % kTcStages;
      ok = mbar_wait_warp(&sm.empty[st], ((k / kTcStages) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      if (it >= items) {
        if (elect_one()) {
          sm.stage_item[st] = -1;
          mbar_arrive(&sm.full[st]);
        }
        __syncwarp();
        break;
      }
      if (it < surr_items) {
        const int slot = it / T, tile = it - slot * T;
        const int h = __ldg(a.head_ids + s_first + slot);
        if (h != cur_h) {  // this head's weights into the next slot
          ++fill;
          cur_h = h;
          const int ws = fill & 1;
          if (fill >= 2) {  // the MMAs of fill - 2 (same slot) have completed
            ok = mbar_wait_warp(&sm.w_empty[ws], ((fill - 2) >> 1) & 1, err, abort_flag);
            if (!ok) break;
          }
          if (elect_one()) {
            mbar_arrive_expect_tx(&sm.w_full[ws], kW1Bytes + kW2Bytes);
            tma_load_2d(sm.w1[ws], &maps.g1, &sm.w_full[ws], 0, h * 64);
            tma_load_2d(sm.w1[ws] + 64 * 64, &maps.d1, &sm.w_full[ws], 0, h * 64);
            tma_load_2d(sm.w2[ws], &maps.g2, &sm.w_full[ws], 0, h * 64);
            tma_load_2d(sm.w2[ws] + 64 * 64, &maps.d2, &sm.w_full[ws], 0, h * 64);
          }
          __syncwarp();
        }
        if (elect_one()) {
          sm.stage_item[st] = it;
          sm.stage_fill[st] = fill;
          sm.stage_head[st] = h;
          mbar_arrive_expect_tx(&sm.full[st], kVTileBytes);
          tma_load_2d(sm.v[st], &maps.v, &sm.full[st], (2 * H + h) * 64, tile * kTcTile);
        }
        __syncwarp();
        tma_k[st] = k;
      } else {
        const int slot = (it - surr_items) / Tm;
        const int h = __ldg(a.head_ids + m_first + slot);
        if (elect_one()) {
          sm.stage_item[st] = it;
          sm.stage_fill[st] = -1;
          sm.stage_head[st] = h;
          mbar_arrive(&sm.full[st]);
        }
        __syncwarp();
      }
    }
    if (!ok && lane == 0) {  // let issued copies land before the CTA releases its smem
      for (int s = 0; s < kTcStages; ++s)
        if (tma_k[s] >= 0)
          for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.full[s], (tma_k[s] / kTcStages) & 1); ++t) {}
      for (int f = fill; f >= 0 && f >= fill - 1; --f)
        for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.w_full[f & 1], (f >> 1) & 1); ++t) {}
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    // A polling loop over two independent kinds of work, issued as soon as each is ready:
    // the first layer of the next tile (its V tile loaded, its accumulator free, its weights
    // loaded) and the second layer of the oldest tile whose H is written.  Tying them to one
    // order would make a group's second layer wait for the other group's epilogue.
    const uint32_t id1 = idesc_bf16(128, 128, 0, 0);  // V (K-major) x W1v^T (K-major)
    const uint32_t id2 = idesc_bf16(128, 64, 0, 0);   // H (TMEM) x W2^T (K-major)
    bool ok = true;
    int k = 0;                        // next tile for the first layer
    bool feeding = true;              // false once the stop item has been read
    int waited_fill = -1;             // newest weight fill known to be loaded
    int cur_fill = -1;                // fill of the newest surrogate tile
    int release = -1;                 // a finished fill whose slot is released once its
                                      // tiles' second layers are issued
    int qk[2], qfill[2];              // tiles waiting for their second layer (oldest first)
    uint32_t qsur[2];
    int qn = 0;
    uint32_t sur_cnt[kTcGroups] = {0u, 0u};  // surrogate tiles sent to group g
    int last_kind[kTcGroups] = {-1, -1};        // kind of group g's last tile (1 surrogate, 0 mean)
    int last_sur[kTcGroups] = {0, 0};           // its index among the group's surrogate tiles
    // Tile kk may go to its group once the group's previous tile no longer needs what tile kk
    // overwrites: its second layer has completed (its H lies in the half that tile kk's first
    // layer writes, and its item was read before), or, for a mean tile, the group has started
    // it (so it has finished the tile before, whose results lie in that half).
    auto group_free = [&](int kk) -> bool {
      const int gb = kk & 1, jj = kk >> 1;
      if (jj == 0) return true;
      if (last_kind[gb] == 1) return mbar_test_wait(&sm.d2_full[gb], (uint32_t)last_sur[gb] & 1);
      return mbar_test_wait(&sm.taken[gb], (uint32_t)(jj - 1) & 1);
    };
    unsigned long long t0 = 0;
    for (uint32_t spin = 1;; ++spin) {
      bool progress = false;
      if (qn > 0) {  // second layer of the oldest waiting tile
        const int pb = qk[0] & 1;
        const bool ready = __shfl_sync(0xffffffffu, (int)mbar_test_wait(&sm.h_full[pb], qsur[0] & 1), 0);
        if (ready) {
          tc_fence_after();
          // Local tile j of group pb: D2 into the main half (j & 1), H read from the other one.
          const uint32_t t_main = tmem + pb * 256 + ((qk[0] >> 1) & 1) * 128;
          const uint32_t t_h = tmem + pb * 256 + (((qk[0] >> 1) & 1) ^ 1) * 128;
          const uint64_t dg = sdesc_sw128(smem_u32(sm.w2[qfill[0] & 1]));
          const uint64_t dd = sdesc_sw128(smem_u32(sm.w2[qfill[0] & 1] + 64 * 64));
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)  // gamma: hidden units 0..63 = H columns 0..31
              tc_mma_ts(t_main, t_h + 8 * kk, dg + 2 * kk, id2, kk > 0 ? 1u : 0u);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)  // delta: hidden units 64..127 = H columns 32..63
              tc_mma_ts(t_main + 64, t_h + 32 + 8 * kk, dd + 2 * kk, id2, kk > 0 ? 1u : 0u);
            tc_commit(&sm.d2_full[pb]);
          }
          __syncwarp();
          qk[0] = qk[1];
          qfill[0] = qfill[1];
          qsur[0] = qsur[1];
          --qn;
          if (release >= 0 && (qn == 0 || qfill[0] != release)) {
            // The weights of that fill are no longer read once these second layers are done.
            if (elect_one()) tc_commit(&sm.w_empty[release & 1]);
            __syncwarp();
            release = -1;
          }
          progress = true;
        }
      }
      if (feeding && qn < 2) {  // first layer of tile k
        const int st = k % kTcStages, b = k & 1;
        const bool ready = __shfl_sync(
            0xffffffffu, (int)(mbar_test_wait(&sm.full[st], (k / kTcStages) & 1) && group_free(k)), 0);
        if (ready) {
          const int it = *reinterpret_cast<volatile int*>(&sm.stage_item[st]);
          const int fill = *reinterpret_cast<volatile int*>(&sm.stage_fill[st]);
          const int head = *reinterpret_cast<volatile int*>(&sm.stage_head[st]);
          if (it < 0) {
            feeding = false;
            progress = true;
          } else if (fill < 0 || fill == waited_fill ||
                     __shfl_sync(0xffffffffu, (int)mbar_test_wait(&sm.w_full[fill & 1], (fill >> 1) & 1), 0)) {
            if (fill >= 0) waited_fill = fill;
            tc_fence_after();
            if (fill >= 0) {
              const uint64_t da = sdesc_sw128(smem_u32(sm.v[st]));
              const uint64_t db = sdesc_sw128(smem_u32(sm.w1[fill & 1]));
              const uint32_t t_main = tmem + b * 256 + ((k >> 1) & 1) * 128;
              if (elect_one()) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)  // K = 64 channels: 4 x K16, +32 bytes per step
                  tc_mma_ss(t_main, da + 2 * kk, db + 2 * kk, id1, kk > 0 ? 1u : 0u);
                tc_commit(&sm.empty[st]);
                tc_commit(&sm.d1_full[b]);
              }
            } else if (elect_one()) {  // a mean tile: no MMA, release the stage and stand in
              mbar_arrive(&sm.empty[st]);
              mbar_arrive(&sm.d1_full[b]);
            }
            __syncwarp();
            if (elect_one()) {
              sm.acc_item[b] = it;
              sm.acc_head[b] = head;
              mbar_arrive(&sm.d1_full[b]);  // releases acc_item / acc_head to the group
            }
            __syncwarp();
            if (fill >= 0) {
              if (cur_fill >= 0 && fill != cur_fill) {  // cur_fill has no more tiles
                if (qn == 0) {
                  if (elect_one()) tc_commit(&sm.w_empty[cur_fill & 1]);
                  __syncwarp();
                } else {
                  release = cur_fill;
                }
              }
              cur_fill = fill;
              qk[qn] = k;
              qfill[qn] = fill;
              qsur[qn] = sur_cnt[b];
              last_sur[b] = (int)sur_cnt[b]++;
              ++qn;
            }
            last_kind[b] = fill >= 0 ? 1 : 0;
            ++k;
            progress = true;
          }
        }
      }
      if (!feeding && qn == 0) break;
      if (progress) {
        t0 = 0;
        continue;
      }
      __nanosleep(32);  // leave the issue slots to the epilogue warps on this sub-partition
      if ((spin & 255u) == 0) {  // bounded: give up after kWaitLimitNs without progress
        if (*abort_flag) {
          ok = false;
          break;
        }
        const unsigned long long now = global_timer_ns();
        if (t0 == 0) {
          t0 = now;
        } else if (now - t0 > kWaitLimitNs) {
          if (lane == 0) {
            atomicOr(err, VP_DEVERR_WAIT_TIMEOUT);
            *abort_flag = 1;
          }
          ok = false;
          break;
        }
      }
    }
    // No more items: a stop for each group (tiles k and k + 1).
    for (int kk = k; ok && kk < k + kTcGroups; ++kk) {
      const int b = kk & 1;
      for (uint32_t sp = 1; !__shfl_sync(0xffffffffu, (int)group_free(kk), 0); ++sp) {
        __nanosleep(32);
        if ((sp & 255u) == 0) {
          const unsigned long long now = global_timer_ns();
          if (*abort_flag || (t0 != 0 && now - t0 > kWaitLimitNs)) {
            if (lane == 0 && !*abort_flag) {
              atomicOr(err, VP_DEVERR_WAIT_TIMEOUT);
              *abort_flag = 1;
            }
            ok = false;
            break;
          }
          if (t0 == 0) t0 = now;
        }
      }
      if (!ok) break;
      if (elect_one()) {
        sm.acc_item[b] = -1;
        mbar_arrive(&sm.d1_full[b]);
        mbar_arrive(&sm.d1_full[b]);
      }
      __syncwarp();
    }
    if (!ok) {
      if (elect_one()) {
        tc_commit(&sm.drain);
        for (int t = 0; t < 1000000 && !mbar_try_wait(&sm.drain, 0); ++t) {}
      }
      __syncwarp();
    }
  } else {
    // ------------------------------------------------------------ epilogue groups
    const int e = warp - 2;
    const int g = e / (4 * kTcParts), part = (e % (4 * kTcParts)) >> 2;
    const int gt = tid - 64 - kGroupThreads * g;  // 0 .. kGroupThreads - 1 within the group
    const int quarter = warp & 3;                 // TMEM lanes this warp may access
    const int row = quarter * 32 + lane;          // token row of the tile = TMEM lane
    const uint32_t t_grp = tmem + ((uint32_t)(quarter * 32) << 16) + g * 256;
    unsigned char* yrow = reinterpret_cast<unsigned char*>(sm.ys[g]) + row * 128;
    // This warp's share of a row: hidden-unit chunks [g0, g1) of 16 (first layer, H) and
    // output-column chunks [f0, f1) of 16 (second layer, y).
    const int g0 = part_begin(part, 8), g1 = part_begin(part + 1, 8);
    const int f0 = part_begin(kTcParts - 1 - part, 4), f1 = part_begin(kTcParts - part, 4);
    uint32_t sj = 0;  // surrogate tiles of this group
    bool ok = true;
    for (uint32_t j = 0;; ++j) {
      ok = group_all(mbar_wait_warp(&sm.d1_full[g], j & 1, err, abort_flag), g);
      if (!ok) break;
      tc_fence_after();
      const int it = *reinterpret_cast<volatile int*>(&sm.acc_item[g]);
      if (it < 0) break;
      const int h = *reinterpret_cast<volatile int*>(&sm.acc_head[g]);
      const bool surr = it < surr_items;
      const int tile = surr ? it % T : (it - surr_items) % Tm;  // a mean item spans kMeanRows rows
      const int slot = surr ? it / T : 0;  // surrogate head slot: its vectors
      const float* c1 = sm.c1[slot];
      const float* b2 = sm.b2[slot];
      const float* cx = sm.cx[slot];
      // This tile's halves of the group's columns: D1 / D2 in the main one (j & 1), H in the
      // first 64 columns of the other.
      const uint32_t t_acc = t_grp + (j & 1) * 128;
      const uint32_t t_h = t_grp + ((j & 1) ^ 1) * 128;
      if (surr) {
        // H = 2 GELU(D1 + c1) as bf16 pairs (the factor 2 is exact in bf16 and is taken out
        // of the second layer's results): chunk c of 16 hidden units (D1 columns 16 c ..)
        // into H columns 8 c .. + 8.  Each chunk's TMEM load is in flight while the chunk
        // before it is computed.
        float vb[2][16];
        tmem_ld16(t_acc + 16 * g0, vb[0]);
#pragma unroll
        for (int i = 0; i < kMaxGChunks; ++i) {
          const int c = g0 + i;
          if (c >= g1) break;
          tmem_wait_ld();
          if (c + 1 < g1) tmem_ld16(t_acc + 16 * (c + 1), vb[(i + 1) & 1]);
          uint32_t hw[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float2 cc = *reinterpret_cast<const float2*>(&c1[16 * c + 2 * q]);
            const float2 x = gelu2_as2(fadd2(make_float2(vb[i & 1][2 * q], vb[i & 1][2 * q + 1]), cc));
            hw[q] = pack_bf16x2(x.x, x.y);
          }
          tmem_st8(t_h + 8 * c, hw);
        }
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&sm.h_full[g]);
        ok = mbar_wait_warp(&sm.d2_full[g], sj & 1, err, abort_flag);
        ++sj;
      }
      if (!surr) {
        // Broadcast(mean of V_h) straight to Y (no staging: a store pipeline two tiles deep
        // per SM would hold these pure-write tiles back): eight threads per row, each a 16-byte
        // chunk, so that a warp writes whole 128-byte rows.
        ok = group_all(ok, g);
        if (!ok) break;
        if (gt == 0) mbar_arrive(&sm.taken[g]);  // every thread has read this tile's item
        const int jc = gt & 7;
        const float4 m0 = __ldg(reinterpret_cast<const float4*>(a.mean_v + h * 64) + 2 * jc);
        const float4 m1 = __ldg(reinterpret_cast<const float4*>(a.mean_v + h * 64) + 2 * jc + 1);
        const uint4 val = make_uint4(pack_bf16x2(m0.x, m0.y), pack_bf16x2(m0.z, m0.w),
                                     pack_bf16x2(m1.x, m1.y), pack_bf16x2(m1.z, m1.w));
        for (int r = gt >> 3; r < kMeanRows; r += kGroupThreads / 8) {
          const int grow = tile * kMeanRows + r;
          if (grow < a.N) *(reinterpret_cast<uint4*>(a.y + ((size_t)grow * H + h) * 64) + jc) = val;
        }
        continue;
      }
      // The staging buffer is free once the previous store from it has read it.
      if (gt == 0) tma_store_wait_read<0>();
      ok = group_all(ok, g);
      if (!ok) break;
      if (gt == 0) mbar_arrive(&sm.taken[g]);  // every thread has read this tile's item
      {
        // y = C + sigma(D2g + b2g) (.) (D2d + b2d) for chunk c of 16 output columns, from
        // D2' = 2 D2: sigma(u) = 1 / (1 + 2^(-log2(e) u)) with the exponent
        // -log2(e) / 2 D2g' + nbg, nbg = -log2(e) b2g held per head.
        tc_fence_after();
        const float kS = -0.5f * 1.4426950408889634f;
#pragma unroll
        for (int i = 0; i < kMaxFChunks; ++i) {
          const int c = f0 + i;
          if (c >= f1) break;
          float og[16], od[16];
          tmem_ld16(t_acc + 16 * c, og);
          tmem_ld16(t_acc + 64 + 16 * c, od);
          tmem_wait_ld();
          uint32_t yw[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const int col = 16 * c + 2 * q;
            const float2 C = *reinterpret_cast<const float2*>(&cx[col]);
            const float2 nbg = *reinterpret_cast<const float2*>(&b2[col]);
            const float2 bd = *reinterpret_cast<const float2*>(&b2[64 + col]);
            const float2 ea = ffma2(make_float2(og[2 * q], og[2 * q + 1]), make_float2(kS, kS), nbg);
            const float2 den = fadd2(make_float2(fast_exp2(ea.x), fast_exp2(ea.y)), make_float2(1.f, 1.f));
            float2 sg;
            asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(sg.x) : "f"(den.x));
            asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(sg.y) : "f"(den.y));
            const float2 dl = ffma2(make_float2(od[2 * q], od[2 * q + 1]), make_float2(0.5f, 0.5f), bd);
            const float2 y2 = ffma2(sg, dl, C);
            yw[q] = pack_bf16x2(y2.x, y2.y);
          }
#pragma unroll
          for (int q = 0; q < 2; ++q) {  // 16-byte chunk jc of the row sits at chunk jc ^ (row & 7)
            const int jc = 2 * c + q;
            *reinterpret_cast<uint4*>(yrow + ((jc ^ (row & 7)) << 4)) =
                make_uint4(yw[4 * q], yw[4 * q + 1], yw[4 * q + 2], yw[4 * q + 3]);
          }
        }
        tc_fence_before();
      }
      fence_proxy_async_smem();
      group_all(true, g);
      if (gt == 0) {
        tma_store_2d(&maps.y, sm.ys[g], h * 64, tile * kTcTile);
        tma_store_commit();
      }
    }
    if (gt == 0) tma_store_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTcTmemCols);
  }
  // Do not complete before the full-attention grid: later work in the stream reads all of Y.
  if (tid == 0) asm volatile("griddepcontrol.wait;" ::: "memory");
}

}  // namespace

size_t cheap_heads_tc_smem() { return sizeof(TcSmem) + 1024; }

cudaError_t launch_cheap_heads_tc(const HeadAttnArgs& a, int num_sms, cudaStream_t st) {
  TcMaps maps;
  cudaError_t e;
  const uint64_t H = (uint64_t)a.H;
  if ((e = make_tmap_bf16_2d(&maps.v, a.qkv, 3 * H * 64, (uint64_t)a.N, 3 * H * 64, 64, kTcTile)) !=
      cudaSuccess)
    return e;
  if ((e = make_tmap_bf16_2d(&maps.y, a.y, H * 64, (uint64_t)a.N, H * 64, 64, kTcTile)) != cudaSuccess)
    return e;
  // Layer-1 weights [H][64][128]: the value half is columns 0..63; layer 2 [H][64][64].
  if ((e = make_tmap_bf16_2d(&maps.g1, a.sw.g1_w, 128, H * 64, 128, 64, 64)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16_2d(&maps.d1, a.sw.d1_w, 128, H * 64, 128, 64, 64)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16_2d(&maps.g2, a.sw.g2_w, 64, H * 64, 64, 64, 64)) != cudaSuccess) return e;
  if ((e = make_tmap_bf16_2d(&maps.d2, a.sw.d2_w, 64, H * 64, 64, 64, 64)) != cudaSuccess) return e;
  const int smem = (int)cheap_heads_tc_smem();
  if ((e = cudaFuncSetAttribute(cheap_heads_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                smem)) != cudaSuccess)
    return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(num_sms);
  cfg.blockDim = dim3(kTcThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, cheap_heads_tc_kernel, maps, a);
}

}  // namespace vp
