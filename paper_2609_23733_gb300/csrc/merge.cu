// Token merging (ToMe) around the routed attention of a global block: the paper combines
// VGGT-Prime with the token merging of FastVGGT (75 % and 90 % of the tokens merged) without
// defining it; the reading here (vp_merge_options):
//   destinations: every special token, every token of the first view, and every stride-th
//     patch token of the other views; all other tokens are sources;
//   metric: the block's keys averaged over heads, k_i = mean_h (x~_i W_k,h^T + b_k,h), as a
//     unit vector (ToMe's similarity);
//   matching: every source joins the destination of largest cosine similarity (ties: the
//     lowest destination), over all destinations of all views;
//   merge: a merged token is the mean of its destination and the sources that joined it;
//   unmerge: every token takes its merged token's attention output.
// Kernels: the head-mean key weights, the metric GEMM (gemm_kernel), unit metric rows of the
// sources and of the destinations with the destination table, the matching (tcgen05 scores of
// 128 sources x 256 destinations per MMA group with a running argmax in the epilogue, work
// split evenly over the SMs), resolving and counting each token's merged row, scan and fill
// of each merged token's members, their mean, and the unmerge fused with LayerScale, the
// residual add and the block's second LayerNorm.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

// Destination test and merged row of token i (MergeGeo: views of P tokens, ps special tokens,
// every stride-th patch of views 1.. is a destination, Dv destinations per such view).
__device__ __forceinline__ int merged_row(const MergeGeo& g, int i) {
  const int v = i / g.P, t = i - v * g.P;
  if (v == 0) return t;
  const int base = g.P + (v - 1) * g.Dv;
  if (t < g.ps) return base + t;
  const int p = t - g.ps;
  return p % g.stride == 0 ? base + g.ps + p / g.stride : -1;
}

// Sources in token order: view v >= 1 holds Sv = P - Dv of them, the patches q = t - ps with
// q % stride != 0.  Index of source token i (merged_row(g, i) < 0) among all sources:
__device__ __forceinline__ int source_index(const MergeGeo& g, int i) {
  const int v = i / g.P, q = i - v * g.P - g.ps;
  return (v - 1) * g.Sv + q - q / g.stride - 1;
}

// Head-mean key weights: wbar[c][k] = mean_h W_qkv[D + 64 h + c][k], bbar[c] likewise.
__global__ void metric_weights_kernel(const __nv_bfloat16* w_qkv, const float* b_qkv, int H,
                                      int D, __nv_bfloat16* wbar, float* bbar) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= 64 * D) return;
  const int c = idx / D, k = idx - c * D;
  float s = 0.f;
  for (int h = 0; h < H; ++h) s += __bfloat162float(w_qkv[(size_t)(D + 64 * h + c) * D + k]);
  wbar[idx] = __float2bfloat16_rn(s / (float)H);
  if (k == 0) {
    float b = 0.f;
    if (b_qkv)
      for (int h = 0; h < H; ++h) b += b_qkv[D + 64 * h + c];
    bbar[c] = b / (float)H;
  }
}

// Eight lanes per token (16 bytes each, four tokens per warp): the metric row as a unit vector
// (bf16), stored by source index for a source and by merged row for a destination; the
// merged row of every token (-1 for sources) and the token of every merged row.
__global__ void merge_setup_kernel(MergeGeo g, const __nv_bfloat16* kbar, __nv_bfloat16* m_src,
                                   __nv_bfloat16* m_dst, int* row_of, int* dst_tok) {
  const int sub = threadIdx.x & 7;
  const int i = blockIdx.x * (blockDim.x >> 3) + (threadIdx.x >> 3);
  if (i >= g.N) return;  // whole groups of eight lanes leave together
  const uint4 u = reinterpret_cast<const uint4*>(kbar + (size_t)i * 64)[sub];
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) ss += bf16_lo(w[k]) * bf16_lo(w[k]) + bf16_hi(w[k]) * bf16_hi(w[k]);
  // the warp's tokens that exist: a prefix of its four groups of eight lanes
  const int live = min(4, g.N - (i - (int)((threadIdx.x & 31) >> 3)));
  const unsigned mask = live == 4 ? 0xffffffffu : (1u << (8 * live)) - 1u;
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) ss += __shfl_xor_sync(mask, ss, o);
  const float inv = ss > 0.f ? rsqrtf(ss) : 0.f;
  uint32_t mu[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) mu[k] = pack_bf16x2(bf16_lo(w[k]) * inv, bf16_hi(w[k]) * inv);
  const int r = merged_row(g, i);
  __nv_bfloat16* dst = r >= 0 ? m_dst + (size_t)r * 64 : m_src + (size_t)source_index(g, i) * 64;
  reinterpret_cast<uint4*>(dst)[sub] = make_uint4(mu[0], mu[1], mu[2], mu[3]);
  if (sub == 0) {
    row_of[i] = r;
    if (r >= 0) dst_tok[r] = i;
  }
}

// Matching on the tensor cores: scores S = M_src M_dst^T (cosines of unit keys) of 128 source
// rows against chunks of 256 destinations, with a running argmax over the chunks.  The work
// units (source tile, destination chunk) are split evenly over the CTAs (one per SM): CTA b
// takes units [b U / G, (b + 1) U / G), runs of ascending chunks of one tile or more
// (segments), so that no SM idles through a partial last round.  Each segment's best per row
// goes into a 64-bit atomic maximum of (score, lowest column), which also joins the rows whose
// chunks two CTAs share.
//   warp 0      TMA: a segment's 128 source rows (16 KB, two buffers) and destination chunks
//               (256 rows x 64 channels, 32 KB, 128-byte swizzle) through a kMatchStages ring;
//   warp 1      TMEM owner;
//   warps 1-2   MMA issue: four tcgen05.mma M128 N256 K16 per chunk into one of two 256-column
//               fp32 accumulators (the epilogue of one chunk overlaps the MMAs of the next),
//               warp 1 the even chunks (accumulator 0), warp 2 the odd ones: a chunk's waits,
//               MMA and commit instructions take one warp about 800 clocks, more than the MMAs
//               themselves (512);
//   warps 4-19  argmax: a source row (TMEM lane) and a quarter of each chunk's columns per
//               thread, loaded into registers (two tcgen05.ld.red of 32 columns, which also
//               return each 32-column piece's maximum) before the accumulator is released; a
//               piece whose max beats the row's best is copied to the
//               thread's slot in shared memory, and the column is looked up there once, at the
//               end of the segment.  Chunks ascend within a segment, so the first piece that
//               reaches a score holds its lowest column.
constexpr int kMatchStages = 4;
constexpr int kMatchN = 256;
constexpr int kMatchParts = 4;                // column parts of a chunk (argmax warps per TMEM lane quarter)
constexpr int kMatchWarps = 4 * kMatchParts;  // argmax warps
constexpr int kMatchThreads = 128 + 32 * kMatchWarps;
constexpr uint32_t kMatchTmemCols = 512;

struct MatchSmem {
  __nv_bfloat16 src[2][128 * 64];
  __nv_bfloat16 dst[kMatchStages][kMatchN * 64];
  float4 stash[kMatchWarps][32][8];  // each argmax thread's best piece, 16-byte slots rotated by lane
  uint64_t src_full[2], src_empty[2];
  uint64_t dst_full[kMatchStages], dst_empty[kMatchStages];
  uint64_t acc_full[2], acc_empty[2], drain[2];
  uint32_t tmem_base;
  int abort_flag;
};

// The run of units starting at unit u of a CTA's range [u, u_end): tile t, chunks [c0, c1).
struct Segment {
  int t, c0, c1;
};
__device__ __forceinline__ Segment segment_at(long long u, long long u_end, int n_chunks) {
  Segment sg;
  sg.t = (int)(u / n_chunks);
  sg.c0 = (int)(u - (long long)sg.t * n_chunks);
  sg.c1 = (int)min((long long)n_chunks, (long long)sg.c0 + (u_end - u));
  return sg;
}

// (score, column) as one 64-bit key that orders like the argmax: higher score first, then the
// lower column.  Float bits made monotone: negative values inverted, positive ones offset.
// -0 and +0 are the same score, so -0 is keyed as +0 (else +0 at a higher column would beat
// an equal -0 and break the lowest-column rule).
__device__ __forceinline__ unsigned long long match_key(float v, int col) {
  uint32_t b = __float_as_uint(v);
  if (b == 0x80000000u) b = 0u;
  const uint32_t ord = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ((unsigned long long)ord << 32) | (unsigned long long)(~(uint32_t)col);
}

__global__ void __launch_bounds__(kMatchThreads, 1)
    tome_match_kernel(const __grid_constant__ CUtensorMap tmap_src,
                      const __grid_constant__ CUtensorMap tmap_dst, MergeGeo g,
                      unsigned long long* best, unsigned int* err) {
  extern __shared__ unsigned char smem_raw[];
  MatchSmem& sm = *reinterpret_cast<MatchSmem*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int n_tiles = (g.Ns + 127) / 128;
  const int n_chunks = (g.Np + kMatchN - 1) / kMatchN;
  const long long n_units = (long long)n_tiles * n_chunks;
  const long long u_begin = n_units * blockIdx.x / gridDim.x;
  const long long u_end = n_units * (blockIdx.x + 1) / gridDim.x;
  if (u_begin >= u_end) return;  // uniform across the CTA
  const int warp = warp_uniform_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  if (threadIdx.x == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.src_full[b], 1);
      mbar_init(&sm.src_empty[b], 2);  // both MMA warps
      mbar_init(&sm.acc_full[b], 1);
      mbar_init(&sm.acc_empty[b], 32 * kMatchWarps);
    }
    for (int s = 0; s < kMatchStages; ++s) {
      mbar_init(&sm.dst_full[s], 1);
      mbar_init(&sm.dst_empty[s], 1);
    }
    mbar_init(&sm.drain[0], 1);
    mbar_init(&sm.drain[1], 1);
    sm.abort_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
    tma_prefetch_desc(&tmap_src);
    tma_prefetch_desc(&tmap_dst);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kMatchTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, sm.tmem_base, 0);

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    uint32_t lc = 0, sc = 0;  // destination chunks / source tiles issued
    bool ok = true;
    for (long long u = u_begin; u < u_end && ok;) {
      const Segment sg = segment_at(u, u_end, n_chunks);
      const int sb = sc & 1;
      ok = mbar_wait_warp(&sm.src_empty[sb], ((sc >> 1) & 1) ^ 1, err, abort_flag);
      if (!ok) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&sm.src_full[sb], 128 * 64 * 2);
        tma_load_2d(sm.src[sb], &tmap_src, &sm.src_full[sb], 0, sg.t * 128);
      }
      __syncwarp();
      ++sc;
      for (int ch = sg.c0; ch < sg.c1; ++ch, ++lc) {
        const int st = lc % kMatchStages;
        ok = mbar_wait_warp(&sm.dst_empty[st], ((lc / kMatchStages) & 1) ^ 1, err, abort_flag);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(&sm.dst_full[st], kMatchN * 64 * 2);
          tma_load_2d(sm.dst[st], &tmap_dst, &sm.dst_full[st], 0, ch * kMatchN);
        }
        __syncwarp();
      }
      u += sg.c1 - sg.c0;
    }
    if (!ok && lane == 0) {  // let issued copies land before the CTA releases its smem
      for (int b = 0; b < 2; ++b) {
        if (sc > (uint32_t)b) {
          const uint32_t last = (sc - 1 - b) / 2 * 2 + b;  // last tile load into buffer b
          for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.src_full[b], (last >> 1) & 1); ++k) {}
        }
      }
      for (int s = 0; s < kMatchStages; ++s) {
        if (lc > (uint32_t)s) {
          const uint32_t last = (lc - 1 - s) / kMatchStages * kMatchStages + s;
          for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.dst_full[s], (last / kMatchStages) & 1); ++k) {}
        }
      }
    }
  } else if (warp == 1 || warp == 2) {
    // ------------------------------------------------------------ MMA issue
    // Warp 1 issues the even chunks, warp 2 the odd ones (ac & 1 picks the accumulator and the
    // warp); both walk all units so that their counters agree, and both commit the release of
    // a segment's source tile (its mbarrier counts two).
    const uint32_t mine = (uint32_t)(warp - 1);
    const uint32_t idesc = idesc_bf16(128, kMatchN, 0, 0);
    uint32_t lc = 0, sc = 0, ac = 0;
    bool ok = true;
    for (long long u = u_begin; u < u_end && ok; ++sc) {
      const Segment sg = segment_at(u, u_end, n_chunks);
      const int sb = sc & 1;
      ok = mbar_wait_warp(&sm.src_full[sb], (sc >> 1) & 1, err, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint64_t da = sdesc_sw128(smem_u32(sm.src[sb]));
      for (int ch = sg.c0; ch < sg.c1; ++ch, ++lc, ++ac) {
        if ((ac & 1) != mine) continue;  // the other warp's chunk
        const int st = lc % kMatchStages;
        const uint32_t ab = ac & 1;
        ok = mbar_wait_warp(&sm.dst_full[st], (lc / kMatchStages) & 1, err, abort_flag) &&
             mbar_wait_warp(&sm.acc_empty[ab], ((ac >> 1) & 1) ^ 1, err, abort_flag);
        if (!ok) break;
        tc_fence_after();
        const uint64_t db = sdesc_sw128(smem_u32(sm.dst[st]));
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // K = 64 channels: 4 x K16, +32 bytes per step
            tc_mma_ss(tmem + ab * kMatchN, da + 2 * kk, db + 2 * kk, idesc, kk > 0 ? 1u : 0u);
          tc_commit(&sm.acc_full[ab]);
          tc_commit(&sm.dst_empty[st]);
        }
        __syncwarp();
      }
      if (!ok) break;
      if (elect_one()) tc_commit(&sm.src_empty[sb]);  // this warp's MMAs on the source tile
      __syncwarp();
      u += sg.c1 - sg.c0;
    }
    if (!ok) {
      if (elect_one()) {
        tc_commit(&sm.drain[mine]);
        for (int k = 0; k < 1000000 && !mbar_try_wait(&sm.drain[mine], 0); ++k) {}
      }
      __syncwarp();
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ running argmax
    constexpr int kCols = kMatchN / kMatchParts;  // columns of a part
    const int aw = warp - 4;
    const int quarter = warp & 3, part = aw >> 2;
    const int rit = quarter * 32 + lane;  // row in the tile
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16) + part * kCols;
    float4* slot = sm.stash[aw][lane];
    uint32_t ac = 0;
    bool ok = true;
    for (long long u = u_begin; u < u_end && ok;) {
      const Segment sg = segment_at(u, u_end, n_chunks);
      float bv = -INFINITY;
      int bcol = -1;  // first column of the stashed piece
      for (int ch = sg.c0; ch < sg.c1; ++ch, ++ac) {
        const uint32_t ab = ac & 1;
        ok = mbar_wait_warp(&sm.acc_full[ab], (ac >> 1) & 1, err, abort_flag);
        if (!ok) break;
        tc_fence_after();
        const int c0 = ch * kMatchN + part * kCols;  // first destination of the part
        const int valid = g.Np - c0;                 // columns past it hold no destination
        // Both pieces into registers, then the accumulator goes back to the MMA warp at once:
        // the max trees below overlap the next chunks' MMAs.
        // Each piece's maximum comes with its load (tcgen05.ld.red).
        float v[kCols / 32][32], pm[kCols / 32];
#pragma unroll
        for (int p = 0; p < kCols / 32; ++p) tmem_ld32_max(t_lane + ab * kMatchN + 32 * p, v[p], pm[p]);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(&sm.acc_empty[ab]);
#pragma unroll
        for (int p = 0; p < kCols / 32; ++p) {
          float* x = v[p];
          float mx = pm[p];
          if (32 * p + 32 > valid) {  // columns past the last destination: masked, then a tree
#pragma unroll
            for (int k = 0; k < 32; ++k)
              if (32 * p + k >= valid) x[k] = -INFINITY;
            float q[4];  // four independent 3-input max chains, then a short tree
#pragma unroll
            for (int k = 0; k < 4; ++k) q[k] = fmaxf(x[k], x[k + 4]);
#pragma unroll
            for (int k = 8; k < 32; k += 8)
#pragma unroll
              for (int e = 0; e < 4; ++e) q[e] = fmax3(q[e], x[k + e], x[k + 4 + e]);
            mx = fmax3(q[0], q[1], fmaxf(q[2], q[3]));
          }
          if (mx > bv) {  // a strictly better piece: keep its scores
            bv = mx;
            bcol = c0 + 32 * p;
#pragma unroll
            for (int j = 0; j < 8; ++j)
              slot[(j + lane) & 7] = make_float4(x[4 * j], x[4 * j + 1], x[4 * j + 2], x[4 * j + 3]);
          }
        }
      }
      if (!ok) break;
      u += sg.c1 - sg.c0;
      const int row = sg.t * 128 + rit;
      if (bcol >= 0 && row < g.Ns) {  // the lowest column of the kept piece that holds bv
        float x[32];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float4 f = slot[(j + lane) & 7];
          x[4 * j] = f.x;
          x[4 * j + 1] = f.y;
          x[4 * j + 2] = f.z;
          x[4 * j + 3] = f.w;
        }
        int k_best = 31;
#pragma unroll
        for (int k = 31; k >= 0; --k)
          if (x[k] == bv) k_best = k;
        atomicMax(best + row, match_key(bv, bcol + k_best));
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kMatchTmemCols);
  }
}

// The merged row of every token -- its own for a destination, the matched destination for a
// source -- counted per merged row.
__global__ void merge_resolve_kernel(MergeGeo g, const int* row_of, const unsigned long long* best,
                                     int* assign, int* cnt) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= g.N) return;
  int r = row_of[i];
  if (r < 0) {
    const unsigned long long k = best[source_index(g, i)];
    r = k ? (int)~(uint32_t)k : 0;  // no score compared (NaN metric): any valid row
    if (r < 0 || r >= g.Np) r = 0;
  }
  assign[i] = r;
  atomicAdd(cnt + r, 1);
}

// Exclusive scan of cnt[0..n) into offs[0..n] in one block of 1024 threads, 4,096 entries a
// round: four per thread (one 16-byte load, the next round's in flight), a warp scan of the
// thread totals, a scan of the 32 warp totals, and the carry of the rounds before.
__global__ void __launch_bounds__(1024) scan_kernel(int n, const int* cnt, int* offs) {
  __shared__ int warp_ex[32];
  __shared__ int round_total;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  auto load4 = [&](int base) {
    const int i = base + 4 * tid;
    if (i + 3 < n) return *reinterpret_cast<const int4*>(cnt + i);
    int4 r = make_int4(0, 0, 0, 0);
    if (i < n) r.x = cnt[i];
    if (i + 1 < n) r.y = cnt[i + 1];
    if (i + 2 < n) r.z = cnt[i + 2];
    return r;
  };
  int carry = 0;
  int4 nxt = load4(0);
  for (int base = 0; base < n; base += 4096) {
    const int4 c = nxt;
    if (base + 4096 < n) nxt = load4(base + 4096);
    const int s1 = c.x, s2 = s1 + c.y, s3 = s2 + c.z, tot = s3 + c.w;
    int incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) warp_ex[wid] = incl;
    __syncthreads();
    if (wid == 0) {
      const int w = warp_ex[lane];
      int wi = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += y;
      }
      warp_ex[lane] = wi - w;
      if (lane == 31) round_total = wi;
    }
    __syncthreads();
    const int ex = carry + warp_ex[wid] + incl - tot;
    const int i = base + 4 * tid;
    if (i + 3 < n) {
      *reinterpret_cast<int4*>(offs + i) = make_int4(ex, ex + s1, ex + s2, ex + s3);
    } else {
      if (i < n) offs[i] = ex;
      if (i + 1 < n) offs[i + 1] = ex + s1;
      if (i + 2 < n) offs[i + 2] = ex + s2;
    }
    carry += round_total;
    __syncthreads();  // warp_ex and round_total are rewritten in the next round
  }
  if (tid == 0) offs[n] = carry;
}

__global__ void merge_fill_kernel(int N, const int* assign, const int* offs, int* fill,
                                  int* members) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N) return;
  const int r = assign[i];
  members[offs[r] + atomicAdd(fill + r, 1)] = i;
}

// The merged tokens: the mean of each merged row's members' rows of LN1(x), normalised on the
// fly (the LN1 output is not stored): per member, its mean and 1 / sqrt(var + eps) from the
// (mean, M2) of its 128-column blocks, then (x - mu) rstd summed in fp32; at the end
// gamma (.) sum / count + beta.  The member list (grouped by merged row) is cut into chunks of
// kMeanChunk consecutive entries, one warp each, so that every warp reads the same number of
// rows however unevenly the sources chose their destinations (later blocks put hundreds of
// sources on a few destinations).  A merged row whose members all lie in the chunk is written
// there.  A row that crosses a chunk boundary leaves its chunk's part of the sum in a slot
// (slot 1 of its first chunk, slot 0 of every later one) and counts its members off fill[r],
// which holds the row's member count; the chunk that brings it to 0 adds the row's slots in
// chunk order and writes the mean.  D = 256 C; lane l holds 16-byte chunks c 32 + l.
constexpr int kMeanChunk = 32;
static_assert(kMeanChunk == 32, "merge_slot_bytes counts chunks of 32 entries");
constexpr int kMeanInFlight = 2;  // member rows whose loads are in flight together

template <int C>
__device__ __forceinline__ void store_mean(const float (&acc)[C][8], float inv, int lane,
                                           const float* gamma, const float* beta,
                                           __nv_bfloat16* dst) {
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int col = (c * 32 + lane) * 8;
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(gamma + col));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(gamma + col) + 1);
    const float4 b0 = __ldg(reinterpret_cast<const float4*>(beta + col));
    const float4 b1 = __ldg(reinterpret_cast<const float4*>(beta + col) + 1);
    const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
    const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
    uint4 o;
    o.x = pack_bf16x2(fmaf(gg[0], acc[c][0] * inv, bb[0]), fmaf(gg[1], acc[c][1] * inv, bb[1]));
    o.y = pack_bf16x2(fmaf(gg[2], acc[c][2] * inv, bb[2]), fmaf(gg[3], acc[c][3] * inv, bb[3]));
    o.z = pack_bf16x2(fmaf(gg[4], acc[c][4] * inv, bb[4]), fmaf(gg[5], acc[c][5] * inv, bb[5]));
    o.w = pack_bf16x2(fmaf(gg[6], acc[c][6] * inv, bb[6]), fmaf(gg[7], acc[c][7] * inv, bb[7]));
    *reinterpret_cast<uint4*>(dst + col) = o;
  }
}

// The members [a, b) of the chunk (entries q0 + a .. q0 + b - 1 of the list) that belong to
// merged row r, summed in acc: the row's mean if the chunk holds all of its members, else the
// chunk's slot and the count-off described above.
template <int C>
__device__ __forceinline__ void flush_row(float (&acc)[C][8], int r, int a, int b, int ch, int q0,
                                          int nm, int lane, const int* offs, int* fill,
                                          float* slots, const float* gamma, const float* beta,
                                          __nv_bfloat16* xm) {
  constexpr int D = 256 * C;
  const int first = __ldg(offs + r), last = __ldg(offs + r + 1);
  if (first < q0 || last > q0 + nm) {  // the row crosses a chunk boundary
    float* slot = slots + ((size_t)ch * 2 + (first < q0 ? 0 : 1)) * D;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      float4* d = reinterpret_cast<float4*>(slot + (c * 32 + lane) * 8);
      d[0] = make_float4(acc[c][0], acc[c][1], acc[c][2], acc[c][3]);
      d[1] = make_float4(acc[c][4], acc[c][5], acc[c][6], acc[c][7]);
    }
    __threadfence();
    __syncwarp();
    int done = 0;
    if (lane == 0) done = atomicSub(fill + r, b - a) == b - a;
    if (!__shfl_sync(0xffffffffu, done, 0)) return;  // another chunk of the row finishes it
    __threadfence();
    const int c0 = first / kMeanChunk, c1 = (last - 1) / kMeanChunk;
#pragma unroll
    for (int c = 0; c < C; ++c)
#pragma unroll
      for (int k = 0; k < 8; ++k) acc[c][k] = 0.f;
#pragma unroll 1
    for (int cc = c0; cc <= c1; ++cc) {
      const float* sl = slots + ((size_t)cc * 2 + (cc == c0 ? 1 : 0)) * D;
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const float4* q = reinterpret_cast<const float4*>(sl + (c * 32 + lane) * 8);
        const float4 u0 = __ldcg(q), u1 = __ldcg(q + 1);
        acc[c][0] += u0.x;
        acc[c][1] += u0.y;
        acc[c][2] += u0.z;
        acc[c][3] += u0.w;
        acc[c][4] += u1.x;
        acc[c][5] += u1.y;
        acc[c][6] += u1.z;
        acc[c][7] += u1.w;
      }
    }
  }
  store_mean<C>(acc, 1.f / (float)(last - first), lane, gamma, beta, xm + (size_t)r * D);
}

// Two CTAs per SM at D = 1,024: the accumulator, two rows in flight and the slot path fit in
// 128 registers without spills (three CTAs spill and measured 1 ms slower per S = 100 forward).
template <int C>
__global__ void __launch_bounds__(256, C <= 2 ? 3 : (C <= 4 ? 2 : 1))
    merge_mean_kernel(int N, const __nv_bfloat16* x, const float2* part, const float* gamma,
                      const float* beta, float eps, const int* offs, const int* members,
                      const int* assign, int* fill, float* slots, __nv_bfloat16* xm) {
  constexpr int D = 256 * C, NB = D / 128;  // 128-column blocks of a row (NB <= 32)
  const int lane = threadIdx.x & 31;
  const int ch = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int q0 = ch * kMeanChunk;
  if (q0 >= N) return;
  const int nm = min(kMeanChunk, N - q0);
  const int mine = lane < nm ? __ldg(members + q0 + lane) : 0;  // one coalesced load
  const int my_row = lane < nm ? __ldg(assign + mine) : -1;
  float acc[C][8];
#pragma unroll
  for (int c = 0; c < C; ++c)
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[c][k] = 0.f;
  int cur = __shfl_sync(0xffffffffu, my_row, 0), run0 = 0;  // the current row and its first entry
  // Entries 0 .. nm - 1, then a sentinel entry nm that ends the last row (one flush site).
  for (int k = 0; k <= nm; k += kMeanInFlight) {  // the rows' loads issued before any arithmetic
    uint4 u[kMeanInFlight][C];
    float2 ps[kMeanInFlight];
#pragma unroll
    for (int j = 0; j < kMeanInFlight; ++j) {
      const int i = __shfl_sync(0xffffffffu, mine, min(k + j, nm - 1));
#pragma unroll
      for (int c = 0; c < C; ++c)
        u[j][c] = __ldg(reinterpret_cast<const uint4*>(x + (size_t)i * D + (c * 32 + lane) * 8));
      ps[j] = lane < NB ? __ldg(part + (size_t)i * NB + lane) : make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int j = 0; j < kMeanInFlight; ++j) {
      const int e = k + j;
      if (e > nm) break;  // uniform across the warp
      const int re = __shfl_sync(0xffffffffu, my_row, min(e, nm - 1));
      const int r = e < nm ? re : -1;
      if (r != cur) {  // the entries of row cur end here
        flush_row<C>(acc, cur, run0, e, ch, q0, nm, lane, offs, fill, slots, gamma, beta, xm);
#pragma unroll
        for (int c = 0; c < C; ++c)
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) acc[c][kk] = 0.f;
        cur = r;
        run0 = e;
      }
      if (e == nm) break;
      float sm = ps[j].x;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
      const float mu = sm / (float)NB;
      const float d = ps[j].x - mu;
      float m2 = lane < NB ? ps[j].y + 128.f * d * d : 0.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) m2 += __shfl_xor_sync(0xffffffffu, m2, o);
      const float rstd = rsqrtf(m2 / (float)D + eps);
      const float nmr = -mu * rstd;
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t w[4] = {u[j][c].x, u[j][c].y, u[j][c].z, u[j][c].w};
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          acc[c][2 * kk] += fmaf(bf16_lo(w[kk]), rstd, nmr);
          acc[c][2 * kk + 1] += fmaf(bf16_hi(w[kk]), rstd, nmr);
        }
      }
    }
  }
}

// The end of a merged block's attention branch and its second LayerNorm, one warp per token:
// x[i] <- bf16(x[i] + ls (.) a[assign[i]]) (unmerge, LayerScale, residual add) and
// z[i] = LN(x[i]) (gamma, beta, eps) from the stored bf16 values, in one pass over the rows
// (the LayerNorm kernel's arithmetic: fp32 mean, then the biased variance about it).
template <int C>
__global__ void __launch_bounds__(256, 4) unmerge_ln_kernel(int N, const int* assign,
                                                            const __nv_bfloat16* a, const float* ls,
                                                            const float* g, const float* b,
                                                            float eps, __nv_bfloat16* x,
                                                            __nv_bfloat16* z) {
  constexpr int D = 256 * C;
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (i >= N) return;
  const int r = assign[i];
  uint4 ua[C], ux[C];
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int col = (c * 32 + lane) * 8;
    ua[c] = __ldg(reinterpret_cast<const uint4*>(a + (size_t)r * D + col));
    ux[c] = *reinterpret_cast<const uint4*>(x + (size_t)i * D + col);
  }
  uint32_t o[4 * C];  // the new residual row, bf16 pairs
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int col = (c * 32 + lane) * 8;
    const float4 l0 = __ldg(reinterpret_cast<const float4*>(ls + col));
    const float4 l1 = __ldg(reinterpret_cast<const float4*>(ls + col) + 1);
    const float lw[8] = {l0.x, l0.y, l0.z, l0.w, l1.x, l1.y, l1.z, l1.w};
    const uint32_t wa[4] = {ua[c].x, ua[c].y, ua[c].z, ua[c].w};
    const uint32_t wx[4] = {ux[c].x, ux[c].y, ux[c].z, ux[c].w};
#pragma unroll
    for (int k = 0; k < 4; ++k)
      o[4 * c + k] = pack_bf16x2(fmaf(lw[2 * k], bf16_lo(wa[k]), bf16_lo(wx[k])),
                                 fmaf(lw[2 * k + 1], bf16_hi(wa[k]), bf16_hi(wx[k])));
    *reinterpret_cast<uint4*>(x + (size_t)i * D + col) =
        make_uint4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < 4 * C; ++k) {
    s += bf16_lo(o[k]);
    s += bf16_hi(o[k]);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  const float mean = s * (1.f / D);
  float q = 0.f;
#pragma unroll
  for (int k = 0; k < 4 * C; ++k) {
    const float t0 = bf16_lo(o[k]) - mean, t1 = bf16_hi(o[k]) - mean;
    q += t0 * t0;
    q += t1 * t1;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) q += __shfl_xor_sync(0xffffffffu, q, off);
  const float rstd = rsqrtf(q * (1.f / D) + eps);
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int col = (c * 32 + lane) * 8;
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(g + col));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(g + col) + 1);
    const float4 b0 = __ldg(reinterpret_cast<const float4*>(b + col));
    const float4 b1 = __ldg(reinterpret_cast<const float4*>(b + col) + 1);
    const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
    const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
    uint32_t y[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
      y[k] = pack_bf16x2((bf16_lo(o[4 * c + k]) - mean) * rstd * gg[2 * k] + bb[2 * k],
                         (bf16_hi(o[4 * c + k]) - mean) * rstd * gg[2 * k + 1] + bb[2 * k + 1]);
    *reinterpret_cast<uint4*>(z + (size_t)i * D + col) = make_uint4(y[0], y[1], y[2], y[3]);
  }
}

}  // namespace

MergeGeo make_merge_geo(int N, int P, int ps, int stride) {
  MergeGeo g;
  g.N = N;
  g.P = P;
  g.ps = ps;
  g.stride = stride;
  g.Dv = ps + (P - ps + stride - 1) / stride;
  g.Sv = P - g.Dv;
  g.Np = N <= P ? N : P + (N / P - 1) * g.Dv;
  g.Ns = N - g.Np;
  return g;
}

cudaError_t launch_merge_prepare(const MergeGeo& g, int H, const __nv_bfloat16* x,
                                 const MergeLn& ln, const __nv_bfloat16* w_qkv,
                                 const float* b_qkv, const MergeScratch& s, int num_sms,
                                 cudaStream_t st) {
  const int D = 64 * H;
  prof_before(VP_KERNEL_MERGE, st);
  metric_weights_kernel<<<(64 * D + 255) / 256, 256, 0, st>>>(w_qkv, b_qkv, H, D, s.wbar, s.bbar);
  prof_after(st);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // The metric of LN1(x) with LN1 folded into its weights, as in the QKV projection.
  if ((e = launch_ln_fold_weights(64, D, s.wbar, ln.g, ln.b, s.bbar, ln.w_fold, ln.c_fold,
                                  ln.b_fold, st)) != cudaSuccess)
    return e;
  LinearArgs la{};
  la.M = g.N;
  la.N = 64;
  la.K = D;
  la.A = x;
  la.W = ln.w_fold;
  la.bias = ln.b_fold;
  la.ln_part = ln.part;
  la.ln_c = ln.c_fold;
  la.ln_eps = ln.eps;
  la.act = VP_ACT_NONE;
  la.out = s.kbar;
  la.err = s.err;
  e = launch_linear(la, num_sms, st);
  if (e != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  merge_setup_kernel<<<(g.N + 31) / 32, 256, 0, st>>>(g, s.kbar, s.m_src, s.m_dst, s.row_of,
                                                      s.dst_tok);
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (g.Ns > 0) {  // one view, or stride 1: every token is a destination
    CUtensorMap tsrc, tdst;  // unit metric rows, 64 channels (128 bytes), 128-byte swizzle
    if ((e = make_tmap_bf16_2d(&tsrc, s.m_src, 64, (uint64_t)g.Ns, 64, 64, 128)) != cudaSuccess)
      return e;
    if ((e = make_tmap_bf16_2d(&tdst, s.m_dst, 64, (uint64_t)g.Np, 64, 64, kMatchN)) != cudaSuccess)
      return e;
    const int smem = (int)sizeof(MatchSmem) + 1024;
    if ((e = cudaFuncSetAttribute(tome_match_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  smem)) != cudaSuccess)
      return e;
    const long long units =
        (long long)((g.Ns + 127) / 128) * ((g.Np + kMatchN - 1) / kMatchN);
    prof_before(VP_KERNEL_MERGE, st);
    e = cudaMemsetAsync(s.best, 0, (size_t)g.Ns * sizeof(unsigned long long), st);
    if (e == cudaSuccess) {
      tome_match_kernel<<<(int)min((long long)num_sms, units), kMatchThreads, smem, st>>>(
          tsrc, tdst, g, s.best, s.err);
      e = cudaGetLastError();
    }
    prof_after(st);
    if (e != cudaSuccess) return e;
  }
  if ((e = cudaMemsetAsync(s.cnt, 0, (size_t)g.Np * sizeof(int), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(s.fill, 0, (size_t)g.Np * sizeof(int), st)) != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  merge_resolve_kernel<<<(g.N + 255) / 256, 256, 0, st>>>(g, s.row_of, s.best, s.assign, s.cnt);
  scan_kernel<<<1, 1024, 0, st>>>(g.Np, s.cnt, s.offs);
  merge_fill_kernel<<<(g.N + 255) / 256, 256, 0, st>>>(g.N, s.assign, s.offs, s.fill, s.members);
  prof_extra_launch();
  prof_extra_launch();
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  const int grid = ((g.N + kMeanChunk - 1) / kMeanChunk + 7) / 8;  // a warp per chunk
#define VP_MEAN(C_)                                                                              \
  merge_mean_kernel<C_><<<grid, 256, 0, st>>>(g.N, x, ln.part, ln.g, ln.b, ln.eps, s.offs,       \
                                              s.members, s.assign, s.fill, s.slots, s.xm)
  switch (D / 256) {
    case 1: VP_MEAN(1); break;
    case 2: VP_MEAN(2); break;
    case 3: VP_MEAN(3); break;
    case 4: VP_MEAN(4); break;
    case 8: VP_MEAN(8); break;
#undef VP_MEAN
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

cudaError_t launch_unmerge_ln(int N, int D, const int* assign, const __nv_bfloat16* a,
                              const float* ls, const float* g, const float* b, float eps,
                              __nv_bfloat16* x, __nv_bfloat16* z, cudaStream_t st) {
  prof_before(VP_KERNEL_MERGE, st);
  const int grid = (N + 7) / 8;
  switch (D / 256) {
    case 1: unmerge_ln_kernel<1><<<grid, 256, 0, st>>>(N, assign, a, ls, g, b, eps, x, z); break;
    case 2: unmerge_ln_kernel<2><<<grid, 256, 0, st>>>(N, assign, a, ls, g, b, eps, x, z); break;
    case 3: unmerge_ln_kernel<3><<<grid, 256, 0, st>>>(N, assign, a, ls, g, b, eps, x, z); break;
    case 4: unmerge_ln_kernel<4><<<grid, 256, 0, st>>>(N, assign, a, ls, g, b, eps, x, z); break;
    case 8: unmerge_ln_kernel<8><<<grid, 256, 0, st>>>(N, assign, a, ls, g, b, eps, x, z); break;
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

}  // namespace vp
