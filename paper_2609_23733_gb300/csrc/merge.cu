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
// Kernels: the head-mean key weights, the metric GEMM (gemm_kernel), unit metric rows and the
// destination table, the matching (mma.sync tiles of 16 sources x 64 destinations with a
// running argmax; the max of a thread's 16 scores is taken first and the index searched only
// when it improves), counting / scan / fill of each merged token's members, their mean, and
// the unmerge fused with LayerScale and the residual add.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace vp {

namespace {

// D (16 x 8, fp32) += A (16 x 16, bf16, row) B (16 x 8, bf16, col): one warp, mma.sync.
__device__ __forceinline__ void mma16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

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

// One warp per token: the metric row as a unit vector (bf16), the merged row of every token
// (-1 for sources), and for destinations their metric row and token index by merged row.
__global__ void merge_setup_kernel(MergeGeo g, const __nv_bfloat16* kbar, __nv_bfloat16* m,
                                   __nv_bfloat16* m_dst, int* row_of, int* dst_tok) {
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (i >= g.N) return;
  const uint32_t u = reinterpret_cast<const uint32_t*>(kbar + (size_t)i * 64)[lane];
  const float a = bf16_lo(u), b = bf16_hi(u);
  float ss = a * a + b * b;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float inv = ss > 0.f ? rsqrtf(ss) : 0.f;
  const uint32_t mu = pack_bf16x2(a * inv, b * inv);
  reinterpret_cast<uint32_t*>(m + (size_t)i * 64)[lane] = mu;
  const int r = merged_row(g, i);
  if (r >= 0) reinterpret_cast<uint32_t*>(m_dst + (size_t)r * 64)[lane] = mu;
  if (lane == 0) {
    row_of[i] = r;
    if (r >= 0) dst_tok[r] = i;
  }
}

constexpr int kMatchWarps = 8;     // 16 source rows per warp
constexpr int kMatchDst = 64;      // destinations per shared-memory tile
constexpr int kMatchStride = 72;   // padded bf16 row: conflict-free fragment loads

// assign[i] = merged row of token i's destination: its own for destinations, the argmax of
// the cosine similarity over all destinations for sources.
__global__ void __launch_bounds__(32 * kMatchWarps) tome_match_kernel(
    MergeGeo g, const __nv_bfloat16* m, const __nv_bfloat16* m_dst, const int* row_of,
    int* assign) {
  __shared__ __align__(16) __nv_bfloat16 sd[kMatchDst * kMatchStride];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int r0 = (blockIdx.x * kMatchWarps + warp) * 16;  // this warp's 16 source rows
  // A fragments (16 rows x 64 channels), kept in registers for the whole sweep.
  uint32_t af[4][4];
  {
    const int ra = min(r0 + gq, g.N - 1), rb = min(r0 + gq + 8, g.N - 1);
    const uint32_t* pa = reinterpret_cast<const uint32_t*>(m + (size_t)ra * 64);
    const uint32_t* pb = reinterpret_cast<const uint32_t*>(m + (size_t)rb * 64);
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      af[kk][0] = __ldg(pa + 8 * kk + tq);
      af[kk][1] = __ldg(pb + 8 * kk + tq);
      af[kk][2] = __ldg(pa + 8 * kk + tq + 4);
      af[kk][3] = __ldg(pb + 8 * kk + tq + 4);
    }
  }
  float bv0 = -INFINITY, bv1 = -INFINITY;
  int bi0 = 0, bi1 = 0;  // a valid row even if no score compares (NaN metric)
  for (int n0 = 0; n0 < g.Np; n0 += kMatchDst) {
    __syncthreads();  // the previous tile is no longer read
    for (int q = threadIdx.x; q < kMatchDst * 8; q += blockDim.x) {  // 16-byte pieces
      const int rr = q >> 3, cc = q & 7;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (n0 + rr < g.Np) v = __ldg(reinterpret_cast<const uint4*>(m_dst + (size_t)(n0 + rr) * 64) + cc);
      *reinterpret_cast<uint4*>(&sd[rr * kMatchStride + cc * 8]) = v;
    }
    __syncthreads();
    float c[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      c[j][0] = c[j][1] = c[j][2] = c[j][3] = 0.f;
      const uint32_t* brow = reinterpret_cast<const uint32_t*>(&sd[(8 * j + gq) * kMatchStride]);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        mma16816(c[j], af[kk], brow[8 * kk + tq], brow[8 * kk + tq + 4]);
      if (n0 + 8 * j + 2 * tq >= g.Np) c[j][0] = c[j][2] = -INFINITY;
      if (n0 + 8 * j + 2 * tq + 1 >= g.Np) c[j][1] = c[j][3] = -INFINITY;
    }
    float m0 = c[0][0], m1 = c[0][2];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      m0 = fmax3(m0, c[j][0], c[j][1]);
      m1 = fmax3(m1, c[j][2], c[j][3]);
    }
    if (m0 > bv0) {  // first column (lowest index) holding the new maximum
      int best = 0x7fffffff;
#pragma unroll
      for (int j = 7; j >= 0; --j) {
        if (c[j][1] == m0) best = n0 + 8 * j + 2 * tq + 1;
        if (c[j][0] == m0) best = n0 + 8 * j + 2 * tq;
      }
      bv0 = m0;
      bi0 = best;
    }
    if (m1 > bv1) {
      int best = 0x7fffffff;
#pragma unroll
      for (int j = 7; j >= 0; --j) {
        if (c[j][3] == m1) best = n0 + 8 * j + 2 * tq + 1;
        if (c[j][2] == m1) best = n0 + 8 * j + 2 * tq;
      }
      bv1 = m1;
      bi1 = best;
    }
  }
  // Across the four threads of a row: larger score, then lower index.
#pragma unroll
  for (int o = 1; o < 4; o <<= 1) {
    const float v0 = __shfl_xor_sync(0xffffffffu, bv0, o), v1 = __shfl_xor_sync(0xffffffffu, bv1, o);
    const int i0 = __shfl_xor_sync(0xffffffffu, bi0, o), i1 = __shfl_xor_sync(0xffffffffu, bi1, o);
    if (v0 > bv0 || (v0 == bv0 && i0 < bi0)) { bv0 = v0; bi0 = i0; }
    if (v1 > bv1 || (v1 == bv1 && i1 < bi1)) { bv1 = v1; bi1 = i1; }
  }
  if (tq == 0) {
    const int ra = r0 + gq, rb = r0 + gq + 8;
    if (ra < g.N) assign[ra] = row_of[ra] >= 0 ? row_of[ra] : bi0;
    if (rb < g.N) assign[rb] = row_of[rb] >= 0 ? row_of[rb] : bi1;
  }
}

__global__ void merge_count_kernel(int N, const int* assign, int* cnt) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < N) atomicAdd(cnt + assign[i], 1);
}

// Exclusive scan of cnt[0..n) into offs[0..n] in one block of 1024 threads: each thread sums
// a contiguous run, the block scans the run totals, then each thread writes its run.
__global__ void __launch_bounds__(1024) scan_kernel(int n, const int* cnt, int* offs) {
  __shared__ int part[1024];
  const int tid = threadIdx.x;
  const int per = (n + 1023) / 1024;
  const int b = min(n, tid * per), e = min(n, b + per);
  int s = 0;
  for (int k = b; k < e; ++k) s += cnt[k];
  part[tid] = s;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {  // Hillis-Steele inclusive scan
    const int v = tid >= o ? part[tid - o] : 0;
    __syncthreads();
    part[tid] += v;
    __syncthreads();
  }
  int run = part[tid] - s;
  for (int k = b; k < e; ++k) {
    offs[k] = run;
    run += cnt[k];
  }
  if (tid == 1023) offs[n] = part[1023];
}

__global__ void merge_fill_kernel(int N, const int* assign, const int* offs, int* fill,
                                  int* members) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N) return;
  const int r = assign[i];
  members[offs[r] + atomicAdd(fill + r, 1)] = i;
}

// One warp per merged token: the fp32 mean of its members' rows of x~ (D = 256 C; lane l
// holds 16-byte chunks c 32 + l).
template <int C>
__global__ void merge_mean_kernel(int Np, const __nv_bfloat16* xt, const int* offs,
                                  const int* members, __nv_bfloat16* xm) {
  constexpr int D = 256 * C;
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= Np) return;
  const int b = offs[r], e = offs[r + 1];
  float acc[C][8];
#pragma unroll
  for (int c = 0; c < C; ++c)
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[c][k] = 0.f;
  for (int q = b; q < e; ++q) {
    const int i = members[q];
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(xt + (size_t)i * D + (c * 32 + lane) * 8));
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        acc[c][2 * k] += bf16_lo(w[k]);
        acc[c][2 * k + 1] += bf16_hi(w[k]);
      }
    }
  }
  const float inv = 1.f / (float)(e - b);
#pragma unroll
  for (int c = 0; c < C; ++c) {
    uint4 o;
    o.x = pack_bf16x2(acc[c][0] * inv, acc[c][1] * inv);
    o.y = pack_bf16x2(acc[c][2] * inv, acc[c][3] * inv);
    o.z = pack_bf16x2(acc[c][4] * inv, acc[c][5] * inv);
    o.w = pack_bf16x2(acc[c][6] * inv, acc[c][7] * inv);
    *reinterpret_cast<uint4*>(xm + (size_t)r * D + (c * 32 + lane) * 8) = o;
  }
}

// x[i] <- x[i] + ls (.) a[assign[i]]: the unmerge, LayerScale and residual add of the block's
// attention branch; one warp per token.
template <int C>
__global__ void unmerge_residual_kernel(int N, const int* assign, const __nv_bfloat16* a,
                                        const float* ls, __nv_bfloat16* x) {
  constexpr int D = 256 * C;
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (i >= N) return;
  const int r = assign[i];
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const int col = (c * 32 + lane) * 8;
    const uint4 ua = __ldg(reinterpret_cast<const uint4*>(a + (size_t)r * D + col));
    uint4* px = reinterpret_cast<uint4*>(x + (size_t)i * D + col);
    const uint4 ux = *px;
    const float4 l0 = __ldg(reinterpret_cast<const float4*>(ls + col));
    const float4 l1 = __ldg(reinterpret_cast<const float4*>(ls + col) + 1);
    const float lw[8] = {l0.x, l0.y, l0.z, l0.w, l1.x, l1.y, l1.z, l1.w};
    const uint32_t wa[4] = {ua.x, ua.y, ua.z, ua.w}, wx[4] = {ux.x, ux.y, ux.z, ux.w};
    uint32_t o[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
      o[k] = pack_bf16x2(fmaf(lw[2 * k], bf16_lo(wa[k]), bf16_lo(wx[k])),
                         fmaf(lw[2 * k + 1], bf16_hi(wa[k]), bf16_hi(wx[k])));
    *px = make_uint4(o[0], o[1], o[2], o[3]);
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
  g.Np = N <= P ? N : P + (N / P - 1) * g.Dv;
  return g;
}

cudaError_t launch_merge_prepare(const MergeGeo& g, int H, const __nv_bfloat16* xt,
                                 const __nv_bfloat16* w_qkv, const float* b_qkv,
                                 const MergeScratch& s, int num_sms, cudaStream_t st) {
  const int D = 64 * H;
  prof_before(VP_KERNEL_MERGE, st);
  metric_weights_kernel<<<(64 * D + 255) / 256, 256, 0, st>>>(w_qkv, b_qkv, H, D, s.wbar, s.bbar);
  prof_after(st);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  LinearArgs la{};
  la.M = g.N;
  la.N = 64;
  la.K = D;
  la.A = xt;
  la.W = s.wbar;
  la.bias = s.bbar;
  la.act = VP_ACT_NONE;
  la.out = s.kbar;
  la.err = s.err;
  e = launch_linear(la, num_sms, st);
  if (e != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  merge_setup_kernel<<<(g.N + 7) / 8, 256, 0, st>>>(g, s.kbar, s.m, s.m_dst, s.row_of, s.dst_tok);
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  tome_match_kernel<<<(g.N + 16 * kMatchWarps - 1) / (16 * kMatchWarps), 32 * kMatchWarps, 0, st>>>(
      g, s.m, s.m_dst, s.row_of, s.assign);
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(s.cnt, 0, (size_t)g.Np * sizeof(int), st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(s.fill, 0, (size_t)g.Np * sizeof(int), st)) != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  merge_count_kernel<<<(g.N + 255) / 256, 256, 0, st>>>(g.N, s.assign, s.cnt);
  scan_kernel<<<1, 1024, 0, st>>>(g.Np, s.cnt, s.offs);
  merge_fill_kernel<<<(g.N + 255) / 256, 256, 0, st>>>(g.N, s.assign, s.offs, s.fill, s.members);
  prof_extra_launch();
  prof_extra_launch();
  prof_after(st);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  prof_before(VP_KERNEL_MERGE, st);
  switch (D / 256) {
    case 1: merge_mean_kernel<1><<<(g.Np + 7) / 8, 256, 0, st>>>(g.Np, xt, s.offs, s.members, s.xm); break;
    case 2: merge_mean_kernel<2><<<(g.Np + 7) / 8, 256, 0, st>>>(g.Np, xt, s.offs, s.members, s.xm); break;
    case 3: merge_mean_kernel<3><<<(g.Np + 7) / 8, 256, 0, st>>>(g.Np, xt, s.offs, s.members, s.xm); break;
    case 4: merge_mean_kernel<4><<<(g.Np + 7) / 8, 256, 0, st>>>(g.Np, xt, s.offs, s.members, s.xm); break;
    case 8: merge_mean_kernel<8><<<(g.Np + 7) / 8, 256, 0, st>>>(g.Np, xt, s.offs, s.members, s.xm); break;
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

cudaError_t launch_unmerge_residual(int N, int D, const int* assign, const __nv_bfloat16* a,
                                    const float* ls, __nv_bfloat16* x, cudaStream_t st) {
  prof_before(VP_KERNEL_MERGE, st);
  switch (D / 256) {
    case 1: unmerge_residual_kernel<1><<<(N + 7) / 8, 256, 0, st>>>(N, assign, a, ls, x); break;
    case 2: unmerge_residual_kernel<2><<<(N + 7) / 8, 256, 0, st>>>(N, assign, a, ls, x); break;
    case 3: unmerge_residual_kernel<3><<<(N + 7) / 8, 256, 0, st>>>(N, assign, a, ls, x); break;
    case 4: unmerge_residual_kernel<4><<<(N + 7) / 8, 256, 0, st>>>(N, assign, a, ls, x); break;
    case 8: unmerge_residual_kernel<8><<<(N + 7) / 8, 256, 0, st>>>(N, assign, a, ls, x); break;
    default: prof_after(st); return cudaErrorInvalidValue;
  }
  prof_after(st);
  return cudaGetLastError();
}

}  // namespace vp
