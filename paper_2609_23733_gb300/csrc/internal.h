// Internal launchers and workspace layout of the sm_103a library (not part of the ABI).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "vp.h"

namespace vp {

constexpr int kHeadDim = 64;
constexpr int kHidden = 64;
constexpr int kMaxHeads = 32;
constexpr int kQTile = 128;          // query rows per full-attention work item
constexpr int kPoolSplitMax = 64;    // CTAs per head in the pooling sweep
constexpr int kKeySplitMax = 64;     // CTAs per head in the key sweep
constexpr int kPoolPartial = 2 + kHeadDim;          // (max, sum, sum p q[64])
constexpr int kKeyPartial = 2 + 2 * kHeadDim;       // (max, sum, sum p v[64], sum v[64])

// Router scratch carved from the caller's workspace (all device pointers).
struct RouterScratch {
  unsigned int* err;            // device error word (first 256 bytes of the workspace)
  unsigned int* counters;       // [2 * kMaxHeads + 2] last-CTA counters, zeroed per call
  float* pool_part;             // [H][kPoolSplitMax][kPoolPartial]
  float* key_part;              // [H][kKeySplitMax][kKeyPartial]
  float* q_pool;                // [H][64]
  float* key_stats;             // [H][2] (global max of scaled logits, sum of exp)
  float* s;                     // [H]
  int32_t* modes;               // [H]
  float* ctx;                   // [H][64]
  float* mean_v;                // [H][64]
  int32_t* head_ids;            // [H]
  int32_t* offsets;             // [4]
  unsigned int* cheap_counter;  // work counter of the cheap head modes
  float* lin_state;             // [H][kLinState] linear-attention state (after the router part)
  float* fa_part;               // [kFaTailUnits][4 chains][128 rows][64] split-tail partial O
  float* fa_stats;              // [kFaTailUnits][4 chains][128 rows][4] (m, l, xmax, -)
  unsigned int* fa_count;       // [kFaTailUnits][4 chains][4 quarters] split arrivals
  float* wo_bias;               // [kMaxHeads * 64] W_O bias with the mean heads folded in
};

// Full attention splits the work items of its last, partial round along the keys over the
// CTAs that would otherwise idle; the partial results need this much scratch (units = groups
// x splits of that round, at most one per CTA).
constexpr int kFaTailUnits = 512;
constexpr size_t kFaPartFloats = (size_t)kFaTailUnits * 4 * 128 * 64;
constexpr size_t kFaStatsFloats = (size_t)kFaTailUnits * 4 * 128 * 4;
constexpr size_t kFaCountWords = (size_t)kFaTailUnits * 4 * 4;

// Linear-attention state of one head (the §5 compute-mode ablation): S_h [64 c][64 e] =
// sum_j phi(k_j)[c] v_j[e], then z_h [64] = sum_j phi(k_j), fp32.
constexpr int kLinState = 64 * 64 + 64;

// Bytes of the router's scratch (what vp_router touches): laid out for kMaxHeads heads
// whatever H is (carve_router_scratch).
constexpr size_t router_scratch_bytes(int /*H*/) {
  return ((size_t)256                                           // error word
          + 512                                                 // counters
          + (size_t)kMaxHeads * kPoolSplitMax * kPoolPartial * 4
          + (size_t)kMaxHeads * kKeySplitMax * kKeyPartial * 4
          + (size_t)kMaxHeads * 64 * 4 * 3                      // q_pool, ctx, mean_v
          + (size_t)kMaxHeads * 4 * 4                           // key_stats, s, modes
          + 256                                                 // head_ids, offsets
          + 4095) & ~(size_t)4095;
}
// Router scratch + linear-attention state: the workspace of the head modes.
size_t heads_scratch_bytes(int H);
RouterScratch carve_router_scratch(void* ws, int H);

struct RouterArgs {
  int N, H;
  float tau_low, tau_high;
  uint32_t variant;  // VP_VARIANT_* bits
  const __nv_bfloat16* qkv;
  const __nv_bfloat16* W;
  const __nv_bfloat16* U;
  const __nv_bfloat16* w;
  const float* bW;
  const float* bU;
  const float* beta;
  const int32_t* force_modes;
  // Outputs (NULL = do not copy out); the scratch copies are always written.
  float* s_out;
  int32_t* modes_out;
  float* q_pool_out;
  float* ctx_out;
  float* mean_v_out;
  float* r_out;
};

cudaError_t launch_router(const RouterArgs& a, const RouterScratch& sc, int num_sms,
                          cudaStream_t st);

// Host-side argument checks shared by the router entry points (api.cu): dims (shape, taus,
// variant bits), router weights (presence, 16-byte alignment of W and U), and the
// RouterArgs of a call (outputs left NULL).
vp_status check_dims(const vp_dims* dm);
vp_status check_router_weights(const vp_router_weights* rw);
RouterArgs make_router_args(const vp_dims* dm, const vp_bf16* qkv, const vp_router_weights* rw,
                            const int32_t* force_modes);
cudaError_t launch_bin_heads(int H, int N, const int32_t* modes, int32_t* head_ids,
                             int32_t* offsets, int32_t* work, int32_t* n_work, cudaStream_t st);

struct SurrogateArgs {
  const __nv_bfloat16* g1_w; const float* g1_b;
  const __nv_bfloat16* g2_w; const float* g2_b;
  const __nv_bfloat16* d1_w; const float* d1_b;
  const __nv_bfloat16* d2_w; const float* d2_b;
};

struct HeadAttnArgs {
  int N, H;
  const __nv_bfloat16* qkv;
  const int32_t* head_ids;
  const int32_t* offsets;
  const float* ctx;
  const float* mean_v;
  SurrogateArgs sw;
  __nv_bfloat16* y;
  float* s_attn;                // [H] MaxAttn saliency of the full heads, or NULL
  uint32_t variant;             // VP_VARIANT_* bits
  float* lin_state;             // [H][kLinState] (VP_VARIANT_LINEAR_ATTENTION only)
  float* fa_part;               // split-tail scratch of the full-attention kernel
  float* fa_stats;
  unsigned int* fa_count;       // zeroed by the launcher
  unsigned int* err;
  unsigned int* cheap_counter;  // one word of scratch, zeroed by the launcher
  int skip_mean_y;              // 1: the mean heads' rows of Y are not written (folded into W_O)
};

// Full-mode heads (attn_full.cu).
cudaError_t launch_full_heads(const HeadAttnArgs& a, int num_sms, cudaStream_t st);
// Surrogate (§4.3, the method's form and the mean-context ablation) and mean heads on the
// tensor cores, queued behind the full-attention kernel (heads_cheap_tc.cu).
cudaError_t launch_cheap_heads_tc(const HeadAttnArgs& a, int num_sms, cudaStream_t st);
// §5 linear-attention state of every surrogate head into a.lin_state (zeroed by the caller),
// on the tensor cores (linear_attn_tc.cu).
cudaError_t launch_linear_state_tc(const HeadAttnArgs& a, int num_sms, cudaStream_t st);
// §5 linear-attention output of every surrogate head from that state, y_i = phi(q_i)^T S /
// phi(q_i)^T z, on the tensor cores (linear_attn_tc.cu).
cudaError_t launch_linear_apply_tc(const HeadAttnArgs& a, int num_sms, cudaStream_t st);
// All heads of a layer: full-mode heads, then surrogate and mean heads overlapped with the
// full-attention tail (heads_cheap.cu).
cudaError_t launch_heads(const HeadAttnArgs& a, int num_sms, cudaStream_t st);

struct LinearArgs {
  int M, N, K;
  const __nv_bfloat16* A;
  const __nv_bfloat16* W;
  const float* bias;
  int act;
  const float* scale;
  const __nv_bfloat16* residual;
  __nv_bfloat16* out;
  unsigned int* err;   // may be NULL (vp_linear has no workspace): a private word is used
  // LayerNorm folded into the projection (A is the un-normalised residual stream): with
  // W' = W diag(gamma), c = W' 1 and bias' = b + W beta prepared by launch_ln_fold_weights,
  //   LN(A) W^T + b = rstd_r (A W'^T - mu_r c^T) + bias',
  // mu_r, rstd_r combined from ln_part (K % 128 == 0).  ln_part NULL: no LayerNorm.
  const float2* ln_part;  // [M][K / 128] (mean, M2) of the 128-column blocks of A's rows
  const float* ln_c;      // [N] column sums of W'
  float ln_eps;
  float2* part_out;       // [M][N / 128] (mean, M2) blocks of the output rows, or NULL (N % 128 == 0)
  // QKV projection with qk-norm and / or 2-D RoPE (vp_qk_options) on its first qk_cols = 2D
  // columns (Q | K; a multiple of 256, so a tile half holds two whole heads of Q or of K):
  // LayerNorm over each head's 64 channels with qn_* / kn_* ([64], NULL: none), then the
  // rotation by rope_cs [pos][16] (cos, sin) at the token's (row, column) position.
  int qk_cols;
  const float* qn_g;
  const float* qn_b;
  const float* kn_g;
  const float* kn_b;
  float qk_eps;
  const float2* rope_cs;  // NULL: no RoPE
  int tok_per_view, patch_start, grid_w;
  const int32_t* tok_index;  // RoPE: token index of output row r (merged tokens), or NULL (r)
  // K-blocks left out (W_O with mean heads folded into its bias): the 64-column blocks kb =
  // skip_ids[skip_off[0] .. skip_off[1]) of A and W contribute nothing (K == 64 x blocks <=
  // 32 x 64; no LayerNorm fold, no qk columns).  NULL: none.
  const int32_t* skip_ids;
  const int32_t* skip_off;
};
cudaError_t launch_linear(const LinearArgs& a, int num_sms, cudaStream_t st);

// W_O's bias with the mean heads folded in (Algorithm 1, step 3): a mean head's output is the
// same row mu_h = bf16(mean_v[h]) for every token, so its part of Y W_O^T is one vector:
//   bias_out[n] = b_o[n] + sum over mean heads h of sum_k mu_h[k] W_O[n][64 h + k]
// (mean heads: head_ids[offsets[0] .. offsets[1]); b_o NULL: 0).  W_O [D][H 64] bf16.
cudaError_t launch_wo_mean_fold(int D, int H, const __nv_bfloat16* w_o, const float* b_o,
                                const float* mean_v, const int32_t* head_ids,
                                const int32_t* offsets, float* bias_out, cudaStream_t st);

// Per-row LayerNorm statistics as (mean, M2) of 128-column blocks: x [M][D] bf16 ->
// part [M][D / 128] float2 (D % 256 == 0, D <= 4096).
cudaError_t launch_ln_partials(int M, int D, const __nv_bfloat16* x, float2* part, cudaStream_t st);
// The folded LayerNorm's weights for a projection W [Nout][K] (nn.Linear layout):
// Wp = W diag(g) (bf16), c[o] = sum_k Wp[o][k] (of the bf16 Wp), bp[o] = b[o] + sum_k W[o][k] beta[k]
// (b NULL: 0).  K % 256 == 0, K <= 4096.
// cos / sin of p * base^(-i / 16), p = 0 .. max_pos, i = 0 .. 15: table [max_pos + 1][16].
cudaError_t launch_rope_table(int max_pos, float base, float2* table, cudaStream_t st);
cudaError_t launch_ln_fold_weights(int Nout, int K, const __nv_bfloat16* W, const float* g,
                                   const float* beta, const float* b, __nv_bfloat16* Wp,
                                   float* c, float* bp, cudaStream_t st);

// Token merging around a block's attention (merge.cu, vp_merge_options).
struct MergeGeo {
  int N, P, ps, stride;
  int Dv;  // destinations per view after the first
  int Sv;  // sources per view after the first (P - Dv)
  int Np;  // merged tokens
  int Ns;  // sources (N - Np)
};
MergeGeo make_merge_geo(int N, int P, int ps, int stride);
struct MergeScratch {
  __nv_bfloat16* wbar;   // [64][D] head-mean key weights
  float* bbar;           // [64]
  __nv_bfloat16* kbar;   // [N][64] metric
  __nv_bfloat16* m_src;  // [Ns][64] unit metric of the sources (in token order)
  __nv_bfloat16* m_dst;  // [Np][64] unit metric of the destinations (by merged row)
  int* row_of;           // [N] merged row of a destination, -1 for sources
  int* dst_tok;          // [Np] token of merged row
  int* assign;           // [N] merged row every token joins
  int* cnt;              // [Np]
  int* offs;             // [Np + 1]
  int* fill;             // [Np]
  int* members;          // [N]
  unsigned long long* best;  // [Ns] matching: (score, destination) keys, 0 before the matching
  __nv_bfloat16* xm;     // [Np][D] merged tokens
  float* slots;          // [ceil(N / 32)][2][D] partial sums of the merged tokens (merge means)
  unsigned int* err;
};
// Bytes of MergeScratch::slots for N tokens of D channels.
inline size_t merge_slot_bytes(size_t N, size_t D) { return (N + 31) / 32 * 2 * D * sizeof(float); }
// LN1 of the merging, folded (its output is never stored): the row statistics of x and the
// scratch of the folded metric weights.
struct MergeLn {
  const float2* part;        // [N][D / 128] (mean, M2) of x's 128-column blocks
  const float* g;            // [D] LN1 gamma
  const float* b;            // [D] LN1 beta
  float eps;
  __nv_bfloat16* w_fold;     // [64][D] head-mean key weights with gamma folded in
  float* c_fold;             // [64] their row sums
  float* b_fold;             // [64] folded bias
};
// x [N][D] (the block's input) -> s.assign, s.dst_tok, s.xm (D = 64 H, D % 256 == 0).
cudaError_t launch_merge_prepare(const MergeGeo& g, int H, const __nv_bfloat16* x,
                                 const MergeLn& ln, const __nv_bfloat16* w_qkv,
                                 const float* b_qkv, const MergeScratch& s, int num_sms,
                                 cudaStream_t st);
// x[i] = bf16(x[i] + ls (.) a[assign[i]]) and z[i] = LN(x[i]) (g, b, eps) over N rows of D
// channels.
cudaError_t launch_unmerge_ln(int N, int D, const int* assign, const __nv_bfloat16* a,
                              const float* ls, const float* g, const float* b, float eps,
                              __nv_bfloat16* x, __nv_bfloat16* z, cudaStream_t st);

// Copy of `bytes` (a multiple of 16; both addresses 16-byte aligned and device-visible, e.g.
// pinned host memory) by the SMs (host_copy.cu).
cudaError_t launch_host_copy(const void* src, void* dst, size_t bytes, int num_sms,
                             cudaStream_t st);

// One warp waiting on an mbarrier that never completes, bounded by limit_ns (self-test of the
// wait limit; sets VP_DEVERR_WAIT_TIMEOUT in *err).
cudaError_t launch_wait_selftest(unsigned int* err, unsigned long long limit_ns, cudaStream_t st);

cudaError_t launch_layer_norm(int M, int D, const __nv_bfloat16* x, const float* g,
                              const float* b, float eps, __nv_bfloat16* out, cudaStream_t st);

// Host-side TMA descriptor creation (driver entry point fetched at run time).
// 2-D bf16 tensor [rows][cols] with a row pitch of `pitch_elems`, box of box_cols x box_rows,
// 128-byte swizzle, zero fill out of bounds.
cudaError_t make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows,
                              uint64_t pitch_elems, uint32_t box_cols, uint32_t box_rows,
                              int swizzle_bytes = 128);

// Launch profiler hooks (no-ops unless vp_profile_begin is active).
void prof_before(int kind, cudaStream_t st);
void prof_after(cudaStream_t st);
void prof_extra_launch();  // one more kernel inside the current bracket

int device_sm_count();
bool device_is_sm103();

}  // namespace vp
