/*
 * vp.h -- C ABI of the GB300 (sm_103a) library for VGGT-Prime's compute-adaptive
 * mixture-of-heads global attention.
 *
 * The method (VGGT-Prime, arXiv 2609.23733):
 *   - §4.1 (head saliency): per head h, gated attention pooling of the queries
 *       alpha_{h,i} = softmax_i( w_h^T (tanh(W_h q_{h,i}) (.) sigma(U_h q_{h,i})) ),
 *       q_pool_h = sum_i alpha_{h,i} q_{h,i},
 *     a single-query attention of q_pool_h over all N keys, r_h = softmax_j(c q_pool . k_j),
 *     and the saliency s_h = max_j r_h(j).
 *   - §4.2 (head routing, routing equation): full softmax attention if s_h >= tau_high,
 *     surrogate attention if tau_low < s_h < tau_high, mean pooling if s_h <= tau_low.
 *   - §4.3 (surrogate attention): C_h = r_h V_h, z_i = [v_i, C_h],
 *     y_i = C_h + sigma(MLP_gamma(z_i)) (.) MLP_delta(z_i).
 *   - Algorithm 1 (App. B): LN1 -> QKV -> router -> routed heads -> concat -> W_O ->
 *     LayerScale + residual -> LN2 -> FFN -> LayerScale + residual.
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller, unless a comment
 *     says "host".  The library never allocates or frees memory; scratch space is the
 *     caller's workspace (vp_workspace_size).  Dense tensors are row-major and
 *     contiguous; bf16 values are passed as their 16-bit patterns (vp_bf16).
 *   - stream is a cudaStream_t passed as void* (NULL = the legacy default stream).
 *     Calls enqueue kernels and return; they never synchronise the host.
 *   - Arguments are validated on the host before anything is enqueued; a failed
 *     check returns a status and enqueues nothing.  VP_ERR_CUDA reports a launch
 *     error.  Kernels that wait on asynchronous copies give up after a bounded
 *     time and record VP_DEVERR_* bits in a device error word inside the workspace
 *     (read it with vp_read_device_error); they never trap.
 *   - Shapes: head dim d = 64, router / surrogate hidden width L = 64, 1 <= H <= 32.
 *     Token-major layouts: QKV is [N][3][H][d] (Q|K|V, head, channel), the head
 *     outputs Y are [N][H][d] (= Concat(Y_1..Y_H), [N][D] with D = H d).
 */
#ifndef VP_H_
#define VP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t vp_bf16; /* bfloat16 bit pattern */

typedef enum vp_status {
  VP_OK = 0,
  VP_ERR_INVALID_ARG = 1,        /* null pointer where one is required, bad enum */
  VP_ERR_UNSUPPORTED_SHAPE = 2,  /* d != 64, L != 64, H outside 1..32, N < 1, ... */
  VP_ERR_ALIGNMENT = 3,          /* a pointer is not 16-byte aligned */
  VP_ERR_CUDA = 4,               /* a CUDA call or launch failed */
  VP_ERR_DEVICE_TIMEOUT = 5,     /* a kernel gave up waiting (see device error word) */
  VP_ERR_WORKSPACE = 6,          /* workspace missing or smaller than vp_workspace_size */
  VP_ERR_UNSUPPORTED_DEVICE = 7, /* the current device is not sm_103 */
  VP_ERR_STATIC_SCRATCH = 8      /* vp_router_noalloc: the call needs more scratch than its
                                    fixed buffer holds */
} vp_status;

/* Routed computation modes, §4.2 routing equation. */
typedef enum vp_mode { VP_MODE_MEAN = 0, VP_MODE_SURROGATE = 1, VP_MODE_FULL = 2 } vp_mode;

/* Bits of the device error word. */
#define VP_DEVERR_WAIT_TIMEOUT 1u   /* an mbarrier wait hit its time limit */
#define VP_DEVERR_NAN_SALIENCY 2u   /* a saliency was NaN; that head was routed to full */

typedef struct vp_dims {
  int32_t N;        /* tokens = views S x tokens per view P, all views at once (Algorithm 1) */
  int32_t H;        /* heads */
  int32_t d;        /* head dim, must be 64 */
  int32_t L;        /* router and surrogate hidden width, must be 64 (App. B) */
  float tau_low;    /* 0.01 in the paper (§4.2) */
  float tau_high;   /* 0.20 in the paper (§4.2); tau_low == tau_high gives the two-branch
                       router of §5's compute-mode ablation (mean and full only) */
  uint32_t variant; /* 0 = the method; else an OR of VP_VARIANT_* (§5 ablations) */
} vp_dims;

/* Ablation variants of §5 (vp_dims.variant).  Component ablation: */
#define VP_VARIANT_MEAN_QPOOL 1u        /* router: mean of the queries instead of the gated
                                           attention pooling (alpha = 1/N) */
#define VP_VARIANT_MEAN_CONTEXT 2u      /* surrogate: C_h = mean of V_h instead of r_h V_h */
#define VP_VARIANT_NO_RESIDUAL 4u       /* surrogate: y_i = C_h, no token-wise correction */
/* Compute-mode ablation: surrogate heads run linear attention (Katharopoulos et al. 2020,
   phi(x) = elu(x) + 1): y_i = phi(q_i)^T S_h / phi(q_i)^T z_h with S_h = sum_j phi(k_j) v_j^T,
   z_h = sum_j phi(k_j).  Not combinable with MEAN_CONTEXT or NO_RESIDUAL. */
#define VP_VARIANT_LINEAR_ATTENTION 8u

/* Router parameters (§4.1), per head; all device pointers. */
typedef struct vp_router_weights {
  const vp_bf16* W;     /* [H][L][d]  W_h */
  const vp_bf16* U;     /* [H][L][d]  U_h */
  const vp_bf16* w;     /* [H][L]     w_h */
  const float* bW;      /* [H][L] bias inside tanh, or NULL (zero; the paper writes none) */
  const float* bU;      /* [H][L] bias inside sigma, or NULL */
  const float* beta;    /* [H] routing-attention temperature, or NULL (1).  The routing
                           logits are beta_h / sqrt(d) * q_pool . k_j; the paper states no
                           scale, and beta_h = 1 gives full attention's 1/sqrt(d). */
} vp_router_weights;

/* Surrogate MLPs (§4.3), per head: Linear(2d -> L) -> GELU(erf) -> Linear(L -> d).
   The first layer's input is z = [v_i, C_h] (value first, context second). */
typedef struct vp_surrogate_weights {
  const vp_bf16* g1_w;  /* [H][L][2d] MLP_gamma layer 1 */
  const float* g1_b;    /* [H][L] */
  const vp_bf16* g2_w;  /* [H][d][L]  MLP_gamma layer 2 */
  const float* g2_b;    /* [H][d] */
  const vp_bf16* d1_w;  /* [H][L][2d] MLP_delta layer 1 */
  const float* d1_b;    /* [H][L] */
  const vp_bf16* d2_w;  /* [H][d][L]  MLP_delta layer 2 */
  const float* d2_b;    /* [H][d] */
} vp_surrogate_weights;

/*
 * Positional information and qk-norm of the QKV step (Algorithm 1 step (2): Q, K, V <-
 * QKV_h(X~) with positional information P).  The paper names P but does not define it; this
 * is the library's reading, applied in the QKV projection's epilogue before the router sees
 * Q and K:
 *   qk-norm: q_h <- LayerNorm_d(q_h) (.) q_norm_g + q_norm_b over each head's d channels
 *     (biased variance, norm_eps), the [d] parameters shared by all heads; likewise k.
 *   2-D rotary position embedding (RoFormer's rotation applied per image axis): a token's
 *     position inside its view is (0, 0) for the patch_start special tokens and
 *     (r + 1, c + 1) for patch r * grid_w + c.  Channels [0, d/2) rotate with the row and
 *     [d/2, d) with the column: within a half, channels i and i + d/4 (i < d/4) turn by the
 *     angle pos * rope_base^(-4 i / d), (a, b) -> (a cos - b sin, b cos + a sin).
 * Tokens are numbered view after view, tokens_per_view per view.  Positions up to
 * VP_ROPE_MAX_POS (grid rows + 1 and grid_w + 1).
 */
#define VP_ROPE_MAX_POS 1023
typedef struct vp_qk_options {
  const float* q_norm_g; const float* q_norm_b;  /* [d], or NULL: no q-norm (both or neither) */
  const float* k_norm_g; const float* k_norm_b;  /* [d], or NULL: no k-norm */
  float norm_eps;
  int32_t rope;             /* 1: 2-D rotary position embedding of q and k, 0: none */
  int32_t tokens_per_view;  /* P (N must be a multiple of it) */
  int32_t patch_start;      /* special tokens at the start of a view (camera + registers) */
  int32_t grid_w;           /* patches per grid row */
  float rope_base;          /* frequency base */
} vp_qk_options;

/*
 * Token merging around a block's attention (the paper's "VGGT-Prime & Token Merging": ToMe as
 * used by FastVGGT, 75 % or 90 % of the tokens merged; the paper gives no further detail, so
 * this is the library's reading, applied to LN1(X) of a block of vp_global_stack):
 *   destinations: the patch_start special tokens of every view, every token of the first
 *     view, and patch tokens p % stride == 0 of the other views; all others are sources
 *     (stride 4 merges ~75 % of the tokens, 10 ~90 %);
 *   metric: the head mean of the block's keys, mean_h (x~ W_k,h^T + b_k,h), as a unit vector;
 *   matching: every source joins the destination of largest cosine similarity over all
 *     destinations (ties: lowest merged row);
 *   merged token: the mean of a destination and the sources that joined it; the routed
 *     attention (QKV, router, modes, W_O) runs on the merged tokens in destination order,
 *     positions (vp_qk_options) taken from each destination's own token;
 *   unmerge: X_i += LS1 (.) A[merged row of i] for every token.
 * tokens_per_view must divide N.  assign_out: [N] int32 device buffer receiving the merged row
 * every token joined, or NULL.
 */
typedef struct vp_merge_options {
  int32_t stride;
  int32_t tokens_per_view;
  int32_t patch_start;
  int32_t* assign_out;
} vp_merge_options;

/* One global block of Algorithm 1; matrices in the nn.Linear layout [out][in]. */
typedef struct vp_layer_weights {
  const float* ln1_g; const float* ln1_b;       /* [D] */
  const vp_bf16* w_qkv; const float* b_qkv;     /* [3D][D], [3D]; rows ordered (Q|K|V, head, channel) */
  const vp_bf16* w_o; const float* b_o;         /* [D][D], [D] */
  const float* ls1;                             /* [D] LayerScale 1 */
  const float* ln2_g; const float* ln2_b;       /* [D] */
  const vp_bf16* w_fc1; const float* b_fc1;     /* [4D][D], [4D] */
  const vp_bf16* w_fc2; const float* b_fc2;     /* [D][4D], [D] */
  const float* ls2;                             /* [D] LayerScale 2 */
  vp_router_weights router;
  vp_surrogate_weights surrogate;
  const vp_qk_options* qk;                      /* HOST pointer: positional encoding and
                                                   qk-norm of the QKV step, or NULL (none) */
  const vp_merge_options* merge;                /* HOST pointer: token merging around the
                                                   block's attention, or NULL (none) */
} vp_layer_weights;

/* Workspace kinds for vp_workspace_size. */
#define VP_WS_ROUTER 0   /* vp_router, vp_head_attention (router scratch + linear-attention state) */
#define VP_WS_LAYER 1    /* vp_moh_global_attention */
#define VP_WS_STACK 2    /* vp_global_stack */
#define VP_WS_STACK_MERGE 3  /* vp_global_stack with token merging in some block */

/* Epilogues of vp_linear. */
#define VP_ACT_NONE 0
#define VP_ACT_GELU 1

/* Human-readable name of a status code (static string). */
const char* vp_status_string(vp_status s);

/* Bytes of workspace a call of kind `what` needs for these dims (host; writes *bytes). */
vp_status vp_workspace_size(const vp_dims* dims, int32_t what, size_t* bytes);

/* Reads and clears the device error word of a workspace: enqueues a copy on `stream`,
   synchronises that stream, writes the VP_DEVERR_* bits to *host_bits (host pointer).
   Returns VP_ERR_DEVICE_TIMEOUT if the wait-timeout bit was set, else VP_OK. */
vp_status vp_read_device_error(void* ws, size_t ws_bytes, uint32_t* host_bits, void* stream);

/*
 * vp_router -- §4.1 router and §4.2 routing for all heads of one layer.
 *   qkv        [N][3][H][d] bf16 (only Q and K, and V for ctx / mean_v, are read)
 *   force_modes [H] int32 or NULL: when given, modes[h] = force_modes[h] (values 0..2)
 *              instead of the §4.2 decision; s, q_pool and ctx are still computed.
 *   s          [H] float: saliency s_h = max_j r_h(j) (required)
 *   modes      [H] int32: routed mode (vp_mode) (required).  A NaN saliency routes to
 *              full and sets VP_DEVERR_NAN_SALIENCY.
 *   q_pool     [H][d] float or NULL: pooled queries
 *   ctx        [H][d] float or NULL: C_h = r_h V_h (§4.3)
 *   mean_v     [H][d] float or NULL: (1/N) sum_i V_{h,i}
 *   r          [H][N] float or NULL: routing vectors (costs an extra pass over K)
 *   ws         workspace of at least vp_workspace_size(dims, VP_WS_ROUTER) bytes
 */
vp_status vp_router(const vp_dims* dims, const vp_bf16* qkv, const vp_router_weights* rw,
                    const int32_t* force_modes, float* s, int32_t* modes, float* q_pool,
                    float* ctx, float* mean_v, float* r, void* ws, size_t ws_bytes, void* stream);

/*
 * vp_bin_heads -- groups heads by routed mode (§4.2: each head runs its case's
 * operator).  head_ids[H]: heads of mode 0 (mean), then 1 (surrogate), then 2 (full),
 * ascending head index inside each group; offsets[4]: group m is
 * head_ids[offsets[m] .. offsets[m+1]).  work (or NULL): [H * ceil(N/128)][2] int32
 * (head, query tile) pairs for the full-mode heads, head-major, tiles ascending;
 * n_work (or NULL): [1] int32 count of valid pairs.  One warp; no host sync.
 */
vp_status vp_bin_heads(int32_t H, int32_t N, const int32_t* modes, int32_t* head_ids,
                       int32_t* offsets, int32_t* work, int32_t* n_work, void* stream);

/*
 * vp_head_attention -- the routed head outputs Y (Algorithm 1 step 2), given the bins
 * of vp_bin_heads and the router's ctx / mean_v:
 *   full heads:      Y_h = softmax(Q_h K_h^T / sqrt d) V_h  (tcgen05 flash attention)
 *   surrogate heads: Y_h = C_h + sigma(MLP_gamma[v, C]) (.) MLP_delta[v, C]   (§4.3)
 *   mean heads:      Y_h = Broadcast(mean_v_h)
 *   y [N][H][d] bf16 (every head column is written).
 *   s_attn [H] float or NULL: the MaxAttn saliency s_h^attn = max_{i,j} A_h[i, j] of every
 *   full head (§3 "Head Saliency", defined in the appendix on saliency metrics: the largest
 *   entry of the head's post-softmax attention matrix), computed exactly, as a by-product of
 *   the flash kernel, from each query row's softmax denominator relative to its true maximum
 *   (max_j A_ij = 1 / sum_j exp(S_ij - max_j S_ij)).  Heads not in full mode get 0 (their
 *   attention matrix is never formed): force every head to full mode to obtain the exact
 *   saliency of all heads, e.g. to compare it with the router's estimate s_h.
 */
vp_status vp_head_attention(const vp_dims* dims, const vp_bf16* qkv, const int32_t* head_ids,
                            const int32_t* offsets, const float* ctx, const float* mean_v,
                            const vp_surrogate_weights* sw, vp_bf16* y, float* s_attn, void* ws,
                            size_t ws_bytes, void* stream);

/*
 * vp_linear -- out = residual + scale (.) act(A W^T + bias), the dense projections of
 * Algorithm 1 (QKV, W_O, FFN) on tcgen05 tensor cores with fp32 accumulation.
 *   A [M][K] bf16, W [Nout][K] bf16 (nn.Linear layout), bias [Nout] float or NULL,
 *   act VP_ACT_NONE / VP_ACT_GELU, scale [Nout] float or NULL (1), residual [M][Nout]
 *   bf16 or NULL (0; may alias out), out [M][Nout] bf16.  K % 8 == 0, Nout % 8 == 0; every
 *   pointer 16-byte aligned (the epilogue reads bias and scale four floats at a time).
 */
vp_status vp_linear(int32_t M, int32_t Nout, int32_t K, const vp_bf16* A, const vp_bf16* W,
                    const float* bias, int32_t act, const float* scale, const vp_bf16* residual,
                    vp_bf16* out, void* stream);

/* vp_layer_norm -- out = LN(x) over rows of length D (biased variance, eps), bf16 in/out,
   gamma / beta [D] float (Algorithm 1 steps 1 and 4).  D in {256, 512, 768, 1024, 2048, 4096};
   all pointers 16-byte aligned. */
vp_status vp_layer_norm(int32_t M, int32_t D, const vp_bf16* x, const float* gamma,
                        const float* beta, float eps, vp_bf16* out, void* stream);

/*
 * vp_moh_global_attention -- one routed global-attention layer, Algorithm 1 steps 2-3 up
 * to W_O (no LayerNorm, LayerScale or residual): out = Concat(Y_h) W_O^T + b_o, with
 * QKV = x W_qkv^T + b_qkv, router, bins and per-mode heads in between.
 *   x [N][D] bf16; out [N][D] bf16; force_modes [H] or NULL (see vp_router).
 *   qkv_out [N][3D] / y_out [N][D] bf16 or NULL: copies of the intermediates (debug).
 *   s_out [H] float / modes_out [H] int32 or NULL; s_attn_out [H] float or NULL: MaxAttn
 *   saliency of the full heads (see vp_head_attention).
 *   qk: HOST pointer, positional encoding and qk-norm of the QKV step (vp_qk_options), or
 *   NULL (none).
 */
vp_status vp_moh_global_attention(const vp_dims* dims, const vp_bf16* x, const vp_bf16* w_qkv,
                                  const float* b_qkv, const vp_bf16* w_o, const float* b_o,
                                  const vp_router_weights* rw, const vp_surrogate_weights* sw,
                                  const vp_qk_options* qk, const int32_t* force_modes, vp_bf16* out, vp_bf16* qkv_out,
                                  vp_bf16* y_out, float* s_out, float* s_attn_out,
                                  int32_t* modes_out, void* ws, size_t ws_bytes, void* stream);

/*
 * vp_global_stack -- n_layers global blocks (Algorithm 1) applied in place to x_inout
 * [N][D] bf16.  layers: HOST array of n_layers vp_layer_weights (their tensors are device
 * pointers).  force_modes [n_layers][H] int32 or NULL; modes_out / s_out / s_attn_out
 * [n_layers][H] or NULL (s_attn_out: MaxAttn saliency of the full heads, see
 * vp_head_attention).  ln_eps: LayerNorm epsilon (the paper does not state it; 1e-6 in the tests).
 * Every weight, bias, LayerNorm and LayerScale pointer must be 16-byte aligned.
 */
vp_status vp_global_stack(const vp_dims* dims, int32_t n_layers, vp_bf16* x_inout,
                          const vp_layer_weights* layers, const int32_t* force_modes,
                          int32_t* modes_out, float* s_out, float* s_attn_out, float ln_eps,
                          void* ws, size_t ws_bytes, void* stream);

/*
 * vp_global_stack_host -- vp_global_stack for tokens that live in host memory: copies x_in
 * (HOST pointer, [N][D] bf16) into x_dev (device, [N][D] bf16, caller-owned), runs the
 * n_layers blocks on x_dev in place, and copies the result to x_out (HOST pointer, [N][D]
 * bf16; may equal x_in).  Both copies are done by the library's own kernel, which reads and
 * writes the host memory through its device-visible address, so x_in and x_out must be
 * page-locked (cudaHostAlloc, cudaHostRegister, or a framework's pinned allocator): other
 * host memory returns VP_ERR_INVALID_ARG.  Everything is enqueued on `stream` and the call
 * returns without waiting: x_in is read, and x_out written, while the stream runs, so the caller
 * leaves both untouched (and allocated) until the stream has completed; x_out is then complete.
 * The other arguments are those of vp_global_stack.  All pointers 16-byte aligned.
 */
vp_status vp_global_stack_host(const vp_dims* dims, int32_t n_layers, const vp_bf16* x_in,
                               vp_bf16* x_out, vp_bf16* x_dev, const vp_layer_weights* layers,
                               const int32_t* force_modes, int32_t* modes_out, float* s_out,
                               float* s_attn_out, float ln_eps, void* ws, size_t ws_bytes,
                               void* stream);

/*
 * vp_router_noalloc -- vp_router without a workspace, for callers that cannot allocate
 * device memory when they call the router (for example a plug-in inside a host framework
 * whose memory pool already reserves the GPU's memory and forbids raw cudaMalloc, or a
 * service that must not allocate once it is running).  The paper has no counterpart: this
 * is an interface choice of the library, not a step of the method.
 *   Arguments, checks and outputs are those of vp_router, minus ws / ws_bytes (dims->variant
 *   included; H outside 1..32 is VP_ERR_UNSUPPORTED_SHAPE); the results are the same.  The
 *   router's scratch comes from one fixed device buffer inside the library, large enough for
 *   up to 32 heads (about 1.56 MiB, held on every GPU that loads the library until the
 *   process exits); a call that would need more returns VP_ERR_STATIC_SCRATCH.  The call
 *   allocates nothing itself (no cudaMalloc, cudaFree or allocating library routine).
 *   Set-up: the first call on a device (or the first after a device reset) looks up the
 *   buffer's device address with that device current.  CUDA loads a library's device code
 *   lazily by default, so that first call is also when the runtime loads the router's kernels
 *   and places the fixed buffer in device memory: make it before a host framework reserves
 *   the GPU's memory for its own pool, and before any stream capture.
 *   All calls on a device share the buffer, which keeps the last call's contents; the parts
 *   that must start at zero are cleared at the start of every call.  Calls that overlap on
 *   the GPU (unordered streams or host threads) race on the buffer: serialise them.
 *   Device error bits (a wait that timed out, a NaN saliency) accumulate in the buffer's
 *   error word until vp_router_noalloc_error reads them.
 */
vp_status vp_router_noalloc(const vp_dims* dims, const vp_bf16* qkv, const vp_router_weights* rw,
                            const int32_t* force_modes, float* s, int32_t* modes, float* q_pool,
                            float* ctx, float* mean_v, float* r, void* stream);

/* Reads and clears the device error word of vp_router_noalloc's fixed buffer on the current
   device, as vp_read_device_error does for a workspace: enqueues a copy on `stream`,
   synchronises that stream, writes the VP_DEVERR_* bits to *host_bits (host pointer).
   Returns VP_ERR_DEVICE_TIMEOUT if the wait-timeout bit was set, else VP_OK.  Allocates
   nothing. */
vp_status vp_router_noalloc_error(uint32_t* host_bits, void* stream);

/* Kernel classes reported by the launch profiler. */
#define VP_KERNEL_GEMM 0
#define VP_KERNEL_ROUTER_POOL 1
#define VP_KERNEL_ROUTER_KEYS 2
#define VP_KERNEL_ROUTER_R 3
#define VP_KERNEL_BIN_HEADS 4
#define VP_KERNEL_ATTN_FULL 5   /* all heads of a layer: full-attention kernel + cheap-heads
                                   kernel overlapping its tail, timed as one bracket */
#define VP_KERNEL_SURROGATE 6   /* (unused: surrogate and mean heads are timed with class 5) */
#define VP_KERNEL_MEAN 7
#define VP_KERNEL_LAYER_NORM 8  /* LayerNorm, and the stack's LN1 statistics pass and QKV
                                   weight fold */
#define VP_KERNEL_MERGE 9       /* token merging (vp_merge_options) and the unmerge */
#define VP_KERNEL_HOST_COPY 10  /* host <-> device copies of vp_global_stack_host */
#define VP_KERNEL_CLASSES 11

/*
 * Launch profiler (for benchmarks; not part of the method).  Between vp_profile_begin and
 * vp_profile_end every kernel the library launches on the calling host thread's current
 * device is bracketed by two CUDA events recorded on the launch's own stream.  Events are
 * created in vp_profile_begin (max_launches pairs) and destroyed in vp_profile_end; launches
 * beyond max_launches are counted but not timed.
 * vp_profile_end waits for the last recorded event, then writes (host pointers):
 *   n_launches[1]            kernels launched while profiling (all classes)
 *   launches[VP_KERNEL_CLASSES]  launches per class
 *   ms[VP_KERNEL_CLASSES]    summed event time per class, milliseconds
 */
vp_status vp_profile_begin(int32_t max_launches);
vp_status vp_profile_end(int32_t* n_launches, int32_t* launches, float* ms);

/*
 * Self-test of the bounded device waits (failure handling; not part of the method).
 * Enqueues on `stream` one warp that waits on an mbarrier nothing arrives on, with a time
 * limit of limit_ns nanoseconds instead of the kernels' 4 s, so that the wait gives up,
 * sets VP_DEVERR_WAIT_TIMEOUT in the workspace's error word and returns, leaving the context
 * usable; vp_read_device_error then reports VP_ERR_DEVICE_TIMEOUT.  The kernel runs for at
 * least limit_ns.
 *   ws, ws_bytes  any workspace of this library (its error word is the first 4 bytes; >= 256 B)
 *   limit_ns      1e6 .. 2e9 (1 ms .. 2 s), else VP_ERR_INVALID_ARG before any launch
 */
vp_status vp_selftest_wait_timeout(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* VP_H_ */
