// C ABI of the library (include/vp.h): argument checks, workspace carving, launches.
// Every entry point validates its arguments on the host before it enqueues anything and
// returns a vp_status; kernels run on the caller's stream and nothing here synchronises
// the host (except vp_read_device_error, whose purpose is to read the device error word).
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <string.h>

#include <mutex>

#include "internal.h"
#include "vp.h"

namespace vp {

// ------------------------------------------------------------------ device queries
namespace {
struct DevInfo {
  int sms = 0;
  int sm103 = -1;
};
DevInfo g_dev[64];
std::mutex g_dev_mu;

DevInfo& dev_info() {
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DevInfo& d = g_dev[dev & 63];
  if (d.sm103 < 0) {
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
    d.sm103 = (major == 10 && minor == 3) ? 1 : 0;
  }
  return d;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;
std::once_flag g_encode_once;
}  // namespace

// ------------------------------------------------------------------ launch profiler
namespace {
struct ProfRecord {
  int kind;
  cudaEvent_t start, stop;
};
struct Profiler {
  bool active = false;
  int max = 0, used = 0, launches = 0;
  int per_class[VP_KERNEL_CLASSES] = {};
  ProfRecord* rec = nullptr;
  cudaEvent_t pending = nullptr;  // start event of the launch being bracketed
  int pending_kind = -1;
};
thread_local Profiler g_prof;
}  // namespace

void prof_before(int kind, cudaStream_t st) {
  Profiler& p = g_prof;
  if (!p.active) return;
  ++p.launches;
  ++p.per_class[kind];
  p.pending = nullptr;
  if (p.used < p.max) {
    ProfRecord& r = p.rec[p.used];
    r.kind = kind;
    cudaEventRecord(r.start, st);
    p.pending = r.stop;
    p.pending_kind = kind;
  }
}

void prof_extra_launch() {
  if (g_prof.active) ++g_prof.launches;
}

void prof_after(cudaStream_t st) {
  Profiler& p = g_prof;
  if (!p.active || !p.pending) return;
  cudaEventRecord(p.pending, st);
  p.pending = nullptr;
  ++p.used;
}

int device_sm_count() { return dev_info().sms; }
bool device_is_sm103() { return dev_info().sm103 == 1; }

cudaError_t make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows,
                              uint64_t pitch_elems, uint32_t box_cols, uint32_t box_rows,
                              int swizzle_bytes) {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<EncodeTiledFn>(fn);
  });
  if (!g_encode) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {pitch_elems * 2};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                        : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                              : CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// ------------------------------------------------------------------ shared argument checks
// (also used by the fixed-scratch router, router_noalloc.cu)
vp_status check_dims(const vp_dims* dm) {
  if (!dm) return VP_ERR_INVALID_ARG;
  if (dm->d != kHeadDim || dm->L != kHidden || dm->H < 1 || dm->H > kMaxHeads || dm->N < 1)
    return VP_ERR_UNSUPPORTED_SHAPE;
  if (!(dm->tau_low == dm->tau_low) || !(dm->tau_high == dm->tau_high)) return VP_ERR_INVALID_ARG;
  const uint32_t known = VP_VARIANT_MEAN_QPOOL | VP_VARIANT_MEAN_CONTEXT | VP_VARIANT_NO_RESIDUAL |
                         VP_VARIANT_LINEAR_ATTENTION;
  if (dm->variant & ~known) return VP_ERR_INVALID_ARG;
  if ((dm->variant & VP_VARIANT_LINEAR_ATTENTION) &&
      (dm->variant & (VP_VARIANT_MEAN_CONTEXT | VP_VARIANT_NO_RESIDUAL)))
    return VP_ERR_INVALID_ARG;  // those two modify the §4.3 surrogate, which linear attention replaces
  return VP_OK;
}

vp_status check_router_weights(const vp_router_weights* rw) {
  if (!rw || !rw->W || !rw->U || !rw->w) return VP_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(rw->W) & 15u) || (reinterpret_cast<uintptr_t>(rw->U) & 15u))
    return VP_ERR_ALIGNMENT;
  return VP_OK;
}

RouterArgs make_router_args(const vp_dims* dm, const vp_bf16* qkv, const vp_router_weights* rw,
                            const int32_t* force_modes) {
  RouterArgs a{};
  a.N = dm->N;
  a.H = dm->H;
  a.tau_low = dm->tau_low;
  a.tau_high = dm->tau_high;
  a.variant = dm->variant;
  a.qkv = reinterpret_cast<const __nv_bfloat16*>(qkv);
  a.W = reinterpret_cast<const __nv_bfloat16*>(rw->W);
  a.U = reinterpret_cast<const __nv_bfloat16*>(rw->U);
  a.w = reinterpret_cast<const __nv_bfloat16*>(rw->w);
  a.bW = rw->bW;
  a.bU = rw->bU;
  a.beta = rw->beta;
  a.force_modes = force_modes;
  return a;
}

}  // namespace vp

using namespace vp;

namespace {

constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

vp_status check_device() {
  if (!device_is_sm103()) return VP_ERR_UNSUPPORTED_DEVICE;
  return VP_OK;
}

// RoPE cos / sin table (vp_qk_options), [VP_ROPE_MAX_POS + 1][16] float2.
constexpr size_t kRopeTableBytes = (size_t)(VP_ROPE_MAX_POS + 1) * 16 * sizeof(float2);

size_t layer_ws_bytes(const vp_dims* dm) {
  const size_t N = dm->N, D = (size_t)dm->H * kHeadDim;
  return heads_scratch_bytes(dm->H) + align_up(kRopeTableBytes) + align_up(N * 3 * D * 2) +
         align_up(N * D * 2);
}

// The stack's LayerNorm scratch: LN1's row statistics (per 128-column block), the current
// block's folded QKV weights with their column sums and biases, and the LN2 output.
size_t ln_scratch_bytes(size_t N, size_t D) {
  return align_up(N * (D / 128) * sizeof(float2)) + align_up(3 * D * D * 2) +
         2 * align_up(3 * D * sizeof(float)) + align_up(N * D * 2);
}

size_t stack_ws_bytes(const vp_dims* dm) {
  const size_t N = dm->N, D = (size_t)dm->H * kHeadDim;
  // LayerNorm scratch + one region shared by {QKV, Y} and the FFN hidden layer.
  return heads_scratch_bytes(dm->H) + align_up(kRopeTableBytes) + ln_scratch_bytes(N, D) +
         align_up(N * 4 * D * 2);
}

// Token-merging scratch (vp_merge_options): metric weights and rows, the destination and
// membership tables, the merged tokens and their attention output (whose region holds the
// partial sums of the merged tokens before the attention writes it).
size_t merge_scratch_bytes(size_t N, size_t D) {
  return align_up(64 * D * 2) + align_up(64 * sizeof(float)) + 3 * align_up(N * 64 * 2) +
         7 * align_up((N + 1) * sizeof(int)) + align_up(N * sizeof(unsigned long long)) +
         align_up(N * D * 2) + align_up(std::max(N * D * 2, merge_slot_bytes(N, D)));
}

size_t stack_merge_ws_bytes(const vp_dims* dm) {
  const size_t N = dm->N, D = (size_t)dm->H * kHeadDim;
  return stack_ws_bytes(dm) + merge_scratch_bytes(N, D);
}

vp_status check_merge(const vp_merge_options* mo, const vp_dims* dm) {
  if (!mo) return VP_OK;
  if (mo->stride < 1 || mo->tokens_per_view < 1 || mo->patch_start < 0 ||
      mo->patch_start > mo->tokens_per_view)
    return VP_ERR_INVALID_ARG;
  if (dm->N % mo->tokens_per_view != 0) return VP_ERR_UNSUPPORTED_SHAPE;
  return VP_OK;
}

// Host-side checks of vp_qk_options; *max_pos: the largest position index a token takes.
vp_status check_qk(const vp_qk_options* qk, const vp_dims* dm, int* max_pos) {
  *max_pos = 0;
  if (!qk) return VP_OK;
  if (!qk->q_norm_g != !qk->q_norm_b || !qk->k_norm_g != !qk->k_norm_b) return VP_ERR_INVALID_ARG;
  if ((qk->q_norm_g && (!aligned16(qk->q_norm_g) || !aligned16(qk->q_norm_b))) ||
      (qk->k_norm_g && (!aligned16(qk->k_norm_g) || !aligned16(qk->k_norm_b))))
    return VP_ERR_ALIGNMENT;
  if ((qk->q_norm_g || qk->k_norm_g) && !(qk->norm_eps >= 0.f)) return VP_ERR_INVALID_ARG;
  if (qk->rope != 0 && qk->rope != 1) return VP_ERR_INVALID_ARG;
  if (qk->rope) {
    if (qk->tokens_per_view < 1 || qk->patch_start < 0 || qk->grid_w < 1 ||
        qk->patch_start > qk->tokens_per_view || !(qk->rope_base > 0.f))
      return VP_ERR_INVALID_ARG;
    if (dm->N % qk->tokens_per_view != 0) return VP_ERR_UNSUPPORTED_SHAPE;
    const int patches = qk->tokens_per_view - qk->patch_start;
    const int rows = (patches + qk->grid_w - 1) / qk->grid_w;
    *max_pos = rows > qk->grid_w ? rows : qk->grid_w;
    if (*max_pos > VP_ROPE_MAX_POS) return VP_ERR_UNSUPPORTED_SHAPE;
  }
  return VP_OK;
}

// The QKV projection's qk-norm / RoPE settings and the device RoPE table.
struct QkArgs {
  const vp_qk_options* o;
  const float2* table;
  const int32_t* tok_index;  // token of each row (merged tokens), or NULL
};

void set_qk(LinearArgs& la, const QkArgs* qk, int D) {
  if (!qk || !qk->o) return;
  const vp_qk_options& o = *qk->o;
  if (!o.q_norm_g && !o.k_norm_g && !o.rope) return;
  la.qk_cols = 2 * D;
  la.qn_g = o.q_norm_g;
  la.qn_b = o.q_norm_b;
  la.kn_g = o.k_norm_g;
  la.kn_b = o.k_norm_b;
  la.qk_eps = o.norm_eps;
  if (o.rope) {
    la.rope_cs = qk->table;
    la.tok_per_view = o.tokens_per_view;
    la.patch_start = o.patch_start;
    la.grid_w = o.grid_w;
    la.tok_index = qk->tok_index;
  }
}

// Row widths the LayerNorm kernel is instantiated for.
bool ln_width_supported(int D) {
  return D == 256 || D == 512 || D == 768 || D == 1024 || D == 2048 || D == 4096;
}

vp_status from_cuda(cudaError_t e) { return e == cudaSuccess ? VP_OK : VP_ERR_CUDA; }

#define VP_TRY(x)                      \
  do {                                 \
    vp_status _s = (x);                \
    if (_s != VP_OK) return _s;        \
  } while (0)

vp_status check_surrogate_weights(const vp_surrogate_weights* sw) {
  if (!sw || !sw->g1_w || !sw->g1_b || !sw->g2_w || !sw->g2_b || !sw->d1_w || !sw->d1_b ||
      !sw->d2_w || !sw->d2_b)
    return VP_ERR_INVALID_ARG;
  if (!aligned16(sw->g1_w) || !aligned16(sw->g2_w) || !aligned16(sw->d1_w) || !aligned16(sw->d2_w))
    return VP_ERR_ALIGNMENT;
  return VP_OK;
}

SurrogateArgs make_surrogate_args(const vp_surrogate_weights* sw) {
  SurrogateArgs s;
  s.g1_w = reinterpret_cast<const __nv_bfloat16*>(sw->g1_w);
  s.g1_b = sw->g1_b;
  s.g2_w = reinterpret_cast<const __nv_bfloat16*>(sw->g2_w);
  s.g2_b = sw->g2_b;
  s.d1_w = reinterpret_cast<const __nv_bfloat16*>(sw->d1_w);
  s.d1_b = sw->d1_b;
  s.d2_w = reinterpret_cast<const __nv_bfloat16*>(sw->d2_w);
  s.d2_b = sw->d2_b;
  return s;
}

// Runs the three mode kernels for bins already in device memory.
// skip_mean_y: the mean heads' rows of Y are left unwritten (their part of W_O is folded into
// its bias, launch_wo_mean_fold).
vp_status run_heads(const vp_dims* dm, const __nv_bfloat16* qkv, const int32_t* head_ids,
                    const int32_t* offsets, const float* ctx, const float* mean_v,
                    const vp_surrogate_weights* sw, __nv_bfloat16* y, float* s_attn,
                    const RouterScratch& sc, cudaStream_t st, bool skip_mean_y = false) {
  HeadAttnArgs ha{};
  ha.N = dm->N;
  ha.H = dm->H;
  ha.qkv = qkv;
  ha.head_ids = head_ids;
  ha.offsets = offsets;
  // §5 component ablation "Context": the surrogate's context is the mean-pooled value vector.
  ha.ctx = (dm->variant & VP_VARIANT_MEAN_CONTEXT) ? mean_v : ctx;
  ha.mean_v = mean_v;
  ha.variant = dm->variant;
  ha.lin_state = sc.lin_state;
  ha.fa_part = sc.fa_part;
  ha.fa_stats = sc.fa_stats;
  ha.fa_count = sc.fa_count;
  ha.sw = make_surrogate_args(sw);
  ha.y = y;
  ha.s_attn = s_attn;
  ha.err = sc.err;
  ha.cheap_counter = sc.cheap_counter;
  ha.skip_mean_y = skip_mean_y ? 1 : 0;
  return from_cuda(launch_heads(ha, device_sm_count(), st));
}

// QKV projection -> router -> bins -> heads -> W_O (+ optional LayerScale / residual).
// A mean head's rows of Y are all mu_h = bf16(mean of V_h), so its part of Y W_O^T is the
// same vector for every token: it goes into W_O's bias (launch_wo_mean_fold) and the W_O GEMM
// leaves that head's 64 K columns out; its rows of Y are written only when the caller asked
// for Y (keep_mean_y).
// LayerNorm folded into a layer's QKV projection: xin is then the raw residual stream and
// w_qkv / b_qkv the folded weights (see LinearArgs).
struct LnFold {
  const float2* part_in;
  const float* c;
  float eps;
};

vp_status run_layer(const vp_dims* dm, const __nv_bfloat16* xin, const vp_bf16* w_qkv,
                    const float* b_qkv, const vp_bf16* w_o, const float* b_o, const float* ls1,
                    const __nv_bfloat16* residual, const vp_router_weights* rw,
                    const vp_surrogate_weights* sw, const int32_t* force_modes,
                    __nv_bfloat16* out, __nv_bfloat16* qkv, __nv_bfloat16* y, float* s_out,
                    float* s_attn_out, int32_t* modes_out, const RouterScratch& sc,
                    cudaStream_t st, const LnFold* fold = nullptr, const QkArgs* qk = nullptr,
                    bool keep_mean_y = false) {
  const int N = dm->N, D = dm->H * kHeadDim;
  const int sms = device_sm_count();
  LinearArgs la{};
  la.M = N;
  la.N = 3 * D;
  la.K = D;
  la.A = xin;
  la.W = reinterpret_cast<const __nv_bfloat16*>(w_qkv);
  la.bias = b_qkv;
  la.act = VP_ACT_NONE;
  la.out = qkv;
  la.err = sc.err;
  if (fold) {
    la.ln_part = fold->part_in;
    la.ln_c = fold->c;
    la.ln_eps = fold->eps;
  }
  set_qk(la, qk, D);
  VP_TRY(from_cuda(launch_linear(la, sms, st)));
  RouterArgs ra = make_router_args(dm, reinterpret_cast<const vp_bf16*>(qkv), rw, force_modes);
  ra.s_out = s_out;
  ra.modes_out = modes_out;
  VP_TRY(from_cuda(launch_router(ra, sc, sms, st)));
  prof_before(VP_KERNEL_GEMM, st);  // W_O's bias, counted with the projections
  const cudaError_t ef = launch_wo_mean_fold(D, dm->H, reinterpret_cast<const __nv_bfloat16*>(w_o),
                                             b_o, sc.mean_v, sc.head_ids, sc.offsets, sc.wo_bias, st);
  prof_after(st);
  VP_TRY(from_cuda(ef));
  VP_TRY(run_heads(dm, qkv, sc.head_ids, sc.offsets, sc.ctx, sc.mean_v, sw, y, s_attn_out, sc,
                   st, !keep_mean_y));
  LinearArgs lo{};
  lo.M = N;
  lo.N = D;
  lo.K = D;
  lo.A = y;
  lo.W = reinterpret_cast<const __nv_bfloat16*>(w_o);
  lo.bias = sc.wo_bias;  // b_O + the mean heads' rows of Y times W_O
  lo.skip_ids = sc.head_ids;  // the mean heads' K columns left out
  lo.skip_off = sc.offsets;
  lo.act = VP_ACT_NONE;
  lo.scale = ls1;
  lo.residual = residual;
  lo.out = out;
  lo.err = sc.err;
  VP_TRY(from_cuda(launch_linear(lo, sms, st)));
  return VP_OK;
}

__device__ unsigned int g_linear_err;  // error word of vp_linear (it has no workspace)

}  // namespace

extern "C" {

const char* vp_status_string(vp_status s) {
  switch (s) {
    case VP_OK: return "ok";
    case VP_ERR_INVALID_ARG: return "invalid argument";
    case VP_ERR_UNSUPPORTED_SHAPE: return "unsupported shape";
    case VP_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
    case VP_ERR_CUDA: return "CUDA error";
    case VP_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case VP_ERR_WORKSPACE: return "workspace missing or too small";
    case VP_ERR_UNSUPPORTED_DEVICE: return "device is not sm_103";
    case VP_ERR_STATIC_SCRATCH: return "needs more scratch than the fixed no-allocation buffer holds";
  }
  return "unknown status";
}

vp_status vp_workspace_size(const vp_dims* dims, int32_t what, size_t* bytes) {
  VP_TRY(check_dims(dims));
  if (!bytes) return VP_ERR_INVALID_ARG;
  switch (what) {
    case VP_WS_ROUTER: *bytes = heads_scratch_bytes(dims->H); break;
    case VP_WS_LAYER: *bytes = layer_ws_bytes(dims); break;
    case VP_WS_STACK: *bytes = stack_ws_bytes(dims); break;
    case VP_WS_STACK_MERGE: *bytes = stack_merge_ws_bytes(dims); break;
    default: return VP_ERR_INVALID_ARG;
  }
  return VP_OK;
}

vp_status vp_profile_begin(int32_t max_launches) {
  Profiler& p = g_prof;
  if (p.active || max_launches < 0 || max_launches > (1 << 20)) return VP_ERR_INVALID_ARG;
  p = Profiler();
  p.rec = new ProfRecord[max_launches > 0 ? max_launches : 1];
  for (int i = 0; i < max_launches; ++i) {
    if (cudaEventCreate(&p.rec[i].start) != cudaSuccess ||
        cudaEventCreate(&p.rec[i].stop) != cudaSuccess) {
      for (int j = 0; j <= i; ++j) {
        cudaEventDestroy(p.rec[j].start);
        cudaEventDestroy(p.rec[j].stop);
      }
      delete[] p.rec;
      p.rec = nullptr;
      return VP_ERR_CUDA;
    }
  }
  p.max = max_launches;
  p.active = true;
  return VP_OK;
}

vp_status vp_profile_end(int32_t* n_launches, int32_t* launches, float* ms) {
  Profiler& p = g_prof;
  if (!p.active) return VP_ERR_INVALID_ARG;
  p.active = false;
  vp_status st = VP_OK;
  float acc[VP_KERNEL_CLASSES] = {};
  if (p.used > 0 && cudaEventSynchronize(p.rec[p.used - 1].stop) != cudaSuccess) st = VP_ERR_CUDA;
  for (int i = 0; i < p.used && st == VP_OK; ++i) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, p.rec[i].start, p.rec[i].stop) != cudaSuccess) st = VP_ERR_CUDA;
    acc[p.rec[i].kind] += t;
  }
  for (int i = 0; i < p.max; ++i) {
    cudaEventDestroy(p.rec[i].start);
    cudaEventDestroy(p.rec[i].stop);
  }
  delete[] p.rec;
  p.rec = nullptr;
  if (n_launches) *n_launches = p.launches;
  for (int k = 0; k < VP_KERNEL_CLASSES; ++k) {
    if (launches) launches[k] = p.per_class[k];
    if (ms) ms[k] = acc[k];
  }
  return st;
}

vp_status vp_read_device_error(void* ws, size_t ws_bytes, uint32_t* host_bits, void* stream) {
  if (!ws || !host_bits || ws_bytes < 256) return VP_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t bits = 0;
  if (cudaMemcpyAsync(&bits, ws, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess) return VP_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return VP_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, 4, st) != cudaSuccess) return VP_ERR_CUDA;
  *host_bits = bits;
  return (bits & VP_DEVERR_WAIT_TIMEOUT) ? VP_ERR_DEVICE_TIMEOUT : VP_OK;
}

vp_status vp_selftest_wait_timeout(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream) {
  if (!ws || ws_bytes < 256 || !aligned16(ws)) return VP_ERR_INVALID_ARG;
  if (limit_ns < 1000000 || limit_ns > 2000000000) return VP_ERR_INVALID_ARG;
  VP_TRY(check_device());
  return from_cuda(launch_wait_selftest(static_cast<unsigned int*>(ws),
                                        (unsigned long long)limit_ns,
                                        static_cast<cudaStream_t>(stream)));
}

vp_status vp_router(const vp_dims* dims, const vp_bf16* qkv, const vp_router_weights* rw,
                    const int32_t* force_modes, float* s, int32_t* modes, float* q_pool,
                    float* ctx, float* mean_v, float* r, void* ws, size_t ws_bytes, void* stream) {
  VP_TRY(check_dims(dims));
  if (!qkv || !s || !modes) return VP_ERR_INVALID_ARG;
  if (!aligned16(qkv)) return VP_ERR_ALIGNMENT;
  VP_TRY(check_router_weights(rw));
  if (!ws || ws_bytes < router_scratch_bytes(dims->H)) return VP_ERR_WORKSPACE;
  VP_TRY(check_device());
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  RouterScratch sc = carve_router_scratch(ws, dims->H);
  RouterArgs a = make_router_args(dims, qkv, rw, force_modes);
  a.s_out = s;
  a.modes_out = modes;
  a.q_pool_out = q_pool;
  a.ctx_out = ctx;
  a.mean_v_out = mean_v;
  a.r_out = r;
  return from_cuda(launch_router(a, sc, device_sm_count(), st));
}

vp_status vp_bin_heads(int32_t H, int32_t N, const int32_t* modes, int32_t* head_ids,
                       int32_t* offsets, int32_t* work, int32_t* n_work, void* stream) {
  if (H < 1 || H > kMaxHeads || N < 1) return VP_ERR_UNSUPPORTED_SHAPE;
  if (!modes || !head_ids || !offsets) return VP_ERR_INVALID_ARG;
  VP_TRY(check_device());
  return from_cuda(launch_bin_heads(H, N, modes, head_ids, offsets, work, n_work,
                                    static_cast<cudaStream_t>(stream)));
}

vp_status vp_head_attention(const vp_dims* dims, const vp_bf16* qkv, const int32_t* head_ids,
                            const int32_t* offsets, const float* ctx, const float* mean_v,
                            const vp_surrogate_weights* sw, vp_bf16* y, float* s_attn, void* ws,
                            size_t ws_bytes, void* stream) {
  VP_TRY(check_dims(dims));
  if (!qkv || !head_ids || !offsets || !ctx || !mean_v || !y) return VP_ERR_INVALID_ARG;
  if (!aligned16(qkv) || !aligned16(y)) return VP_ERR_ALIGNMENT;
  VP_TRY(check_surrogate_weights(sw));
  if (!ws || ws_bytes < heads_scratch_bytes(dims->H)) return VP_ERR_WORKSPACE;
  VP_TRY(check_device());
  RouterScratch sc = carve_router_scratch(ws, dims->H);
  return run_heads(dims, reinterpret_cast<const __nv_bfloat16*>(qkv), head_ids, offsets, ctx,
                   mean_v, sw, reinterpret_cast<__nv_bfloat16*>(y), s_attn, sc,
                   static_cast<cudaStream_t>(stream));
}

vp_status vp_linear(int32_t M, int32_t Nout, int32_t K, const vp_bf16* A, const vp_bf16* W,
                    const float* bias, int32_t act, const float* scale, const vp_bf16* residual,
                    vp_bf16* out, void* stream) {
  if (M < 1 || Nout < 8 || K < 8 || Nout % 8 || K % 8) return VP_ERR_UNSUPPORTED_SHAPE;
  if (!A || !W || !out) return VP_ERR_INVALID_ARG;
  if (act != VP_ACT_NONE && act != VP_ACT_GELU) return VP_ERR_INVALID_ARG;
  if (!aligned16(A) || !aligned16(W) || !aligned16(out) || (residual && !aligned16(residual)) ||
      (bias && !aligned16(bias)) || (scale && !aligned16(scale)))
    return VP_ERR_ALIGNMENT;
  VP_TRY(check_device());
  unsigned int* err = nullptr;
  if (cudaGetSymbolAddress(reinterpret_cast<void**>(&err), g_linear_err) != cudaSuccess)
    return VP_ERR_CUDA;
  LinearArgs la{};
  la.M = M;
  la.N = Nout;
  la.K = K;
  la.A = reinterpret_cast<const __nv_bfloat16*>(A);
  la.W = reinterpret_cast<const __nv_bfloat16*>(W);
  la.bias = bias;
  la.act = act;
  la.scale = scale;
  la.residual = reinterpret_cast<const __nv_bfloat16*>(residual);
  la.out = reinterpret_cast<__nv_bfloat16*>(out);
  la.err = err;
  return from_cuda(launch_linear(la, device_sm_count(), static_cast<cudaStream_t>(stream)));
}

vp_status vp_layer_norm(int32_t M, int32_t D, const vp_bf16* x, const float* gamma,
                        const float* beta, float eps, vp_bf16* out, void* stream) {
  if (M < 1 || !ln_width_supported(D)) return VP_ERR_UNSUPPORTED_SHAPE;
  if (!x || !gamma || !beta || !out) return VP_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(out) || !aligned16(gamma) || !aligned16(beta))
    return VP_ERR_ALIGNMENT;
  VP_TRY(check_device());
  return from_cuda(launch_layer_norm(M, D, reinterpret_cast<const __nv_bfloat16*>(x), gamma, beta,
                                     eps, reinterpret_cast<__nv_bfloat16*>(out),
                                     static_cast<cudaStream_t>(stream)));
}

vp_status vp_moh_global_attention(const vp_dims* dims, const vp_bf16* x, const vp_bf16* w_qkv,
                                  const float* b_qkv, const vp_bf16* w_o, const float* b_o,
                                  const vp_router_weights* rw, const vp_surrogate_weights* sw,
                                  const vp_qk_options* qk, const int32_t* force_modes,
                                  vp_bf16* out, vp_bf16* qkv_out, vp_bf16* y_out, float* s_out,
                                  float* s_attn_out, int32_t* modes_out, void* ws, size_t ws_bytes,
                                  void* stream) {
  VP_TRY(check_dims(dims));
  if (!x || !w_qkv || !w_o || !out) return VP_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(w_qkv) || !aligned16(w_o) || !aligned16(out) ||
      (qkv_out && !aligned16(qkv_out)) || (y_out && !aligned16(y_out)) ||
      (b_qkv && !aligned16(b_qkv)) || (b_o && !aligned16(b_o)))
    return VP_ERR_ALIGNMENT;
  VP_TRY(check_router_weights(rw));
  VP_TRY(check_surrogate_weights(sw));
  int max_pos = 0;
  VP_TRY(check_qk(qk, dims, &max_pos));
  if (!ws || ws_bytes < layer_ws_bytes(dims)) return VP_ERR_WORKSPACE;
  VP_TRY(check_device());
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t N = dims->N, D = (size_t)dims->H * kHeadDim;
  RouterScratch sc = carve_router_scratch(ws, dims->H);
  char* p = static_cast<char*>(ws) + heads_scratch_bytes(dims->H);
  float2* rope = reinterpret_cast<float2*>(p);
  p += align_up(kRopeTableBytes);
  if (qk && qk->rope) VP_TRY(from_cuda(launch_rope_table(max_pos, qk->rope_base, rope, st)));
  const QkArgs qa{qk, rope, nullptr};
  __nv_bfloat16* qkv = reinterpret_cast<__nv_bfloat16*>(p);
  p += align_up(N * 3 * D * 2);
  __nv_bfloat16* y = reinterpret_cast<__nv_bfloat16*>(p);
  if (qkv_out) qkv = reinterpret_cast<__nv_bfloat16*>(qkv_out);
  if (y_out) y = reinterpret_cast<__nv_bfloat16*>(y_out);
  return run_layer(dims, reinterpret_cast<const __nv_bfloat16*>(x), w_qkv, b_qkv, w_o, b_o,
                   nullptr, nullptr, rw, sw, force_modes, reinterpret_cast<__nv_bfloat16*>(out),
                   qkv, y, s_out, s_attn_out, modes_out, sc, st, nullptr, &qa, y_out != nullptr);
}

// The host-side checks of vp_global_stack (also run by vp_global_stack_host before it
// enqueues anything); *any_merge: some block merges tokens.
static vp_status check_stack(const vp_dims* dims, int32_t n_layers, const vp_bf16* x_inout,
                             const vp_layer_weights* layers, size_t ws_bytes, const void* ws,
                             bool* any_merge_out) {
  VP_TRY(check_dims(dims));
  if (n_layers < 1 || !x_inout || !layers) return VP_ERR_INVALID_ARG;
  if (!aligned16(x_inout)) return VP_ERR_ALIGNMENT;
  const int D = dims->H * kHeadDim;
  if (!ln_width_supported(D)) return VP_ERR_UNSUPPORTED_SHAPE;
  bool any_merge = false;
  for (int l = 0; l < n_layers; ++l) {
    const vp_layer_weights& w = layers[l];
    if (!w.ln1_g || !w.ln1_b || !w.w_qkv || !w.w_o || !w.ls1 || !w.ln2_g || !w.ln2_b ||
        !w.w_fc1 || !w.w_fc2 || !w.ls2)
      return VP_ERR_INVALID_ARG;
    if (!aligned16(w.w_qkv) || !aligned16(w.w_o) || !aligned16(w.w_fc1) || !aligned16(w.w_fc2) ||
        !aligned16(w.ls1) || !aligned16(w.ls2) || !aligned16(w.ln1_g) || !aligned16(w.ln1_b) ||
        !aligned16(w.ln2_g) || !aligned16(w.ln2_b) || (w.b_qkv && !aligned16(w.b_qkv)) ||
        (w.b_o && !aligned16(w.b_o)) || (w.b_fc1 && !aligned16(w.b_fc1)) ||
        (w.b_fc2 && !aligned16(w.b_fc2)))
      return VP_ERR_ALIGNMENT;
    VP_TRY(check_router_weights(&w.router));
    VP_TRY(check_surrogate_weights(&w.surrogate));
    int max_pos = 0;
    VP_TRY(check_qk(w.qk, dims, &max_pos));
    VP_TRY(check_merge(w.merge, dims));
    any_merge = any_merge || w.merge != nullptr;
  }
  if (!ws || ws_bytes < (any_merge ? stack_merge_ws_bytes(dims) : stack_ws_bytes(dims)))
    return VP_ERR_WORKSPACE;
  *any_merge_out = any_merge;
  return check_device();
}

vp_status vp_global_stack(const vp_dims* dims, int32_t n_layers, vp_bf16* x_inout,
                          const vp_layer_weights* layers, const int32_t* force_modes,
                          int32_t* modes_out, float* s_out, float* s_attn_out, float ln_eps,
                          void* ws, size_t ws_bytes, void* stream) {
  bool any_merge = false;
  VP_TRY(check_stack(dims, n_layers, x_inout, layers, ws_bytes, ws, &any_merge));
  const int D = dims->H * kHeadDim;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t N = dims->N;
  RouterScratch sc = carve_router_scratch(ws, dims->H);
  char* p = static_cast<char*>(ws) + heads_scratch_bytes(dims->H);
  float2* rope = reinterpret_cast<float2*>(p);
  p += align_up(kRopeTableBytes);
  const vp_qk_options* rope_built = nullptr;  // the options the table was last built for
  // LayerNorm scratch (see ln_scratch_bytes).  LN1 is folded into the QKV projection, which
  // then reads the raw residual stream; its row statistics come from the kernel that last
  // wrote the stream (the previous block's FFN-down, or a statistics pass for the first
  // block).  LN2 stays a kernel of its own: folded into the FFN-up projection it costs that
  // GEMM's GELU epilogue more than the LayerNorm pass it saves.
  float2* part = reinterpret_cast<float2*>(p);  // LN1 input statistics
  p += align_up(N * (D / 128) * sizeof(float2));
  __nv_bfloat16* wq = reinterpret_cast<__nv_bfloat16*>(p);  // [3D][D] folded W_qkv
  p += align_up((size_t)3 * D * D * 2);
  float* cq = reinterpret_cast<float*>(p);
  p += align_up((size_t)3 * D * sizeof(float));
  float* bq = reinterpret_cast<float*>(p);
  p += align_up((size_t)3 * D * sizeof(float));
  __nv_bfloat16* zt = reinterpret_cast<__nv_bfloat16*>(p);  // LN2 output
  p += align_up(N * D * 2);
  __nv_bfloat16* qkv = reinterpret_cast<__nv_bfloat16*>(p);
  __nv_bfloat16* y = reinterpret_cast<__nv_bfloat16*>(p + align_up(N * 3 * D * 2));
  __nv_bfloat16* hid = reinterpret_cast<__nv_bfloat16*>(p);  // reuses the QKV / Y region
  p += align_up(N * 4 * D * 2);
  MergeScratch ms{};  // after the stack's own regions (VP_WS_STACK_MERGE)
  if (any_merge) {
    ms.wbar = reinterpret_cast<__nv_bfloat16*>(p);
    p += align_up(64 * D * 2);
    ms.bbar = reinterpret_cast<float*>(p);
    p += align_up(64 * sizeof(float));
    __nv_bfloat16** rows64[3] = {&ms.kbar, &ms.m_src, &ms.m_dst};
    for (__nv_bfloat16** q : rows64) {
      *q = reinterpret_cast<__nv_bfloat16*>(p);
      p += align_up(N * 64 * 2);
    }
    int** ints[7] = {&ms.row_of, &ms.dst_tok, &ms.assign, &ms.cnt, &ms.offs, &ms.fill, &ms.members};
    for (int** q : ints) {
      *q = reinterpret_cast<int*>(p);
      p += align_up((N + 1) * sizeof(int));
    }
    ms.best = reinterpret_cast<unsigned long long*>(p);
    p += align_up(N * sizeof(unsigned long long));
    ms.xm = reinterpret_cast<__nv_bfloat16*>(p);
    p += align_up(N * D * 2);
    ms.err = sc.err;
  }
  __nv_bfloat16* merged_out = any_merge ? reinterpret_cast<__nv_bfloat16*>(p) : nullptr;  // [Np][D]
  ms.slots = reinterpret_cast<float*>(merged_out);  // free until the block's attention writes it
  __nv_bfloat16* x = reinterpret_cast<__nv_bfloat16*>(x_inout);
  const int sms = device_sm_count();
  VP_TRY(from_cuda(launch_ln_partials(dims->N, D, x, part, st)));
  for (int l = 0; l < n_layers; ++l) {
    const vp_layer_weights& w = layers[l];
    if (!w.merge)
      VP_TRY(from_cuda(launch_ln_fold_weights(3 * D, D,
                                              reinterpret_cast<const __nv_bfloat16*>(w.w_qkv),
                                              w.ln1_g, w.ln1_b, w.b_qkv, wq, cq, bq, st)));
    if (w.qk && w.qk->rope &&
        !(rope_built && rope_built->rope_base == w.qk->rope_base &&
          rope_built->tokens_per_view == w.qk->tokens_per_view &&
          rope_built->patch_start == w.qk->patch_start && rope_built->grid_w == w.qk->grid_w)) {
      int max_pos = 0;
      VP_TRY(check_qk(w.qk, dims, &max_pos));
      VP_TRY(from_cuda(launch_rope_table(max_pos, w.qk->rope_base, rope, st)));
      rope_built = w.qk;
    }
    const int32_t* fm = force_modes ? force_modes + (size_t)l * dims->H : nullptr;
    float* s_l = s_out ? s_out + (size_t)l * dims->H : nullptr;
    float* sa_l = s_attn_out ? s_attn_out + (size_t)l * dims->H : nullptr;
    int32_t* m_l = modes_out ? modes_out + (size_t)l * dims->H : nullptr;
    if (w.merge) {
      // (1) X~ = LN1(X), folded into the key metric and the merged tokens (not stored); merge
      // X~ (vp_merge_options); (2)-(3) routed attention of the merged tokens; unmerge:
      // X_i += LS1 (.) A[merged row of i].  The folded metric weights use the QKV fold's
      // scratch, which merged blocks do not need.
      const MergeGeo g = make_merge_geo(dims->N, w.merge->tokens_per_view, w.merge->patch_start,
                                        w.merge->stride);
      const MergeLn mln{part, w.ln1_g, w.ln1_b, ln_eps, wq, cq, bq};
      VP_TRY(from_cuda(launch_merge_prepare(g, dims->H, x, mln,
                                            reinterpret_cast<const __nv_bfloat16*>(w.w_qkv),
                                            w.b_qkv, ms, sms, st)));
      if (w.merge->assign_out)
        VP_TRY(from_cuda(cudaMemcpyAsync(w.merge->assign_out, ms.assign, N * sizeof(int),
                                         cudaMemcpyDeviceToDevice, st)));
      vp_dims dm = *dims;
      dm.N = g.Np;
      const QkArgs qm{w.qk, rope, ms.dst_tok};
      VP_TRY(run_layer(&dm, ms.xm, w.w_qkv, w.b_qkv, w.w_o, w.b_o, nullptr, nullptr, &w.router,
                       &w.surrogate, fm, merged_out, qkv, y, s_l, sa_l, m_l, sc, st, nullptr, &qm));
      // unmerge, X_attn = X + LS1 (.) A, and (4)'s Z~ = LN2(X_attn) in one pass
      VP_TRY(from_cuda(launch_unmerge_ln(dims->N, D, ms.assign, merged_out, w.ls1, w.ln2_g,
                                         w.ln2_b, ln_eps, x, zt, st)));
    } else {
      const QkArgs qa{w.qk, rope, nullptr};
      // (1)-(3) X <- X + LS1 (Y W_O + b_O) in place, Y the routed attention of LN1(X)
      const LnFold fold{part, cq, ln_eps};
      VP_TRY(run_layer(dims, x, reinterpret_cast<const vp_bf16*>(wq), bq, w.w_o, w.b_o, w.ls1, x,
                       &w.router, &w.surrogate, fm, x, qkv, y, s_l, sa_l, m_l, sc, st, &fold, &qa));
    }
    // (4) Z~ = LN2(X_attn) (done above for a merged block); X <- X_attn + LS2 FFN(Z~)
    if (!w.merge)
      VP_TRY(from_cuda(launch_layer_norm(dims->N, D, x, w.ln2_g, w.ln2_b, ln_eps, zt, st)));
    LinearArgs f1{};
    f1.M = dims->N;
    f1.N = 4 * D;
    f1.K = D;
    f1.A = zt;
    f1.W = reinterpret_cast<const __nv_bfloat16*>(w.w_fc1);
    f1.bias = w.b_fc1;
    f1.act = VP_ACT_GELU;
    f1.out = hid;
    f1.err = sc.err;
    VP_TRY(from_cuda(launch_linear(f1, sms, st)));
    LinearArgs f2{};
    f2.M = dims->N;
    f2.N = D;
    f2.K = 4 * D;
    f2.A = hid;
    f2.W = reinterpret_cast<const __nv_bfloat16*>(w.w_fc2);
    f2.bias = w.b_fc2;
    f2.act = VP_ACT_NONE;
    f2.scale = w.ls2;
    f2.residual = x;
    f2.out = x;
    f2.err = sc.err;
    f2.part_out = part;  // the next block's LN1 statistics
    VP_TRY(from_cuda(launch_linear(f2, sms, st)));
  }
  return VP_OK;
}

// A host pointer the GPU can read and write (page-locked), as a device-visible address.
static vp_status device_view_of_host(const void* p, void** dev) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();  // clear the error of an unknown pointer
    return VP_ERR_INVALID_ARG;
  }
  if (at.type != cudaMemoryTypeHost || !at.devicePointer) return VP_ERR_INVALID_ARG;
  *dev = at.devicePointer;
  return VP_OK;
}

vp_status vp_global_stack_host(const vp_dims* dims, int32_t n_layers, const vp_bf16* x_in,
                               vp_bf16* x_out, vp_bf16* x_dev, const vp_layer_weights* layers,
                               const int32_t* force_modes, int32_t* modes_out, float* s_out,
                               float* s_attn_out, float ln_eps, void* ws, size_t ws_bytes,
                               void* stream) {
  if (!x_in || !x_out || !x_dev) return VP_ERR_INVALID_ARG;
  if (!aligned16(x_in) || !aligned16(x_out)) return VP_ERR_ALIGNMENT;
  bool any_merge = false;
  VP_TRY(check_stack(dims, n_layers, x_dev, layers, ws_bytes, ws, &any_merge));
  void* in_dev = nullptr;
  void* out_dev = nullptr;
  VP_TRY(device_view_of_host(x_in, &in_dev));
  VP_TRY(device_view_of_host(x_out, &out_dev));
  const size_t bytes = (size_t)dims->N * dims->H * kHeadDim * sizeof(vp_bf16);  // a multiple of 16
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int sms = device_sm_count();
  VP_TRY(from_cuda(launch_host_copy(in_dev, x_dev, bytes, sms, st)));
  VP_TRY(vp_global_stack(dims, n_layers, x_dev, layers, force_modes, modes_out, s_out, s_attn_out,
                         ln_eps, ws, ws_bytes, stream));
  return from_cuda(launch_host_copy(x_dev, out_dev, bytes, sms, st));
}

}  // extern "C"
