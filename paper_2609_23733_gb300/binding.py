"""Thin ctypes binding of the C ABI in include/vp.h.

Functions carry the ABI's names and only marshal arguments: torch tensors become raw
device pointers, the current torch CUDA stream becomes the cudaStream_t, and a non-zero
vp_status raises VPError.  Every computation runs inside libvp.so; if the library is not
built (``__graft_entry__.build()``) the first call raises instead of falling back.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, Structure, c_char_p, c_float, c_int32, c_int64, c_size_t, c_uint32, c_void_p

import numpy as np
import torch

from .build import LIB

VP_MODE_MEAN, VP_MODE_SURROGATE, VP_MODE_FULL = 0, 1, 2
VP_WS_ROUTER, VP_WS_LAYER, VP_WS_STACK, VP_WS_STACK_MERGE = 0, 1, 2, 3
VP_ACT_NONE, VP_ACT_GELU = 0, 1
VP_DEVERR_WAIT_TIMEOUT, VP_DEVERR_NAN_SALIENCY = 1, 2
VP_VARIANT_MEAN_QPOOL, VP_VARIANT_MEAN_CONTEXT, VP_VARIANT_NO_RESIDUAL, VP_VARIANT_LINEAR_ATTENTION = 1, 2, 4, 8
KERNEL_CLASSES = ["gemm", "router_pool", "router_keys", "router_r", "bin_heads", "attn_full",
                  "surrogate", "mean", "layer_norm", "merge", "host_copy"]

STATUS = {0: "VP_OK", 1: "VP_ERR_INVALID_ARG", 2: "VP_ERR_UNSUPPORTED_SHAPE", 3: "VP_ERR_ALIGNMENT",
          4: "VP_ERR_CUDA", 5: "VP_ERR_DEVICE_TIMEOUT", 6: "VP_ERR_WORKSPACE",
          7: "VP_ERR_UNSUPPORTED_DEVICE", 8: "VP_ERR_STATIC_SCRATCH"}


class VPError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)}")


class VpDims(Structure):
    _fields_ = [("N", c_int32), ("H", c_int32), ("d", c_int32), ("L", c_int32),
                ("tau_low", c_float), ("tau_high", c_float), ("variant", c_uint32)]


class VpRouterWeights(Structure):
    _fields_ = [(n, c_void_p) for n in ("W", "U", "w", "bW", "bU", "beta")]


class VpSurrogateWeights(Structure):
    _fields_ = [(n, c_void_p) for n in ("g1_w", "g1_b", "g2_w", "g2_b", "d1_w", "d1_b", "d2_w", "d2_b")]


class VpQkOptions(Structure):
    _fields_ = [(n, c_void_p) for n in ("q_norm_g", "q_norm_b", "k_norm_g", "k_norm_b")] + \
               [("norm_eps", c_float), ("rope", c_int32), ("tokens_per_view", c_int32),
                ("patch_start", c_int32), ("grid_w", c_int32), ("rope_base", c_float)]


class VpMergeOptions(Structure):
    _fields_ = [("stride", c_int32), ("tokens_per_view", c_int32), ("patch_start", c_int32),
                ("assign_out", c_void_p)]


class VpLayerWeights(Structure):
    _fields_ = [(n, c_void_p) for n in ("ln1_g", "ln1_b", "w_qkv", "b_qkv", "w_o", "b_o", "ls1",
                                        "ln2_g", "ln2_b", "w_fc1", "b_fc1", "w_fc2", "b_fc2", "ls2")] + \
               [("router", VpRouterWeights), ("surrogate", VpSurrogateWeights),
                ("qk", POINTER(VpQkOptions)), ("merge", POINTER(VpMergeOptions))]


_lib = None

# (name, restype, argtypes)
_SIGS = [
    ("vp_status_string", c_char_p, [c_int32]),
    ("vp_workspace_size", c_int32, [POINTER(VpDims), c_int32, POINTER(c_size_t)]),
    ("vp_read_device_error", c_int32, [c_void_p, c_size_t, POINTER(c_uint32), c_void_p]),
    ("vp_selftest_wait_timeout", c_int32, [c_void_p, c_size_t, c_int64, c_void_p]),
    ("vp_router", c_int32, [POINTER(VpDims), c_void_p, POINTER(VpRouterWeights), c_void_p, c_void_p,
                            c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_size_t,
                            c_void_p]),
    ("vp_router_noalloc", c_int32, [POINTER(VpDims), c_void_p, POINTER(VpRouterWeights), c_void_p,
                                    c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                    c_void_p]),
    ("vp_router_noalloc_error", c_int32, [POINTER(c_uint32), c_void_p]),
    ("vp_bin_heads", c_int32, [c_int32, c_int32, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                               c_void_p]),
    ("vp_head_attention", c_int32, [POINTER(VpDims), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                    POINTER(VpSurrogateWeights), c_void_p, c_void_p, c_void_p, c_size_t,
                                    c_void_p]),
    ("vp_linear", c_int32, [c_int32, c_int32, c_int32, c_void_p, c_void_p, c_void_p, c_int32, c_void_p,
                            c_void_p, c_void_p, c_void_p]),
    ("vp_layer_norm", c_int32, [c_int32, c_int32, c_void_p, c_void_p, c_void_p, c_float, c_void_p,
                                c_void_p]),
    ("vp_moh_global_attention", c_int32, [POINTER(VpDims), c_void_p, c_void_p, c_void_p, c_void_p,
                                          c_void_p, POINTER(VpRouterWeights),
                                          POINTER(VpSurrogateWeights), POINTER(VpQkOptions), c_void_p,
                                          c_void_p, c_void_p,
                                          c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_size_t,
                                          c_void_p]),
    ("vp_global_stack_host", c_int32, [POINTER(VpDims), c_int32, c_void_p, c_void_p, c_void_p,
                                       POINTER(VpLayerWeights), c_void_p, c_void_p, c_void_p, c_void_p,
                                       c_float, c_void_p, c_size_t, c_void_p]),
    ("vp_profile_begin", c_int32, [c_int32]),
    ("vp_profile_end", c_int32, [POINTER(c_int32), POINTER(c_int32), POINTER(c_float)]),
    ("vp_global_stack", c_int32, [POINTER(VpDims), c_int32, c_void_p, POINTER(VpLayerWeights),
                                  c_void_p, c_void_p, c_void_p, c_void_p, c_float, c_void_p, c_size_t,
                                  c_void_p]),
]
EXPORTS = [s[0] for s in _SIGS]


def lib():
    """Load libvp.so (once).  Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is missing: build it with __graft_entry__.build()")
        handle = ctypes.CDLL(LIB)
        for name, res, args in _SIGS:
            f = getattr(handle, name)
            f.restype = res
            f.argtypes = args
        _lib = handle
    return _lib


def _check(status: int, where: str):
    if status != 0:
        raise VPError(status, where)


def _p(t):
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        if t.device.type != "cuda":
            raise ValueError("device tensors are required (the library has no CPU path)")
        if not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
        return t.data_ptr()
    return int(t)


def _host_p(t):
    """Address of a page-locked, contiguous CPU tensor (a host buffer the GPU can reach)."""
    if not isinstance(t, torch.Tensor) or t.device.type != "cpu":
        raise ValueError("a CPU tensor is required")
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return t.data_ptr()


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def dims(N, H=16, d=64, L=64, tau_low=0.01, tau_high=0.20, variant=0) -> VpDims:
    return VpDims(int(N), int(H), int(d), int(L), float(tau_low), float(tau_high), int(variant))


# The weight and option structs hold raw device addresses.  Each keeps a reference to the
# tensors it points into (``_keep``), so that a struct built from a temporary dict does not
# outlive its memory: a freed tensor's block is handed to the next allocation (a workspace,
# say), and the library would then read that as weights.  A struct copied into another one
# (``lw.router = ...``) or into a ctypes array does not carry the reference: the outer struct
# or the caller's list does.
def router_weights(w: dict) -> VpRouterWeights:
    rw = VpRouterWeights(_p(w["r_W"]), _p(w["r_U"]), _p(w["r_w"]), _p(w.get("r_bW")),
                         _p(w.get("r_bU")), _p(w.get("r_beta")))
    rw._keep = w
    return rw


def surrogate_weights(w: dict) -> VpSurrogateWeights:
    sw = VpSurrogateWeights(*[_p(w[k]) for k in ("s_g1_w", "s_g1_b", "s_g2_w", "s_g2_b",
                                                  "s_d1_w", "s_d1_b", "s_d2_w", "s_d2_b")])
    sw._keep = w
    return sw


def qk_options(w: dict = None, norm_eps: float = 1e-6, rope: bool = False, tokens_per_view: int = 1,
               patch_start: int = 0, grid_w: int = 1, rope_base: float = 100.0) -> VpQkOptions:
    """vp_qk_options from device tensors w["q_norm_g"], ... (each pair optional) and the
    RoPE token layout."""
    w = w or {}
    o = VpQkOptions(*[_p(w.get(k)) for k in ("q_norm_g", "q_norm_b", "k_norm_g", "k_norm_b")])
    o.norm_eps = norm_eps
    o.rope = 1 if rope else 0
    o.tokens_per_view = tokens_per_view
    o.patch_start = patch_start
    o.grid_w = grid_w
    o.rope_base = rope_base
    o._keep = w
    return o


def merge_options(stride: int, tokens_per_view: int, patch_start: int = 5, assign_out=None) -> VpMergeOptions:
    """vp_merge_options; assign_out: int32 device tensor [N] or None."""
    mo = VpMergeOptions(stride, tokens_per_view, patch_start, _p(assign_out))
    mo._keep = assign_out
    return mo


def layer_weights(w: dict, qk: VpQkOptions = None, merge: VpMergeOptions = None) -> VpLayerWeights:
    lw = VpLayerWeights(*[_p(w[k]) for k in ("ln1_g", "ln1_b", "w_qkv", "b_qkv", "w_o", "b_o", "ls1",
                                             "ln2_g", "ln2_b", "w_fc1", "b_fc1", "w_fc2", "b_fc2",
                                             "ls2")])
    lw.router = router_weights(w)
    lw.surrogate = surrogate_weights(w)
    lw._keep = w
    if qk is not None:
        lw.qk = ctypes.pointer(qk)
        lw._qk_keep = qk  # the struct must outlive the call
    if merge is not None:
        lw.merge = ctypes.pointer(merge)
        lw._merge_keep = merge
    return lw


def to_device(w: dict, device="cuda") -> dict:
    """Upload a parameter dict from ``synth`` (bf16 bits as uint16, fp32 arrays)."""
    out = {}
    for k, v in w.items():
        v = np.ascontiguousarray(v)
        t = torch.from_numpy(v.view(np.int16)).view(torch.bfloat16) if v.dtype == np.uint16 else torch.from_numpy(v)
        out[k] = t.to(device)
    return out


def bf16_from_bits(u, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(u).view(np.int16)).view(torch.bfloat16).to(device)


def bits_from_bf16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


# ---------------------------------------------------------------- ABI wrappers
def vp_status_string(status: int) -> str:
    return lib().vp_status_string(int(status)).decode()


def vp_workspace_size(dm: VpDims, what: int) -> int:
    n = c_size_t(0)
    _check(lib().vp_workspace_size(ctypes.byref(dm), int(what), ctypes.byref(n)), "vp_workspace_size")
    return n.value


def workspace(dm: VpDims, what: int, device="cuda") -> torch.Tensor:
    """A zeroed device workspace of the size the library asks for."""
    return torch.zeros(vp_workspace_size(dm, what), dtype=torch.uint8, device=device)


def vp_selftest_wait_timeout(ws: torch.Tensor, limit_ns: int, stream=None):
    """Enqueues the library's bounded-wait self-test: a wait that nothing satisfies gives up
    after limit_ns and sets the timeout bit of ws's error word."""
    _check(lib().vp_selftest_wait_timeout(_p(ws), ws.numel(), int(limit_ns), _stream(stream)),
           "vp_selftest_wait_timeout")


def vp_read_device_error(ws: torch.Tensor, stream=None) -> int:
    bits = c_uint32(0)
    st = lib().vp_read_device_error(_p(ws), ws.numel(), ctypes.byref(bits), _stream(stream))
    if st not in (0, 5):
        _check(st, "vp_read_device_error")
    return bits.value


def vp_router(dm, qkv, rw: VpRouterWeights, force_modes, s, modes, q_pool, ctx, mean_v, r, ws, stream=None):
    _check(lib().vp_router(ctypes.byref(dm), _p(qkv), ctypes.byref(rw), _p(force_modes), _p(s), _p(modes),
                           _p(q_pool), _p(ctx), _p(mean_v), _p(r), _p(ws), ws.numel(), _stream(stream)),
           "vp_router")


def vp_router_noalloc(dm, qkv, rw: VpRouterWeights, force_modes, s, modes, q_pool, ctx, mean_v, r,
                      stream=None):
    """vp_router without a workspace: scratch comes from a fixed buffer inside the library,
    for callers that cannot allocate device memory (see include/vp.h)."""
    _check(lib().vp_router_noalloc(ctypes.byref(dm), _p(qkv), ctypes.byref(rw), _p(force_modes), _p(s),
                                   _p(modes), _p(q_pool), _p(ctx), _p(mean_v), _p(r), _stream(stream)),
           "vp_router_noalloc")


def vp_router_noalloc_error(stream=None) -> int:
    """Reads and clears the device error bits of vp_router_noalloc's fixed buffer."""
    bits = c_uint32(0)
    st = lib().vp_router_noalloc_error(ctypes.byref(bits), _stream(stream))
    if st not in (0, 5):
        _check(st, "vp_router_noalloc_error")
    return bits.value


def vp_bin_heads(H, N, modes, head_ids, offsets, work=None, n_work=None, stream=None):
    _check(lib().vp_bin_heads(int(H), int(N), _p(modes), _p(head_ids), _p(offsets), _p(work), _p(n_work),
                              _stream(stream)), "vp_bin_heads")


def vp_head_attention(dm, qkv, head_ids, offsets, ctx, mean_v, sw: VpSurrogateWeights, y, ws, stream=None,
                      s_attn=None):
    _check(lib().vp_head_attention(ctypes.byref(dm), _p(qkv), _p(head_ids), _p(offsets), _p(ctx), _p(mean_v),
                                   ctypes.byref(sw), _p(y), _p(s_attn), _p(ws), ws.numel(), _stream(stream)),
           "vp_head_attention")


def vp_linear(A, W, bias=None, act=VP_ACT_NONE, scale=None, residual=None, out=None, stream=None):
    M, K = A.shape
    Nout = W.shape[0]
    if out is None:
        out = torch.empty((M, Nout), dtype=torch.bfloat16, device=A.device)
    _check(lib().vp_linear(M, Nout, K, _p(A), _p(W), _p(bias), int(act), _p(scale), _p(residual), _p(out),
                           _stream(stream)), "vp_linear")
    return out


def vp_layer_norm(x, gamma, beta, eps=1e-6, out=None, stream=None):
    M, D = x.shape
    if out is None:
        out = torch.empty_like(x)
    _check(lib().vp_layer_norm(M, D, _p(x), _p(gamma), _p(beta), float(eps), _p(out), _stream(stream)),
           "vp_layer_norm")
    return out


def vp_moh_global_attention(dm, x, w_qkv, b_qkv, w_o, b_o, rw, sw, force_modes, out, qkv_out, y_out,
                            s_out, modes_out, ws, stream=None, s_attn_out=None, qk=None):
    _check(lib().vp_moh_global_attention(ctypes.byref(dm), _p(x), _p(w_qkv), _p(b_qkv), _p(w_o), _p(b_o),
                                         ctypes.byref(rw), ctypes.byref(sw),
                                         ctypes.byref(qk) if qk is not None else None,
                                         _p(force_modes), _p(out),
                                         _p(qkv_out), _p(y_out), _p(s_out), _p(s_attn_out), _p(modes_out),
                                         _p(ws), ws.numel(), _stream(stream)), "vp_moh_global_attention")


def vp_global_stack(dm, x_inout, layers, force_modes, modes_out, s_out, ln_eps, ws, stream=None,
                    s_attn_out=None):
    arr = (VpLayerWeights * len(layers))(*layers)
    _check(lib().vp_global_stack(ctypes.byref(dm), len(layers), _p(x_inout), arr, _p(force_modes),
                                 _p(modes_out), _p(s_out), _p(s_attn_out), float(ln_eps), _p(ws), ws.numel(),
                                 _stream(stream)), "vp_global_stack")


def vp_global_stack_host(dm, x_in, x_out, x_dev, layers, force_modes, modes_out, s_out, ln_eps, ws,
                         stream=None, s_attn_out=None):
    """vp_global_stack on tokens in page-locked host memory (x_in, x_out: pinned CPU tensors);
    x_dev is the device buffer the blocks run on."""
    arr = (VpLayerWeights * len(layers))(*layers)
    _check(lib().vp_global_stack_host(ctypes.byref(dm), len(layers), _host_p(x_in), _host_p(x_out), _p(x_dev), arr,
                                      _p(force_modes), _p(modes_out), _p(s_out), _p(s_attn_out), float(ln_eps),
                                      _p(ws), ws.numel(), _stream(stream)), "vp_global_stack_host")


def vp_profile_begin(max_launches: int):
    _check(lib().vp_profile_begin(int(max_launches)), "vp_profile_begin")


def vp_profile_end():
    """Returns (total launches, {class: launches}, {class: summed ms})."""
    n = c_int32(0)
    cnt = (c_int32 * len(KERNEL_CLASSES))()
    ms = (c_float * len(KERNEL_CLASSES))()
    _check(lib().vp_profile_end(ctypes.byref(n), cnt, ms), "vp_profile_end")
    return n.value, dict(zip(KERNEL_CLASSES, list(cnt))), dict(zip(KERNEL_CLASSES, list(ms)))
