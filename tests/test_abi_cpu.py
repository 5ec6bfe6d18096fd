"""The C ABI without a GPU: the library builds for sm_103a, loads, exports every function
include/vp.h declares, and rejects bad arguments on the host before touching a device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vp.h")


@pytest.fixture(scope="module")
def vp():
    from paper_2609_23733_gb300 import binding, build
    if not os.path.exists(build.LIB):
        build.build()
    return binding


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:vp_status|const char\*)\s+(vp_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("vp_router", "vp_bin_heads", "vp_moh_global_attention", "vp_global_stack",
                     "vp_workspace_size", "vp_status_string", "vp_head_attention", "vp_linear",
                     "vp_layer_norm", "vp_router_noalloc"):
        assert required in names


def test_library_exports_every_declared_function(vp):
    lib = vp.lib()
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) == set(vp.EXPORTS)


def test_status_strings(vp):
    for code in range(9):
        assert vp.vp_status_string(code) not in ("", "unknown status")
    assert vp.vp_status_string(99) == "unknown status"


def test_workspace_sizes(vp):
    small = vp.dims(1044)
    big = vp.dims(137400)
    r = vp.vp_workspace_size(small, vp.VP_WS_ROUTER)
    assert r == vp.vp_workspace_size(big, vp.VP_WS_ROUTER)  # router scratch is independent of N
    assert vp.vp_workspace_size(big, vp.VP_WS_LAYER) >= r + 137400 * 4 * 1024 * 2
    # stack: {QKV, Y} / FFN hidden region, the LN2 output, LN1 row statistics (8 blocks of
    # (mean, M2) per row) and one block's folded QKV weights
    assert vp.vp_workspace_size(big, vp.VP_WS_STACK) >= (r + 137400 * 5 * 1024 * 2 + 137400 * 8 * 8
                                                         + 3 * 1024 * 1024 * 2)
    with pytest.raises(vp.VPError) as e:
        vp.vp_workspace_size(vp.dims(100, d=32), vp.VP_WS_ROUTER)
    assert e.value.status == 2
    with pytest.raises(vp.VPError) as e:
        vp.vp_workspace_size(vp.dims(100, H=33), vp.VP_WS_ROUTER)
    assert e.value.status == 2
    with pytest.raises(vp.VPError) as e:
        vp.vp_workspace_size(small, 7)
    assert e.value.status == 1


def test_host_side_validation(vp):
    lib = vp.lib()
    A = 0x10000  # aligned fake device addresses: the checks below fail before any access
    dm = vp.dims(300)
    rw = vp.VpRouterWeights(A, A, A, None, None, None)
    null_rw = vp.VpRouterWeights(None, A, A, None, None, None)
    bad = vp.dims(300, d=32)
    # vp_router: missing dims / bad shape / null output / bad alignment / small workspace
    assert lib.vp_router(None, A, ctypes.byref(rw), None, A, A, None, None, None, None, A, 1 << 30, None) == 1
    assert lib.vp_router(ctypes.byref(bad), A, ctypes.byref(rw), None, A, A, None, None, None, None, A, 1 << 30, None) == 2
    assert lib.vp_router(ctypes.byref(dm), A, ctypes.byref(rw), None, None, A, None, None, None, None, A, 1 << 30, None) == 1
    assert lib.vp_router(ctypes.byref(dm), A + 8, ctypes.byref(rw), None, A, A, None, None, None, None, A, 1 << 30, None) == 3
    assert lib.vp_router(ctypes.byref(dm), A, ctypes.byref(null_rw), None, A, A, None, None, None, None, A, 1 << 30, None) == 1
    assert lib.vp_router(ctypes.byref(dm), A, ctypes.byref(rw), None, A, A, None, None, None, None, A, 16, None) == 6
    # vp_router_noalloc: the checks of vp_router (H outside 1..32 is a shape error, as there;
    # unknown or conflicting variant bits; missing outputs or weights; alignment)
    na = lambda d, q=A, r=rw, s=A: lib.vp_router_noalloc(None if d is None else ctypes.byref(d), q,
                                                         ctypes.byref(r), None, s, A, None, None, None,
                                                         None, None)
    assert na(None) == 1
    assert na(vp.dims(300, H=33)) == 2
    assert na(bad) == 2
    assert na(vp.dims(300, variant=16)) == 1
    assert na(vp.dims(300, variant=8 | 2)) == 1
    assert na(dm, s=None) == 1
    assert na(dm, r=null_rw) == 1
    assert na(dm, q=A + 8) == 3
    # its error reader needs somewhere to write the bits
    assert lib.vp_router_noalloc_error(None, None) == 1
    # vp_global_stack_host: missing buffers, misaligned host buffers (before any device query)
    hs = lambda a, b, c: lib.vp_global_stack_host(ctypes.byref(dm), 1, a, b, c, None, None, None, None, None,
                                                  ctypes.c_float(1e-6), A, 1 << 30, None)
    assert hs(None, A, A) == 1 and hs(A, None, A) == 1 and hs(A, A, None) == 1
    assert hs(A + 8, A, A) == 3 and hs(A, A + 4, A) == 3
    # vp_linear: shapes and alignment
    assert lib.vp_linear(100, 12, 64, A, A, None, 0, None, None, A, None) == 2
    assert lib.vp_linear(100, 256, 60, A, A, None, 0, None, None, A, None) == 2
    assert lib.vp_linear(100, 256, 64, None, A, None, 0, None, None, A, None) == 1
    assert lib.vp_linear(100, 256, 64, A, A, None, 2, None, None, A, None) == 1
    assert lib.vp_linear(100, 256, 64, A, A, A + 4, 0, None, None, A, None) == 3
    # vp_layer_norm: unsupported width
    assert lib.vp_layer_norm(10, 1000, A, A, A, ctypes.c_float(1e-6), A, None) == 2
    # vp_bin_heads: no heads
    assert lib.vp_bin_heads(0, 10, A, A, A, None, None, None) == 2
    # vp_global_stack: no layers
    assert lib.vp_global_stack(ctypes.byref(dm), 0, A, None, None, None, None, None, ctypes.c_float(1e-6), A,
                               1 << 30, None) == 1


def test_valid_call_without_a_gpu_reports_the_device(vp):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    lib = vp.lib()
    A = 0x10000
    rw = vp.VpRouterWeights(A, A, A, None, None, None)
    st = lib.vp_router(ctypes.byref(vp.dims(300)), A, ctypes.byref(rw), None, A, A, None, None, None, None,
                       A, 1 << 30, None)
    assert st == 7  # VP_ERR_UNSUPPORTED_DEVICE: nothing was enqueued


def _fake_layer(vp, A, qk=None, merge=None):
    lw = vp.VpLayerWeights(*([A] * 14))
    lw.router = vp.VpRouterWeights(A, A, A, None, None, None)
    lw.surrogate = vp.VpSurrogateWeights(*([A] * 8))
    if qk is not None:
        lw.qk = ctypes.pointer(qk)
        lw._keep_qk = qk
    if merge is not None:
        lw.merge = ctypes.pointer(merge)
        lw._keep_merge = merge
    return lw


def test_stack_options_validated_on_the_host(vp):
    """vp_qk_options and vp_merge_options are checked before the workspace and the device:
    the expected status comes back without a GPU."""
    lib = vp.lib()
    A = 0x10000
    P = 261
    dm = vp.dims(4 * P)
    big = 1 << 40

    def stack(lw, n_tokens=4 * P):
        d = vp.dims(n_tokens)
        arr = (vp.VpLayerWeights * 1)(lw)
        return lib.vp_global_stack(ctypes.byref(d), 1, A, arr, None, None, None, None, ctypes.c_float(1e-6), A,
                                   big, None)

    # qk-norm: a scale without a shift
    half = vp.VpQkOptions(A, None, None, None, 1e-6, 0, 1, 0, 1, 100.0)
    assert stack(_fake_layer(vp, A, qk=half)) == 1
    # misaligned norm parameters
    mis = vp.VpQkOptions(A + 4, A, None, None, 1e-6, 0, 1, 0, 1, 100.0)
    assert stack(_fake_layer(vp, A, qk=mis)) == 3
    # RoPE: views that do not tile N, a zero-width grid, positions past the table
    assert stack(_fake_layer(vp, A, qk=vp.VpQkOptions(None, None, None, None, 1e-6, 1, 300, 5, 16, 100.0))) == 2
    assert stack(_fake_layer(vp, A, qk=vp.VpQkOptions(None, None, None, None, 1e-6, 1, P, 5, 0, 100.0))) == 1
    assert stack(_fake_layer(vp, A, qk=vp.VpQkOptions(None, None, None, None, 1e-6, 1, 4096, 0, 2, 100.0)),
                 n_tokens=4096) == 2
    # merging: stride 0, views that do not tile N, more special tokens than a view holds
    assert stack(_fake_layer(vp, A, merge=vp.VpMergeOptions(0, P, 5, None))) == 1
    assert stack(_fake_layer(vp, A, merge=vp.VpMergeOptions(4, 300, 5, None))) == 2
    assert stack(_fake_layer(vp, A, merge=vp.VpMergeOptions(4, P, P + 1, None))) == 1
    # merging needs the larger workspace kind
    need = vp.vp_workspace_size(dm, vp.VP_WS_STACK_MERGE)
    assert need > vp.vp_workspace_size(dm, vp.VP_WS_STACK)
    arr = (vp.VpLayerWeights * 1)(_fake_layer(vp, A, merge=vp.VpMergeOptions(4, P, 5, None)))
    assert lib.vp_global_stack(ctypes.byref(dm), 1, A, arr, None, None, None, None, ctypes.c_float(1e-6), A,
                               vp.vp_workspace_size(dm, vp.VP_WS_STACK), None) == 6


def test_option_struct_layouts(vp):
    # field order and sizes of the C structs (vp.h)
    assert ctypes.sizeof(vp.VpQkOptions) == 4 * 8 + 4 + 4 * 4 + 4
    assert ctypes.sizeof(vp.VpMergeOptions) == 3 * 4 + 4 + 8
    assert ctypes.sizeof(vp.VpLayerWeights) == 14 * 8 + 6 * 8 + 8 * 8 + 2 * 8


def test_weight_structs_keep_their_tensors(vp):
    """A struct built from a temporary dict keeps the buffers it points into alive: freed,
    their memory would go to the next allocation and be read as weights.  (Stand-in buffers
    that only carry an address: the binding takes device tensors, and there is no device here.)"""
    import gc
    import weakref

    import synth

    class Buf:  # an address, like a device tensor's data_ptr()
        def __init__(self, addr):
            self.addr = addr

        def __int__(self):
            return self.addr

    names = list(synth.make_layer_weights(synth.rng(3), block=True)) + ["q_norm_g", "q_norm_b"]

    def fresh():
        return {k: Buf(4096 * (i + 1)) for i, k in enumerate(names)}

    built, refs = {}, {}
    for kind, make in (("layer", vp.layer_weights), ("router", vp.router_weights),
                       ("surrogate", vp.surrogate_weights), ("qk", vp.qk_options)):
        w = fresh()
        refs[kind] = weakref.ref(w["r_U"] if kind == "router" else w["s_d2_b"] if kind == "surrogate"
                                 else w["q_norm_g"] if kind == "qk" else w["b_qkv"])
        built[kind] = make(w)
        del w
    assign = Buf(1 << 30)
    refs["merge"] = weakref.ref(assign)
    built["merge"] = vp.merge_options(4, 261, 5, assign)
    del assign
    gc.collect()
    for kind, r in refs.items():
        assert r() is not None, kind
    assert built["layer"].b_qkv == int(refs["layer"]())
    assert built["router"].U == int(refs["router"]())
    assert built["surrogate"].d2_b == int(refs["surrogate"]())
    assert built["qk"].q_norm_g == int(refs["qk"]())
    assert built["merge"].assign_out == 1 << 30


def test_wait_selftest_validated_on_the_host(vp):
    lib = vp.lib()
    buf = (ctypes.c_uint8 * 4096)()
    A = ctypes.c_void_p(((ctypes.addressof(buf) + 255) // 256) * 256)
    for limit in (0, 999_999, 2_000_000_001, -5):  # outside 1 ms .. 2 s
        assert lib.vp_selftest_wait_timeout(A, 1024, limit, None) == 1
    assert lib.vp_selftest_wait_timeout(None, 1024, 50_000_000, None) == 1
    assert lib.vp_selftest_wait_timeout(A, 128, 50_000_000, None) == 1  # no room for the error word
