"""GB300 (sm_103a) library for VGGT-Prime's compute-adaptive mixture-of-heads global
attention: router (§4.1), routing (§4.2), full / surrogate (§4.3) / mean heads, and the
Algorithm 1 block, behind the C ABI of include/vp.h.  ``binding`` is the ctypes layer."""
from . import binding
from .binding import (VPError, dims, layer_weights, router_weights, surrogate_weights, to_device,
                      vp_bin_heads, vp_global_stack, vp_head_attention, vp_layer_norm, vp_linear,
                      vp_moh_global_attention, vp_read_device_error, vp_router, vp_status_string,
                      vp_workspace_size, workspace)

__all__ = ["binding", "VPError", "dims", "layer_weights", "router_weights", "surrogate_weights",
           "to_device", "vp_bin_heads", "vp_global_stack", "vp_head_attention", "vp_layer_norm",
           "vp_linear", "vp_moh_global_attention", "vp_read_device_error", "vp_router",
           "vp_status_string", "vp_workspace_size", "workspace"]
