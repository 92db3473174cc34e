"""GB300-native Mixture-of-Sparse-Attention (MoSA) layer, arXiv 2505.00315.

The layer runs in libmosa.so (hand-written CUDA for sm_103a behind the C ABI
of include/mosa.h).  This package holds the thin Python binding with the
same call names, the seeded synthetic workloads and the FLOP model.  The
binding is imported lazily so that ``workloads`` and ``flops`` work on a
machine without a GPU.
"""
from __future__ import annotations

__all__ = ["mosa_forward", "mosa_forward_with_indices", "mosa_backward", "mosa_topk",
           "mosa_workspace_bytes", "mosa_check_status", "alloc_workspace", "make_shape",
           "MosaShape", "MosaError", "load", "mosa_kernel_launches", "mosa_profile_stages",
           "mosa_profile_read", "mosa_profile_spans", "mosa_profile_timeline",
           "mosa_profile_timeline_read", "mosa_profile_spans_copy", "mosa_stage_name", "mosa_stage_engine", "stage_impl",
           "mosa_route_noalloc", "mosa_adaptive_k", "MosaHybridShape", "make_hybrid_shape",
           "mosa_hybrid_workspace_bytes", "alloc_hybrid_workspace", "mosa_hybrid_forward",
           "mosa_hybrid_backward"]


def __getattr__(name):
    if name in __all__:
        from . import _binding
        return getattr(_binding, name)
    raise AttributeError(name)
