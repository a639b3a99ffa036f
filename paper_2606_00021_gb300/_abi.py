"""ctypes declarations of the libsense C ABI (include/sense.h)."""
from __future__ import annotations

import ctypes as C
import os

from . import _build

c_i32, c_i64, c_u32, c_size, c_p = C.c_int32, C.c_int64, C.c_uint32, C.c_size_t, C.c_void_p


class GateParams(C.Structure):
    _fields_ = [("gamma", C.c_float), ("topk", c_i32), ("window", c_i32),
                ("tau", c_i32), ("flags", c_u32)]


# name -> (restype, argtypes); every symbol declared in include/sense.h
SIGNATURES = {
    "sense_version": (c_i32, []),
    "sense_status_string": (C.c_char_p, [c_i32]),
    "sense_last_error": (C.c_char_p, []),
    "sense_device_status": (c_i32, [c_p, C.POINTER(c_u32), c_i32]),
    "sense_datastore_build": (c_i32, [c_p, c_i32, c_i64, c_i32, c_p, c_i32, c_u32, c_p,
                                      C.POINTER(c_p)]),
    "sense_datastore_destroy": (c_i32, [c_p]),
    "sense_datastore_keys": (c_p, [c_p]),
    "sense_retrieve_workspace_bytes": (c_size, [c_p, c_i32, c_i32]),
    "sense_retrieve_topk": (c_i32, [c_p, c_p, c_i32, c_i32, c_p, c_p, c_p, c_size, c_p]),
    "sense_retrieve_topk_noalloc": (c_i32, [c_p, c_p, c_i32, c_i32, c_p, c_p, c_p]),
    "sense_retrieve_noalloc_status": (c_i32, [c_p, C.POINTER(c_u32), c_i32]),
    "sense_retrieve_noalloc_selftest": (c_i32, [c_p, c_i64]),
    "sense_ann_draft_workspace_bytes": (c_size, [c_p, c_i32, c_i32, c_i32, c_i32]),
    "sense_ann_draft": (c_i32, [c_p, c_p, c_p, c_i32, c_p, c_p, c_i32, c_i32, c_i32, c_i32, c_u32,
                                c_p, c_size, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p]),
    "sense_rescore_topk": (c_i32, [c_p, c_p, c_i32, c_p, c_i32, c_i32, c_p, c_p, c_p]),
    "sense_gather_drafts": (c_i32, [c_p, c_p, c_i32, c_i32, c_p, c_i32, c_u32, c_p, c_p]),
    "sense_build_tree": (c_i32, [c_p, c_i32, c_i32, c_i32, c_i32, c_u32, c_p, c_p, c_p, c_p,
                                 c_p, c_p, c_p]),
    "sense_draft": (c_i32, [c_p, c_p, c_i32, c_i32, c_p, c_size, c_i32, c_u32, c_p, c_p, c_p, c_p,
                            c_p, c_p, c_p, c_p, c_p, c_p]),
    "sense_tree_mask_full": (c_i32, [c_p, c_p, c_i32, c_i32, c_p, c_i32, c_p, c_p]),
    "sense_project": (c_i32, [c_p, c_i64, c_i32, c_p, c_i32, c_p, c_u32, c_p, c_p]),
    "sense_kmeans_workspace_bytes": (c_size, [c_i64, c_i32, c_i32]),
    "sense_kmeans": (c_i32, [c_p, c_i64, c_i32, c_i32, c_i32, c_i32, c_u32, c_p, c_p, c_p, c_p,
                             c_size, c_p]),
    "sense_ivf_residuals": (c_i32, [c_p, c_i64, c_i32, c_p, c_i32, c_p, c_p, c_p]),
    "sense_ivf_build": (c_i32, [c_p, c_i64, c_i32, c_p, c_i32, c_p, c_i32, c_p, C.POINTER(c_p)]),
    "sense_ivf_destroy": (c_i32, [c_p]),
    "sense_ivf_arrays": (c_i32, [c_p, C.POINTER(c_i64), C.POINTER(c_p), C.POINTER(c_p),
                                 C.POINTER(c_p)]),
    "sense_ivf_search_workspace_bytes": (c_size, [c_p, c_i32, c_i32, c_i32]),
    "sense_ivf_search": (c_i32, [c_p, c_p, c_i32, c_i32, c_i32, c_p, c_p, c_p, c_p, c_size, c_p]),
    "sense_ctx_create": (c_i32, [c_i32, c_i32, c_i32, C.POINTER(c_p)]),
    "sense_ctx_destroy": (c_i32, [c_p]),
    "sense_ctx_reset": (c_i32, [c_p, c_p]),
    "sense_ctx_count": (c_i32, [c_p, c_p, C.POINTER(c_i64)]),
    "sense_ctx_append": (c_i32, [c_p, c_p, c_p, c_i32, c_p]),
    "sense_ctx_append_path": (c_i32, [c_p, c_p, c_p, c_i32, c_p, c_i32, c_p, c_p, c_p, c_p]),
    "sense_ctx_search_workspace_bytes": (c_size, [c_p, c_i32, c_i32]),
    "sense_ctx_search": (c_i32, [c_p, c_p, c_i32, c_i32, C.c_float, c_p, c_p, c_p, c_p, c_size,
                                 c_p]),
    "sense_hybrid_drafts": (c_i32, [c_p, c_p, c_p, c_i32, c_p, c_p, c_i32, c_i32, c_p, c_i32,
                                    c_u32, c_p, c_p]),
    "sense_ann_search": (c_i32, [c_p, c_p, c_p, c_i32, c_p, c_p, c_i32, c_i32, c_i32, c_p, c_size,
                                 c_p, c_p, c_p]),
    "sense_dyn_draft": (c_i32, [c_p, c_p, c_p, c_i32, c_p, c_p, c_i32, c_i32, C.c_float, c_p,
                                c_i32, c_u32, c_i32, c_u32, c_p, c_size, c_p, c_p, c_p, c_p, c_p,
                                c_p, c_p, c_p, c_p, c_p, c_p]),
    "sense_tree_attention_workspace_bytes": (c_size, [c_i32, c_i32, c_i32]),
    "sense_tree_attention": (c_i32, [c_p, c_p, c_p, c_i32, c_i32, c_i32, c_i32, c_i32, c_p, c_i32,
                                     C.c_float, c_p, c_p, c_size, c_p]),
    "sense_soft_gate_workspace_bytes": (c_size, [c_i32, c_i32, c_i32]),
    "sense_soft_gate": (c_i32, [c_p, c_p, c_p, c_p, c_i32, c_i32, c_i32, c_i32, c_p, c_p, c_i32,
                                c_p, c_p, c_i32, C.POINTER(GateParams), c_p, c_p, c_p, c_p, c_p,
                                c_p, c_p, c_p, c_p, c_size, c_p]),
    "sense_selftest_timeout": (c_i32, [c_p, c_i64]),
    "sense_profile_filter": (c_i32, [C.c_char_p]),
    "sense_profile_enable": (c_i32, [c_i32]),
    "sense_profile_count": (c_i32, []),
    "sense_profile_name": (C.c_char_p, [c_i32]),
    "sense_profile_query": (c_i32, [C.c_char_p, C.POINTER(C.c_double), C.POINTER(c_i64)]),
}

_lib = None


def load(build_if_missing: bool = True) -> C.CDLL:
    """Loads the in-tree libsense.so (building it first if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB):
        if not build_if_missing:
            raise RuntimeError(f"libsense.so is missing at {_build.LIB}; run the build first")
        _build.build()
    lib = C.CDLL(_build.LIB)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib
