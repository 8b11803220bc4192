"""ctypes declarations of libumim's C ABI (include/umim.h).

Loading fails loudly when the shared library has not been built: there is
no CPU or PyTorch fallback for any call.
"""
import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libumim.so")
DEBUG_LIB_PATH = os.path.join(HERE, "libumim_debug.so")   # the same calls built with UMIM_DEBUG

c_i32 = ctypes.c_int32
c_i64 = ctypes.c_int64
c_ptr = ctypes.c_void_p
c_size = ctypes.c_size_t


class MergeWeightsC(ctypes.Structure):
    _fields_ = [
        ("w_kv", c_ptr), ("b_kv", c_ptr), ("ln_kv_gamma", c_ptr), ("ln_kv_beta", c_ptr),
        ("query", c_ptr), ("w_o", c_ptr), ("b_o", c_ptr), ("ln_o_gamma", c_ptr), ("ln_o_beta", c_ptr),
        ("d_model", c_i32), ("n_heads", c_i32), ("ln_eps", ctypes.c_float),
    ]


class PagedKVC(ctypes.Structure):
    _fields_ = [
        ("base", c_ptr), ("n_layers", c_i32), ("n_pages", c_i32), ("n_kv_heads", c_i32),
        ("page_size", c_i32), ("head_dim", c_i32),
    ]


# name -> (restype, argtypes), exactly as declared in include/umim.h
SIGNATURES = {
    "umim_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "umim_version": (ctypes.c_int, []),
    "umim_merge_spans_workspace_size": (c_size, [c_i64, c_i32, c_i32]),
    "umim_merge_spans": (ctypes.c_int, [c_ptr, c_i64, c_ptr, c_i64, c_ptr, c_i32,
                                        ctypes.POINTER(MergeWeightsC), c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_build_compressed_workspace_size": (c_size, [c_i32, c_i32]),
    "umim_build_compressed": (ctypes.c_int, [c_ptr, c_i64, c_i32, c_ptr, c_i32, c_i32, c_ptr, c_ptr, c_ptr,
                                             c_i32, c_ptr, c_ptr, c_i64, c_ptr, c_ptr, c_ptr, c_size, c_ptr,
                                             c_ptr]),
    "umim_kv_rollback_workspace_size": (c_size, [c_i32, c_i32, c_i32, c_i32, c_i32, c_i32]),
    "umim_kv_rollback": (ctypes.c_int, [ctypes.POINTER(PagedKVC), c_ptr, c_i32, c_ptr, c_i32, c_ptr, c_ptr,
                                        c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_kv_rollback_rope": (ctypes.c_int, [ctypes.POINTER(PagedKVC), c_ptr, c_i32, c_ptr, c_i32, c_ptr, c_ptr,
                                             c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_i32, c_ptr, c_ptr, c_size, c_ptr,
                                             c_ptr]),
    "umim_kv_append": (ctypes.c_int, [ctypes.POINTER(PagedKVC), c_ptr, c_i32, c_ptr, c_i32, c_ptr, c_ptr, c_ptr,
                                      c_ptr, c_ptr]),
    "umim_decode_append_merge": (ctypes.c_int, [ctypes.POINTER(PagedKVC), c_ptr, c_i32, c_ptr, c_i32, c_ptr, c_ptr,
                                                c_ptr, c_ptr, c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_ptr, c_ptr]),
    "umim_decode_layer_step_workspace_size": (c_size, [c_i32, c_i32, c_i32]),
    "umim_decode_layer_step": (ctypes.c_int, [c_ptr, c_i32, ctypes.POINTER(PagedKVC), c_i32, c_ptr, c_i32, c_ptr,
                                              c_i32, c_ptr, c_ptr, c_i64, c_ptr, c_ptr, c_ptr, c_i32, c_ptr, c_ptr,
                                              c_i32, c_ptr, ctypes.c_float, c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_selftest_bounded_wait": (ctypes.c_int, [c_i32, ctypes.c_uint32, c_ptr, c_ptr, c_ptr, c_ptr]),
    "umim_prefill_attention_workspace_size": (c_size, [c_i32, c_i32, c_i32, c_i32]),
    "umim_prefill_attention": (ctypes.c_int, [c_ptr, c_ptr, c_ptr, c_i32, c_i32, c_i32, c_i32, c_ptr, c_i32,
                                              ctypes.c_float, c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_rule_table_bytes": (c_size, [c_i64]),
    "umim_rules_build": (ctypes.c_int, [c_ptr, c_size, c_ptr, c_i64, c_ptr, c_ptr]),
    "umim_match_prompts_workspace_size": (c_size, [c_i32, c_i32]),
    "umim_match_prompts": (ctypes.c_int, [c_ptr, c_size, c_ptr, c_i32, c_i32, c_ptr, c_ptr, c_ptr, c_ptr, c_ptr,
                                          c_ptr, c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_match_suffix": (ctypes.c_int, [c_ptr, c_size, c_ptr, c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_ptr, c_ptr,
                                         c_ptr, c_ptr]),
    "umim_lookup_surrogates": (ctypes.c_int, [c_ptr, c_i64, c_i32, c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_ptr]),
    "umim_distill_align_workspace_size": (c_size, [c_i32, c_i32]),
    "umim_distill_align": (ctypes.c_int, [c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_i32, c_ptr, c_ptr, c_ptr, c_i32,
                                          c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_distill_soft_ce_workspace_size": (c_size, [c_i32, c_i32]),
    "umim_distill_soft_ce": (ctypes.c_int, [c_ptr, c_i32, c_ptr, c_i32, c_i32, c_i64, c_ptr, c_ptr, c_i32, c_ptr,
                                            ctypes.c_float, c_ptr, c_ptr, c_ptr, c_ptr, c_size, c_ptr, c_ptr]),
    "umim_decode_attention_workspace_size": (c_size, [c_i32, c_i32, c_i32, c_i32]),
    "umim_decode_attention": (ctypes.c_int, [c_ptr, c_i32, ctypes.POINTER(PagedKVC), c_i32, c_ptr, c_i32,
                                             c_ptr, c_i32, ctypes.c_float, c_ptr, c_ptr, c_size, c_ptr,
                                             c_ptr]),
    "umim_decode_attention_static": (ctypes.c_int, [c_ptr, c_i32, ctypes.POINTER(PagedKVC), c_i32, c_ptr, c_i32,
                                                    c_ptr, c_i32, ctypes.c_float, c_ptr, c_ptr, c_ptr]),
    "umim_debug_build": (ctypes.c_int, []),
    "umim_debug_site_name": (ctypes.c_char_p, [c_i32]),
    "umim_selftest_bounds_check": (ctypes.c_int, [c_ptr, c_i64, c_i64, c_ptr, c_ptr]),
    "umim_trace_start": (ctypes.c_int, [c_i32]),
    "umim_trace_stop": (None, []),
    "umim_trace_read": (c_i32, [ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_char_p), c_i32]),
}

_libs = {}
_active = LIB_PATH


def use_debug(flag: bool) -> None:
    """Route every later call of the binding through libumim_debug.so (True)
    or libumim.so (False, the default).  Both may be loaded at once."""
    global _active
    _active = DEBUG_LIB_PATH if flag else LIB_PATH


def load(path: str = None):
    """Load the active library (or `path`) and declare every entry point;
    raises if it is missing."""
    path = path or _active
    lib = _libs.get(path)
    if lib is not None:
        return lib
    if not os.path.exists(path):
        raise RuntimeError(
            f"{os.path.basename(path)} not found at {path}: build it first "
            "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _libs[path] = lib
    return lib
