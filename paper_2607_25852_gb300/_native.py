"""ctypes declarations of libspec's C ABI (include/spec.h).

Loading fails loudly when the library has not been built: there is no CPU
fallback for any entry point.
"""
import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIBRARY = os.path.join(HERE, "libspec.so")

_P = ctypes.c_void_p
_I = ctypes.c_int
_SZ = ctypes.c_size_t

# name -> (restype, argtypes); the exported surface of include/spec.h
SIGNATURES = {
    "spec_error_string": (ctypes.c_char_p, [_I]),
    "spec_version": (_I, []),
    "spec_pointer_device_readable": (_I, [_P]),
    "spec_budget_from_ratios": (_I, [_I, _I, _P, _P, _I, _P]),
    "spec_allocate_workspace": (_SZ, [_I, _I, _I]),
    "spec_allocate": (_I, [_P, _I, _I, _P, _P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "spec_verify_workspace": (_SZ, [_I, _I, _I]),
    "spec_verify": (_I, [_P, _I, _P, _P, _P, _P, _I, _I, _I, _I, ctypes.c_float, _P, _P, _P,
                         _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "spec_verify_static": (_I, [_P, _I, _P, _P, _P, _P, _I, _I, _I, _I, ctypes.c_float, _P, _P,
                                _P, _P, _P, _P, _P, _P, _P]),
    "spec_commit": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "spec_profile_stream_pass": (_I, [_P, _P]),
    "spec_check_bounded_wait": (_I, [_P, _P]),
    "spec_draft_workspace": (_SZ, [_I, _I, _I]),
    "spec_draft": (_I, [_P, _I, _I, _I, _I, ctypes.c_float, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "spec_markov_workspace": (_SZ, [_I, _I, _I, _I]),
    "spec_markov_draft": (_I, [_P, _I, _P, _P, _I, _P, _I, _I, _I, ctypes.c_float, _P, _P, _P, _P, _P, _P, _P,
                               _P, _P, _SZ, _P]),
    "spec_graph_begin_capture": (_I, [_P]),
    "spec_graph_end_capture": (_I, [_P, _I, ctypes.POINTER(ctypes.c_void_p)]),
    "spec_graph_launch": (_I, [_P, _P]),
    "spec_graph_destroy": (_I, [_P]),
    "spec_select_round": (_I, [_P, _I, _P, _P, _P, _P, _P]),
    "spec_pack_rows": (_I, [_P, _SZ, _I, _I, _P, _P, _I, _P, _P]),
    "spec_shard_workspace": (_SZ, [_I, _I, _I]),
    "spec_shard_stats": (_I, [_P, _I, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, ctypes.c_float, _P, _P,
                              _P, _P, _SZ, _P]),
    "spec_shard_decide": (_I, [_P, _I, _P, _P, _P, _I, _I, _I, _I, ctypes.c_float, _P, _P, _P, _P,
                               _P, _P, _P, _P, _P, _P]),
    "spec_shard_sample": (_I, [_P, _I, _P, _I, _P, _I, _I, _I, _I, _I, ctypes.c_float, _P, _P, _P,
                               _P, _P, _SZ, _P]),
    "spec_shard_finish": (_I, [_P, _I, _P, _I, _I, _I, ctypes.c_float, _P, _P, _P, _P, _P, _P]),
}

_lib = None


def load(path: str = LIBRARY):
    """Load libspec.so (raises if it is missing: build it with __graft_entry__.build())."""
    global _lib
    if _lib is not None and path == LIBRARY:
        return _lib
    if not os.path.exists(path):
        raise ImportError(
            f"{path} is missing: the CUDA library has not been built. "
            "Run `python -c 'import __graft_entry__ as g; g.build()'` first.")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path == LIBRARY:
        _lib = lib
    return lib
