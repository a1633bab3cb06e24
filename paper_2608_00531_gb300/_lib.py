"""ctypes loader for libcure.so (include/cure.h).

The library is built in-tree by ``paper_2608_00531_gb300.build``.  Loading
fails loudly when it is missing: there is no CPU fallback anywhere in the
package.
"""
from __future__ import annotations

import ctypes as C
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libcure.so")

CURE_OK = 0
STATUS = {0: "CURE_OK", 1: "CURE_ERR_INVALID_ARG", 2: "CURE_ERR_CAPACITY", 3: "CURE_ERR_CUDA",
          4: "CURE_ERR_DEVICE_FAULT", 5: "CURE_ERR_UNSUPPORTED"}

DEVERR_PAGE, DEVERR_SLOT, DEVERR_NODES, DEVERR_TOKEN, DEVERR_TIMEOUT = 0x1, 0x2, 0x4, 0x8, 0x10

# every entry point the header declares
EXPORTS = ("cure_score_draft", "cure_build_tree", "cure_tree_attn", "cure_tree_attn_workspace_size",
           "cure_accept", "cure_lm_head_argmax", "cure_lm_head_workspace_size", "cure_selftest_wait_timeout", "cure_sample_target", "cure_resync_kv", "cure_device_error", "cure_status_string",
           "cure_abi_version")


class TreeParams(C.Structure):
    _fields_ = [("batch", C.c_int32), ("block", C.c_int32), ("topk", C.c_int32),
                ("tau", C.c_float), ("budget", C.c_int32), ("branches", C.c_int32),
                ("repair_depth", C.c_int32), ("max_ufp", C.c_int32),
                ("margin_scale", C.c_float), ("branch_min", C.c_int32),
                ("max_depth", C.c_int32), ("beam", C.c_int32)]


class KVDesc(C.Structure):
    _fields_ = [("layout", C.c_int32), ("heads_kv", C.c_int32), ("head_dim", C.c_int32),
                ("page_size", C.c_int32), ("max_len", C.c_int32), ("num_pages", C.c_int32),
                ("block_table", C.c_void_p)]


class CureError(RuntimeError):
    def __init__(self, fn: str, code: int, detail: str = ""):
        super().__init__(f"{fn} returned {STATUS.get(code, code)}" + (f": {detail}" if detail else ""))
        self.code = code


_lib = None

P = C.c_void_p
I32 = C.c_int32


def load() -> C.CDLL:
    """Load libcure.so once; raise when it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = C.CDLL(LIB_PATH)
    lib.cure_score_draft.argtypes = [P, I32, I32, I32, P, P, P, P, P]
    lib.cure_build_tree.argtypes = [C.POINTER(TreeParams), P, P, P, P, P, P, P, P, P, P, P, P, P, P]
    lib.cure_tree_attn.argtypes = [P, P, P, P, P, C.POINTER(KVDesc), P, P, P, I32, I32, I32,
                                   C.c_float, P, P, C.c_size_t, P]
    lib.cure_tree_attn_workspace_size.argtypes = [I32, I32, I32, C.POINTER(KVDesc)]
    lib.cure_tree_attn_workspace_size.restype = C.c_size_t
    lib.cure_accept.argtypes = [P, P, I32, I32, I32, I32, P, P, P, P, P, P, P, P, P, P, P]
    lib.cure_sample_target.argtypes = [P, P, C.c_float, I32, I32, I32, P, P, P]
    lib.cure_lm_head_argmax.argtypes = [P, P, I32, I32, I32, P, P, P, C.c_size_t, P]
    lib.cure_lm_head_workspace_size.argtypes = [I32, I32]
    lib.cure_lm_head_workspace_size.restype = C.c_size_t
    lib.cure_selftest_wait_timeout.argtypes = [C.c_int64, P]
    lib.cure_selftest_wait_timeout.restype = C.c_int
    lib.cure_resync_kv.argtypes = [I32, C.POINTER(C.c_void_p), C.POINTER(C.c_void_p),
                                   C.POINTER(KVDesc), P, P, I32, I32, I32, P, P, P, P, P, P, P,
                                   P, P, P]
    lib.cure_device_error.argtypes = [P, C.POINTER(I32)]
    lib.cure_status_string.argtypes = [C.c_int]
    lib.cure_status_string.restype = C.c_char_p
    lib.cure_abi_version.restype = I32
    for name in ("cure_score_draft", "cure_build_tree", "cure_tree_attn", "cure_accept",
                 "cure_resync_kv", "cure_device_error", "cure_sample_target", "cure_lm_head_argmax"):
        getattr(lib, name).restype = C.c_int
    _lib = lib
    return lib


def check(fn: str, code: int) -> None:
    if code != CURE_OK:
        raise CureError(fn, code)
