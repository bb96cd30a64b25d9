"""ctypes declarations for libtr.so (include/tr.h).  Marshalling only."""
from __future__ import annotations

import ctypes
import os
import re

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtr.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "tr.h")

TR_F32, TR_BF16, TR_F16 = 0, 1, 2
TR_STRIDE_INTERVAL = 1
STRIDE_MODES = {"alg1": 0, "interval": TR_STRIDE_INTERVAL}
TR_STATS_WORDS = 8
TR_STATUS_WORDS = 4
TR_MAX_N = 16384
TR_MAX_D = 16384
STATUS_NAMES = {0: "TR_OK", 1: "TR_ERR_ARG", 2: "TR_ERR_BUDGET", 3: "TR_ERR_DTYPE", 4: "TR_ERR_ALIGN",
                5: "TR_ERR_WORKSPACE", 6: "TR_ERR_CUDA", 7: "TR_ERR_UNSUPPORTED"}


class TrTokens(ctypes.Structure):
    _fields_ = [
        ("x", ctypes.c_void_p),
        ("x_pre", ctypes.c_void_p),
        ("x_post", ctypes.c_void_p),
        ("dtype", ctypes.c_int32),
        ("d", ctypes.c_int32),
        ("batch", ctypes.c_int32),
        ("n", ctypes.c_int32),
        ("cu_seqlens", ctypes.c_void_p),
        ("total", ctypes.c_int32),
        ("max_n", ctypes.c_int32),
        ("flags", ctypes.c_int32),
    ]


TR_ACT = {"gelu": 0, "quick_gelu": 1, "none": 2}


class TrMlp(ctypes.Structure):
    _fields_ = [
        ("x_pre", ctypes.c_void_p),
        ("resid", ctypes.c_void_p),
        ("w1", ctypes.c_void_p),
        ("w2", ctypes.c_void_p),
        ("b1", ctypes.c_void_p),
        ("b2", ctypes.c_void_p),
        ("t", ctypes.c_int32),
        ("d", ctypes.c_int32),
        ("d_hidden", ctypes.c_int32),
        ("act", ctypes.c_int32),
    ]


class TrError(RuntimeError):
    def __init__(self, fn, code, lib):
        self.code = code
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(code, code)} ({lib.tr_status_string(code).decode()})")


_lib = None


def load() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -c \"import __graft_entry__ as g; "
                           f"g.build()\"` (the reducer has no CPU path)")
    lib = ctypes.CDLL(LIB_PATH)
    P, I32, SZ, VP = ctypes.POINTER, ctypes.c_int32, ctypes.c_size_t, ctypes.c_void_p
    tok = P(TrTokens)
    lib.tr_status_string.argtypes, lib.tr_status_string.restype = [I32], ctypes.c_char_p
    lib.tr_version.argtypes, lib.tr_version.restype = [], ctypes.c_char_p
    lib.tr_budgets.argtypes = [I32, P(I32), I32, I32, I32, I32, I32, P(I32), P(I32), P(I32)]
    lib.tr_budgets.restype = I32
    lib.tr_workspace_bytes.argtypes, lib.tr_workspace_bytes.restype = [tok], SZ
    lib.tr_score.argtypes, lib.tr_score.restype = [tok, VP, VP, VP, VP], I32
    lib.tr_select.argtypes = [tok, VP, VP, VP, VP, VP, VP, VP, VP, VP, SZ, VP, VP]
    lib.tr_select.restype = I32
    lib.tr_gather.argtypes, lib.tr_gather.restype = [tok, VP, VP, I32, VP, VP], I32
    lib.tr_select_gather.argtypes = [tok, VP, VP, VP, VP, I32, VP, VP, VP, VP, VP, SZ, VP, VP]
    lib.tr_select_gather.restype = I32
    lib.tr_pipeline_create.argtypes = [P(VP), VP, I32, P(VP), SZ, P(VP)]
    lib.tr_pipeline_create.restype = I32
    lib.tr_pipeline_submit.argtypes = [VP, tok, VP, VP, VP, I32, VP, VP, VP, VP, VP, VP, VP]
    lib.tr_pipeline_submit.restype = I32
    lib.tr_pipeline_wait.argtypes, lib.tr_pipeline_wait.restype = [VP, VP], I32
    lib.tr_pipeline_kernels.argtypes, lib.tr_pipeline_kernels.restype = [VP], ctypes.c_longlong
    lib.tr_pipeline_destroy.argtypes, lib.tr_pipeline_destroy.restype = [VP], I32
    lib.tr_reduce.argtypes = [tok, VP, VP, VP, I32, VP, VP, VP, VP, VP, SZ, VP, VP]
    lib.tr_reduce.restype = I32
    mlp = P(TrMlp)
    lib.tr_mlp_hidden.argtypes, lib.tr_mlp_hidden.restype = [mlp, VP, VP, VP], I32
    lib.tr_mlp_workspace_bytes.argtypes, lib.tr_mlp_workspace_bytes.restype = [mlp], SZ
    lib.tr_mlp_score.argtypes = [mlp, VP, VP, VP, VP, VP, VP, VP, SZ, VP, VP]
    lib.tr_mlp_score.restype = I32
    lib.tr_project_kept.argtypes = [tok, VP, VP, I32, VP, VP, I32, I32, VP, VP, VP]
    lib.tr_project_kept.restype = I32
    lib.tr_project.argtypes = [VP, I32, I32, VP, VP, I32, I32, VP, VP, VP]
    lib.tr_project.restype = I32
    _lib = lib
    return lib


def check(fn: str, code: int):
    if code != 0:
        raise TrError(fn, code, load())


def declared_functions():
    """Names of the functions include/tr.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(tr_[a-z_0-9]+)\s*\(", text, flags=re.M)))
