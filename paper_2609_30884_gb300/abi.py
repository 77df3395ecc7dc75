"""ctypes mirror of include/crf.h and the loader for the in-tree libcrf.so.

Argument marshalling only: every step of the path runs in the CUDA library.
Loading fails loudly when the library has not been built; there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_char_p, c_float, c_int, c_size_t, c_uint32, c_void_p

LIB_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib")
# CRF_LIB_VARIANT=debug selects the build with device-side page-id checks
# (``build.build(debug=True)``); anything else, or unset, the release build.
LIB_PATH = os.path.join(LIB_DIR, "libcrf_debug.so" if os.environ.get("CRF_LIB_VARIANT") == "debug"
                        else "libcrf.so")

OK, EINVAL, ESHAPE, EUNSUPPORTED, ENOMEM, ECUDA, ETIMEOUT = range(7)
STATUS_NAMES = ["CRF_OK", "CRF_EINVAL", "CRF_ESHAPE", "CRF_EUNSUPPORTED", "CRF_ENOMEM",
                "CRF_ECUDA", "CRF_ETIMEOUT"]
NUM_MODULES = 7
PAGE_SIZE = 16
MAX_REQUESTS = 32

# Every symbol include/crf.h declares.
EXPORTS = ("crf_create", "crf_destroy", "crf_last_error", "crf_check", "crf_workspace_size",
           "crf_recompute_window", "crf_drift_workspace_size", "crf_drift",
           "crf_kl_workspace_size", "crf_kl", "crf_kl_logits_noalloc", "crf_profile_enable",
           "crf_profile_read", "crf_decode_workspace_size", "crf_decode_step",
           "crf_selftest_timeout")


class ModelDims(ctypes.Structure):
    _fields_ = [("n_layers", c_int), ("hidden", c_int), ("n_q_heads", c_int),
                ("n_kv_heads", c_int), ("head_dim", c_int), ("ffn", c_int), ("vocab", c_int),
                ("rms_eps", c_float), ("rope_theta", c_float), ("qkv_bias", c_int)]


class LoraDims(ctypes.Structure):
    _fields_ = [("rank", c_int), ("alpha", c_float), ("module_mask", c_uint32)]


class LayerWeights(ctypes.Structure):
    _fields_ = [("W", c_void_p * NUM_MODULES), ("bias", c_void_p * 3), ("ln1", c_void_p),
                ("ln2", c_void_p)]


class Model(ctypes.Structure):
    _fields_ = [("dims", ModelDims), ("layers", POINTER(LayerWeights)), ("embed", c_void_p),
                ("final_norm", c_void_p), ("lm_head", c_void_p)]


class Adapter(ctypes.Structure):
    _fields_ = [("dims", LoraDims), ("A", POINTER(c_void_p)), ("B", POINTER(c_void_p))]


class KVPool(ctypes.Structure):
    _fields_ = [("k_pages", POINTER(c_void_p)), ("v_pages", POINTER(c_void_p)),
                ("num_pages", c_int)]


class Request(ctypes.Structure):
    _fields_ = [("n_tokens", c_int), ("s", c_int), ("e", c_int), ("page_table", c_void_p),
                ("tokens", c_void_p), ("hidden_in", c_void_p),
                ("hidden_out", POINTER(c_void_p)), ("final_hidden_out", c_void_p)]


class DecodeRow(ctypes.Structure):
    _fields_ = [("pos", c_int), ("page_table", c_void_p), ("token", c_void_p)]


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libcrf.so (built by ``paper_2609_30884_gb300.build``); raise if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{os.path.basename(path)} not built at {path}; run "
                           "paper_2609_30884_gb300.build.build()"
                           + ("" if path.endswith("libcrf.so") else " with debug=True"))
    lib = ctypes.CDLL(path)
    P = c_void_p
    sig = {
        "crf_create": ([POINTER(c_void_p), c_int], c_int),
        "crf_destroy": ([P], c_int),
        "crf_last_error": ([], c_char_p),
        "crf_check": ([P, P], c_int),
        "crf_selftest_timeout": ([P, P], c_int),
        "crf_workspace_size": ([P, POINTER(Model), POINTER(LoraDims), POINTER(Request), c_int,
                                POINTER(c_size_t)], c_int),
        "crf_recompute_window": ([P, POINTER(Model), POINTER(Adapter), POINTER(KVPool),
                                  POINTER(Request), c_int, P, c_size_t, P], c_int),
        "crf_drift_workspace_size": ([P, POINTER(ModelDims), POINTER(LoraDims), POINTER(c_size_t)],
                                     c_int),
        "crf_drift": ([P, POINTER(ModelDims), POINTER(Adapter), POINTER(POINTER(Adapter)), P, P,
                       c_size_t, P], c_int),
        "crf_kl_workspace_size": ([P, c_int, c_int, c_int, POINTER(c_size_t)], c_int),
        "crf_decode_workspace_size": ([P, POINTER(Model), POINTER(LoraDims), POINTER(DecodeRow), c_int,
                                       POINTER(c_size_t)], c_int),
        "crf_decode_step": ([P, POINTER(Model), POINTER(Adapter), POINTER(KVPool), POINTER(DecodeRow),
                             c_int, P, P, P, c_size_t, P], c_int),
        "crf_kl": ([P, POINTER(Model), P, P, c_int, c_int, P, P, P, c_size_t, P], c_int),
        "crf_kl_logits_noalloc": ([c_int, P, P, c_int, c_int, P, P], c_int),
        "crf_profile_enable": ([P, c_int, c_int], c_int),
        "crf_profile_read": ([P, c_int, ctypes.c_char_p, POINTER(ctypes.c_double), POINTER(c_int),
                              POINTER(c_int), POINTER(c_int)], c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


class CrfError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"{name}: {message}")


def check(status: int) -> None:
    if status != OK:
        msg = load().crf_last_error()
        raise CrfError(status, msg.decode() if msg else "")
