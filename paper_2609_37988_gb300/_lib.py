"""ctypes binding of ``libkvk.so`` (include/kvk.h).

Argument marshalling only: every step of the decode path runs in the
library's CUDA kernels.  Loading fails loudly when the library is missing;
there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libkvk.so")

KVK_OK = 0
STATUS_NAMES = {
    0: "KVK_OK", 1: "KVK_ERR_INVALID_ARG", 2: "KVK_ERR_INVALID_CONFIG",
    3: "KVK_ERR_INHERITED_LAYER", 4: "KVK_ERR_CAPACITY", 5: "KVK_ERR_UNSUPPORTED",
    6: "KVK_ERR_CUDA", 7: "KVK_ERR_DEVICE",
}
KIND_GQA, KIND_MLA = 0, 1
AXIS_TOKEN, AXIS_CHANNEL = 0, 1
QUANT_GROUPED, QUANT_SYMMETRIC = 0, 1
DTYPE_F32, DTYPE_BF16 = 0, 1


class ModelDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "kind", "n_layers", "n_q_heads", "n_kv_heads", "head_dim",
        "latent_dim", "rope_dim", "max_batch", "max_ctx")]


class LayerCfg(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "inherit", "bits", "group", "key_axis", "value_axis", "width", "evict_capacity",
        "scheme")]


class KVKError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = status
        self.name = STATUS_NAMES.get(status, str(status))
        super().__init__(f"{self.name}: {message}")


_P = ctypes.c_void_p
_I = ctypes.c_int32
_F = ctypes.c_float
_SZ = ctypes.c_size_t

# name -> argument types (all return kvk_status unless listed in _RET)
_SIGS = {
    "kvk_cache_plan": [ctypes.POINTER(ModelDesc), ctypes.POINTER(LayerCfg), ctypes.POINTER(_SZ)],
    "kvk_workspace_size": [ctypes.POINTER(ModelDesc), _I, ctypes.POINTER(_SZ)],
    "kvk_cache_create": [ctypes.POINTER(ModelDesc), ctypes.POINTER(LayerCfg), ctypes.POINTER(_P),
                         _P, _SZ, _I, ctypes.POINTER(_P)],
    "kvk_cache_destroy": [_P],
    "kvk_cache_reset": [_P, _P],
    "kvk_set_wait_limit": [_P, ctypes.c_uint32],
    "kvk_set_decode_schedule": [_P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32],
    "kvk_layer_source": [_P, _I, ctypes.POINTER(_I)],
    "kvk_layer_lengths": [_P, _I, ctypes.POINTER(_P)],
    "kvk_append": [_P, _I, _P, _P, _I, _I, _P, _P],
    "kvk_set_kept": [_P, _I, _P, _P, _P],
    "kvk_evict_scratch_size": [_P, _I, _I, ctypes.POINTER(_SZ)],
    "kvk_evict_window": [_P, _I, _P, _I, _I, _F, _I, _P, _SZ, _P],
    "kvk_export_kept": [_P, _I, _P, _P, ctypes.POINTER(_I), _P],
    "kvk_prefill_scratch_size": [_P, _I, _I, ctypes.POINTER(_SZ)],
    "kvk_prefill_attention": [_P, _I, _P, _I, _I, _F, _P, _P, _SZ, _P],
    "kvk_prefill_attention_mla": [_P, _I, _P, _P, _P, _P, _I, _F, _P, _P, _SZ, _P],
    "kvk_rewind": [_P, _I, _P],
    "kvk_decode_plan_splits": [_P, _I, ctypes.POINTER(_I)],
    "kvk_decode_attention": [_P, _I, _P, _I, _F, _P, _I, _P],
    "kvk_decode_attention_mla": [_P, _I, _P, _P, _P, _P, _F, _P, _I, _P],
    "kvk_decode_partial": [_P, _I, _P, _I, _F, _P, _I, _P],
    "kvk_decode_attention_noalloc": [_P, _I, _P, _I, _F, _P, _I, _P],
    "kvk_splitk_reduce": [_P, _I, _I, _I, _P, _P],
    "kvk_cost": [_P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                 ctypes.POINTER(ctypes.c_double)],
    "kvk_plan_cost": [ctypes.POINTER(ModelDesc), ctypes.POINTER(LayerCfg), ctypes.POINTER(ctypes.c_double),
                      ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)],
    "kvk_export_layer": [_P, _I, _P, _P, _P, _P, _P, _P, _P, _P],
    "kvk_get_device_error": [_P, _P, ctypes.POINTER(_I)],
    "kvk_status_string": [_I],
    "kvk_last_error": [],
    "kvk_version": [],
}
_RET = {"kvk_status_string": ctypes.c_char_p, "kvk_last_error": ctypes.c_char_p,
        "kvk_version": ctypes.c_char_p}

_lib = None


def load(path: str = LIB_PATH):
    """Load the library (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(
            f"{path} is missing: build it with `python -m paper_2609_37988_gb300.build` "
            "(there is no fallback implementation)")
    lib = ctypes.CDLL(path)
    for name, args in _SIGS.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = _RET.get(name, ctypes.c_int32)
    _lib = lib
    return lib


def exported_symbols():
    """Names this binding expects the library to export."""
    return list(_SIGS)


def check(status: int):
    if status != KVK_OK:
        lib = load()
        raise KVKError(status, lib.kvk_last_error().decode())
