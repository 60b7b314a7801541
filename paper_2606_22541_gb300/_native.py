"""ctypes view of libasap_moe.so (argument marshalling only).

Loading fails loudly when the library has not been built: there is no other
implementation of the layer behind this package.
"""
import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libasap_moe.so")

ASAP_OK = 0
ASAP_ERR_INVALID = -1
ASAP_ERR_UNSUPPORTED = -2
ASAP_ERR_WORKSPACE = -3
ASAP_ERR_CUDA = -4
ASAP_ERR_DEVICE_STATUS = -5

STATUS_NAMES = {0: "ASAP_OK", -1: "ASAP_ERR_INVALID", -2: "ASAP_ERR_UNSUPPORTED",
                -3: "ASAP_ERR_WORKSPACE", -4: "ASAP_ERR_CUDA", -5: "ASAP_ERR_DEVICE_STATUS"}


class AsapMoeConfig(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int32), ("n_experts", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("inter", ctypes.c_int32), ("n_shared", ctypes.c_int32), ("shared_inter", ctypes.c_int32),
                ("gating", ctypes.c_int32), ("n_groups", ctypes.c_int32), ("topk_groups", ctypes.c_int32),
                ("route_scale", ctypes.c_float), ("dtype", ctypes.c_int32), ("max_tokens", ctypes.c_int32)]


class AsapMoeWeights(ctypes.Structure):
    _fields_ = [(name, ctypes.c_void_p) for name in (
        "router_w", "router_bias", "w_gate", "w_up", "w_down", "s_gate", "s_up", "s_down",
        "sh_gate", "sh_up", "sh_down", "sh_s_gate", "sh_s_up", "sh_s_down")]


_P = ctypes.c_void_p
_I = ctypes.c_int32
_SZ = ctypes.c_size_t

SIGNATURES = {
    "asap_moe_create": [ctypes.POINTER(AsapMoeConfig), ctypes.POINTER(AsapMoeWeights), ctypes.POINTER(_P)],
    "asap_moe_create_layers": [ctypes.POINTER(AsapMoeConfig), ctypes.POINTER(AsapMoeWeights), _I,
                               ctypes.POINTER(_P)],
    "asap_moe_n_layers": [_P, ctypes.POINTER(_I)],
    "asap_moe_destroy": [_P],
    "asap_moe_time_layer": [_I, ctypes.POINTER(_P)],
    "asap_moe_set_combine": [_P, _I],
    "asap_moe_workspace_size": [ctypes.POINTER(AsapMoeConfig), _I, ctypes.POINTER(_SZ)],
    "asap_moe_check_config": [ctypes.POINTER(AsapMoeConfig)],
    "asap_moe_router_logits": [_P, _P, _I, _P, _P, _SZ, _P],
    "asap_moe_route": [_P, _P, _I, _P, _P, _P, _P, _P, _SZ, _P],
    "asap_moe_route_logits": [_P, _P, _I, _P, _P, _P, _P, _P, _SZ, _P],
    "asap_moe_dispatch": [_P, _P, _I, _P, _P, _P, _P, _P, _P, _SZ, _P],
    "asap_moe_expert_ffn": [_P, _P, _P, _P, _P, _I, _P, _P, _P, _SZ, _P],
    "asap_moe_expert_gate_up": [_P, _P, _P, _P, _P, _I, _P, _P, _P, _SZ, _P],
    "asap_moe_expert_down": [_P, _P, _P, _P, _P, _I, _P, _P, _P, _SZ, _P],
    "asap_moe_combine": [_P, _P, _P, _P, _P, _I, _P, _P],
    "asap_moe_layer": [_P, _P, _I, _P, _P, _SZ, _P],
    "asap_moe_route_noalloc": [_P, _P, _I, _P, _P, _P, _P, _P],
    "asap_moe_layer_batched": [_P, _I, ctypes.POINTER(_P), ctypes.POINTER(_I), ctypes.POINTER(_P), _P, _SZ, _P],
    "asap_moe_layer_dyn": [_P, _P, _P, _I, _P, _P, _SZ, _P],
    "asap_moe_layer_batched_dyn": [_P, _P, _I, ctypes.POINTER(_P), ctypes.POINTER(_I), ctypes.POINTER(_P), _P, _SZ,
                                   _P],
    "asap_moe_set_tiling": [_P, _I],
    "asap_moe_mailbox_create": [_P, _I, _I, _P, ctypes.c_int64, ctypes.POINTER(_P)],
    "asap_moe_mailbox_destroy": [_P],
    "asap_moe_mailbox_post": [_P, _I, _P, _I, _P, _P, _P, ctypes.POINTER(ctypes.c_uint64)],
    "asap_moe_mailbox_serve": [_P, _I, ctypes.c_uint64, _P],
    "asap_moe_mailbox_serve_many": [_P, _I, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_uint64), _P],
    "asap_moe_mailbox_wait": [_P, _I, _P],
    "asap_moe_mailbox_served": [_P, _I, ctypes.POINTER(ctypes.c_uint64)],
    "asap_moe_mailbox_time_gemms": [_P, _P, _P],
    "asap_moe_mailbox_rounds": [_P, ctypes.POINTER(_I), ctypes.POINTER(_I), _I],
    "asap_moe_status": [_P, ctypes.POINTER(ctypes.c_uint32)],
    "asap_moe_last_error": [],
}

_lib = None


def lib():
    """The loaded library (raises ImportError when it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with "
                              "`python -m paper_2606_22541_gb300.build` (the layer has no other backend)")
        L = ctypes.CDLL(LIB_PATH)
        for name, args in SIGNATURES.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = ctypes.c_char_p if name == "asap_moe_last_error" else ctypes.c_int
        _lib = L
    return _lib


class AsapError(RuntimeError):
    def __init__(self, fn, code):
        msg = lib().asap_moe_last_error().decode(errors="replace")
        super().__init__(f"{fn} -> {STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


def check(fn, code):
    if code != ASAP_OK:
        raise AsapError(fn, code)
    return code
