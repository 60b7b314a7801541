"""The C-ABI library loads on a machine without a GPU, exports every entry
point the header declares, and its pure-host calls (config checks, workspace
sizing, argument validation) behave as documented.  No compute calls."""
import ctypes
import os
import re

import pytest

from paper_2606_22541_gb300 import _native, build as build_mod
from paper_2606_22541_gb300.configs import CONFIGS, DSV3, TINY
from paper_2606_22541_gb300 import api

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "asap_moe.h")


@pytest.fixture(scope="module")
def L():
    build_mod.build()
    return _native.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(asap_moe_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("asap_moe_route", "asap_moe_dispatch", "asap_moe_expert_ffn",
                     "asap_moe_combine", "asap_moe_layer", "asap_moe_create", "asap_moe_destroy"):
        assert required in names


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name
    assert set(declared_functions()) == set(_native.SIGNATURES)


def test_check_config(L):
    for c in CONFIGS.values():
        code = api.asap_moe_check_config(c, 4096)
        assert code == _native.ASAP_OK, api.asap_moe_last_error()
    from dataclasses import replace
    bad = [replace(TINY, hidden=200), replace(TINY, top_k=9), replace(TINY, inter=100),
           replace(DSV3, n_groups=7), replace(DSV3, topk_groups=0), replace(TINY, n_experts=300),
           replace(TINY, gating="softmax", top_k=0)]
    for b in bad:
        assert api.asap_moe_check_config(b, 16) == _native.ASAP_ERR_INVALID
    assert api.asap_moe_check_config(TINY, 0) == _native.ASAP_ERR_INVALID


def test_workspace_size_fp8(L):
    from paper_2606_22541_gb300.configs import DSV3_FP8
    a = api.asap_moe_workspace_size(DSV3_FP8, 4096)
    b = api.asap_moe_workspace_size(DSV3, 4096)
    # e4m3 rows of x and h plus bf16 expert outputs
    assert a > 4096 * 8 * (7168 + 2048 + 7168 * 2)
    assert a != b


def test_workspace_size(L):
    assert api.asap_moe_workspace_size(TINY, 0, 100) == 0
    a = api.asap_moe_workspace_size(DSV3, 4096)
    b = api.asap_moe_workspace_size(DSV3, 4097)
    assert b > a > 4096 * 8 * 7168 * 2   # at least the grouped hidden states
    assert a % 256 == 0
    with pytest.raises(_native.AsapError):
        api.asap_moe_workspace_size(TINY, 10, 5)


def test_create_rejects_bad_arguments_before_touching_cuda(L):
    c = api.make_config(TINY, 16)
    w = _native.AsapMoeWeights()
    out = ctypes.c_void_p(1234)
    assert L.asap_moe_create(ctypes.byref(c), ctypes.byref(w), ctypes.byref(out)) == _native.ASAP_ERR_INVALID
    assert out.value is None
    assert "required" in api.asap_moe_last_error()
    assert L.asap_moe_create(None, ctypes.byref(w), ctypes.byref(out)) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_destroy(None) == _native.ASAP_OK


def test_calls_reject_null_handle(L):
    assert L.asap_moe_layer(None, None, 1, None, None, 0, None) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_combine(None, None, None, None, None, 1, None, None) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_status(None, None) == _native.ASAP_ERR_INVALID


def test_create_layers_rejects_bad_layer_counts_before_touching_cuda(L):
    c = api.make_config(TINY, 16)
    ws = (_native.AsapMoeWeights * 2)()
    out = ctypes.c_void_p(1234)
    for n in (0, -1, 5000):
        assert L.asap_moe_create_layers(ctypes.byref(c), ws, n, ctypes.byref(out)) == _native.ASAP_ERR_INVALID
        assert out.value is None
    assert L.asap_moe_create_layers(ctypes.byref(c), ws, 2, ctypes.byref(out)) == _native.ASAP_ERR_INVALID
    assert "layer 0" in api.asap_moe_last_error()
    assert L.asap_moe_layer_dyn(None, None, None, 1, None, None, 0, None) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_layer_batched_dyn(None, None, 1, None, None, None, None, 0, None) == _native.ASAP_ERR_INVALID
    n = ctypes.c_int32(0)
    assert L.asap_moe_n_layers(None, ctypes.byref(n)) == _native.ASAP_ERR_INVALID


def test_tiling_modes_match_the_header(L):
    text = open(HEADER).read()
    vals = {m: int(v) for m, v in re.findall(r"ASAP_TILING_(\w+)\s*=\s*(\d+)", text)}
    assert vals == {"AUTO": api.TILING_AUTO, "SINGLE": api.TILING_SINGLE, "PAIRED": api.TILING_PAIRED}
    # a NULL handle is rejected on the host
    assert L.asap_moe_set_tiling(None, api.TILING_AUTO) == _native.ASAP_ERR_INVALID


def test_time_layer_validates_its_request(L):
    arr = (ctypes.c_void_p * 7)()
    assert L.asap_moe_time_layer(-1, arr) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_time_layer(7, arr) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_time_layer(2, None) == _native.ASAP_ERR_INVALID
    assert L.asap_moe_time_layer(0, None) == _native.ASAP_OK
    # NULL entries are allowed (skipped when the layer records them); a
    # failing layer call takes the request and records nothing
    assert L.asap_moe_time_layer(6, arr) == _native.ASAP_OK
    assert L.asap_moe_layer(None, None, 1, None, None, 0, None) == _native.ASAP_ERR_INVALID


def test_combine_modes_match_the_header(L):
    text = open(HEADER).read()
    vals = {m: int(v) for m, v in re.findall(r"ASAP_COMBINE_(\w+)\s*=\s*(\d+)", text)}
    assert vals == {"SEPARATE": api.COMBINE_SEPARATE, "FUSED": api.COMBINE_FUSED}
    assert L.asap_moe_set_combine(None, api.COMBINE_FUSED) == _native.ASAP_ERR_INVALID
