"""The one-launch routing path (router GEMM split over a thread-block cluster,
gating and scan in the same kernel) against the float64 oracle and against
the composed route (router logits, then routing from those logits), at a
hidden size where the router's K slices take every cluster size the kernel
has (1, 2 and 4) and at token counts with ragged last tiles."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import DSV3

from _helpers import bf16_to_f64, weights_f64, compare_rows, routing_check

pytestmark = pytest.mark.gpu

DEV = "cuda"

# H = 2048: 32 k-blocks, so the router splits K into up to 4 slices; n picks
# 4 slices up to 38 tiles of 128 tokens, 2 up to 76, then 1.
DS_ROUTE = inputs.small_variant(DSV3, name="dsv3_route", hidden=2048, inter=128, shared_inter=128,
                                microbatches=[700, 10000])
DS_ROUTE_G4 = inputs.small_variant(DS_ROUTE, name="dsv3_route_g4", n_groups=4, topk_groups=2, top_k=6)
DS_ROUTE_G1 = inputs.small_variant(DS_ROUTE, name="dsv3_route_g1", n_groups=1, topk_groups=1)
# a selection bias (it moves the selection keys and group scores, not the weights)
DS_ROUTE_BIAS = inputs.small_variant(DS_ROUTE, name="dsv3_route_bias")
SIZES = [1, 33, 130, 700, 5000, 10000]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


_cache = {}


def case(cfg):
    if cfg.name not in _cache:
        w = inputs.make_weights(cfg, DEV)
        if cfg is DS_ROUTE_BIAS:
            g = torch.Generator(device=DEV).manual_seed(4242)
            w["router_bias"] = 0.05 * torch.randn(cfg.n_experts, generator=g, device=DEV)
        _cache[cfg.name] = (w, api.asap_moe_create(cfg, w, max(SIZES)), weights_f64(w))
    return _cache[cfg.name]


def bias_of(w):
    b = w.get("router_bias")
    return None if b is None else b.cpu().numpy().astype(np.float32).astype(np.float64)


def outputs(n, cfg):
    k, E = cfg.top_k, cfg.n_experts
    return (torch.full((n, k), -7, dtype=torch.int32, device=DEV),
            torch.full((n, k), -7.0, dtype=torch.float32, device=DEV),
            torch.full((E,), -7, dtype=torch.int32, device=DEV),
            torch.full((E + 1,), -7, dtype=torch.int32, device=DEV))


@pytest.mark.parametrize("cfg", [DS_ROUTE, DS_ROUTE_G4, DS_ROUTE_G1, DS_ROUTE_BIAS], ids=lambda c: c.name)
@pytest.mark.parametrize("n", SIZES)
def test_fused_route_against_oracle_and_composed_route(cfg, n):
    w, h, wf = case(cfg)
    x = inputs.make_tokens(cfg, n, 3, DEV)
    got = outputs(n, cfg)
    api.asap_moe_route(h, x, *got, api.workspace(h, n))
    # the composed route: logits (same K slices, added in order), then gating
    logits = torch.empty((n, cfg.n_experts), dtype=torch.float32, device=DEV)
    api.asap_moe_router_logits(h, x, logits, api.workspace(h, n))
    ref = outputs(n, cfg)
    api.asap_moe_route_logits(h, logits, *ref, api.workspace(h, n))
    torch.cuda.synchronize()
    for a, b in zip(got, ref):
        assert torch.equal(a, b)
    idx, wt, counts, offsets = (t.cpu().numpy() for t in got)
    xf = bf16_to_f64(x)
    L = oracle.router_logits(xf, wf["router_w"])
    eps = oracle.logit_error_bound(xf, wf["router_w"])
    ocfg = cfg.oracle_cfg()
    bias = bias_of(w)
    idx_ref, w_ref = oracle.route(L, ocfg, bias)
    ig = idx.astype(np.int64)
    decided = routing_check(L, eps, ocfg, ig, wt.astype(np.float64), w_ref, idx_ref, bias=bias)
    assert np.array_equal(counts, np.bincount(ig.reshape(-1), minlength=cfg.n_experts))
    assert offsets[0] == 0 and np.array_equal(np.diff(offsets), counts) and offsets[-1] == ig.size
    if decided.all():
        assert np.array_equal(counts, oracle.expert_counts(idx_ref, cfg.n_experts))
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"device status word {word:#x}"


@pytest.mark.parametrize("n", [700, 5000])
def test_layer_on_fused_route_against_oracle(n):
    """The layer's dispatch places rows by the fused kernel's chunk bases."""
    cfg = DS_ROUTE
    w, h, wf = case(cfg)
    x = inputs.make_tokens(cfg, n, 4, DEV)
    out = torch.empty_like(x)
    api.asap_moe_layer(h, x, out, api.workspace(h, n))
    torch.cuda.synchronize()
    xf = bf16_to_f64(x)
    r = oracle.moe_layer(xf, wf["router_w"], wf["w_gate"], wf["w_up"], wf["w_down"], cfg.oracle_cfg(),
                         shared=(wf["sh_gate"], wf["sh_up"], wf["sh_down"]))
    eps = oracle.logit_error_bound(xf, wf["router_w"])
    decided = np.array([oracle.token_decided(r["logits"][t], eps[t], cfg.oracle_cfg()) for t in range(n)])
    compare_rows(bf16_to_f64(out)[decided], r["y"][decided])
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"device status word {word:#x}"


def test_fused_route_on_concurrent_streams_equals_serial():
    """Micro-batches routed on four streams at once (each with its own
    workspace) give what they give one after the other."""
    cfg = DS_ROUTE
    w, h, wf = case(cfg)
    sizes = [700, 4096, 33, 5000]
    xs = [inputs.make_tokens(cfg, n, i, DEV) for i, n in enumerate(sizes)]
    serial = []
    for x in xs:
        o = outputs(x.shape[0], cfg)
        api.asap_moe_route(h, x, *o, api.workspace(h, x.shape[0]))
        serial.append(o)
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in xs]
    wss = [api.workspace(h, x.shape[0]) for x in xs]
    conc = [outputs(x.shape[0], cfg) for x in xs]
    torch.cuda.synchronize()
    for rep in range(3):
        for x, s, ws, o in zip(xs, streams, wss, conc):
            with torch.cuda.stream(s):
                api.asap_moe_route(h, x, *o, ws, stream=s)
    torch.cuda.synchronize()
    for a, b in zip(serial, conc):
        for u, v in zip(a, b):
            assert torch.equal(u, v)
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"device status word {word:#x}"
