"""asap_moe_route_noalloc: routing for callers that cannot allocate device
memory (their HBM belongs to another allocator, or allocating on that path is
not allowed).  It must give exactly what asap_moe_route gives, call after
call, although its scratch lives in one static array that every call reuses.

This file is collected last so that a run stopping at its first failure has
already run every other test; it also passes on its own in a fresh process."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import DSV3, MIXTRAL

from _helpers import bf16_to_f64, routing_check

pytestmark = pytest.mark.gpu

DEV = "cuda"
# E = 256 grouped sigmoid gating runs the one-launch route: two micro-batches
# of different lengths.  At hidden 512 the router has one K slice; at 2048 it
# splits K into 4 slices over a thread-block cluster (700 and 4096 tokens).
CFG = inputs.small_variant(DSV3, name="dsv3_noalloc", hidden=512, inter=256, shared_inter=256,
                           microbatches=[700, 301])
CFG_WIDE = inputs.small_variant(DSV3, name="dsv3_noalloc_wide", hidden=2048, inter=128, shared_inter=128,
                                microbatches=[700, 4096])
# The router, gate and scan kernels one after the other: E = 256 with
# softmax-renorm gating (tensor-core router, K of hidden 2048 split 4 ways at
# every length here) and an 8-expert softmax-renorm layer (mma.sync router,
# one K slice).
CFG_RENORM = inputs.small_variant(DSV3, name="e256_renorm_noalloc", hidden=2048, inter=128, shared_inter=128,
                                  gating="softmax_renorm", n_groups=1, topk_groups=1, route_scale=1.0,
                                  microbatches=[4096, 2048, 333])
CFG_E8 = inputs.small_variant(MIXTRAL, name="e8_renorm_noalloc", hidden=1024, inter=256,
                              microbatches=[4096, 517])


@pytest.fixture(scope="module", params=[CFG, CFG_WIDE, CFG_RENORM, CFG_E8], ids=lambda c: c.name)
def handle(request):
    import __graft_entry__
    __graft_entry__.build()
    cfg = request.param
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, max(cfg.microbatches))
    h.test_cfg = cfg
    h.router_w = w["router_w"]
    yield h
    h.close()


def _outputs(cfg, n):
    k, E = cfg.top_k, cfg.n_experts
    return (torch.full((n, k), -7, dtype=torch.int32, device=DEV),
            torch.full((n, k), -7.0, dtype=torch.float32, device=DEV),
            torch.full((E,), -7, dtype=torch.int32, device=DEV),
            torch.full((E + 1,), -7, dtype=torch.int32, device=DEV))


def test_noalloc_route_equals_route_on_consecutive_calls(handle):
    cfg = handle.test_cfg
    for i, n in enumerate(cfg.microbatches):       # calls in a row
        x = inputs.make_tokens(cfg, n, i, DEV)
        ref = _outputs(cfg, n)
        api.asap_moe_route(handle, x, *ref, api.workspace(handle, n))
        got = _outputs(cfg, n)
        api.asap_moe_route_noalloc(handle, x, *got)
        torch.cuda.synchronize()
        for a, b in zip(ref, got):
            assert torch.equal(a, b)
        if i == 0:
            # and the routing itself against the oracle (certified comparison)
            xf = bf16_to_f64(x)
            wr = bf16_to_f64(handle.router_w)
            L = oracle.router_logits(xf, wr)
            eps = oracle.logit_error_bound(xf, wr)
            ocfg = cfg.oracle_cfg()
            idx_ref, w_ref = oracle.route(L, ocfg)
            ig = got[0].cpu().numpy().astype(np.int64)
            routing_check(L, eps, ocfg, ig, got[1].cpu().numpy().astype(np.float64), w_ref, idx_ref)
            assert np.array_equal(got[2].cpu().numpy(), np.bincount(ig.reshape(-1), minlength=cfg.n_experts))
    code, word = api.asap_moe_status(handle)
    assert code == 0 and word == 0


def test_noalloc_route_rejects_more_tokens_than_its_scratch(handle):
    from paper_2606_22541_gb300._native import AsapError
    big = inputs.small_variant(handle.test_cfg, name=handle.test_cfg.name + "_big")
    w = inputs.make_weights(big, DEV)
    h = api.asap_moe_create(big, w, 5000)
    try:
        x = inputs.make_tokens(big, 4097, 0, DEV)
        with pytest.raises(AsapError, match="static routing scratch"):
            api.asap_moe_route_noalloc(h, x, *_outputs(big, 4097))
    finally:
        h.close()
