"""asap_moe_route_noalloc: routing for callers that cannot allocate device
memory (their HBM belongs to another allocator, or allocating on that path is
not allowed).  It must give exactly what asap_moe_route gives, call after
call, although its scratch lives in one static array that every call reuses.

This file is collected last so that a run stopping at its first failure has
already run every other test; it also passes on its own in a fresh process."""
import pytest
import torch

from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import DSV3

pytestmark = pytest.mark.gpu

DEV = "cuda"
# E = 256 puts the router on the tensor core; two micro-batches of different
# lengths.  At hidden 512 the router has one K slice; at 2048 it splits K into
# 4 slices over a thread-block cluster (700 and 4096 tokens).
CFG = inputs.small_variant(DSV3, name="dsv3_noalloc", hidden=512, inter=256, shared_inter=256,
                           microbatches=[700, 301])
CFG_WIDE = inputs.small_variant(DSV3, name="dsv3_noalloc_wide", hidden=2048, inter=128, shared_inter=128,
                                microbatches=[700, 4096])


@pytest.fixture(scope="module", params=[CFG, CFG_WIDE], ids=lambda c: c.name)
def handle(request):
    import __graft_entry__
    __graft_entry__.build()
    cfg = request.param
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, max(cfg.microbatches))
    h.test_cfg = cfg
    yield h
    h.close()


def _outputs(n):
    k, E = CFG.top_k, CFG.n_experts
    return (torch.full((n, k), -7, dtype=torch.int32, device=DEV),
            torch.full((n, k), -7.0, dtype=torch.float32, device=DEV),
            torch.full((E,), -7, dtype=torch.int32, device=DEV),
            torch.full((E + 1,), -7, dtype=torch.int32, device=DEV))


def test_noalloc_route_equals_route_on_consecutive_calls(handle):
    cfg = handle.test_cfg
    for i, n in enumerate(cfg.microbatches):       # two calls in a row
        x = inputs.make_tokens(cfg, n, i, DEV)
        ref = _outputs(n)
        api.asap_moe_route(handle, x, *ref, api.workspace(handle, n))
        got = _outputs(n)
        api.asap_moe_route_noalloc(handle, x, *got)
        torch.cuda.synchronize()
        for a, b in zip(ref, got):
            assert torch.equal(a, b)
    code, word = api.asap_moe_status(handle)
    assert code == 0 and word == 0


def test_noalloc_route_rejects_more_tokens_than_its_scratch(handle):
    from paper_2606_22541_gb300._native import AsapError
    big = inputs.small_variant(handle.test_cfg, name="dsv3_noalloc_big")
    w = inputs.make_weights(big, DEV)
    h = api.asap_moe_create(big, w, 5000)
    try:
        x = inputs.make_tokens(big, 4097, 0, DEV)
        with pytest.raises(AsapError, match="static routing scratch"):
            api.asap_moe_route_noalloc(h, x, *_outputs(4097))
    finally:
        h.close()
