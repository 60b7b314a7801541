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
# E = 256 puts the router on the tensor-core GEMM, the path whose logits go
# into the static scratch; two micro-batches of different lengths
CFG = inputs.small_variant(DSV3, name="dsv3_noalloc", hidden=512, inter=256, shared_inter=256,
                           microbatches=[700, 301])


@pytest.fixture(scope="module")
def handle():
    import __graft_entry__
    __graft_entry__.build()
    w = inputs.make_weights(CFG, DEV)
    h = api.asap_moe_create(CFG, w, max(CFG.microbatches))
    yield h
    h.close()


def _outputs(n):
    k, E = CFG.top_k, CFG.n_experts
    return (torch.full((n, k), -7, dtype=torch.int32, device=DEV),
            torch.full((n, k), -7.0, dtype=torch.float32, device=DEV),
            torch.full((E,), -7, dtype=torch.int32, device=DEV),
            torch.full((E + 1,), -7, dtype=torch.int32, device=DEV))


def test_noalloc_route_equals_route_on_consecutive_calls(handle):
    for i, n in enumerate(CFG.microbatches):       # two calls in a row
        x = inputs.make_tokens(CFG, n, i, DEV)
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
    big = inputs.small_variant(CFG, name="dsv3_noalloc_big")
    w = inputs.make_weights(big, DEV)
    h = api.asap_moe_create(big, w, 5000)
    try:
        x = inputs.make_tokens(big, 4097, 0, DEV)
        with pytest.raises(AsapError, match="static routing scratch"):
            api.asap_moe_route_noalloc(h, x, *_outputs(4097))
    finally:
        h.close()
