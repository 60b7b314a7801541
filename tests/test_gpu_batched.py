"""asap_moe_layer_batched: several ready micro-batches served in one pass
give, for every micro-batch, the same bits as asap_moe_layer on it alone."""
import pytest
import torch

from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import DSV3, STRESS, DSV3_FP8, MIXTRAL

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _check(cfg, lengths):
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, sum(lengths))
    xs = [inputs.make_tokens(cfg, n, i, DEV) for i, n in enumerate(lengths)]
    ref = []
    for x in xs:
        o = torch.empty_like(x)
        if x.shape[0]:
            api.asap_moe_layer(h, x, o, api.workspace(h, x.shape[0]))
        ref.append(o)
    outs = [torch.full_like(x, 3.0) for x in xs]
    api.asap_moe_layer_batched(h, xs, outs, api.workspace(h, sum(lengths)))
    torch.cuda.synchronize()
    for a, b in zip(ref, outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0
    h.close()


@pytest.mark.parametrize("cfg,lengths", [
    (inputs.small_variant(DSV3, name="b_ds", hidden=512, inter=256, shared_inter=256), [300, 0, 77, 1, 129]),
    (inputs.small_variant(STRESS, name="b_st", hidden=512, inter=256, shared_inter=256), [700, 33, 5]),
    (inputs.small_variant(MIXTRAL, name="b_mx", hidden=1024, inter=512), [1000, 333]),
    (inputs.small_variant(DSV3_FP8, name="b_f8", hidden=512, inter=256, shared_inter=256), [300, 77, 2]),
], ids=["dsv3_small", "stress_small", "mixtral_small", "fp8_small"])
def test_batched_equals_separate_calls(cfg, lengths):
    _check(cfg, lengths)


@pytest.mark.parametrize("cfg", [DSV3, STRESS, MIXTRAL, DSV3_FP8], ids=lambda c: c.name)
def test_batched_full_size(cfg):
    _check(cfg, cfg.microbatches)
