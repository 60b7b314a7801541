"""The seeded input generators follow their documented recipe (CPU only):
reproducible from the seed, one routed expert regenerable on its own, the
documented standard deviations, the FP8 block quantisation (s = amax / 448 per
128 x 128 block, the block's largest value at +-448) and the Zipf logit bias
(zero mean, log-probabilities of a power law under a seeded permutation)."""
import numpy as np
import torch

from paper_2606_22541_gb300 import inputs
from paper_2606_22541_gb300.configs import DSV3_FP8, MIXTRAL, STRESS, TINY

CPU = "cpu"


def small(cfg, **kw):
    base = dict(hidden=256, n_experts=8, inter=128, shared_inter=128 if cfg.n_shared else 0, microbatches=[64])
    base.update(kw)
    return inputs.small_variant(cfg, **base)


def test_tokens_are_reproducible_and_distinct_per_microbatch():
    cfg = small(MIXTRAL)
    a = inputs.make_tokens(cfg, 64, 0, CPU)
    assert torch.equal(a, inputs.make_tokens(cfg, 64, 0, CPU))
    assert not torch.equal(a, inputs.make_tokens(cfg, 64, 1, CPU))
    assert a.dtype == torch.bfloat16 and tuple(a.shape) == (64, 256)


def test_one_expert_can_be_regenerated_alone():
    stack = inputs.expert_stack_bf16(4, 16, 32, 0.5, 77, CPU)
    for e in range(4):
        assert torch.equal(stack[e], inputs.randn_bf16((16, 32), 0.5, 77 * 1000 + e, CPU))


def test_documented_standard_deviations():
    H, I = 1024, 512
    cfg = small(MIXTRAL, hidden=H, inter=I, n_experts=2)
    w = inputs.make_weights(cfg, CPU)
    x = inputs.make_tokens(cfg, 512, 0, CPU).float()
    assert abs(x.std().item() - 1.0) < 0.02 and abs(x.mean().item()) < 0.02
    for name, std in (("w_gate", 1 / np.sqrt(H)), ("w_up", 1 / np.sqrt(H)), ("w_down", 1 / np.sqrt(I)),
                      ("router_w", 1 / np.sqrt(H))):
        got = w[name].float().std().item()
        assert abs(got / std - 1.0) < 0.03, (name, got, std)
    # the tiny layer's router is N(0, 0.02)
    wt = inputs.make_weights(inputs.small_variant(TINY, microbatches=[8]), CPU)
    assert abs(wt["router_w"].float().std().item() / 0.02 - 1.0) < 0.05


def test_fp8_block_quantisation_recipe():
    g = torch.Generator().manual_seed(5)
    w = torch.randn(256, 384, generator=g) * 0.03
    w[0:128, 128:256] = 0.0                                   # an all-zero block gets scale 1
    q, s = inputs.quantize_block128_e4m3(w)
    assert q.dtype == torch.float8_e4m3fn and tuple(s.shape) == (2, 3)
    blocks = w.reshape(2, 128, 3, 128)
    amax = blocks.abs().amax(dim=(1, 3))
    expect = torch.where(amax > 0, amax / 448.0, torch.ones_like(amax))
    assert torch.equal(s, expect)
    deq = (q.float().reshape(2, 128, 3, 128) * s[:, None, :, None])
    qb = q.float().reshape(2, 128, 3, 128)
    for i in range(2):
        for j in range(3):
            if amax[i, j] > 0:
                assert qb[i, :, j, :].abs().max().item() == 448.0   # the block maximum maps to 448
                rel = (deq[i, :, j, :] - blocks[i, :, j, :]).abs() / amax[i, j]
                # e4m3 keeps 3 mantissa bits: each value's rounding error is at most 2^-4 of its
                # magnitude (or of the block amax in the subnormal range), hence of the block amax
                assert rel.max().item() <= 2.0 ** -4
            else:
                assert torch.all(qb[i, :, j, :] == 0)


def test_fp8_weights_are_blocks_of_the_bf16_recipe_shape():
    cfg = small(DSV3_FP8, hidden=256, inter=128, n_experts=2, shared_inter=128)
    w = inputs.make_weights(cfg, CPU)
    assert w["w_gate"].dtype == torch.float8_e4m3fn and tuple(w["s_gate"].shape) == (2, 1, 2)
    assert tuple(w["s_down"].shape) == (2, 2, 1) and tuple(w["sh_s_down"].shape) == (2, 1)


def test_zipf_bias_is_a_permuted_power_law_with_zero_mean():
    E, s = 64, 1.1
    b = inputs.zipf_logit_bias(E, s, 1234)
    assert abs(b.mean()) < 1e-12
    assert np.allclose(b, inputs.zipf_logit_bias(E, s, 1234))
    r = np.arange(1, E + 1)
    lp = -s * np.log(r)
    lp -= np.log(np.exp(lp).sum())
    assert np.allclose(np.sort(b)[::-1], np.sort(lp - lp.mean())[::-1])   # a permutation of ln p_r
    assert not np.allclose(b, lp - lp.mean())                             # and not the identity order


def test_zipf_workload_plants_the_bias_in_channel_0():
    cfg = small(STRESS, n_experts=16)
    x = inputs.make_tokens(cfg, 32, 0, CPU)
    assert torch.all(x[:, 0] == 1.0)
    wr = inputs.router_weights_bf16(cfg, CPU)
    b = torch.tensor(cfg.zipf_beta * inputs.zipf_logit_bias(16, cfg.zipf_s, cfg.seed)).to(torch.bfloat16)
    assert torch.equal(wr[:, 0], b)
    assert 0.0 < cfg.zipf_beta < 1.0


def test_layer_seeds():
    cfg = small(MIXTRAL)
    assert inputs.layer_config(cfg, 0) is cfg
    assert inputs.layer_config(cfg, 3).seed == cfg.seed + 3 * 7919
    w0, w1 = inputs.make_layer_weights(cfg, 2, CPU)
    assert not torch.equal(w0["w_gate"], w1["w_gate"])
    assert torch.equal(w0["w_gate"], inputs.make_weights(cfg, CPU)["w_gate"])
