"""The layer against the float64 oracle on seeded random shapes: expert
counts from 8 to 256, top-k 1..8, the three gating rules with random group
counts, hidden sizes that do and do not split the router's K, with and
without a shared expert, ragged token counts (some large enough for the
paired-m-tile GEMMs).  Each case also runs with single and with paired
m-tiles forced, which must give the same bits.  Each case is drawn from its
own seed, so a failure names a reproducible shape."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import LayerConfig

from _helpers import bf16_to_f64, weights_f64, compare_rows, routing_check

pytestmark = pytest.mark.gpu

DEV = "cuda"
N_CASES = 48


def random_config(i):
    rng = np.random.default_rng(5000 + i)
    E = int(rng.choice([8, 16, 32, 64, 128, 256]))
    gating = str(rng.choice(["softmax", "softmax_renorm", "sigmoid_grouped"]))
    top_k = int(rng.integers(1, min(8, E) + 1))
    H = int(rng.choice([256, 512, 768, 2048]))
    I = int(rng.choice([128, 256, 384]))
    shared = int(rng.integers(0, 2))
    Is = int(rng.choice([128, 256])) if shared else 0
    n_groups, topk_groups = 1, 1
    if gating == "sigmoid_grouped":
        # a group count that divides E with >= 2 experts per group, and
        # enough kept groups to hold top_k experts
        n_groups = int(rng.choice([g for g in (1, 2, 4, 8, 16, 32) if E % g == 0 and E // g >= 2]))
        gsz = E // n_groups
        topk_groups = int(rng.integers(-(-top_k // gsz), n_groups + 1))
    n = int(rng.integers(1, 1200))
    return LayerConfig(f"rand{i}", hidden=H, n_experts=E, top_k=top_k, inter=I, n_shared=shared,
                       shared_inter=Is, gating=gating, n_groups=n_groups, topk_groups=topk_groups,
                       route_scale=float(rng.choice([1.0, 2.5])), microbatches=[n], seed=7000 + i)


# fixed shapes the draws may miss: E = 256 with grouped gating through the
# one-launch route (8 groups, K split over a cluster) and through the gate
# kernels (16 groups), E = 256 softmax-renorm with a shared expert, and a
# Mixtral-like shape with segments of about 275 rows (a paired and a half tile
# each with paired m-tiles)
FIXED = [
    LayerConfig("fixed_g8", hidden=2048, n_experts=256, top_k=8, inter=128, n_shared=1, shared_inter=128,
                gating="sigmoid_grouped", n_groups=8, topk_groups=4, route_scale=2.5, microbatches=[777], seed=7101),
    LayerConfig("fixed_g16", hidden=768, n_experts=256, top_k=6, inter=256, n_shared=0, shared_inter=0,
                gating="sigmoid_grouped", n_groups=16, topk_groups=3, route_scale=1.0, microbatches=[333], seed=7102),
    LayerConfig("fixed_renorm256", hidden=512, n_experts=256, top_k=8, inter=128, n_shared=1, shared_inter=256,
                gating="softmax_renorm", microbatches=[401], seed=7103),
    LayerConfig("fixed_pair8", hidden=768, n_experts=8, top_k=2, inter=384, n_shared=0, shared_inter=0,
                gating="softmax", microbatches=[1100], seed=7104),
]
CASES = [random_config(i) for i in range(N_CASES)] + FIXED


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("cfg", CASES, ids=lambda c: c.name)
def test_random_shape_layer_matches_oracle(cfg):
    n = cfg.microbatches[0]
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, n)
    try:
        x = inputs.make_tokens(cfg, n, 0, DEV)
        out = torch.empty_like(x)
        api.asap_moe_layer(h, x, out, api.workspace(h, n))
        forced = {}
        for mode in (api.TILING_SINGLE, api.TILING_PAIRED):
            api.asap_moe_set_tiling(h, mode)
            forced[mode] = torch.empty_like(x)
            api.asap_moe_layer(h, x, forced[mode], api.workspace(h, n))
        api.asap_moe_set_tiling(h, api.TILING_AUTO)
        k, E = cfg.top_k, cfg.n_experts
        idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
        wt = torch.empty((n, k), dtype=torch.float32, device=DEV)
        counts = torch.empty(E, dtype=torch.int32, device=DEV)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
        api.asap_moe_route(h, x, idx, wt, counts, offsets, api.workspace(h, n))
        torch.cuda.synchronize()
        for mode, o in forced.items():
            assert torch.equal(o.view(torch.int16), out.view(torch.int16)), f"tiling mode {mode}"
        wf = weights_f64(w)
        xf = bf16_to_f64(x)
        ocfg = cfg.oracle_cfg()
        shared = (wf["sh_gate"], wf["sh_up"], wf["sh_down"]) if cfg.n_shared else None
        r = oracle.moe_layer(xf, wf["router_w"], wf["w_gate"], wf["w_up"], wf["w_down"], ocfg, shared=shared)
        eps = oracle.logit_error_bound(xf, wf["router_w"])
        ig = idx.cpu().numpy().astype(np.int64)
        decided = routing_check(r["logits"], eps, ocfg, ig, wt.cpu().numpy().astype(np.float64), r["w"], r["idx"])
        cg = counts.cpu().numpy()
        assert np.array_equal(cg, np.bincount(ig.reshape(-1), minlength=E))
        assert np.array_equal(offsets.cpu().numpy(), np.concatenate([[0], np.cumsum(cg)]))
        if decided.any():
            compare_rows(bf16_to_f64(out)[decided], r["y"][decided])
        code, word = api.asap_moe_status(h)
        assert code == 0 and word == 0, f"{cfg}: device status word {word:#x}"
    finally:
        h.close()
