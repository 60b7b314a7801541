"""Parity of the CUDA path (through the C ABI) with the float64 oracle, on
seeded inputs: each step and the whole layer, shapes spanning several tiles
with ragged tails, edge cases, and the multi-stream submission model."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import TINY, MIXTRAL, DSV3, DSV3_FP8, STRESS

from _helpers import bf16_to_f64, weights_f64, compare_rows, routing_check

pytestmark = pytest.mark.gpu

DEV = "cuda"

# Reduced shapes of the Mixtral and DeepSeek-V3 layers: several 128-row tiles,
# ragged segments, empty experts, the tensor-core router (E = 256) and the
# shared expert, small enough for the oracle to finish in seconds.
MX_SMALL = inputs.small_variant(MIXTRAL, name="mixtral_small", hidden=1024, inter=512, microbatches=[1000, 333])
DS_SMALL = inputs.small_variant(DSV3, name="dsv3_small", hidden=512, inter=256, shared_inter=256,
                                microbatches=[300, 77])
ST_SMALL = inputs.small_variant(STRESS, name="stress_small", hidden=512, inter=256, shared_inter=256,
                                microbatches=[700, 129, 1])
SMALL = [TINY, MX_SMALL, DS_SMALL, ST_SMALL]
# Shapes outside the 32-lane-team gate (expert counts and groups that are not
# powers of two): routed by the warp-per-token gate kernel.
ODD_SOFTMAX = inputs.small_variant(TINY, name="odd_softmax", n_experts=12, top_k=3, gating="softmax_renorm",
                                   microbatches=[200, 33])
ODD_GROUPED = inputs.small_variant(DSV3, name="odd_grouped", hidden=256, n_experts=24, top_k=4, inter=128,
                                   shared_inter=128, n_groups=3, topk_groups=2, microbatches=[200, 33])
ODD = [ODD_SOFTMAX, ODD_GROUPED]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


class Case:
    """Weights on the GPU, their float64 copies and a handle."""
    _cache = {}

    @classmethod
    def get(cls, cfg):
        if cfg.name not in cls._cache:
            cls._cache[cfg.name] = cls(cfg)
        return cls._cache[cfg.name]

    def __init__(self, cfg):
        self.cfg = cfg
        self.w = inputs.make_weights(cfg, DEV)
        self.h = api.asap_moe_create(cfg, self.w, max(cfg.microbatches))
        self.wf = weights_f64(self.w)
        self.ocfg = cfg.oracle_cfg()
        self.shared = (self.wf["sh_gate"], self.wf["sh_up"], self.wf["sh_down"]) if cfg.n_shared else None

    def tokens(self, i, n=None):
        n = self.cfg.microbatches[i] if n is None else n
        return inputs.make_tokens(self.cfg, n, i, DEV)

    def ws(self, n):
        return api.workspace(self.h, n)


def run_route(c, x):
    n = x.shape[0]
    k, E = c.cfg.top_k, c.cfg.n_experts
    idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
    w = torch.empty((n, k), dtype=torch.float32, device=DEV)
    counts = torch.empty(E, dtype=torch.int32, device=DEV)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
    api.asap_moe_route(c.h, x, idx, w, counts, offsets, c.ws(n))
    torch.cuda.synchronize()
    return idx, w, counts, offsets


def assert_clean(c):
    code, word = api.asap_moe_status(c.h)
    assert code == 0 and word == 0, f"device status word {word:#x}"


# ---------------------------------------------------------------- routing

@pytest.mark.parametrize("cfg", SMALL, ids=lambda c: c.name)
def test_router_logits_within_bound(cfg):
    c = Case.get(cfg)
    x = c.tokens(0)
    logits = torch.empty((x.shape[0], cfg.n_experts), dtype=torch.float32, device=DEV)
    api.asap_moe_router_logits(c.h, x, logits, c.ws(x.shape[0]))
    torch.cuda.synchronize()
    xf = bf16_to_f64(x)
    L = oracle.router_logits(xf, c.wf["router_w"])
    eps = oracle.logit_error_bound(xf, c.wf["router_w"])
    err = np.abs(logits.cpu().numpy().astype(np.float64) - L)
    assert (err <= eps).all(), f"max err/bound {float((err / eps).max()):.3f}"
    assert_clean(c)


# router widths: E = 8, 16, 32, 64 run the mma.sync router (16 tokens per CTA,
# K split over 8 warps), E = 24 and 128 the CUDA-core one; ragged token counts
# cover the CTA's 16-token tail
ROUTER_E = [inputs.small_variant(MIXTRAL, name=f"router_e{E}", hidden=768, n_experts=E, top_k=2, inter=128,
                                 microbatches=[1000]) for E in (8, 16, 24, 32, 64, 128)]


@pytest.mark.parametrize("cfg", ROUTER_E, ids=lambda c: c.name)
def test_router_logits_widths_within_bound(cfg):
    c = Case.get(cfg)
    for n in (1, 15, 17, 100, 1000):
        x = c.tokens(0, n)
        logits = torch.full((n, cfg.n_experts), float("nan"), dtype=torch.float32, device=DEV)
        api.asap_moe_router_logits(c.h, x, logits, c.ws(n))
        torch.cuda.synchronize()
        xf = bf16_to_f64(x)
        L = oracle.router_logits(xf, c.wf["router_w"])
        eps = oracle.logit_error_bound(xf, c.wf["router_w"])
        err = np.abs(logits.cpu().numpy().astype(np.float64) - L)
        assert (err <= eps).all(), f"n={n}: max err/bound {float(np.nanmax(err / eps)):.3f}"
    assert_clean(c)


def test_set_tiling_rejects_unknown_mode():
    from paper_2606_22541_gb300._native import AsapError
    c = Case.get(TINY)
    with pytest.raises(AsapError):
        api.asap_moe_set_tiling(c.h, 3)
    api.asap_moe_set_tiling(c.h, api.TILING_AUTO)


@pytest.mark.parametrize("cfg", SMALL + ODD, ids=lambda c: c.name)
def test_route_matches_oracle(cfg):
    c = Case.get(cfg)
    for i in range(len(cfg.microbatches)):
        x = c.tokens(i)
        idx, w, counts, offsets = run_route(c, x)
        xf = bf16_to_f64(x)
        L = oracle.router_logits(xf, c.wf["router_w"])
        eps = oracle.logit_error_bound(xf, c.wf["router_w"])
        idx_ref, w_ref = oracle.route(L, c.ocfg)
        ig = idx.cpu().numpy().astype(np.int64)
        decided = routing_check(L, eps, c.ocfg, ig, w.cpu().numpy().astype(np.float64), w_ref, idx_ref)
        # counts / offsets: the histogram of the returned idx and its scan
        cg = counts.cpu().numpy()
        og = offsets.cpu().numpy()
        assert np.array_equal(cg, np.bincount(ig.reshape(-1), minlength=cfg.n_experts))
        assert og[0] == 0 and np.array_equal(np.diff(og), cg) and og[-1] == ig.size
        if decided.all():
            assert np.array_equal(cg, oracle.expert_counts(idx_ref, cfg.n_experts))
            assert np.array_equal(og, oracle.expert_offsets(oracle.expert_counts(idx_ref, cfg.n_experts)))
    assert_clean(c)


def test_route_logits_exact_ties():
    c = Case.get(TINY)
    n, E = 130, TINY.n_experts
    rng = np.random.default_rng(7)
    L = np.round(rng.normal(0, 1, (n, E)) * 2) / 2          # many exact ties
    L[5] = 0.0                                              # every expert tied
    L[6] = [1, 1, 1, 0, 0, 0, 0, 0]
    lg = torch.tensor(L, dtype=torch.float32, device=DEV)
    idx = torch.empty((n, 2), dtype=torch.int32, device=DEV)
    w = torch.empty((n, 2), dtype=torch.float32, device=DEV)
    counts = torch.empty(E, dtype=torch.int32, device=DEV)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
    api.asap_moe_route_logits(c.h, lg, idx, w, counts, offsets, c.ws(n))
    torch.cuda.synchronize()
    idx_ref, w_ref = oracle.route(L, c.ocfg)
    assert np.array_equal(idx.cpu().numpy(), idx_ref)
    assert np.allclose(w.cpu().numpy(), w_ref, rtol=1e-6, atol=0)
    assert list(idx_ref[5]) == [0, 1] and list(idx_ref[6]) == [0, 1]
    assert np.array_equal(counts.cpu().numpy(), oracle.expert_counts(idx_ref, E))
    assert np.array_equal(offsets.cpu().numpy(), oracle.expert_offsets(oracle.expert_counts(idx_ref, E)))


def test_route_logits_grouped_exact_ties_and_all_to_one_group():
    c = Case.get(DS_SMALL)
    n, E = 70, 256
    rng = np.random.default_rng(8)
    L = np.round(rng.normal(0, 1, (n, E)) * 4) / 4
    L[0] = 0.0                       # everything tied: groups 0-3, experts 0..7
    L[1] = -5.0
    L[1, 64:72] = 3.0                # one group holds all 8 picks
    L[2] = -5.0
    L[2, 200] = 4.0                  # a single hot expert
    lg = torch.tensor(L, dtype=torch.float32, device=DEV)
    idx = torch.empty((n, 8), dtype=torch.int32, device=DEV)
    w = torch.empty((n, 8), dtype=torch.float32, device=DEV)
    counts = torch.empty(E, dtype=torch.int32, device=DEV)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
    api.asap_moe_route_logits(c.h, lg, idx, w, counts, offsets, c.ws(n))
    torch.cuda.synchronize()
    idx_ref, w_ref = oracle.route(L, c.ocfg)
    # float32 sigmoid may merge logits the float64 one separates; the
    # quarter-step logits here keep every tie exact or well separated
    eps = np.zeros_like(L)
    ig = idx.cpu().numpy().astype(np.int64)
    routing_check(L, eps, c.ocfg, ig, w.cpu().numpy().astype(np.float64), w_ref, idx_ref)
    assert list(idx_ref[0]) == list(range(8))
    assert list(idx_ref[1]) == list(range(64, 72))
    # constructed exact ties resolve bit-exactly by the lower-index rule
    for t in range(3):
        assert list(ig[t]) == list(idx_ref[t])


# ---------------------------------------------------------------- dispatch / combine

def test_gate_kernels_agree():
    """The 32-lane-team gate and the warp-per-token gate (taken for logits
    that are not 16-byte aligned) route the same logits to the same experts
    with the same weights (grouped sigmoid: the same arithmetic in the same
    order)."""
    c = Case.get(DS_SMALL)
    n, k, E = 300, DS_SMALL.top_k, DS_SMALL.n_experts
    x = c.tokens(0, n)
    logits = torch.empty((n, E), dtype=torch.float32, device=DEV)
    api.asap_moe_router_logits(c.h, x, logits, c.ws(n))
    raw = torch.empty(n * E + 1, dtype=torch.float32, device=DEV)
    shifted = raw[1:].view(n, E)                              # 4-byte offset: warp-per-token gate
    shifted.copy_(logits)
    outs = []
    for lg in (logits, shifted):
        idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
        w = torch.empty((n, k), dtype=torch.float32, device=DEV)
        counts = torch.empty(E, dtype=torch.int32, device=DEV)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
        api.asap_moe_route_logits(c.h, lg, idx, w, counts, offsets, c.ws(n))
        outs.append((idx, w, counts, offsets))
    torch.cuda.synchronize()
    for a, b in zip(*outs):
        assert torch.equal(a, b)
    assert_clean(c)


@pytest.mark.parametrize("cfg", [TINY, DS_SMALL], ids=lambda c: c.name)
def test_dispatch_exact(cfg):
    c = Case.get(cfg)
    n, k, E, H = 333, cfg.top_k, cfg.n_experts, cfg.hidden
    if n > max(cfg.microbatches):
        n = max(cfg.microbatches)
    rng = np.random.default_rng(9)
    idx_np = np.array([rng.permutation(E)[:k] for _ in range(n)], np.int64).reshape(n, k)
    idx_np[: n // 3, 0] = 1                     # make expert 1 hot
    idx_np[: n // 3, 1:] = np.array([rng.permutation(np.arange(2, E))[:k - 1] for _ in range(n // 3)])
    x = c.tokens(0, n)
    idx = torch.tensor(idx_np, dtype=torch.int32, device=DEV)
    x_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
    perm_src = torch.empty(n * k, dtype=torch.int32, device=DEV)
    perm_dst = torch.empty((n, k), dtype=torch.int32, device=DEV)
    api.asap_moe_dispatch(c.h, x, idx, x_perm, perm_src, perm_dst, c.ws(n))
    torch.cuda.synchronize()
    src_ref, dst_ref = oracle.permutation(idx_np, E)
    assert np.array_equal(perm_src.cpu().numpy(), src_ref)
    assert np.array_equal(perm_dst.cpu().numpy(), dst_ref)
    assert np.array_equal(bf16_to_f64(x_perm), oracle.dispatch(bf16_to_f64(x), src_ref))
    assert_clean(c)


@pytest.mark.parametrize("cfg", [TINY, DS_SMALL], ids=lambda c: c.name)
def test_identity_experts_return_k_x(cfg):
    """dispatch then combine with y_perm = x_perm and unit weights gives k*x
    exactly (k a power of two, so k*x is a bf16 value)."""
    c = Case.get(cfg)
    n, k, E, H = max(cfg.microbatches), cfg.top_k, cfg.n_experts, cfg.hidden
    x = c.tokens(1 if len(cfg.microbatches) > 1 else 0, n)
    idx, w, counts, offsets = run_route(c, x)
    x_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
    perm_src = torch.empty(n * k, dtype=torch.int32, device=DEV)
    perm_dst = torch.empty((n, k), dtype=torch.int32, device=DEV)
    api.asap_moe_dispatch(c.h, x, idx, x_perm, perm_src, perm_dst, c.ws(n))
    out = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
    ones = torch.ones((n, k), dtype=torch.float32, device=DEV)
    api.asap_moe_combine(c.h, x_perm, None, ones, perm_dst, out)
    torch.cuda.synchronize()
    assert np.array_equal(bf16_to_f64(out), k * bf16_to_f64(x))
    assert_clean(c)


@pytest.mark.parametrize("cfg", [TINY, DS_SMALL], ids=lambda c: c.name)
def test_combine_matches_oracle(cfg):
    c = Case.get(cfg)
    n, k, H = 150, cfg.top_k, cfg.hidden
    n = min(n, max(cfg.microbatches))
    rng = np.random.default_rng(10)
    y_perm = inputs.randn_bf16((n * k, H), 1.0, 77, DEV)
    y_sh = inputs.randn_bf16((n, H), 1.0, 78, DEV)
    perm = rng.permutation(n * k).reshape(n, k)
    w_np = rng.uniform(0.01, 1.0, (n, k)).astype(np.float32)
    out = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
    api.asap_moe_combine(c.h, y_perm, y_sh, torch.tensor(w_np, device=DEV),
                         torch.tensor(perm, dtype=torch.int32, device=DEV), out)
    torch.cuda.synchronize()
    ref = oracle.combine(bf16_to_f64(y_perm), w_np.astype(np.float64), perm, bf16_to_f64(y_sh))
    g = bf16_to_f64(out)
    # fp32 accumulation then one bf16 rounding: within one bf16 ulp of the
    # exact sum plus the fp32 accumulation error
    tol = np.abs(ref) * 2.0 ** -8 + 1e-5 * (np.abs(bf16_to_f64(y_perm)).max() * k + 1)
    assert (np.abs(g - ref) <= tol).all()
    assert_clean(c)


# ---------------------------------------------------------------- expert FFN

@pytest.mark.parametrize("cfg", SMALL, ids=lambda c: c.name)
def test_expert_ffn_matches_oracle(cfg):
    """Grouped GEMMs on oracle-made segments: empty experts, one hot expert,
    segments that are not multiples of 128 rows."""
    c = Case.get(cfg)
    n, k, E, H = max(cfg.microbatches), cfg.top_k, cfg.n_experts, cfg.hidden
    rng = np.random.default_rng(11)
    counts = rng.multinomial(n * k, np.r_[0.3, np.full(E - 1, 0.7 / (E - 1))])
    counts[E // 2 + 1] += counts[E // 2]      # one empty expert, total kept at n*k
    counts[E // 2] = 0
    offsets_np = oracle.expert_offsets(counts)
    x = c.tokens(0, n)
    x_perm = inputs.randn_bf16((n * k, H), 1.0, 90, DEV)
    y_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
    y_sh = torch.empty((n, H), dtype=torch.bfloat16, device=DEV) if cfg.n_shared else None
    offsets = torch.tensor(offsets_np, dtype=torch.int32, device=DEV)
    api.asap_moe_expert_ffn(c.h, x_perm, offsets, x, y_perm, y_sh, c.ws(n))
    torch.cuda.synchronize()
    ref = oracle.expert_ffn(bf16_to_f64(x_perm), offsets_np, c.wf["w_gate"], c.wf["w_up"], c.wf["w_down"])
    compare_rows(bf16_to_f64(y_perm), ref)
    if cfg.n_shared:
        compare_rows(bf16_to_f64(y_sh), oracle.swiglu(bf16_to_f64(x), *c.shared))
    assert_clean(c)


def test_expert_ffn_segment_tails_at_mma_boundaries():
    """Segments whose last 128-row half holds 1, 63, 64, 65, 127 or 128 rows,
    with one, two and three 128-row halves (a half of at most 64 rows takes
    M = 64 MMAs): single and paired m-tiles give the same bits, equal to the
    oracle's values."""
    cfg = DS_SMALL
    c = Case.get(cfg)
    n, k, E, H = max(cfg.microbatches), cfg.top_k, cfg.n_experts, cfg.hidden
    sizes = [1, 63, 64, 65, 127, 128, 129, 191, 192, 193, 257, 320, 321, 0, 2]
    counts = np.zeros(E, np.int64)
    counts[:len(sizes)] = sizes
    counts[E - 1] = n * k - counts.sum()          # the rest in the last expert
    assert counts[E - 1] >= 0
    offsets_np = oracle.expert_offsets(counts)
    x = c.tokens(0, n)
    x_perm = inputs.randn_bf16((n * k, H), 1.0, 92, DEV)
    offsets = torch.tensor(offsets_np, dtype=torch.int32, device=DEV)
    outs = []
    try:
        for mode in (api.TILING_SINGLE, api.TILING_PAIRED):
            api.asap_moe_set_tiling(c.h, mode)
            y_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
            y_sh = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
            api.asap_moe_expert_ffn(c.h, x_perm, offsets, x, y_perm, y_sh, c.ws(n))
            outs.append(y_perm)
        torch.cuda.synchronize()
    finally:
        api.asap_moe_set_tiling(c.h, api.TILING_AUTO)
    assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))
    lim = int(offsets_np[len(sizes)])               # the boundary segments
    ref = oracle.expert_ffn(bf16_to_f64(x_perm[:lim]), offsets_np[:len(sizes) + 1], c.wf["w_gate"], c.wf["w_up"],
                            c.wf["w_down"])
    compare_rows(bf16_to_f64(outs[1][:lim]), ref)
    assert_clean(c)


@pytest.mark.parametrize("hot", ["first", "middle", "last"])
def test_expert_ffn_all_rows_in_one_expert(hot):
    """Every routed row in one expert, every other segment empty, with single
    and with paired m-tiles: the same bits both ways and the oracle's values."""
    cfg = DS_SMALL
    c = Case.get(cfg)
    n, k, E, H = max(cfg.microbatches), cfg.top_k, cfg.n_experts, cfg.hidden
    e_hot = {"first": 0, "middle": E // 2, "last": E - 1}[hot]
    counts = np.zeros(E, np.int64)
    counts[e_hot] = n * k
    offsets_np = oracle.expert_offsets(counts)
    x = c.tokens(0, n)
    x_perm = inputs.randn_bf16((n * k, H), 1.0, 91, DEV)
    offsets = torch.tensor(offsets_np, dtype=torch.int32, device=DEV)
    outs = []
    try:
        for mode in (api.TILING_SINGLE, api.TILING_PAIRED):
            api.asap_moe_set_tiling(c.h, mode)
            y_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
            y_sh = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
            api.asap_moe_expert_ffn(c.h, x_perm, offsets, x, y_perm, y_sh, c.ws(n))
            outs.append((y_perm, y_sh))
    finally:
        api.asap_moe_set_tiling(c.h, api.TILING_AUTO)
    torch.cuda.synchronize()
    for a, b in zip(outs[0], outs[1]):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    ref = oracle.expert_ffn(bf16_to_f64(x_perm), offsets_np, c.wf["w_gate"], c.wf["w_up"], c.wf["w_down"])
    compare_rows(bf16_to_f64(outs[1][0]), ref)
    compare_rows(bf16_to_f64(outs[1][1]), oracle.swiglu(bf16_to_f64(x), *c.shared))
    assert_clean(c)


# ---------------------------------------------------------------- whole layer

def oracle_layer(c, x):
    return oracle.moe_layer(bf16_to_f64(x), c.wf["router_w"], c.wf["w_gate"], c.wf["w_up"], c.wf["w_down"],
                            c.ocfg, shared=c.shared)


@pytest.mark.parametrize("cfg", SMALL + ODD, ids=lambda c: c.name)
def test_layer_matches_oracle(cfg):
    c = Case.get(cfg)
    for i, n in enumerate(cfg.microbatches):
        x = c.tokens(i)
        out = torch.empty((n, cfg.hidden), dtype=torch.bfloat16, device=DEV)
        api.asap_moe_layer(c.h, x, out, c.ws(n))
        torch.cuda.synchronize()
        r = oracle_layer(c, x)
        idx, w, _, _ = run_route(c, x)
        xf = bf16_to_f64(x)
        eps = oracle.logit_error_bound(xf, c.wf["router_w"])
        decided = routing_check(r["logits"], eps, c.ocfg, idx.cpu().numpy().astype(np.int64),
                                w.cpu().numpy().astype(np.float64), r["w"], r["idx"])
        compare_rows(bf16_to_f64(out)[decided], r["y"][decided])
    assert_clean(c)


@pytest.mark.parametrize("cfg", [TINY, DS_SMALL, ST_SMALL] + ODD, ids=lambda c: c.name)
def test_route_equals_route_logits_of_router_logits(cfg):
    """asap_moe_route == asap_moe_route_logits(asap_moe_router_logits(x))."""
    c = Case.get(cfg)
    x = c.tokens(0)
    n, k, E = x.shape[0], cfg.top_k, cfg.n_experts
    a = run_route(c, x)
    logits = torch.empty((n, E), dtype=torch.float32, device=DEV)
    api.asap_moe_router_logits(c.h, x, logits, c.ws(n))
    b = (torch.empty((n, k), dtype=torch.int32, device=DEV), torch.empty((n, k), dtype=torch.float32, device=DEV),
         torch.empty(E, dtype=torch.int32, device=DEV), torch.empty(E + 1, dtype=torch.int32, device=DEV))
    api.asap_moe_route_logits(c.h, logits, *b, c.ws(n))
    torch.cuda.synchronize()
    for u, v in zip(a, b):
        assert torch.equal(u, v)


@pytest.mark.parametrize("cfg", [TINY, DS_SMALL], ids=lambda c: c.name)
def test_layer_equals_composed_calls_bit_for_bit(cfg):
    c = Case.get(cfg)
    n, k, E, H = cfg.microbatches[0], cfg.top_k, cfg.n_experts, cfg.hidden
    x = c.tokens(0)
    ws = c.ws(n)
    out = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
    api.asap_moe_layer(c.h, x, out, ws)
    idx, w, counts, offsets = run_route(c, x)
    x_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
    perm_src = torch.empty(n * k, dtype=torch.int32, device=DEV)
    perm_dst = torch.empty((n, k), dtype=torch.int32, device=DEV)
    api.asap_moe_dispatch(c.h, x, idx, x_perm, perm_src, perm_dst, ws)
    y_perm = torch.empty_like(x_perm)
    y_sh = torch.empty((n, H), dtype=torch.bfloat16, device=DEV) if cfg.n_shared else None
    api.asap_moe_expert_ffn(c.h, x_perm, offsets, x, y_perm, y_sh, ws)
    out2 = torch.empty_like(out)
    api.asap_moe_combine(c.h, y_perm, y_sh, w, perm_dst, out2)
    torch.cuda.synchronize()
    assert torch.equal(out.view(torch.int16), out2.view(torch.int16))
    assert_clean(c)


@pytest.mark.parametrize("cfg", [DS_SMALL, inputs.small_variant(DSV3_FP8, name="fp8_timing", hidden=512, inter=256,
                                                                 shared_inter=256, microbatches=[300])],
                         ids=lambda c: c.name)
def test_layer_timing_events_mark_its_steps_and_change_no_bit(cfg):
    """asap_moe_time_layer: the next layer call records the six events in
    order around its five steps, on its own stream, and computes the same
    bits; the request is used once (the call after it records nothing)."""
    h = api.asap_moe_create(cfg, inputs.make_weights(cfg, DEV), max(cfg.microbatches))
    n, H = cfg.microbatches[0], cfg.hidden
    x = inputs.make_tokens(cfg, n, 0, DEV)
    ws = api.workspace(h, n)
    s = torch.cuda.Stream()
    ref = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
    api.asap_moe_layer(h, x, ref, ws)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
    api.asap_moe_time_layer(ev)
    out = torch.empty_like(ref)
    with torch.cuda.stream(s):
        torch.cuda._sleep(1_000_000)              # the recorded events must wait for the layer's stream
        api.asap_moe_layer(h, x, out, ws, stream=s)
    torch.cuda.synchronize()
    d = [ev[j].elapsed_time(ev[j + 1]) for j in range(5)]
    assert all(v > 0 for v in d), d
    assert torch.equal(ref.view(torch.int16), out.view(torch.int16))
    late = torch.cuda.Event(enable_timing=True)
    late.record()
    out2 = torch.empty_like(ref)
    api.asap_moe_layer(h, x, out2, ws)               # no request pending: ev keep their times
    torch.cuda.synchronize()
    assert ev[5].elapsed_time(late) >= 0
    assert torch.equal(ref.view(torch.int16), out2.view(torch.int16))
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"device status word {word:#x}"
    h.close()


@pytest.mark.parametrize("cfg", SMALL + ODD, ids=lambda c: c.name)
def test_fused_combine_is_bit_identical(cfg):
    """ASAP_COMBINE_FUSED (the combine inside the down GEMM's epilogue, the
    last arrival of each token slice summing it) against the separate combine
    kernel: every micro-batch of the configuration, the same bits; tiny
    micro-batches too (1 and 2 tokens, single tiles with M = 64 tails)."""
    c = Case.get(cfg)
    H = cfg.hidden
    for n in list(cfg.microbatches) + [1, 2]:
        x = c.tokens(0, n)
        ws = c.ws(n)
        ref = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
        api.asap_moe_layer(c.h, x, ref, ws)
        api.asap_moe_set_combine(c.h, api.COMBINE_FUSED)
        try:
            out = torch.full_like(ref, 5.0)
            api.asap_moe_layer(c.h, x, out, ws)
            torch.cuda.synchronize()
        finally:
            api.asap_moe_set_combine(c.h, api.COMBINE_SEPARATE)
        assert torch.equal(ref.view(torch.int16), out.view(torch.int16)), (cfg.name, n)
    assert_clean(c)


@pytest.mark.parametrize("cfg", [DS_SMALL, ST_SMALL], ids=lambda c: c.name)
def test_streams_concurrent_equals_serial_and_token_independent(cfg):
    """Micro-batches submitted on their own streams with no host barrier give
    the same bits as one stream; a token's output does not depend on the
    micro-batch it arrived in."""
    c = Case.get(cfg)
    xs = [c.tokens(i) for i in range(len(cfg.microbatches))]
    wss = [c.ws(x.shape[0]) for x in xs]
    serial = []
    for x, ws in zip(xs, wss):
        o = torch.empty_like(x)
        api.asap_moe_layer(c.h, x, o, ws)
        serial.append(o)
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in xs]
    conc = [torch.empty_like(x) for x in xs]
    for x, o, ws, s in zip(xs, conc, wss, streams):
        s.wait_stream(torch.cuda.current_stream())
        api.asap_moe_layer(c.h, x, o, ws, stream=s)
    torch.cuda.synchronize()
    for a, b in zip(serial, conc):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    # regroup: the first 50 tokens of micro-batch 0 as a batch of their own
    x0 = xs[0][:50].contiguous()
    o0 = torch.empty_like(x0)
    api.asap_moe_layer(c.h, x0, o0, c.ws(50))
    torch.cuda.synchronize()
    assert torch.equal(o0.view(torch.int16), serial[0][:50].view(torch.int16))
    assert_clean(c)


# 8 experts, top-2, 1100 tokens: about 275 routed rows per expert, so with
# paired tiles every segment takes one full paired tile and one half tile.
MX_PAIR = inputs.small_variant(MIXTRAL, name="mixtral_pair", hidden=512, inter=512, microbatches=[1100])


@pytest.mark.parametrize("cfg", [MX_PAIR, DS_SMALL], ids=lambda c: c.name)
def test_paired_m_tiles_match_oracle_and_single_tiles(cfg):
    """The paired-tile GEMMs (with half tiles at the segment tails, and on
    the shared expert's rows) against the oracle, and bit for bit against the
    single-tile GEMMs and the automatic choice."""
    c = Case.get(cfg)
    x = c.tokens(0)
    n = x.shape[0]
    outs = {}
    try:
        for mode in (api.TILING_SINGLE, api.TILING_PAIRED, api.TILING_AUTO):
            api.asap_moe_set_tiling(c.h, mode)
            outs[mode] = torch.empty_like(x)
            api.asap_moe_layer(c.h, x, outs[mode], c.ws(n))
    finally:
        api.asap_moe_set_tiling(c.h, api.TILING_AUTO)
    torch.cuda.synchronize()
    out = outs[api.TILING_PAIRED]
    assert torch.equal(out.view(torch.int16), outs[api.TILING_SINGLE].view(torch.int16))
    assert torch.equal(out.view(torch.int16), outs[api.TILING_AUTO].view(torch.int16))
    r = oracle_layer(c, x)
    eps = oracle.logit_error_bound(bf16_to_f64(x), c.wf["router_w"])
    decided = np.array([oracle.token_decided(r["logits"][t], eps[t], c.ocfg) for t in range(n)])
    compare_rows(bf16_to_f64(out)[decided], r["y"][decided])
    assert_clean(c)


def test_edge_sizes():
    c = Case.get(DS_SMALL)
    H = DS_SMALL.hidden
    # n = 0 is a no-op
    x = c.tokens(0, 1)
    out = torch.full((1, H), 7.0, dtype=torch.bfloat16, device=DEV)
    api.asap_moe_layer(c.h, x[:0], out[:0], None)
    # n = 1 and the maximum n
    for n in (1, max(DS_SMALL.microbatches)):
        x = c.tokens(0, n)
        out = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
        api.asap_moe_layer(c.h, x, out, c.ws(n))
        torch.cuda.synchronize()
        r = oracle_layer(c, x)
        eps = oracle.logit_error_bound(bf16_to_f64(x), c.wf["router_w"])
        dec = np.array([oracle.token_decided(r["logits"][t], eps[t], c.ocfg) for t in range(n)])
        compare_rows(bf16_to_f64(out)[dec], r["y"][dec])
    # n > max_tokens and a short workspace are rejected without launching
    from paper_2606_22541_gb300._native import AsapError
    big = c.tokens(0, max(DS_SMALL.microbatches) + 1)
    with pytest.raises(AsapError):
        api.asap_moe_layer(c.h, big, torch.empty_like(big), c.ws(max(DS_SMALL.microbatches)))
    x = c.tokens(0, 10)
    with pytest.raises(AsapError):
        api.asap_moe_layer(c.h, x, torch.empty_like(x), c.ws(5))
    assert_clean(c)


def test_bad_indices_are_reported_not_trapped():
    c = Case.get(TINY)
    n, k, H = 20, 2, TINY.hidden
    x = c.tokens(0, n)
    idx = torch.zeros((n, k), dtype=torch.int32, device=DEV)
    idx[:, 1] = 1
    idx[3, 0] = 99                                           # out of range
    x_perm = torch.zeros((n * k, H), dtype=torch.bfloat16, device=DEV)
    perm_src = torch.empty(n * k, dtype=torch.int32, device=DEV)
    perm_dst = torch.empty((n, k), dtype=torch.int32, device=DEV)
    api.asap_moe_dispatch(c.h, x, idx, x_perm, perm_src, perm_dst, c.ws(n))
    code, word = api.asap_moe_status(c.h)
    assert code != 0 and (word & 1)
    assert perm_dst[3, 0].item() == -1
    code, word = api.asap_moe_status(c.h)                   # cleared by the read
    assert code == 0 and word == 0


@pytest.mark.parametrize("bad", ["decreasing", "past_rows", "negative"])
def test_bad_offsets_are_reported_and_computed_nothing(bad):
    """Offsets the grouped GEMMs cannot use (the kernels' own checks, no
    out-of-range access) leave the routed outputs untouched and set status
    bit 8; the shared expert (problem 1) is still computed."""
    c = Case.get(DS_SMALL)
    cfg = DS_SMALL
    n, k, E, H = 64, cfg.top_k, cfg.n_experts, cfg.hidden
    x = c.tokens(0, n)
    offs = torch.arange(E + 1, dtype=torch.int32, device=DEV) * 2   # offsets[E] = 512 = n * k
    if bad == "decreasing":
        offs[10] = 30
    elif bad == "past_rows":
        offs[E] = n * k + 128
    else:
        offs[0] = -128
    x_perm = c.tokens(1, n * k)
    y = torch.full((n * k, H), 7.0, dtype=torch.bfloat16, device=DEV)
    y_sh = torch.zeros((n, H), dtype=torch.bfloat16, device=DEV)
    api.asap_moe_expert_ffn(c.h, x_perm, offs, x, y, y_sh, c.ws(n))
    code, word = api.asap_moe_status(c.h)
    assert code != 0 and word == 8, word
    assert bool((y == 7.0).all())
    compare_rows(bf16_to_f64(y_sh), oracle.swiglu(bf16_to_f64(x), *c.shared))
    assert_clean(c)


@pytest.mark.parametrize("cfg", [MX_SMALL, DS_SMALL], ids=lambda c: c.name)
def test_ffn_halves_equal_expert_ffn_and_h_matches_oracle(cfg):
    """gate_up then down give the same bits as expert_ffn; the intermediate h
    matches silu(X Wg^T) * (X Wu^T) of the oracle."""
    c = Case.get(cfg)
    n, k, H, I = max(cfg.microbatches), cfg.top_k, cfg.hidden, cfg.inter
    x = c.tokens(0, n)
    idx, w, counts, offsets = run_route(c, x)
    x_perm = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
    perm_src = torch.empty(n * k, dtype=torch.int32, device=DEV)
    perm_dst = torch.empty((n, k), dtype=torch.int32, device=DEV)
    ws = c.ws(n)
    api.asap_moe_dispatch(c.h, x, idx, x_perm, perm_src, perm_dst, ws)
    y1 = torch.empty_like(x_perm)
    ysh1 = torch.empty((n, H), dtype=torch.bfloat16, device=DEV) if cfg.n_shared else None
    api.asap_moe_expert_ffn(c.h, x_perm, offsets, x, y1, ysh1, ws)
    hb = torch.empty((n * k, I), dtype=torch.bfloat16, device=DEV)
    hsh = torch.empty((n, cfg.shared_inter), dtype=torch.bfloat16, device=DEV) if cfg.n_shared else None
    api.asap_moe_expert_gate_up(c.h, x_perm, offsets, x, hb, hsh)
    y2 = torch.empty_like(x_perm)
    ysh2 = torch.empty_like(ysh1) if cfg.n_shared else None
    api.asap_moe_expert_down(c.h, hb, offsets, hsh, n, y2, ysh2)
    # the same halves with a workspace: tiles claimed dynamically, same bits
    hb3 = torch.empty_like(hb)
    hsh3 = torch.empty_like(hsh) if cfg.n_shared else None
    api.asap_moe_expert_gate_up(c.h, x_perm, offsets, x, hb3, hsh3, ws=ws)
    y3 = torch.empty_like(x_perm)
    ysh3 = torch.empty_like(ysh1) if cfg.n_shared else None
    api.asap_moe_expert_down(c.h, hb3, offsets, hsh3, n, y3, ysh3, ws=ws)
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))
    assert torch.equal(y1.view(torch.int16), y3.view(torch.int16))
    assert torch.equal(hb.view(torch.int16), hb3.view(torch.int16))
    if cfg.n_shared:
        assert torch.equal(ysh1.view(torch.int16), ysh2.view(torch.int16))
        assert torch.equal(ysh1.view(torch.int16), ysh3.view(torch.int16))
    off = offsets.cpu().numpy()
    xp = bf16_to_f64(x_perm)
    hg = bf16_to_f64(hb)
    for e in range(cfg.n_experts):
        a, b = off[e], off[e + 1]
        if b > a:
            X = xp[a:b]
            ref = oracle.silu(X @ c.wf["w_gate"][e].T) * (X @ c.wf["w_up"][e].T)
            compare_rows(hg[a:b], ref, rel_norm=5e-3)
    assert_clean(c)


def test_create_waits_for_weights_still_being_written():
    """Weights produced by kernels still running on another stream are read
    only after they are complete (create synchronises first)."""
    cfg = inputs.small_variant(TINY, name="tiny_race")
    w = inputs.make_weights(cfg, DEV)
    ref = api.asap_moe_create(cfg, w, 160)
    x = inputs.make_tokens(cfg, 160, 0, DEV)
    out_ref = torch.empty_like(x)
    api.asap_moe_layer(ref, x, out_ref, api.workspace(ref, 160))
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    w2 = {}
    with torch.cuda.stream(side):
        torch.cuda._sleep(50_000_000)                 # keep the side stream busy
        for k_, v in w.items():
            if v is not None:
                w2[k_] = torch.zeros_like(v)
                w2[k_].copy_(v)                      # the copy lands after the sleep
    h2 = api.asap_moe_create(cfg, w2, 160)
    out = torch.empty_like(x)
    api.asap_moe_layer(h2, x, out, api.workspace(h2, 160))
    torch.cuda.synchronize()
    assert torch.equal(out.view(torch.int16), out_ref.view(torch.int16))
    ref.close()
    h2.close()
