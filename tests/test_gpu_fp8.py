"""FP8 configuration (e4m3 expert weights with fp32 128 x 128 block scales,
e4m3 activations per token per 128 channels) through the C ABI against the
float64 oracle, which emulates the activation quantisation."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import DSV3_FP8, LayerConfig

from _helpers import bf16_to_f64, routing_check, sample_tokens

pytestmark = pytest.mark.gpu

DEV = "cuda"
REL_NORM_FP8 = 3e-2
F8_SMALL = inputs.small_variant(DSV3_FP8, name="fp8_small", hidden=512, inter=256, shared_inter=256,
                                microbatches=[300, 77])


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def e4m3_to_f64(t):
    return oracle.e4m3_bits_to_f64(t.detach().contiguous().view(torch.uint8).cpu().numpy())


def dequant_expert(w, e):
    """Float64 weights of routed expert e, decoded by the oracle."""
    return (oracle.dequant_blocks(e4m3_to_f64(w["w_gate"][e]), w["s_gate"][e].cpu().numpy()),
            oracle.dequant_blocks(e4m3_to_f64(w["w_up"][e]), w["s_up"][e].cpu().numpy()),
            oracle.dequant_blocks(e4m3_to_f64(w["w_down"][e]), w["s_down"][e].cpu().numpy()))


def shared_expert(w):
    return (oracle.dequant_blocks(e4m3_to_f64(w["sh_gate"]), w["sh_s_gate"].cpu().numpy()),
            oracle.dequant_blocks(e4m3_to_f64(w["sh_up"]), w["sh_s_up"].cpu().numpy()),
            oracle.dequant_blocks(e4m3_to_f64(w["sh_down"]), w["sh_s_down"].cpu().numpy()))


def compare_fp8(g, r):
    g = np.asarray(g, np.float64)
    r = np.asarray(r, np.float64)
    norm = float(np.linalg.norm(g - r) / np.linalg.norm(r))
    rms = np.sqrt(np.mean(r * r, axis=-1, keepdims=True))
    worst = float((np.abs(g - r) / np.maximum(np.abs(r), rms)).max())
    assert norm <= REL_NORM_FP8, f"normwise {norm:.3e}"
    assert worst <= 0.5, f"elementwise {worst:.3e}"   # gross-error guard; the fp8 bound is normwise
    return norm, worst


@pytest.fixture(scope="module")
def small():
    w = inputs.make_weights(F8_SMALL, DEV)
    h = api.asap_moe_create(F8_SMALL, w, max(F8_SMALL.microbatches))
    yield w, h
    h.close()


def test_dispatch_quantises_like_the_oracle(small):
    w, h = small
    cfg = F8_SMALL
    n, k, E, H = 300, cfg.top_k, cfg.n_experts, cfg.hidden
    x = inputs.make_tokens(cfg, n, 0, DEV)
    rng = np.random.default_rng(3)
    idx_np = np.array([rng.permutation(E)[:k] for _ in range(n)], np.int64)
    xq = torch.empty((n * k, H), dtype=torch.uint8, device=DEV)
    xs = torch.empty((n * k, H // 128), dtype=torch.float32, device=DEV)
    ps = torch.empty(n * k, dtype=torch.int32, device=DEV)
    pd = torch.empty((n, k), dtype=torch.int32, device=DEV)
    api.asap_moe_dispatch(h, x, torch.tensor(idx_np, dtype=torch.int32, device=DEV), xq, ps, pd,
                          api.workspace(h, n), x_perm_scales=xs)
    torch.cuda.synchronize()
    src, dst = oracle.permutation(idx_np, E)
    assert np.array_equal(ps.cpu().numpy(), src)
    q_ref, s_ref = oracle.quantize_rows_e4m3(oracle.dispatch(bf16_to_f64(x), src))
    q = e4m3_to_f64(xq)
    s = xs.cpu().numpy().astype(np.float64)
    assert np.allclose(s, s_ref, rtol=1e-6, atol=0)
    diff = q != q_ref
    assert diff.mean() < 1e-3, diff.mean()
    # where the float32 and float64 quotients straddle a rounding boundary,
    # the two picks are neighbouring e4m3 values
    assert np.all(np.abs(q[diff] - q_ref[diff]) <= np.abs(q_ref[diff]) * 2.0 ** -3 + 2.0 ** -9)


def test_fp8_layer_matches_oracle(small):
    w, h = small
    cfg = F8_SMALL
    ocfg = cfg.oracle_cfg()
    wr = bf16_to_f64(w["router_w"])
    shared = shared_expert(w)
    cache = {}

    def get_expert(e):
        if e not in cache:
            cache[e] = dequant_expert(w, e)
        return cache[e]

    for i, n in enumerate(cfg.microbatches):
        x = inputs.make_tokens(cfg, n, i, DEV)
        out = torch.empty_like(x)
        api.asap_moe_layer(h, x, out, api.workspace(h, n))
        torch.cuda.synchronize()
        xf = bf16_to_f64(x)
        L = oracle.router_logits(xf, wr)
        idx_ref, w_ref = oracle.route(L, ocfg)
        eps = oracle.logit_error_bound(xf, wr)
        dec = np.array([oracle.token_decided(L[t], eps[t], ocfg) for t in range(n)])
        ref = np.zeros((n, cfg.hidden))
        for t in np.nonzero(dec)[0]:
            wg, wu, wd = zip(*[get_expert(int(e)) for e in idx_ref[t]])
            ref[t] = oracle.moe_layer_tokens_fp8(xf[t:t + 1], np.arange(cfg.top_k)[None], w_ref[t:t + 1],
                                                 list(wg), list(wu), list(wd), shared)[0]
        compare_fp8(bf16_to_f64(out)[dec], ref[dec])
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0


def test_fp8_expert_ffn_equals_layer_bits(small):
    w, h = small
    cfg = F8_SMALL
    n, k, E, H = 300, cfg.top_k, cfg.n_experts, cfg.hidden
    x = inputs.make_tokens(cfg, n, 0, DEV)
    ws = api.workspace(h, n)
    out = torch.empty_like(x)
    api.asap_moe_layer(h, x, out, ws)
    idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
    wt = torch.empty((n, k), dtype=torch.float32, device=DEV)
    counts = torch.empty(E, dtype=torch.int32, device=DEV)
    offs = torch.empty(E + 1, dtype=torch.int32, device=DEV)
    api.asap_moe_route(h, x, idx, wt, counts, offs, ws)
    xq = torch.empty((n * k, H), dtype=torch.uint8, device=DEV)
    xs = torch.empty((n * k, H // 128), dtype=torch.float32, device=DEV)
    ps = torch.empty(n * k, dtype=torch.int32, device=DEV)
    pd = torch.empty((n, k), dtype=torch.int32, device=DEV)
    api.asap_moe_dispatch(h, x, idx, xq, ps, pd, ws, x_perm_scales=xs)
    y = torch.empty((n * k, H), dtype=torch.bfloat16, device=DEV)
    ysh = torch.empty((n, H), dtype=torch.bfloat16, device=DEV)
    api.asap_moe_expert_ffn(h, xq, offs, x, y, ysh, ws, x_perm_scales=xs)
    out2 = torch.empty_like(x)
    api.asap_moe_combine(h, y, ysh, wt, pd, out2)
    torch.cuda.synchronize()
    assert torch.equal(out.view(torch.int16), out2.view(torch.int16))


FP8_SAMPLE_PER_MB = 32


def test_fp8_full_size_streams_against_oracle():
    """The FP8 workload at full size (8 x 4096 tokens, each micro-batch on its
    own stream, all in flight at once): routing of every token, and the layer
    output of at least FP8_SAMPLE_PER_MB decided tokens of every micro-batch
    (its last token, the ends of its hottest and coldest expert's segments,
    seeded random tokens) against the oracle's FP8 emulation, each expert
    decoded once."""
    cfg = DSV3_FP8
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, max(cfg.microbatches))
    xs = inputs.make_microbatches(cfg, DEV)
    wss = [api.workspace(h, x.shape[0]) for x in xs]
    streams = [torch.cuda.Stream() for _ in xs]
    outs = [torch.empty_like(x) for x in xs]
    torch.cuda.synchronize()
    for x, o, ws, s in zip(xs, outs, wss, streams):
        api.asap_moe_layer(h, x, o, ws, stream=s)
    torch.cuda.synchronize()
    ocfg = cfg.oracle_cfg()
    wr = bf16_to_f64(w["router_w"])
    shared = shared_expert(w)
    rng = np.random.default_rng(cfg.seed)
    xs_s, idx_s, w_s, g_s = [], [], [], []
    for i, x in enumerate(xs):
        n, k, E = x.shape[0], cfg.top_k, cfg.n_experts
        idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
        wt = torch.empty((n, k), dtype=torch.float32, device=DEV)
        counts = torch.empty(E, dtype=torch.int32, device=DEV)
        offs = torch.empty(E + 1, dtype=torch.int32, device=DEV)
        api.asap_moe_route(h, x, idx, wt, counts, offs, wss[i])
        torch.cuda.synchronize()
        xf = bf16_to_f64(x)
        L = oracle.router_logits(xf, wr)
        eps = oracle.logit_error_bound(xf, wr)
        idx_ref, w_ref = oracle.route(L, ocfg)
        dec = routing_check(L, eps, ocfg, idx.cpu().numpy().astype(np.int64),
                            wt.cpu().numpy().astype(np.float64), w_ref, idx_ref)
        pick = sample_tokens(idx_ref, dec, E, rng, FP8_SAMPLE_PER_MB)
        assert len(pick) >= min(FP8_SAMPLE_PER_MB, int(dec.sum()))
        xs_s.append(xf[pick]); idx_s.append(idx_ref[pick]); w_s.append(w_ref[pick])
        g_s.append(bf16_to_f64(outs[i])[pick])
    x_a, idx_a, w_a, g = map(np.concatenate, (xs_s, idx_s, w_s, g_s))
    ref = oracle.moe_layer_tokens_fp8_by_expert(x_a, idx_a, w_a, lambda e: dequant_expert(w, e), shared)
    lo = 0
    for i, part in enumerate(g_s):            # the bound per micro-batch
        hi = lo + len(part)
        norm, worst = compare_fp8(g[lo:hi], ref[lo:hi])
        print(f"[fp8 mb{i}] {hi - lo} tokens: normwise {norm:.3e} elementwise {worst:.3e}")
        lo = hi
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0
    h.close()


def random_fp8_config(i):
    """A seeded random FP8 layer: 8 to 256 experts, the three gating rules,
    H and I multiples of the 128-channel scale blocks, with and without a
    shared expert, ragged token counts."""
    rng = np.random.default_rng(9000 + i)
    E = int(rng.choice([8, 16, 32, 64, 256]))
    gating = str(rng.choice(["softmax", "softmax_renorm", "sigmoid_grouped"]))
    k = int(rng.integers(1, min(8, E) + 1))
    H = int(rng.choice([256, 512, 1024]))
    I = int(rng.choice([128, 256]))
    sh = int(rng.integers(0, 2))
    Is = int(rng.choice([128, 256])) if sh else 0
    ng, tg = 1, 1
    if gating == "sigmoid_grouped":
        ng = int(rng.choice([g for g in (1, 2, 4, 8) if E % g == 0 and E // g >= 2]))
        tg = int(rng.integers(-(-k // (E // ng)), ng + 1))
    n = int(rng.integers(1, 900))
    return LayerConfig(f"f8rand{i}", hidden=H, n_experts=E, top_k=k, inter=I, n_shared=sh, shared_inter=Is,
                       gating=gating, n_groups=ng, topk_groups=tg, route_scale=float(rng.choice([1.0, 2.5])),
                       dtype="fp8_e4m3_block128", microbatches=[n], seed=9500 + i)


@pytest.mark.parametrize("cfg", [random_fp8_config(i) for i in range(12)], ids=lambda c: c.name)
def test_fp8_random_shapes_against_oracle(cfg):
    """The FP8 layer on seeded random shapes against the oracle's FP8
    emulation, on up to 64 decided tokens (40 more seeds were checked once)."""
    n, k, H = cfg.microbatches[0], cfg.top_k, cfg.hidden
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, n)
    x = inputs.make_tokens(cfg, n, 0, DEV)
    out = torch.empty_like(x)
    api.asap_moe_layer(h, x, out, api.workspace(h, n))
    torch.cuda.synchronize()
    ocfg = cfg.oracle_cfg()
    wr = bf16_to_f64(w["router_w"])
    shared = shared_expert(w) if cfg.n_shared else None
    xf = bf16_to_f64(x)
    L = oracle.router_logits(xf, wr)
    idx_ref, w_ref = oracle.route(L, ocfg)
    eps = oracle.logit_error_bound(xf, wr)
    dec = np.array([oracle.token_decided(L[t], eps[t], ocfg) for t in range(n)])
    cache = {}

    def get_expert(e):
        if e not in cache:
            cache[e] = dequant_expert(w, e)
        return cache[e]

    pick = np.nonzero(dec)[0][:64]
    ref = np.zeros((len(pick), H))
    for j, t in enumerate(pick):
        wg, wu, wd = zip(*[get_expert(int(e)) for e in idx_ref[t]])
        ref[j] = oracle.moe_layer_tokens_fp8(xf[t:t + 1], np.arange(k)[None], w_ref[t:t + 1], list(wg), list(wu),
                                             list(wd), shared)[0]
    compare_fp8(bf16_to_f64(out)[pick], ref)
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0
    h.close()
