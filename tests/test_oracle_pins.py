"""Pins of the float64 oracle against things other than itself: library
conversions, brute force on tiny inputs, closed forms, invariants and a
hand-worked example.  CPU only."""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import formats, gating, layer

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- formats

def test_bf16_decoder_matches_torch_on_every_pattern():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = formats.bf16_bits_to_f64(bits)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])


def test_bf16_decoder_known_values():
    f = formats.bf16_bits_to_f64
    assert f(np.uint16(0x3F80)) == 1.0
    assert f(np.uint16(0xC000)) == -2.0
    assert f(np.uint16(0x0001)) == 2.0 ** -133
    assert f(np.uint16(0x7F7F)) == (2 - 2 ** -7) * 2.0 ** 127
    assert np.isinf(f(np.uint16(0x7F80)))


def test_e4m3_decoder_matches_torch_on_every_pattern():
    bits = np.arange(256, dtype=np.uint8)
    ours = formats.e4m3_bits_to_f64(bits)
    ref = torch.from_numpy(bits).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    assert formats.e4m3_bits_to_f64(np.uint8(0x7E)) == 448.0
    assert formats.e4m3_bits_to_f64(np.uint8(0x01)) == 2.0 ** -9


def test_e4m3_rounding_matches_torch_cast_in_range():
    rng = np.random.default_rng(5)
    v = np.concatenate([rng.normal(0, 30, 20000), rng.normal(0, 0.01, 5000),
                        rng.uniform(-448, 448, 5000)])
    ours = formats.round_to_e4m3_sat(v)
    ref = torch.from_numpy(v).to(torch.float8_e4m3fn).to(torch.float64).numpy()
    assert np.array_equal(ours, ref)


def test_e4m3_rounding_ties_and_saturation():
    r = formats.round_to_e4m3_sat
    assert r(1.0625) == 1.0          # halfway between 1 and 1.125 -> even
    assert r(1.1875) == 1.25         # halfway between 1.125 and 1.25 -> even
    assert r(464.0) == 448.0         # tie between 448 and (absent) 480
    assert r(1e6) == 448.0 and r(-1e6) == -448.0
    assert r(2.0 ** -10) == 0.0      # half the smallest subnormal -> even (0)
    assert r(3 * 2.0 ** -10) == 2 * 2.0 ** -9


# ---------------------------------------------------------------- gating

def _brute_topk_softmax(l, k, renorm):
    """Max-sum subset, ties -> lexicographically smallest index set; slots by
    (-value, index); weights from the softmax written out directly."""
    E = len(l)
    best = None
    for S in itertools.combinations(range(E), k):
        key = (sum(l[i] for i in S), tuple(-i for i in S))
        if best is None or key > best[0]:
            best = (key, S)
    S = sorted(best[1], key=lambda i: (-l[i], i))
    z = sum(math.exp(v) for v in l)
    w = [math.exp(l[i]) / z for i in S]
    if renorm:
        tot = sum(w)
        w = [v / tot for v in w]
    return S, w


@pytest.mark.parametrize("renorm", [False, True])
def test_softmax_topk_matches_brute_force(renorm):
    rng = np.random.default_rng(11)
    for _ in range(300):
        l = rng.normal(0, 1.5, 8)
        idx, w = gating.route_token_softmax(l, 2, renorm)
        S, wb = _brute_topk_softmax(list(l), 2, renorm)
        assert list(idx) == S
        assert np.allclose(w, wb, rtol=1e-13, atol=0)


def test_softmax_topk_exact_ties_lower_index_wins():
    l = np.array([0.5, 1.0, 1.0, 0.2, 1.0, -1.0, 0.0, 1.0])
    idx, _ = gating.route_token_softmax(l, 2, False)
    assert list(idx) == [1, 2]
    S, _ = _brute_topk_softmax(list(l), 3, False)
    idx3, _ = gating.route_token_softmax(l, 3, False)
    assert list(idx3) == S == [1, 2, 4]


def _brute_grouped(l, k, G, kg, scale):
    s = [1 / (1 + math.exp(-v)) for v in l]
    E = len(l)
    gsz = E // G
    gscore = []
    for g in range(G):
        mem = range(g * gsz, (g + 1) * gsz)
        gscore.append(max(s[a] + s[b] for a, b in itertools.combinations(mem, 2)))
    best = None
    for Gs in itertools.combinations(range(G), kg):
        key = (sum(gscore[g] for g in Gs), tuple(-g for g in Gs))
        if best is None or key > best[0]:
            best = (key, Gs)
    cand = [e for g in best[1] for e in range(g * gsz, (g + 1) * gsz)]
    bestS = None
    for S in itertools.combinations(cand, k):
        key = (sum(s[i] for i in S), tuple(-i for i in sorted(S)))
        if bestS is None or key > bestS[0]:
            bestS = (key, S)
    S = sorted(bestS[1], key=lambda i: (-s[i], i))
    tot = sum(s[i] for i in S)
    return S, [s[i] / tot * scale for i in S]


def test_grouped_sigmoid_matches_brute_force():
    rng = np.random.default_rng(12)
    for _ in range(150):
        l = rng.normal(0, 1.0, 16)
        idx, w = gating.route_token_sigmoid_grouped(l, 4, 4, 2, 2.5)
        S, wb = _brute_grouped(list(l), 4, 4, 2, 2.5)
        assert list(idx) == S
        assert np.allclose(w, wb, rtol=1e-13, atol=0)


def _brute_grouped_bias(l, b, k, G, kg, scale):
    """Brute force of the biased rule: experts and groups are chosen by the
    selection score sigmoid(l) + b; the weights use sigmoid(l) alone."""
    s = [1 / (1 + math.exp(-v)) for v in l]
    key = [s[i] + b[i] for i in range(len(l))]
    E = len(l)
    gsz = E // G
    gscore = [max(key[a] + key[c] for a, c in itertools.combinations(range(g * gsz, (g + 1) * gsz), 2))
              for g in range(G)]
    best = None
    for Gs in itertools.combinations(range(G), kg):
        kk = (sum(gscore[g] for g in Gs), tuple(-g for g in Gs))
        if best is None or kk > best[0]:
            best = (kk, Gs)
    cand = [e for g in best[1] for e in range(g * gsz, (g + 1) * gsz)]
    bestS = None
    for S in itertools.combinations(cand, k):
        kk = (sum(key[i] for i in S), tuple(-i for i in sorted(S)))
        if bestS is None or kk > bestS[0]:
            bestS = (kk, S)
    S = sorted(bestS[1], key=lambda i: (-key[i], i))
    tot = sum(s[i] for i in S)
    return S, [s[i] / tot * scale for i in S]


def test_grouped_sigmoid_with_bias_matches_brute_force():
    """The selection bias moves which experts are chosen but not their
    weights; a large bias on a weak expert must select it."""
    rng = np.random.default_rng(14)
    for _ in range(150):
        l = rng.normal(0, 1.0, 16)
        b = rng.normal(0, 0.3, 16)
        idx, w = gating.route_token_sigmoid_grouped(l, 4, 4, 2, 2.5, bias=b)
        S, wb = _brute_grouped_bias(list(l), list(b), 4, 4, 2, 2.5)
        assert list(idx) == S
        assert np.allclose(w, wb, rtol=1e-13, atol=0)
    l = np.zeros(16)
    l[0] = 3.0
    b = np.zeros(16)
    b[9] = 5.0                                   # expert 9 (group 2) wins on its bias alone
    idx, w = gating.route_token_sigmoid_grouped(l, 2, 4, 2, 1.0, bias=b)
    assert list(idx) == [9, 0]
    s = 1 / (1 + np.exp(-l))
    assert np.allclose(w, [s[9] / (s[9] + s[0]), s[0] / (s[9] + s[0])], rtol=1e-13)


def test_grouped_sigmoid_group_tie_lower_group_wins():
    # groups of 4; groups 1 and 2 tie on the top-2 sum, group 0 is best
    l = np.array([3.0, 2.9, -5, -5,   1.0, 0.5, -5, -5,   0.5, 1.0, -5, -5,   -3, -3, -3, -3])
    idx, _ = gating.route_token_sigmoid_grouped(l, 4, 4, 2, 1.0)
    assert list(idx) == [0, 1, 4, 5]
    S, _ = _brute_grouped(list(l), 4, 4, 2, 1.0)
    assert S == [0, 1, 4, 5]


def test_softmax_renorm_with_k_equal_E_is_full_softmax():
    rng = np.random.default_rng(13)
    l = rng.normal(0, 2, 8)
    idx, w = gating.route_token_softmax(l, 8, True)
    p = np.exp(l) / np.exp(l).sum()
    assert np.allclose(w, p[idx], rtol=1e-13)
    assert sorted(idx) == list(range(8))


def test_softmax_variants_agree_on_idx():
    rng = np.random.default_rng(14)
    L = rng.normal(0, 1, (64, 8))
    a, _ = gating.route(L, dict(gating="softmax", top_k=2))
    b, _ = gating.route(L, dict(gating="softmax_renorm", top_k=2))
    assert np.array_equal(a, b)


def test_certified_comparison():
    cfg = dict(gating="softmax", top_k=2)
    l = np.array([1.0, 0.9, 0.5, 0.4, 0.0, -1, -2, -3])
    eps = np.full(8, 1e-3)
    assert gating.token_decided(l, eps, cfg)
    assert gating.token_feasible(l, eps, cfg, [0, 1])
    assert not gating.token_feasible(l, eps, cfg, [1, 0])
    assert not gating.token_feasible(l, eps, cfg, [0, 2])
    l2 = l.copy()
    l2[2] = 0.9 - 5e-4                      # near tie at the k boundary
    assert not gating.token_decided(l2, eps, cfg)
    assert gating.token_feasible(l2, eps, cfg, [0, 2])   # either may win
    assert gating.token_feasible(l2, eps, cfg, [0, 1])
    gcfg = dict(gating="sigmoid_grouped", top_k=4, n_groups=4, topk_groups=2, route_scale=1.0)
    rng = np.random.default_rng(15)
    n_decided = 0
    for _ in range(50):
        lg = rng.normal(0, 1, 16)
        idx, _ = gating.route_token_sigmoid_grouped(lg, 4, 4, 2, 1.0)
        e = np.full(16, 1e-6)
        assert gating.token_feasible(lg, e, gcfg, idx)
        if gating.token_decided(lg, e, gcfg):
            n_decided += 1
            # the next-best expert of the kept groups swapped into the last
            # slot, or a slot swap, must be infeasible for a decided token
            groups = sorted(set((idx // 4).tolist()) | set())
            s = 1 / (1 + np.exp(-lg))
            cand = [c for g in range(4) for c in range(4 * g, 4 * g + 4)
                    if c not in idx and (c // 4) in groups]
            if cand:
                nxt = max(cand, key=lambda c: (s[c], -c))
                wrong = idx.copy()
                wrong[-1] = nxt
                assert not gating.token_feasible(lg, e, gcfg, wrong)
            assert not gating.token_feasible(lg, e, gcfg, idx[[1, 0, 2, 3]])
    assert n_decided > 40


def _bf16_values(a):
    """Round float64 values to bf16 (torch's round-to-nearest-even) and return them as float64."""
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).to(torch.float64).numpy()


def _fp32_truncating_block_sums(prods, block=16):
    """fp32 accumulation as a tensor-core MMA does it: each step adds a block
    of ``block`` products (K of one bf16 MMA) to the accumulator in one
    operation whose result is rounded toward zero (truncated) to fp32."""
    n_blk = prods.shape[-1] // block
    blocks = prods.reshape(*prods.shape[:-1], n_blk, block).astype(np.float64).sum(axis=-1)
    acc = np.zeros(prods.shape[:-1], np.float32)
    for i in range(n_blk):
        t = acc.astype(np.float64) + blocks[..., i]
        f = t.astype(np.float32)
        over = np.abs(f.astype(np.float64)) > np.abs(t)
        f[over] = np.nextafter(f[over], np.float32(0))
        acc = f
    return acc


@pytest.mark.parametrize("case", ["configs", "cancelling"])
def test_logit_error_bound_covers_fp32_accumulation_orders(case):
    """The bound on |fp32 logit - exact logit| that the certified routing
    comparison relies on holds, on inputs drawn like the configs' (x ~ N(0,1),
    router weights ~ N(0, 0.02), bf16) and on rows whose logit nearly cancels,
    for fp32 accumulation of the (exact) bf16 products in every order a router
    kernel may use: sequential, reversed, blocked by the MMA's K = 16, split-K
    slices added in slice order, and MMA steps of 16 products whose sums are
    truncated instead of rounded."""
    rng = np.random.default_rng({"configs": 31, "cancelling": 33}[case])
    n, E, H = 24, 48, 7168
    x, wr = rng.normal(0, 1, (n, H)), rng.normal(0, 0.02, (E, H))
    if case == "cancelling":
        # second half of every weight row cancels the first half's dot with x[0]
        ratio = x[0, :H // 2] / np.where(np.abs(x[0, H // 2:]) < 1e-3, 1.0, x[0, H // 2:])
        wr[:, H // 2:] = np.clip(-wr[:, :H // 2] * ratio[None, :], -0.1, 0.1)
    x, wr = _bf16_values(x), _bf16_values(wr)
    exact = x @ wr.T
    eps = gating.logit_error_bound(x, wr)
    prods = (x[:, None, :] * wr[None, :, :]).astype(np.float32)   # bf16 x bf16 is exact in fp32
    assert np.array_equal(prods.astype(np.float64), x[:, None, :] * wr[None, :, :])
    sums = {
        "sequential": np.cumsum(prods, axis=2, dtype=np.float32)[..., -1],
        "reversed": np.cumsum(prods[..., ::-1], axis=2, dtype=np.float32)[..., -1],
        "k16_blocks": np.cumsum(prods.reshape(n, E, H // 16, 16).sum(axis=3, dtype=np.float32), axis=2,
                                dtype=np.float32)[..., -1],
        "split_k4": np.cumsum(np.stack([np.cumsum(q, axis=2, dtype=np.float32)[..., -1]
                                        for q in np.split(prods, 4, axis=2)], axis=2), axis=2,
                              dtype=np.float32)[..., -1],
        "k16_truncating": _fp32_truncating_block_sums(prods),
    }
    for name, got in sums.items():
        err = np.abs(got.astype(np.float64) - exact)
        assert np.all(err <= eps), (case, name, float((err / eps).max()))


# ---------------------------------------------------------------- counts / permutation

def _random_idx(rng, n, E, k):
    return np.array([rng.permutation(E)[:k] for _ in range(n)], np.int64).reshape(n, k)


def test_counts_offsets_invariants():
    rng = np.random.default_rng(21)
    for n, E, k in [(0, 8, 2), (1, 8, 2), (37, 8, 2), (200, 256, 8)]:
        idx = _random_idx(rng, n, E, k).reshape(n, k)
        c = layer.expert_counts(idx, E)
        o = layer.expert_offsets(c)
        assert c.sum() == n * k and (c >= 0).all()
        assert o[0] == 0 and o[-1] == n * k and (np.diff(o) == c).all()
        assert np.array_equal(c, np.bincount(idx.reshape(-1), minlength=E))


def test_permutation_is_a_stable_bijection():
    rng = np.random.default_rng(22)
    n, E, k = 150, 16, 4
    idx = _random_idx(rng, n, E, k)
    src, dst = layer.permutation(idx, E)
    assert sorted(dst.reshape(-1).tolist()) == list(range(n * k))
    off = layer.expert_offsets(layer.expert_counts(idx, E))
    for t in range(n):
        for j in range(k):
            p = dst[t, j]
            assert src[p] == t
            e = idx[t, j]
            assert off[e] <= p < off[e + 1]
    # stable: inside each segment the (t, j) pairs increase
    pairs = {int(dst[t, j]): (t, j) for t in range(n) for j in range(k)}
    for e in range(E):
        seg = [pairs[p] for p in range(off[e], off[e + 1])]
        assert seg == sorted(seg)


def test_identity_experts_return_k_times_x():
    rng = np.random.default_rng(23)
    n, E, k, H = 64, 8, 2, 32
    bits = rng.integers(0, 65536, (n, H)).astype(np.uint16)
    bits = (bits & 0x3FFF) | 0x3000           # finite, moderate bf16 values
    x = formats.bf16_bits_to_f64(bits)
    idx = _random_idx(rng, n, E, k)
    src, dst = layer.permutation(idx, E)
    xp = layer.dispatch(x, src)
    out = layer.combine(xp, np.ones((n, k)), dst)
    assert np.array_equal(out, k * x)


# ---------------------------------------------------------------- FFN / layer

def test_single_expert_k1_equals_dense_swiglu():
    rng = np.random.default_rng(31)
    n, H, I = 20, 48, 24
    x = rng.normal(0, 1, (n, H))
    wg = rng.normal(0, 0.2, (1, I, H))
    wu = rng.normal(0, 0.2, (1, I, H))
    wd = rng.normal(0, 0.2, (1, H, I))
    wr = rng.normal(0, 0.2, (1, H))
    cfg = dict(n_experts=1, top_k=1, gating="softmax", n_groups=1, topk_groups=1, route_scale=1.0)
    r = layer.moe_layer(x, wr, wg, wu, wd, cfg)
    # dense SwiGLU written independently: per token, per channel sums
    g = np.einsum("ih,nh->ni", wg[0], x)
    u = np.einsum("ih,nh->ni", wu[0], x)
    h = g * u / (1 + np.exp(-g))
    ref = np.einsum("hi,ni->nh", wd[0], h)
    assert np.allclose(r["w"], 1.0)
    assert np.allclose(r["y"], ref, rtol=1e-12, atol=1e-12)


def test_worked_example():
    d = json.load(open(os.path.join(GOLDEN, "worked_layer_example.json")))
    a = lambda k: np.array(d[k], np.float64)
    cfg = dict(n_experts=2, top_k=1, gating="softmax", n_groups=1, topk_groups=1, route_scale=1.0)
    r = layer.moe_layer(a("x"), a("router_w"), a("w_gate"), a("w_up"), a("w_down"), cfg,
                        shared=(a("sh_gate"), a("sh_up"), a("sh_down")))
    p0 = 1 / (1 + math.exp(-2))
    h = 2 / (1 + math.exp(-2))
    hs = -1 / (1 + math.exp(1))
    assert r["idx"].tolist() == d["expected_idx"]
    assert np.allclose(r["y"], [[p0 * h + 2 * hs, 3 * p0 * h]], rtol=1e-14, atol=0)


def test_per_token_independence():
    rng = np.random.default_rng(32)
    n, H, E, k, I = 60, 32, 8, 2, 16
    x = rng.normal(0, 1, (n, H))
    wr = rng.normal(0, 0.3, (E, H))
    wg = rng.normal(0, 0.2, (E, I, H))
    wu = rng.normal(0, 0.2, (E, I, H))
    wd = rng.normal(0, 0.2, (E, H, I))
    cfg = dict(n_experts=E, top_k=k, gating="softmax_renorm", n_groups=1, topk_groups=1, route_scale=1.0)
    full = layer.moe_layer(x, wr, wg, wu, wd, cfg)["y"]
    parts = [layer.moe_layer(x[a:b], wr, wg, wu, wd, cfg)["y"] for a, b in [(0, 7), (7, 33), (33, 60)]]
    assert np.allclose(np.concatenate(parts), full, rtol=1e-12, atol=1e-12)
    some = [3, 17, 59]
    r = layer.moe_layer(x, wr, wg, wu, wd, cfg)
    tok = layer.moe_layer_tokens(x[some], r["idx"][some], r["w"][some], wg, wu, wd)
    assert np.allclose(tok, full[some], rtol=1e-12, atol=1e-12)


def test_expert_major_sampling_equals_token_major():
    rng = np.random.default_rng(34)
    n, H, E, k, I = 12, 16, 6, 3, 8
    x = rng.normal(0, 1, (n, H))
    wg, wu = rng.normal(0, 0.3, (2, E, I, H))
    wd = rng.normal(0, 0.3, (E, H, I))
    sh = (rng.normal(0, 0.2, (I, H)), rng.normal(0, 0.2, (I, H)), rng.normal(0, 0.2, (H, I)))
    idx = np.array([rng.permutation(E)[:k] for _ in range(n)])
    w = rng.uniform(0, 1, (n, k))
    a = layer.moe_layer_tokens(x, idx, w, wg, wu, wd, sh)
    b = layer.moe_layer_tokens_by_expert(x, idx, w, lambda e: (wg[e], wu[e], wd[e]), sh)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12)


def test_shared_expert_enters_once():
    rng = np.random.default_rng(33)
    n, H, E, k, I = 10, 16, 4, 2, 8
    x = rng.normal(0, 1, (n, H))
    wr = rng.normal(0, 0.3, (E, H))
    wg, wu = rng.normal(0, 0.2, (2, E, I, H))
    wd = rng.normal(0, 0.2, (E, H, I))
    sh = (rng.normal(0, 0.2, (I, H)), rng.normal(0, 0.2, (I, H)), rng.normal(0, 0.2, (H, I)))
    cfg = dict(n_experts=E, top_k=k, gating="softmax", n_groups=1, topk_groups=1, route_scale=1.0)
    a = layer.moe_layer(x, wr, wg, wu, wd, cfg)["y"]
    b = layer.moe_layer(x, wr, wg, wu, wd, cfg, shared=sh)["y"]
    assert np.allclose(b - a, layer.swiglu(x, *sh), rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- FP8 emulation

def test_row_quantisation_properties():
    rng = np.random.default_rng(41)
    v = rng.normal(0, 3, (7, 384))
    q, s = layer.quantize_rows_e4m3(v)
    assert s.shape == (7, 3)
    # every q is an e4m3 value and the block max maps to exactly 448
    assert np.array_equal(formats.round_to_e4m3_sat(q), q)
    for b in range(3):
        assert np.allclose(np.abs(q[:, b * 128:(b + 1) * 128]).max(1), 448.0)
    back = q * np.repeat(s, 128, 1)
    # relative error of e4m3 normals is at most 2^-4; subnormals add 2^-10*s
    err = np.abs(back - v)
    bound = np.abs(v) * 2.0 ** -4 + np.repeat(s, 128, 1) * 2.0 ** -10
    assert (err <= bound * (1 + 1e-12)).all()


def test_dequant_blocks_layout():
    q = np.ones((256, 384))
    s = np.arange(6, dtype=np.float64).reshape(2, 3)
    w = layer.dequant_blocks(q, s)
    assert w[0, 0] == 0 and w[127, 383] == 2 and w[128, 0] == 3 and w[255, 383] == 5


def test_fp8_swiglu_within_e4m3_error_of_unquantised():
    """Two e4m3 roundings (x, then h) of about 2^-4 relative each keep the
    result within a few per cent of the unquantised SwiGLU."""
    rng = np.random.default_rng(42)
    H, I = 256, 128
    x = rng.normal(0, 1, (3, H))
    wg, wu = rng.normal(0, 1 / 16, (2, I, H))
    wd = rng.normal(0, 1 / 11.3, (H, I))
    a = layer.swiglu_fp8(x, wg, wu, wd)
    b = layer.swiglu(x, wg, wu, wd)
    assert np.linalg.norm(a - b) / np.linalg.norm(b) < 0.08


# Pins of the FP8 emulation (activation quantisation per token per 128
# channels, s = amax / 448, round to nearest even e4m3, for x before the
# gate/up product and for h before the down product).  Each pin returns
# True when it holds, so the planted-mistake test below can show that a
# missing h quantisation, a 64-channel block or a scale taken over the wrong
# axis fails at least one of them.

def _representable_block(rng, c, width=128):
    """One block of ``width`` values that are e4m3 values times 2^c; the
    first half holds the block maximum 448 * 2^c, the second half peaks at
    320 * 2^c, so only a 128-wide block has a power-of-two scale."""
    e4 = formats.e4m3_bits_to_f64(np.arange(0, 0x7F, dtype=np.uint8))   # finite, >= 0
    e4 = e4[e4 <= 320.0]
    v = rng.choice(e4, width) * rng.choice([-1.0, 1.0], width)
    v[rng.integers(0, width // 2)] = 448.0
    v[width // 2 + rng.integers(0, width // 2)] = -320.0
    return np.ldexp(v, c)


def _fp8_exact_weights(x0, h_target):
    """Gate/up weights that read only channel 0 of x (x0 = x[0], a power of
    two): g = 64 in every channel, where silu(64) == 64 in float64, and
    u = h_target / 64, so silu(g) * u == h_target exactly."""
    I = len(h_target)
    H = 256
    wg = np.zeros((I, H))
    wu = np.zeros((I, H))
    wg[:, 0] = 64.0 / x0
    wu[:, 0] = h_target / 64.0 / x0
    return wg, wu


def _pin_fp8_exact_on_representable_input():
    """x and h whose 128-channel blocks are e4m3 values times power-of-two
    scales equal to amax / 448 quantise without error, so the emulation
    must return the unquantised SwiGLU bit for bit."""
    rng = np.random.default_rng(61)
    x = np.concatenate([_representable_block(rng, -3), _representable_block(rng, 2)])
    x[0] = 256.0 * 2.0 ** -3            # channel 0 is a power of two below the block max
    h = np.concatenate([_representable_block(rng, -5), _representable_block(rng, 1)])
    wg, wu = _fp8_exact_weights(x[0], h)
    wd = rng.normal(0, 0.1, (256, 256))
    a = layer.swiglu_fp8(x[None], wg, wu, wd)
    b = layer.swiglu(x[None], wg, wu, wd)
    return np.array_equal(a, b)


def _pin_fp8_hand_worked_rounding():
    """One token, hand-worked.  x is representable (quantises exactly), g = 64
    everywhere and the down projection is the identity, so the output is
    the quantised h itself.  h has two 128-channel blocks with maxima 448 * 2
    and 448 / 4 (scales 2 and 1/4); the other values, divided by the scale,
    sit on rounding ties or off the grid:
        17 -> 16, 19 -> 20 (ties to the even neighbour, binade [16, 32) step 2),
        1.5 * 2^-9 -> 2^-8 (subnormal tie), 0.3 -> 0.3125 (nearest, step 2^-5),
        -100 -> -96 (step 8: 96 and 104, 100 is a tie -> 96, even),
    and the rest are zero."""
    x = np.zeros(256)
    x[0] = 1.0
    x[1] = 448.0
    x[128] = 448.0 * 2.0 ** -6
    s0, s1 = 2.0, 0.25
    scaled = {0: 448.0, 1: 17.0, 2: 19.0, 3: 1.5 * 2.0 ** -9, 4: 0.3, 5: -100.0,
              64: -19.0, 65: 17.0, 100: -0.3}
    expect_q = {0: 448.0, 1: 16.0, 2: 20.0, 3: 2.0 ** -8, 4: 0.3125, 5: -96.0,
                64: -20.0, 65: 16.0, 100: -0.3125}
    h = np.zeros(256)
    want = np.zeros(256)
    for ch, v in scaled.items():
        h[ch] = v * s0
        want[ch] = expect_q[ch] * s0
        h[128 + ch] = v * s1
        want[128 + ch] = expect_q[ch] * s1
    wg, wu = _fp8_exact_weights(x[0], h)
    y = layer.moe_layer_tokens_fp8(x[None], np.array([[0]]), np.array([[1.0]]),
                                   wg[None], wu[None], np.eye(256)[None])
    return np.array_equal(y[0], want)


_E4M3_TABLE = torch.arange(0, 0x7F, dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float64).numpy()


def _nearest_e4m3(v):
    """Round to e4m3 by search over the table of finite non-negative codes
    (decoded by torch): nearest value, a tie going to the even code; magnitudes
    above 448 saturate."""
    a = np.minimum(np.abs(v), 448.0)
    i = np.clip(np.searchsorted(_E4M3_TABLE, a), 1, len(_E4M3_TABLE) - 1)
    lo, hi = _E4M3_TABLE[i - 1], _E4M3_TABLE[i]
    pick_hi = (hi - a < a - lo) | ((hi - a == a - lo) & (i % 2 == 0))
    return np.copysign(np.where(pick_hi, hi, lo), v)


def _quantize_blocks_by_search(v):
    n, c = v.shape
    blocks = v.reshape(n, c // 128, 128)
    amax = np.abs(blocks).max(axis=2, keepdims=True)
    s = np.where(amax > 0, amax / 448.0, 1.0)
    return (_nearest_e4m3(blocks / s) * s).reshape(n, c)


def _pin_fp8_equals_search_composition():
    """Random inputs: the emulation equals quantise (by table search) ->
    product -> quantise -> product, composed here without the oracle."""
    rng = np.random.default_rng(62)
    n, H, I = 5, 384, 256
    x = rng.normal(0, 1, (n, H))
    x[1, 130:140] *= 40.0                      # one block with a large maximum
    wg, wu = rng.normal(0, 1 / 19.6, (2, I, H))
    wd = rng.normal(0, 1 / 16, (H, I))
    xd = _quantize_blocks_by_search(x)
    g = xd @ wg.T
    hd = _quantize_blocks_by_search(g / (1.0 + np.exp(-g)) * (xd @ wu.T))
    ref = hd @ wd.T
    got = layer.swiglu_fp8(x, wg, wu, wd)
    return np.allclose(got, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())


def test_fp8_swiglu_exact_on_representable_input():
    assert _pin_fp8_exact_on_representable_input()


def test_fp8_hand_worked_rounding_of_h():
    assert _pin_fp8_hand_worked_rounding()


def test_fp8_swiglu_equals_composition_by_table_search():
    assert _pin_fp8_equals_search_composition()


def test_fp8_layer_tokens_weights_and_shared_expert():
    """moe_layer_tokens_fp8: two experts with equal weights and routing
    weights summing to 1 give one expert's output; the shared expert adds
    its own quantised SwiGLU."""
    rng = np.random.default_rng(63)
    n, H, I = 4, 256, 128
    x = rng.normal(0, 1, (n, H))
    wg, wu = rng.normal(0, 1 / 16, (2, 1, I, H))
    wd = rng.normal(0, 1 / 11.3, (1, H, I))
    two = lambda a: np.concatenate([a, a])
    idx = np.tile([[0, 1]], (n, 1))
    w = np.tile([[0.25, 0.75]], (n, 1))
    one = layer.swiglu_fp8(x, wg[0], wu[0], wd[0])
    y = layer.moe_layer_tokens_fp8(x, idx, w, two(wg), two(wu), two(wd))
    assert np.allclose(y, one, rtol=1e-14, atol=1e-14 * np.abs(one).max())
    sh = (rng.normal(0, 1 / 16, (I, H)), rng.normal(0, 1 / 16, (I, H)), rng.normal(0, 1 / 11.3, (H, I)))
    ys = layer.moe_layer_tokens_fp8(x, idx, w, two(wg), two(wu), two(wd), shared=sh)
    assert np.allclose(ys - y, layer.swiglu_fp8(x, *sh), rtol=1e-12, atol=1e-12 * np.abs(ys).max())


def test_fp8_expert_major_equals_token_major():
    rng = np.random.default_rng(64)
    n, H, E, k, I = 9, 256, 5, 3, 128
    x = rng.normal(0, 1, (n, H))
    wg, wu = rng.normal(0, 1 / 16, (2, E, I, H))
    wd = rng.normal(0, 1 / 11.3, (E, H, I))
    sh = (rng.normal(0, 1 / 16, (I, H)), rng.normal(0, 1 / 16, (I, H)), rng.normal(0, 1 / 11.3, (H, I)))
    idx = _random_idx(rng, n, E, k)
    w = rng.uniform(0, 1, (n, k))
    a = layer.moe_layer_tokens_fp8(x, idx, w, wg, wu, wd, sh)
    b = layer.moe_layer_tokens_fp8_by_expert(x, idx, w, lambda e: (wg[e], wu[e], wd[e]), sh)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12 * np.abs(a).max())


def test_fp8_pins_catch_planted_mistakes(monkeypatch):
    """Plant each plausible mistake in the oracle's FP8 emulation and check
    that at least one FP8 pin fails."""
    pins = (_pin_fp8_exact_on_representable_input, _pin_fp8_hand_worked_rounding,
            _pin_fp8_equals_search_composition)
    assert all(p() for p in pins)
    real = layer.quantize_rows_e4m3

    def skip_h(v, block=128):                 # the second call (h) is not quantised
        skip_h.calls += 1
        if skip_h.calls % 2 == 0:
            v = np.asarray(v, np.float64)
            return v.copy(), np.ones((v.shape[0], (v.shape[1] + block - 1) // block))
        return real(v, block)
    skip_h.calls = 0

    # the mistakes below return dequantised values with unit scales, which
    # the emulation multiplies back unchanged
    def block64(v, block=128):                # 64-channel blocks
        q, s = real(v, 64)
        v = np.asarray(v, np.float64)
        return q * np.repeat(s, 64, 1)[:, :v.shape[1]], np.ones((v.shape[0], (v.shape[1] + block - 1) // block))

    def column_scale(v, block=128):           # amax over tokens instead of channels
        v = np.asarray(v, np.float64)
        amax = np.abs(v).max(axis=0, keepdims=True)
        sc = np.where(amax > 0, amax / 448.0, 1.0)
        q = formats.round_to_e4m3_sat(v / sc)
        return q * sc, np.ones((v.shape[0], (v.shape[1] + block - 1) // block))

    for mistake in (skip_h, block64, column_scale):
        monkeypatch.setattr(layer, "quantize_rows_e4m3", mistake)
        assert not all(p() for p in pins), mistake.__name__
        monkeypatch.setattr(layer, "quantize_rows_e4m3", real)
# ---------------------------------------------------------------- paper constants

def test_table1_shapes_are_the_dsv3_configs():
    d = json.load(open(os.path.join(GOLDEN, "table1_dsv3.json")))
    from paper_2606_22541_gb300.configs import DSV3, STRESS, DSV3_FP8
    for c in (DSV3, STRESS, DSV3_FP8):
        assert c.n_experts == d["E_total"] == d["routed_experts"]
        assert c.top_k == d["K"] == d["active_routed_per_token"]
        assert c.hidden == d["H"]
        assert c.n_shared == d["shared_experts"] == d["active_shared_per_token"]


# ---------------------------------------------------------------- planted mistakes

def test_pins_catch_planted_mistakes(monkeypatch):
    """Plant plausible mistakes in the oracle and check a pin notices."""
    rng = np.random.default_rng(51)
    n, H, I = 6, 16, 8
    x = rng.normal(0, 1, (n, H))
    wg, wu = rng.normal(0, 0.3, (2, 1, I, H))
    wd = rng.normal(0, 0.3, (1, H, I))
    cfg = dict(n_experts=1, top_k=1, gating="softmax", n_groups=1, topk_groups=1, route_scale=1.0)
    g = np.einsum("ih,nh->ni", wg[0], x)
    u = np.einsum("ih,nh->ni", wu[0], x)
    ref = np.einsum("hi,ni->nh", wd[0], g * u / (1 + np.exp(-g)))
    good = layer.moe_layer(x, rng.normal(0, 1, (1, H)), wg, wu, wd, cfg)["y"]
    assert np.allclose(good, ref)
    monkeypatch.setattr(layer, "silu", lambda v: v / (1.0 + np.exp(v)))   # sign slip
    bad = layer.moe_layer(x, rng.normal(0, 1, (1, H)), wg, wu, wd, cfg)["y"]
    assert not np.allclose(bad, ref)
    monkeypatch.undo()
    # transposed router operand order would reorder top-k: brute force sees it
    l = np.array([0.1, 2.0, -1.0, 1.5, 0.0, 0.3, -0.2, 0.9])
    S, _ = _brute_topk_softmax(list(l), 2, False)
    monkeypatch.setattr(gating, "_order", lambda keys: np.lexsort((np.arange(len(keys)), np.asarray(keys))))
    idx, _ = gating.route_token_softmax(l, 2, False)
    assert list(idx) != S


def test_router_logits_hand_worked_and_one_hot():
    """router_logits against values worked by hand (the logits are the dot
    products of each token with each expert's router row) and against
    one-hot tokens, which must pick out one router column exactly."""
    x = np.array([[1.0, 2.0, -1.0], [0.5, 0.0, 4.0]])
    wr = np.array([[2.0, 0.0, 1.0], [-1.0, 3.0, 0.5], [0.0, 0.0, 0.0], [1.0, 1.0, 1.0]])
    # token 0: 2 + 0 - 1 = 1; -1 + 6 - 0.5 = 4.5; 0; 1 + 2 - 1 = 2
    # token 1: 1 + 0 + 4 = 5; -0.5 + 0 + 2 = 1.5; 0; 0.5 + 0 + 4 = 4.5
    want = np.array([[1.0, 4.5, 0.0, 2.0], [5.0, 1.5, 0.0, 4.5]])
    assert np.array_equal(oracle.router_logits(x, wr), want)
    rng = np.random.default_rng(3)
    W = rng.standard_normal((6, 5))
    eye = np.eye(5)
    L = oracle.router_logits(eye, W)
    assert L.shape == (5, 6)
    assert np.array_equal(L, W.T)                     # token j = e_j gives column j of Wr
    assert np.array_equal(oracle.router_logits(np.zeros((2, 5)), W), np.zeros((2, 6)))


def test_expert_ffn_hand_worked_segments():
    """expert_ffn on two experts' segments with values worked by hand:
    expert 0 (gate row [1, 0], up row [0, 1], down column [1, 2]) on token
    [1, 2] gives g = 1, u = 2, h = silu(1) * 2 and y = [h, 2h]; expert 1 has
    an empty segment; expert 2 (gate row [0, 0]) gives h = silu(0) * u = 0.
    silu(1) = 1 / (1 + e^-1) exactly as the closed form."""
    wg = np.array([[[1.0, 0.0]], [[5.0, 5.0]], [[0.0, 0.0]]])      # [E=3, I=1, H=2]
    wu = np.array([[[0.0, 1.0]], [[5.0, 5.0]], [[3.0, 4.0]]])
    wd = np.array([[[1.0], [2.0]], [[9.0], [9.0]], [[1.0], [1.0]]])  # [E, H=2, I=1]
    x_perm = np.array([[1.0, 2.0], [7.0, -3.0]])
    offsets = np.array([0, 1, 1, 2])                                 # expert 1's segment is empty
    y = oracle.expert_ffn(x_perm, offsets, wg, wu, wd)
    h = 1.0 / (1.0 + np.exp(-1.0)) * 2.0
    assert np.allclose(y[0], [h, 2.0 * h], rtol=0, atol=1e-15)
    assert np.array_equal(y[1], [0.0, 0.0])
    # callables decode one expert at a time and give the same result
    y2 = oracle.expert_ffn(x_perm, offsets, lambda e: wg[e], lambda e: wu[e], lambda e: wd[e])
    assert np.array_equal(y, y2)
