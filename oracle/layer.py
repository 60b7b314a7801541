"""The expert-side MoE layer, float64, expert by expert.

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg may import this package.

Definition followed (the layer the MoE devices run in ASAP, Sections 3.2 and
3.4.2; model shape from Table 1 and Section 5.1):

    y[t] = sum_{j<k} w[t,j] * FFN_{idx[t,j]}(x[t]) + FFN_shared(x[t])
    FFN_e(v) = Wd_e (silu(Wg_e v) * (Wu_e v)),   silu(g) = g / (1 + exp(-g))

* The MoE side receives per-expert token counts as its metadata (Section
  3.2.1, region 1 of the shared buffer) and the tokens grouped for the experts
  (region 2): ``expert_counts``/``expert_offsets``/``permutation``/``dispatch``.
* The expert computation is a grouped matrix multiplication with the hidden
  states on the left and one layer's expert weights on the right (Section
  3.4.2): ``expert_ffn`` runs it expert by expert over each expert's segment.
* Results go back to the originating tokens through the expert IDs (Section
  3.2.2): ``combine``.

Readings where the paper is silent: a segment lists its (token, slot) pairs
in increasing (t, j) order; the combine adds the k weighted expert rows in
slot order, then the shared expert's row.
"""
import numpy as np

from .formats import round_to_e4m3_sat, E4M3_MAX
from . import gating


def expert_counts(idx, n_experts):
    """counts[e] = number of (t, j) with idx[t, j] == e."""
    idx = np.asarray(idx, np.int64)
    counts = np.zeros(n_experts, np.int64)
    for e in idx.reshape(-1):
        counts[e] += 1
    return counts


def expert_offsets(counts):
    """Exclusive prefix sum with E + 1 entries; offsets[E] = total."""
    off = np.zeros(len(counts) + 1, np.int64)
    for e, c in enumerate(counts):
        off[e + 1] = off[e] + c
    return off


def permutation(idx, n_experts):
    """Position of every (t, j) in the expert-grouped order.

    Returns perm_src [n*k] (position -> token) and perm_dst [n, k]
    ((token, slot) -> position).  Within expert e the pairs occupy
    positions offsets[e] .. offsets[e+1]-1 in increasing (t, j) order."""
    idx = np.asarray(idx, np.int64)
    n, k = idx.shape
    off = expert_offsets(expert_counts(idx, n_experts))
    fill = off[:-1].copy()
    perm_src = np.zeros(n * k, np.int64)
    perm_dst = np.zeros((n, k), np.int64)
    for t in range(n):
        for j in range(k):
            e = idx[t, j]
            p = fill[e]
            fill[e] += 1
            perm_src[p] = t
            perm_dst[t, j] = p
    return perm_src, perm_dst


def dispatch(x, perm_src):
    """x_perm[p] = x[perm_src[p]]: the tokens grouped for the experts."""
    return np.asarray(x, np.float64)[np.asarray(perm_src, np.int64)]


def silu(g):
    return g / (1.0 + np.exp(-g))


def swiglu(X, wg, wu, wd):
    """Rows of X through one SwiGLU FFN: (silu(X Wg^T) * (X Wu^T)) Wd^T."""
    X = np.asarray(X, np.float64)
    return (silu(X @ wg.T) * (X @ wu.T)) @ wd.T


def expert_ffn(x_perm, offsets, wg, wu, wd):
    """Run every expert on its segment of x_perm.

    wg, wu: [E, I, H]; wd: [E, H, I] (float64, or callables e -> matrix so
    large weight sets can be decoded one expert at a time)."""
    x_perm = np.asarray(x_perm, np.float64)
    E = len(offsets) - 1
    y = np.zeros_like(x_perm)   # an expert maps H channels back to H
    for e in range(E):
        a, b = offsets[e], offsets[e + 1]
        if b > a:
            y[a:b] = swiglu(x_perm[a:b], _get(wg, e), _get(wu, e), _get(wd, e))
    return y


def combine(y_perm, w, perm_dst, y_shared=None):
    """out[t] = sum_j w[t,j] * y_perm[perm_dst[t,j]]  (+ y_shared[t])."""
    y_perm = np.asarray(y_perm, np.float64)
    n, k = np.asarray(perm_dst).shape
    out = np.zeros((n, y_perm.shape[1]), np.float64)
    for t in range(n):
        for j in range(k):
            out[t] += w[t, j] * y_perm[perm_dst[t, j]]
        if y_shared is not None:
            out[t] += y_shared[t]
    return out


def _get(wset, e):
    return wset(e) if callable(wset) else wset[e]


def moe_layer(x, router_w, wg, wu, wd, cfg, shared=None, router_bias=None):
    """The whole layer for one micro-batch.

    x: [n, H]; router_w: [E, H]; wg/wu: [E, I, H]; wd: [E, H, I] (float64 or
    per-expert callables); shared: None or (sg [Is, H], su [Is, H], sd [H, Is]);
    cfg: mapping with n_experts, top_k, gating, n_groups, topk_groups,
    route_scale.  Returns a dict of every intermediate the GPU path exposes."""
    x = np.asarray(x, np.float64)
    E = cfg["n_experts"]
    L = gating.router_logits(x, router_w)
    idx, w = gating.route(L, cfg, router_bias)
    counts = expert_counts(idx, E)
    offsets = expert_offsets(counts)
    perm_src, perm_dst = permutation(idx, E)
    x_perm = dispatch(x, perm_src)
    y_perm = expert_ffn(x_perm, offsets, wg, wu, wd)
    y_sh = swiglu(x, *shared) if shared is not None else None
    y = combine(y_perm, w, perm_dst, y_sh)
    return dict(logits=L, idx=idx, w=w, counts=counts, offsets=offsets,
                perm_src=perm_src, perm_dst=perm_dst, y_perm=y_perm,
                y_shared=y_sh, y=y)


def moe_layer_tokens(x_tok, idx, w, wg, wu, wd, shared=None):
    """Layer outputs of a few tokens whose routing is already known (the layer
    is per token, so any subset of a micro-batch can be checked on its own).
    x_tok: [m, H]; idx, w: [m, k]."""
    x_tok = np.asarray(x_tok, np.float64)
    m, k = np.asarray(idx).shape
    out = np.zeros_like(x_tok)
    for t in range(m):
        for j in range(k):
            e = int(idx[t, j])
            out[t] += w[t, j] * swiglu(x_tok[t:t + 1], _get(wg, e), _get(wu, e), _get(wd, e))[0]
        if shared is not None:
            out[t] += swiglu(x_tok[t:t + 1], *shared)[0]
    return out


def moe_layer_tokens_by_expert(x_tok, idx, w, get_expert, shared=None):
    """``moe_layer_tokens`` looping over experts instead of tokens, so a large
    weight set is fetched (decoded) once per expert: get_expert(e) returns
    (Wg_e, Wu_e, Wd_e).  Same definition; the terms of a token are added in
    expert order, then the shared expert."""
    x_tok = np.asarray(x_tok, np.float64)
    idx = np.asarray(idx, np.int64)
    out = np.zeros_like(x_tok)
    for e in np.unique(idx):
        rows, slots = np.nonzero(idx == e)
        wg, wu, wd = get_expert(int(e))
        out[rows] += w[rows, slots][:, None] * swiglu(x_tok[rows], wg, wu, wd)
    if shared is not None:
        out += swiglu(x_tok, *shared)
    return out


# --------------------------------------------------------------------------
# FP8 (e4m3) configuration.  Weights arrive quantised (e4m3 values with one
# float32 scale per 128 x 128 block); activations are quantised on the fly per
# token per 128-channel block: s = amax / 448, q = round_to_e4m3_sat(v / s).
# The oracle emulates that activation rounding in float64 for x (before the
# gate/up GEMM) and for h (before the down GEMM), so the comparison tolerance
# only has to cover accumulation order and rounding-boundary cases.
# --------------------------------------------------------------------------

def quantize_rows_e4m3(v, block=128):
    """Per row, per ``block`` channels: returns (q, s) with v ~= q * s,
    q exact e4m3 values, s = amax / 448 (s = 1 where a block is all zero)."""
    v = np.asarray(v, np.float64)
    n, c = v.shape
    nb = (c + block - 1) // block
    q = np.zeros_like(v)
    s = np.ones((n, nb), np.float64)
    for b in range(nb):
        blk = v[:, b * block:(b + 1) * block]
        amax = np.abs(blk).max(axis=1)
        sc = np.where(amax > 0, amax / E4M3_MAX, 1.0)
        s[:, b] = sc
        q[:, b * block:(b + 1) * block] = round_to_e4m3_sat(blk / sc[:, None])
    return q, s


def dequant_blocks(q, s, block=128):
    """Weight matrix [R, C] from e4m3 values q and per-(block x block) scales
    s [ceil(R/block), ceil(C/block)]."""
    q = np.asarray(q, np.float64)
    rs = np.repeat(np.repeat(np.asarray(s, np.float64), block, 0), block, 1)
    return q * rs[:q.shape[0], :q.shape[1]]


def swiglu_fp8(X, wg, wu, wd, block=128):
    """SwiGLU with the activation quantisation of the FP8 configuration:
    x and h are each rounded per row per 128 channels to e4m3 * scale."""
    xq, xs = quantize_rows_e4m3(X, block)
    xd = xq * np.repeat(xs, block, 1)[:, :xq.shape[1]]
    h = silu(xd @ wg.T) * (xd @ wu.T)
    hq, hs = quantize_rows_e4m3(h, block)
    hd = hq * np.repeat(hs, block, 1)[:, :hq.shape[1]]
    return hd @ wd.T


def moe_layer_tokens_fp8(x_tok, idx, w, wg, wu, wd, shared=None, block=128):
    """FP8 twin of ``moe_layer_tokens``; weights are dequantised float64
    matrices (or per-expert callables returning them)."""
    x_tok = np.asarray(x_tok, np.float64)
    m, k = np.asarray(idx).shape
    out = np.zeros_like(x_tok)
    for t in range(m):
        for j in range(k):
            e = int(idx[t, j])
            out[t] += w[t, j] * swiglu_fp8(x_tok[t:t + 1], _get(wg, e), _get(wu, e), _get(wd, e), block)[0]
        if shared is not None:
            out[t] += swiglu_fp8(x_tok[t:t + 1], *shared, block=block)[0]
    return out


def moe_layer_tokens_fp8_by_expert(x_tok, idx, w, get_expert, shared=None, block=128):
    """``moe_layer_tokens_fp8`` looping over experts instead of tokens, so a
    large weight set is fetched (decoded) once per expert: get_expert(e)
    returns the dequantised (Wg_e, Wu_e, Wd_e).  Same definition (the
    activation quantisation is per row, so an expert's rows are quantised
    together); the terms of a token are added in expert order, then the
    shared expert."""
    x_tok = np.asarray(x_tok, np.float64)
    idx = np.asarray(idx, np.int64)
    out = np.zeros_like(x_tok)
    for e in np.unique(idx):
        rows, slots = np.nonzero(idx == e)
        wg, wu, wd = get_expert(int(e))
        out[rows] += w[rows, slots][:, None] * swiglu_fp8(x_tok[rows], wg, wu, wd, block)
    if shared is not None:
        out += swiglu_fp8(x_tok, *shared, block=block)
    return out
