"""Top-k gating and routing of the MoE layer, float64, one token at a time.

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg may import this package.

What the paper fixes: each token activates K = 8 of E_total = 256 routed experts
(ASAP Table 1) plus one always-active shared expert (Section 5.1, DeepSeek-V3.2).
The paper never writes the gating function down; the three rules below are the
published definitions of the model families the workloads are shaped after,
with these readings of the gaps:

* ``softmax``        p = softmax(L) over all E experts; pick the k largest;
                     weight = the picked p (no renormalisation).
* ``softmax_renorm`` as above, then weight = p / sum of the picked p.
* ``sigmoid_grouped`` s = sigmoid(L); selection score s_b = s + bias (a
                     selection-only correction bias, zero in every workload);
                     experts split into G equal contiguous groups; a group's
                     score is the sum of its two largest s_b; keep the
                     ``topk_groups`` best groups; pick the k largest s_b among
                     their experts; weight = s / sum of the picked s * scale.

Ties: the lower expert index (and the lower group index) wins.  Slot order
within a token: descending selection score, ties by ascending index.  Because
softmax is monotone, selecting on p is the same as selecting on the logits L;
this module selects on L for the two softmax rules.
"""
import numpy as np


def router_logits(x, wr):
    """L[t, e] = sum_h x[t, h] * Wr[e, h]   (x: [n, H], Wr: [E, H], float64)."""
    return np.asarray(x, np.float64) @ np.asarray(wr, np.float64).T


def _order(keys):
    """Indices of ``keys`` sorted by descending value, ties by ascending index."""
    keys = np.asarray(keys)
    return np.lexsort((np.arange(keys.shape[0]), -keys))


def sigmoid(v):
    return 1.0 / (1.0 + np.exp(-np.asarray(v, np.float64)))


def route_token_softmax(l, k, renorm):
    """Route one token.  l: [E] logits.  Returns (idx[k], w[k])."""
    l = np.asarray(l, np.float64)
    idx = _order(l)[:k]
    m = l.max()
    p = np.exp(l - m) / np.exp(l - m).sum()
    w = p[idx]
    if renorm:
        w = w / w.sum()
    return idx.astype(np.int64), w


def route_token_sigmoid_grouped(l, k, n_groups, topk_groups, scale, bias=None):
    """Route one token with grouped sigmoid gating.  Returns (idx[k], w[k])."""
    l = np.asarray(l, np.float64)
    E = l.shape[0]
    s = sigmoid(l)
    sb = s + (0.0 if bias is None else np.asarray(bias, np.float64))
    gsz = E // n_groups
    gscore = np.empty(n_groups)
    for g in range(n_groups):
        members = sb[g * gsz:(g + 1) * gsz]
        top2 = members[_order(members)[:2]]
        gscore[g] = top2.sum()
    kept = _order(gscore)[:topk_groups]
    cand = np.concatenate([np.arange(g * gsz, (g + 1) * gsz) for g in sorted(kept)])
    # rank candidates by (-sb, index); _order breaks ties on position, and
    # ``cand`` is ascending, so position order is index order.
    idx = cand[_order(sb[cand])[:k]]
    w = s[idx] / s[idx].sum() * scale
    return idx.astype(np.int64), w


def route(L, cfg, bias=None):
    """Route every token.  L: [n, E] logits; cfg: mapping with keys gating,
    top_k, n_groups, topk_groups, route_scale.  Returns idx [n, k] int64 and
    w [n, k] float64."""
    L = np.asarray(L, np.float64)
    n = L.shape[0]
    k = cfg["top_k"]
    idx = np.zeros((n, k), np.int64)
    w = np.zeros((n, k), np.float64)
    for t in range(n):
        if cfg["gating"] == "softmax":
            idx[t], w[t] = route_token_softmax(L[t], k, renorm=False)
        elif cfg["gating"] == "softmax_renorm":
            idx[t], w[t] = route_token_softmax(L[t], k, renorm=True)
        elif cfg["gating"] == "sigmoid_grouped":
            idx[t], w[t] = route_token_sigmoid_grouped(
                L[t], k, cfg["n_groups"], cfg["topk_groups"], cfg["route_scale"], bias)
        else:
            raise ValueError(cfg["gating"])
    return idx, w


# --------------------------------------------------------------------------
# Certified comparison of a float32 router against this float64 one.
#
# The GPU forms each logit as a float32 sum of exact bf16*bf16 products in an
# order the tensor core chooses, so a token whose decisive comparisons have a
# margin below the float32 error may legitimately go either way.  The error
# model is a random walk of float32 rounding errors over the sum: one term for
# the spread of the products and one for the partial sums that carry the
# logit's own magnitude through about H/16 accumulation steps,
#     eps[t, e] = 10 * 2^-24 * ( sqrt(H) * ||x[t] * Wr[e]||_2 + sqrt(H/16) * |L[t, e]| ).
# On GB300 the largest observed float32 logit error was below 0.4 eps on every
# workload (DeepSeek-V3 shape: max 1.2e-5, median 1.2e-6).  Tests check the
# GPU's logits against eps element by element, which is what makes the
# decided / undecided split below sound for the data tested.
# --------------------------------------------------------------------------

U32 = 2.0 ** -24


def logit_error_bound(x, wr):
    x = np.asarray(x, np.float64)
    wr = np.asarray(wr, np.float64)
    H = x.shape[1]
    l2 = np.sqrt((x * x) @ (wr * wr).T)
    L = x @ wr.T
    return 10.0 * U32 * (np.sqrt(H) * l2 + np.sqrt(H / 16.0) * np.abs(L))


def _score_bounds(l, eps, cfg, bias):
    """Selection scores of one token and their half-widths."""
    if cfg["gating"] in ("softmax", "softmax_renorm"):
        return l, eps
    s = sigmoid(l)
    sb = s + (0.0 if bias is None else np.asarray(bias, np.float64))
    # sigmoid is increasing: a logit in [l - eps, l + eps] maps into
    # [sigmoid(l - eps), sigmoid(l + eps)]; add a few float32 ulps for the
    # GPU's own evaluation of sigmoid
    r = np.maximum(s - sigmoid(l - eps), sigmoid(l + eps) - s)
    return sb, r + 8.0 * U32


def _decided_greedy(v, r, m):
    """True when picking the top m of v (in order) is unambiguous under
    +-r uncertainty: every adjacent pair in the chosen order and the boundary
    between the m-th and all rejected entries are separated by more than the
    sum of their radii."""
    order = _order(v)
    for j in range(m - 1):
        a, b = order[j], order[j + 1]
        if v[a] - r[a] <= v[b] + r[b]:
            return False
    if m < len(v):
        a = order[m - 1]
        rest = order[m:]
        if np.any(v[a] - r[a] <= v[rest] + r[rest]):
            return False
    return True


def _group_bounds(v, r, n_groups):
    """Lower and upper bounds of each group's score (sum of its two largest
    selection scores) when every member lies in [v - r, v + r].  The sum of
    the two largest entries is monotone in every entry, so the bounds are the
    same statistic of v - r and of v + r; 4 ulps cover the float32 add."""
    E = v.shape[0]
    gsz = E // n_groups
    lo = np.empty(n_groups)
    hi = np.empty(n_groups)
    for g in range(n_groups):
        mv, mr = v[g * gsz:(g + 1) * gsz], r[g * gsz:(g + 1) * gsz]
        lo[g] = np.sort(mv - mr)[-2:].sum() - 4.0 * U32
        hi[g] = np.sort(mv + mr)[-2:].sum() + 4.0 * U32
    return lo, hi


def token_decided(l, eps, cfg, bias=None):
    """Whether every comparison that fixes this token's experts and slot
    order clears the error bound: for grouped gating the kept group set must
    be unambiguous (only the set matters, not the order of kept groups), then
    the top-k among the kept groups' experts and their order."""
    l = np.asarray(l, np.float64)
    v, r = _score_bounds(l, np.asarray(eps, np.float64), cfg, bias)
    k = cfg["top_k"]
    if cfg["gating"] in ("softmax", "softmax_renorm"):
        return _decided_greedy(v, r, k)
    E = v.shape[0]
    G = cfg["n_groups"]
    gsz = E // G
    lo, hi = _group_bounds(v, r, G)
    mid = (lo + hi) / 2.0
    kept = sorted(_order(mid)[:cfg["topk_groups"]])
    dropped = [g for g in range(G) if g not in kept]
    if dropped and min(lo[g] for g in kept) <= max(hi[g] for g in dropped):
        return False
    cand = np.concatenate([np.arange(g * gsz, (g + 1) * gsz) for g in kept])
    return _decided_greedy(v[cand], r[cand], k)


def token_feasible(l, eps, cfg, idx, bias=None):
    """Whether a candidate routing ``idx`` (length k, in slot order) of one
    token is consistent with the logits lying anywhere inside +-eps.

    Checked conditions (necessary for some admissible logits to produce idx):
    slot order is non-increasing within the bounds; every picked expert's
    upper bound reaches every rejected eligible expert's lower bound; for
    grouped gating the picked experts lie in ``topk_groups`` groups whose
    score upper bounds reach every other group's lower bound."""
    l = np.asarray(l, np.float64)
    idx = np.asarray(idx, np.int64)
    v, r = _score_bounds(l, np.asarray(eps, np.float64), cfg, bias)
    k = cfg["top_k"]
    if len(set(idx.tolist())) != k or idx.min() < 0 or idx.max() >= v.shape[0]:
        return False
    for j in range(k - 1):
        if v[idx[j]] + r[idx[j]] < v[idx[j + 1]] - r[idx[j + 1]]:
            return False
    E = v.shape[0]
    if cfg["gating"] in ("softmax", "softmax_renorm"):
        eligible = np.arange(E)
    else:
        G = cfg["n_groups"]
        gsz = E // G
        groups = sorted(set((idx // gsz).tolist()))
        if len(groups) > cfg["topk_groups"]:
            return False
        lo, hi = _group_bounds(v, r, G)
        others = [g for g in range(G) if g not in groups]
        # the picked groups must be completable to a kept set: there must be
        # a choice of (topk_groups - len(groups)) further groups such that
        # every kept group's upper bound reaches every dropped group's lower
        # bound.  Choose the extra groups with the largest upper bounds.
        extra = sorted(others, key=lambda g: (-hi[g], g))[:cfg["topk_groups"] - len(groups)]
        kept = sorted(groups + extra)
        dropped = [g for g in range(G) if g not in kept]
        if dropped and min(hi[g] for g in kept) < max(lo[g] for g in dropped):
            return False
        eligible = np.concatenate([np.arange(g * gsz, (g + 1) * gsz) for g in kept])
    rejected = np.setdiff1d(eligible, idx)
    if rejected.size:
        if np.min(v[idx] + r[idx]) < np.max(v[rejected] - r[rejected]):
            return False
    return True
