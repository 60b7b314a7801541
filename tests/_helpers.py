"""Shared test plumbing: moving torch tensors to the oracle's float64 view
(through the oracle's own bit decoders) and the comparison rules."""
import numpy as np
import torch

import oracle

# Layer-output tolerance for bf16 storage with fp32 accumulation:
# per element |g - r| <= REL_ELEM * max(|r|, rms of r's token row), and per
# micro-batch ||g - r||_F / ||r||_F <= REL_NORM.
REL_ELEM = 2e-2
REL_NORM = 5e-3


def bf16_to_f64(t):
    """Exact float64 values of a bf16 tensor, decoded by the oracle."""
    bits = t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return oracle.bf16_bits_to_f64(bits)


def weights_f64(w, keys=("router_w", "w_gate", "w_up", "w_down", "sh_gate", "sh_up", "sh_down")):
    return {k: bf16_to_f64(w[k]) for k in keys if w.get(k) is not None}


def compare_rows(g, r, rel_elem=REL_ELEM, rel_norm=REL_NORM):
    """Returns (max elementwise ratio, normwise error); asserts both bounds."""
    g = np.asarray(g, np.float64)
    r = np.asarray(r, np.float64)
    assert g.shape == r.shape, (g.shape, r.shape)
    if r.size == 0:
        return 0.0, 0.0
    rms = np.sqrt(np.mean(r * r, axis=-1, keepdims=True))
    den = np.maximum(np.abs(r), rms)
    den = np.where(den > 0, den, 1.0)
    ratio = np.abs(g - r) / den
    worst = float(ratio.max())
    norm = float(np.linalg.norm(g - r) / max(np.linalg.norm(r), 1e-300))
    assert worst <= rel_elem, f"elementwise error {worst:.3e} > {rel_elem} at {np.unravel_index(ratio.argmax(), ratio.shape)}"
    assert norm <= rel_norm, f"normwise error {norm:.3e} > {rel_norm}"
    return worst, norm


def routing_check(L_ref, eps, cfg, idx_gpu, w_gpu, w_ref, idx_ref, bias=None):
    """Certified comparison of GPU routing with the oracle's: decided tokens
    bit-exact (idx), their weights within 1e-5 + 4 * max eps relative (a
    weight moves by at most twice the largest logit error in log space for
    both softmax and normalised sigmoid weights); undecided tokens feasible.
    Returns the boolean decided mask."""
    n = L_ref.shape[0]
    decided = np.array([oracle.token_decided(L_ref[t], eps[t], cfg, bias) for t in range(n)], bool)
    d = decided
    assert np.array_equal(idx_gpu[d], idx_ref[d]), f"{(idx_gpu[d] != idx_ref[d]).any(1).sum()} decided tokens differ"
    if d.any():
        rel = np.abs(w_gpu[d] - w_ref[d]) / np.abs(w_ref[d])
        tol = 1e-5 + 4.0 * eps[d].max(axis=1, keepdims=True)
        assert (rel <= tol).all(), float((rel / tol).max())
    for t in np.nonzero(~d)[0]:
        assert oracle.token_feasible(L_ref[t], eps[t], cfg, idx_gpu[t], bias), f"token {t} infeasible"
    return decided


def sample_tokens(idx_ref, decided, E, rng, count):
    """Decided tokens to compare: the last token, the first and last token
    of the hottest and of the coldest non-empty expert, then random ones."""
    n = idx_ref.shape[0]
    cnt = np.bincount(idx_ref.reshape(-1), minlength=E)
    hot = int(cnt.argmax())
    cold = int(np.where(cnt > 0, cnt, cnt.max() + 1).argmin())
    must = [n - 1]
    for e in (hot, cold):
        toks = np.nonzero((idx_ref == e).any(axis=1))[0]
        must += [int(toks[0]), int(toks[-1])]
    must = sorted({t for t in must if decided[t]})
    rest = np.setdiff1d(np.nonzero(decided)[0], must)
    extra = rng.choice(rest, max(0, min(count - len(must), len(rest))), replace=False)
    return np.unique(np.r_[must, extra]).astype(np.int64)
