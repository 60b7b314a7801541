"""Full-size workloads in the launch configuration bench.py times: every
micro-batch through asap_moe_layer on its own CUDA stream, all in flight at
once.  Routing, counts and offsets are checked for every token; the layer
output on a sample of at least SAMPLE_PER_MB decided tokens per micro-batch
(the oracle decodes each expert once for the whole sample): the micro-batch's
last token, the first and last tokens routed to its most and to its least
loaded expert (the ends of those segments and the last m-tiles of the
grouped GEMMs), and seeded random tokens; concurrent submission must equal
serial submission bit for bit.  A last case runs the largest micro-batch
the stress workload's length recipe allows."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import MIXTRAL, DSV3, STRESS

from _helpers import bf16_to_f64, compare_rows, routing_check, sample_tokens

pytestmark = pytest.mark.gpu

DEV = "cuda"
SAMPLE_PER_MB = 128



@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


# the largest micro-batch the stress workload's length recipe allows (its
# clip at 16384 tokens) through one call: the route without a K split, 512
# dispatch chunks, about 512 rows per expert in the grouped GEMMs
STRESS_MAX = inputs.small_variant(STRESS, name="dsv3_stress_max_microbatch", microbatches=[16384])


@pytest.mark.parametrize("cfg", [MIXTRAL, DSV3, STRESS, STRESS_MAX], ids=lambda c: c.name)
def test_full_size_streams_against_oracle(cfg):
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, max(cfg.microbatches))
    del w
    torch.cuda.empty_cache()
    xs = inputs.make_microbatches(cfg, DEV)
    wss = [api.workspace(h, x.shape[0]) for x in xs]
    streams = [torch.cuda.Stream() for _ in xs]
    conc = [torch.empty_like(x) for x in xs]
    torch.cuda.synchronize()
    for x, o, ws, s in zip(xs, conc, wss, streams):
        api.asap_moe_layer(h, x, o, ws, stream=s)
    torch.cuda.synchronize()
    serial = []
    for x, ws in zip(xs, wss):
        o = torch.empty_like(x)
        api.asap_moe_layer(h, x, o, ws)
        serial.append(o)
    torch.cuda.synchronize()
    for a, b in zip(conc, serial):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))

    ocfg = cfg.oracle_cfg()
    wr = bf16_to_f64(inputs.router_weights_bf16(cfg, DEV))
    shared = tuple(bf16_to_f64(t) for t in inputs.shared_weights_bf16(cfg, DEV)) if cfg.n_shared else None
    rng = np.random.default_rng(cfg.seed)
    samples = []   # (x rows, idx, w, gpu out rows)
    n_undecided = 0
    for i, x in enumerate(xs):
        n, k, E = x.shape[0], cfg.top_k, cfg.n_experts
        idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
        wt = torch.empty((n, k), dtype=torch.float32, device=DEV)
        counts = torch.empty(E, dtype=torch.int32, device=DEV)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
        api.asap_moe_route(h, x, idx, wt, counts, offsets, wss[i])
        torch.cuda.synchronize()
        xf = bf16_to_f64(x)
        L = oracle.router_logits(xf, wr)
        eps = oracle.logit_error_bound(xf, wr)
        lg = torch.empty((n, E), dtype=torch.float32, device=DEV)
        api.asap_moe_router_logits(h, x, lg, wss[i])
        torch.cuda.synchronize()
        err = np.abs(lg.cpu().numpy().astype(np.float64) - L)
        assert (err <= eps).all(), float((err / eps).max())
        # error statistics against two normalisations (diagnostic output)
        l1 = np.abs(xf) @ np.abs(wr).T
        l2 = np.sqrt((xf * xf) @ (wr * wr).T) * np.sqrt(xf.shape[1])
        print(f"[{cfg.name} mb{i}] logit err max {err.max():.3e} med {np.median(err):.3e} "
              f"max err/eps {float((err / eps).max()):.3e} max err/(2^-24 sum|p|) {float((err / (2**-24 * l1)).max()):.3e} "
              f"max err/(2^-24 sqrt(H)|p|_2) {float((err / (2**-24 * l2)).max()):.3e}")
        idx_ref, w_ref = oracle.route(L, ocfg)
        ig = idx.cpu().numpy().astype(np.int64)
        decided = routing_check(L, eps, ocfg, ig, wt.cpu().numpy().astype(np.float64), w_ref, idx_ref)
        n_undecided += int((~decided).sum())
        cg = counts.cpu().numpy()
        og = offsets.cpu().numpy()
        assert np.array_equal(cg, np.bincount(ig.reshape(-1), minlength=E))
        assert og[0] == 0 and np.array_equal(np.diff(og), cg) and og[-1] == n * k
        pick = sample_tokens(idx_ref, decided, E, rng, SAMPLE_PER_MB)
        assert len(pick) >= min(SAMPLE_PER_MB, int(decided.sum()))
        samples.append((xf[pick], idx_ref[pick], w_ref[pick], bf16_to_f64(conc[i])[pick]))
    print(f"[{cfg.name}] undecided tokens {n_undecided} of {sum(cfg.microbatches)}")
    assert n_undecided <= 0.05 * sum(cfg.microbatches), n_undecided

    x_s = np.concatenate([s[0] for s in samples])
    idx_s = np.concatenate([s[1] for s in samples])
    w_s = np.concatenate([s[2] for s in samples])
    g_s = np.concatenate([s[3] for s in samples])

    def get_expert(e):
        return tuple(bf16_to_f64(t) for t in inputs.expert_weights_bf16(cfg, e, DEV))

    ref = oracle.moe_layer_tokens_by_expert(x_s, idx_s, w_s, get_expert, shared)
    lo = 0
    for i, smp in enumerate(samples):          # both bounds per micro-batch
        hi = lo + len(smp[0])
        worst, norm = compare_rows(g_s[lo:hi], ref[lo:hi])
        print(f"[{cfg.name} mb{i}] {hi - lo} tokens: elementwise {worst:.3e} normwise {norm:.3e}")
        lo = hi
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"status {word:#x}"
    h.close()


@pytest.mark.parametrize("cfg,n", [(DSV3, 4096), (MIXTRAL, 3584)], ids=["dsv3_4096", "mixtral_3584"])
def test_fused_combine_full_size_bit_identical(cfg, n):
    """The combine fused into the down GEMM at a full-size micro-batch (every
    256-column slice of every token completed by its last arrival) gives the
    separate combine's bits."""
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, n)
    del w
    x = inputs.make_tokens(cfg, n, 0, DEV)
    ws = api.workspace(h, n)
    ref = torch.empty_like(x)
    api.asap_moe_layer(h, x, ref, ws)
    api.asap_moe_set_combine(h, api.COMBINE_FUSED)
    out = torch.full_like(x, 3.0)
    api.asap_moe_layer(h, x, out, ws)
    torch.cuda.synchronize()
    assert torch.equal(ref.view(torch.int16), out.view(torch.int16))
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"status {word:#x}"
    h.close()
