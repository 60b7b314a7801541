"""The layer-oblivious path (the MoE Super Kernel of Section 3.4.2): one
handle over several layers, the layer id read by the kernels from device
memory.  Each layer's result must equal, bit for bit, a single-layer handle
built from that layer's weights alone (which the other GPU tests hold against
the oracle), whatever the order of the layers, whether the calls were
enqueued before the ids were written, and when replayed from one CUDA graph.
One layer is also checked against the oracle directly."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300.configs import TINY, DSV3, MIXTRAL, DSV3_FP8

from _helpers import bf16_to_f64, weights_f64, compare_rows, routing_check

pytestmark = pytest.mark.gpu

DEV = "cuda"
N_LAYERS = 3
ST_BAD_LAYER = 16
DS_SMALL = inputs.small_variant(DSV3, name="dsv3_small", hidden=512, inter=256, shared_inter=256,
                                microbatches=[300, 77])
MX_SMALL = inputs.small_variant(MIXTRAL, name="mixtral_small", hidden=1024, inter=512, microbatches=[1000, 333])
F8_SMALL = inputs.small_variant(DSV3_FP8, name="fp8_small", hidden=512, inter=256, shared_inter=256,
                                microbatches=[300, 77])
ORDER = [2, 0, 1, 1, 0, 2]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


class Layers:
    """N_LAYERS layers' weights, one multi-layer handle and one single-layer
    handle per layer.  The grouped-sigmoid layers get a selection bias on
    layer 1 only, so the per-layer bias lookup is exercised."""
    _cache = {}

    @classmethod
    def get(cls, cfg):
        if cfg.name not in cls._cache:
            cls._cache[cfg.name] = cls(cfg)
        return cls._cache[cfg.name]

    def __init__(self, cfg):
        self.cfg = cfg
        self.w = inputs.make_layer_weights(cfg, N_LAYERS, DEV)
        if cfg.gating == "sigmoid_grouped":
            g = torch.Generator(device=DEV).manual_seed(4242)
            self.w[1]["router_bias"] = 0.05 * torch.randn(cfg.n_experts, generator=g, device=DEV)
        mt = max(cfg.microbatches)
        self.h = api.asap_moe_create_layers(cfg, self.w, mt)
        self.single = [api.asap_moe_create(cfg, w, mt) for w in self.w]

    def tokens(self, i):
        return inputs.make_tokens(self.cfg, self.cfg.microbatches[i], i, DEV)


def single_out(L, layer, x):
    out = torch.empty_like(x)
    api.asap_moe_layer(L.single[layer], x, out, api.workspace(L.single[layer], x.shape[0]))
    return out


def same_bits(a, b):
    return torch.equal(a.view(torch.int16), b.view(torch.int16))


def assert_clean(h):
    code, word = api.asap_moe_status(h)
    assert code == 0 and word == 0, f"device status word {word:#x}"


@pytest.mark.parametrize("cfg", [TINY, MX_SMALL, DS_SMALL, F8_SMALL], ids=lambda c: c.name)
def test_layer_dyn_equals_single_layer_handles(cfg):
    L = Layers.get(cfg)
    assert api.asap_moe_n_layers(L.h) == N_LAYERS
    xs = [L.tokens(i) for i in range(len(cfg.microbatches))]
    ref = {(l, i): single_out(L, l, x) for l in range(N_LAYERS) for i, x in enumerate(xs)}
    slot = torch.empty(1, dtype=torch.int32, device=DEV)
    for step, l in enumerate(ORDER):
        i = step % len(xs)
        slot.fill_(l)
        out = torch.empty_like(xs[i])
        api.asap_moe_layer_dyn(L.h, slot, xs[i], out, api.workspace(L.h, xs[i].shape[0]))
        torch.cuda.synchronize()
        assert same_bits(out, ref[(l, i)]), (l, i)
    # the layers differ, and the calls without a layer id serve layer 0
    assert not same_bits(ref[(0, 0)], ref[(1, 0)])
    out = torch.empty_like(xs[0])
    api.asap_moe_layer(L.h, xs[0], out, api.workspace(L.h, xs[0].shape[0]))
    torch.cuda.synchronize()
    assert same_bits(out, ref[(0, 0)])
    assert_clean(L.h)


def test_biased_layer_against_oracle():
    """Layer 1 of the DeepSeek-shaped model (with its selection bias) through
    the layer id, against the float64 oracle on that layer's weights."""
    cfg = DS_SMALL
    L = Layers.get(cfg)
    wf = weights_f64(L.w[1])
    bias = L.w[1]["router_bias"].cpu().numpy().astype(np.float32).astype(np.float64)
    ocfg = cfg.oracle_cfg()
    slot = torch.ones(1, dtype=torch.int32, device=DEV)
    for i in range(len(cfg.microbatches)):
        x = L.tokens(i)
        out = torch.empty_like(x)
        api.asap_moe_layer_dyn(L.h, slot, x, out, api.workspace(L.h, x.shape[0]))
        torch.cuda.synchronize()
        xf = bf16_to_f64(x)
        r = oracle.moe_layer(xf, wf["router_w"], wf["w_gate"], wf["w_up"], wf["w_down"], ocfg,
                             shared=(wf["sh_gate"], wf["sh_up"], wf["sh_down"]), router_bias=bias)
        # routing of this call, read back through the single-layer handle of layer 1
        n, k, E = x.shape[0], cfg.top_k, cfg.n_experts
        idx = torch.empty((n, k), dtype=torch.int32, device=DEV)
        w = torch.empty((n, k), dtype=torch.float32, device=DEV)
        counts = torch.empty(E, dtype=torch.int32, device=DEV)
        offs = torch.empty(E + 1, dtype=torch.int32, device=DEV)
        api.asap_moe_route(L.single[1], x, idx, w, counts, offs, api.workspace(L.single[1], n))
        torch.cuda.synchronize()
        eps = oracle.logit_error_bound(xf, wf["router_w"])
        decided = routing_check(r["logits"], eps, ocfg, idx.cpu().numpy().astype(np.int64),
                                w.cpu().numpy().astype(np.float64), r["w"], r["idx"], bias=bias)
        compare_rows(bf16_to_f64(out)[decided], r["y"][decided])
    assert_clean(L.h)


def test_calls_enqueued_before_their_layer_ids_are_written():
    """Every call of a sequence is enqueued first, each with its own id slot;
    a kernel writes all the ids only afterwards (the stream orders it first
    by an event), as a producer that resolves layers late would."""
    cfg = DS_SMALL
    L = Layers.get(cfg)
    xs = [L.tokens(i) for i in range(len(cfg.microbatches))]
    ref = {(l, i): single_out(L, l, x) for l in range(N_LAYERS) for i, x in enumerate(xs)}
    torch.cuda.synchronize()
    producer = torch.cuda.Stream()
    moe = torch.cuda.Stream()
    slots = torch.full((len(ORDER),), -7, dtype=torch.int32, device=DEV)
    sched = torch.tensor(ORDER, dtype=torch.int32, device=DEV)
    written = torch.cuda.Event()
    outs = [torch.empty_like(xs[step % len(xs)]) for step in range(len(ORDER))]
    wss = [api.workspace(L.h, xs[step % len(xs)].shape[0]) for step in range(len(ORDER))]
    torch.cuda.synchronize()
    # the producer writes the ids about a millisecond from now; the whole
    # sequence is enqueued behind its event while the slots still hold -7
    with torch.cuda.stream(producer):
        torch.cuda._sleep(2_000_000)
        slots.copy_(sched)
        written.record(producer)
    moe.wait_event(written)
    for step in range(len(ORDER)):
        i = step % len(xs)
        api.asap_moe_layer_dyn(L.h, slots[step:step + 1], xs[i], outs[step], wss[step], stream=moe)
    torch.cuda.synchronize()
    for step, l in enumerate(ORDER):
        assert same_bits(outs[step], ref[(l, step % len(xs))]), step
    assert_clean(L.h)


@pytest.mark.parametrize("cfg", [DS_SMALL, F8_SMALL], ids=lambda c: c.name)
def test_one_graph_replayed_for_every_layer(cfg):
    L = Layers.get(cfg)
    x = L.tokens(0)
    ref = [single_out(L, l, x) for l in range(N_LAYERS)]
    slot = torch.zeros(1, dtype=torch.int32, device=DEV)
    out = torch.empty_like(x)
    ws = api.workspace(L.h, x.shape[0])
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        api.asap_moe_layer_dyn(L.h, slot, x, out, ws)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        api.asap_moe_layer_dyn(L.h, slot, x, out, ws)
    for l in [1, 2, 0, 2]:
        slot.fill_(l)
        out.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert same_bits(out, ref[l]), l
    assert_clean(L.h)


def test_layers_on_concurrent_streams():
    """Different layers at the same time on different streams, each call
    with its own id slot and workspace, equal the single-layer handles."""
    cfg = DS_SMALL
    L = Layers.get(cfg)
    xs = [L.tokens(i % len(cfg.microbatches)) for i in range(N_LAYERS)]
    ref = [single_out(L, l, xs[l]) for l in range(N_LAYERS)]
    torch.cuda.synchronize()
    slots = torch.tensor([2, 0, 1], dtype=torch.int32, device=DEV)
    order = slots.tolist()
    streams = [torch.cuda.Stream() for _ in range(N_LAYERS)]
    xin = [xs[l] for l in order]                   # stream j serves layer order[j] on its input
    outs = [torch.empty_like(x) for x in xin]
    wss = [api.workspace(L.h, x.shape[0]) for x in xin]
    for rep in range(3):
        for j, st in enumerate(streams):
            api.asap_moe_layer_dyn(L.h, slots[j:j + 1], xin[j], outs[j], wss[j], stream=st)
    torch.cuda.synchronize()
    for j in range(N_LAYERS):
        assert same_bits(outs[j], ref[order[j]]), j
    assert_clean(L.h)


def test_layer_id_out_of_range_is_reported_and_uses_layer_0():
    cfg = DS_SMALL
    L = Layers.get(cfg)
    x = L.tokens(1)
    ref0 = single_out(L, 0, x)
    for bad in (N_LAYERS, -1, 1 << 30):
        slot = torch.full((1,), bad, dtype=torch.int32, device=DEV)
        out = torch.empty_like(x)
        api.asap_moe_layer_dyn(L.h, slot, x, out, api.workspace(L.h, x.shape[0]))
        torch.cuda.synchronize()
        code, word = api.asap_moe_status(L.h)
        assert word & ST_BAD_LAYER, (bad, word)
        assert word & ~ST_BAD_LAYER == 0, word
        assert same_bits(out, ref0)
    assert_clean(L.h)


def test_batched_dyn_equals_per_microbatch_dyn():
    cfg = DS_SMALL
    L = Layers.get(cfg)
    xs = [L.tokens(i) for i in range(len(cfg.microbatches))]
    slot = torch.full((1,), 2, dtype=torch.int32, device=DEV)
    single = []
    for x in xs:
        o = torch.empty_like(x)
        api.asap_moe_layer_dyn(L.h, slot, x, o, api.workspace(L.h, x.shape[0]))
        single.append(o)
    outs = [torch.empty_like(x) for x in xs]
    h2 = api.asap_moe_create_layers(cfg, L.w, sum(cfg.microbatches))
    api.asap_moe_layer_batched_dyn(h2, slot, xs, outs, api.workspace(h2, sum(cfg.microbatches)))
    torch.cuda.synchronize()
    for a, b in zip(outs, single):
        assert same_bits(a, b)
    assert_clean(h2)
    assert_clean(L.h)
    h2.close()


def test_null_or_unaligned_layer_id_is_rejected():
    from paper_2606_22541_gb300._native import AsapError
    L = Layers.get(TINY)
    x = L.tokens(0)
    out = torch.empty_like(x)
    ws = api.workspace(L.h, x.shape[0])
    with pytest.raises(AsapError):
        api.asap_moe_layer_dyn(L.h, None, x, out, ws)
    raw = torch.zeros(8, dtype=torch.uint8, device=DEV)
    with pytest.raises(AsapError):
        api.asap_moe_layer_dyn(L.h, raw[1:], x, out, ws)
