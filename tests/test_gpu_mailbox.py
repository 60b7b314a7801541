"""The mailbox (device-side ready set): DP-group streams post routed
micro-batches into slots; service rounds on the MoE stream claim, on the
device, every post published when they start and serve all of them with one
grouped GEMM pass.  Whichever posts share a round, each output must equal
asap_moe_layer on the same micro-batch bit for bit.  Arrival orders and
delays are driven from the host (posts in random slot order on several
streams, each behind a random GPU sleep); the one failure case is a round
started for a post that is never made, whose bounded wait must run out,
record its status bit and still serve what is ready."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_22541_gb300 import api, inputs
from paper_2606_22541_gb300._native import AsapError
from paper_2606_22541_gb300.configs import DSV3, DSV3_FP8, MIXTRAL, STRESS

from _helpers import bf16_to_f64, compare_rows

pytestmark = pytest.mark.gpu

DEV = "cuda"
ST_MBOX_WAIT = 128

DS = inputs.small_variant(DSV3, name="mbox_ds", hidden=1024, inter=256, shared_inter=256,
                          microbatches=[700, 301, 512, 1000, 96, 333])
MX = inputs.small_variant(MIXTRAL, name="mbox_mx", hidden=1024, inter=512, microbatches=[1000, 333, 64, 517])
F8 = inputs.small_variant(DSV3_FP8, name="mbox_f8", hidden=512, inter=256, shared_inter=256,
                          microbatches=[300, 77, 2, 129])


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


class Case:
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
        self.xs = inputs.make_microbatches(cfg, DEV)
        self.ref = []
        for x in self.xs:
            o = torch.empty_like(x)
            api.asap_moe_layer(self.h, x, o, api.workspace(self.h, x.shape[0]))
            self.ref.append(o)
        torch.cuda.synchronize()


def same_bits(a, b):
    return torch.equal(a.view(torch.int16), b.view(torch.int16))


def assert_clean(h, allowed=0):
    code, word = api.asap_moe_status(h)
    assert word & ~allowed == 0, f"status {word:#x}"
    return word


@pytest.mark.parametrize("cfg", [DS, MX, F8], ids=lambda c: c.name)
def test_all_posted_first_are_served_by_one_round(cfg):
    """Every post published before the first round starts: that round claims
    all of them; the later rounds find nothing left."""
    c = Case.get(cfg)
    n = len(c.xs)
    m = api.asap_moe_mailbox_create(c.h, n, max(cfg.microbatches))
    streams = [torch.cuda.Stream() for _ in range(n)]
    outs = [torch.full_like(x, 7.0) for x in c.xs]
    eps = [api.asap_moe_mailbox_post(m, i, x, o, stream=s) for i, (x, o, s) in enumerate(zip(c.xs, outs, streams))]
    torch.cuda.synchronize()
    server = torch.cuda.Stream()
    for i in range(n):
        api.asap_moe_mailbox_serve(m, i, eps[i], stream=server)
    torch.cuda.synchronize()
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == n and claimed == [n] + [0] * (n - 1)
    for a, b in zip(c.ref, outs):
        assert same_bits(a, b)
    assert [api.asap_moe_mailbox_served(m, i) for i in range(n)] == eps
    assert_clean(c.h)
    m.close()


@pytest.mark.parametrize("cfg", [DS, MX, F8], ids=lambda c: c.name)
def test_random_arrivals_and_delays(cfg):
    """Posts in random slot order on three producer streams, each behind a
    random GPU sleep, every post served right after it was made: the device
    decides how the posts group into rounds; the outputs may not depend on
    it.  Three passes reuse the slots (epochs 1, 2, 3)."""
    c = Case.get(cfg)
    n = len(c.xs)
    rng = np.random.default_rng(7)
    m = api.asap_moe_mailbox_create(c.h, n, max(cfg.microbatches))
    producers = [torch.cuda.Stream() for _ in range(3)]
    server = torch.cuda.Stream()
    consumer = torch.cuda.Stream()
    total_posts = 0
    for rep in range(3):
        outs = [torch.full_like(x, float(rep + 3)) for x in c.xs]
        order = rng.permutation(n)
        for i in order:
            s = producers[int(rng.integers(0, 3))]
            with torch.cuda.stream(s):
                torch.cuda._sleep(int(rng.integers(0, 400_000)))
            if rep > 0:
                api.asap_moe_mailbox_wait(m, int(i), stream=s)   # the slot's previous post is done
            ep = api.asap_moe_mailbox_post(m, int(i), c.xs[i], outs[i], stream=s)
            assert ep == rep + 1
            api.asap_moe_mailbox_serve(m, int(i), ep, stream=server)
            total_posts += 1
        copies = []
        for i in range(n):
            api.asap_moe_mailbox_wait(m, i, stream=consumer)
            with torch.cuda.stream(consumer):
                copies.append(outs[i].clone())
        torch.cuda.synchronize()
        for a, b, cp in zip(c.ref, outs, copies):
            assert same_bits(a, b) and same_bits(a, cp)
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == total_posts and sum(claimed) == total_posts
    print(f"[{cfg.name}] posts per round: {claimed}")
    assert_clean(c.h)
    m.close()


def test_serve_calls_from_several_streams():
    """Serve calls spread over three server streams (a round per post, its
    stream chosen at random): each round waits for the mailbox's previous
    round, so rounds never overlap on the shared server workspace, and the
    outputs stay bit-identical over passes that reuse the slots."""
    c = Case.get(DS)
    n = len(c.xs)
    rng = np.random.default_rng(11)
    m = api.asap_moe_mailbox_create(c.h, n, max(DS.microbatches))
    producers = [torch.cuda.Stream() for _ in range(2)]
    servers = [torch.cuda.Stream() for _ in range(3)]
    for rep in range(3):
        outs = [torch.full_like(x, float(rep + 1)) for x in c.xs]
        for i in rng.permutation(n):
            s = producers[int(rng.integers(0, 2))]
            with torch.cuda.stream(s):
                torch.cuda._sleep(int(rng.integers(0, 200_000)))
            if rep > 0:
                api.asap_moe_mailbox_wait(m, int(i), stream=s)
            ep = api.asap_moe_mailbox_post(m, int(i), c.xs[i], outs[i], stream=s)
            srv = servers[int(rng.integers(0, 3))]
            with torch.cuda.stream(srv):
                torch.cuda._sleep(int(rng.integers(0, 200_000)))
            api.asap_moe_mailbox_serve(m, int(i), ep, stream=srv)
        torch.cuda.synchronize()
        for a, b in zip(c.ref, outs):
            assert same_bits(a, b)
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == 3 * n and sum(claimed) == 3 * n
    assert_clean(c.h)
    m.close()


def test_post_routes_match_layer_routes_at_every_slice_count():
    """A post routes with one CTA per tile adding its K slices in turn; the
    layer call routes with a cluster per tile (one CTA per slice).  Sizes
    chosen so the slice count is 4 (1, 33 and 700 tokens), 2 (5000) and 1
    (10000) at H = 2048: every post's output equals asap_moe_layer's bit for
    bit, all five served by one round."""
    cfg = inputs.small_variant(DSV3, name="mbox_slices", hidden=2048, inter=128, shared_inter=128,
                               microbatches=[1, 33, 700, 5000, 10000])
    c = Case.get(cfg)
    n = len(c.xs)
    m = api.asap_moe_mailbox_create(c.h, n, max(cfg.microbatches))
    streams = [torch.cuda.Stream() for _ in range(n)]
    outs = [torch.full_like(x, 9.0) for x in c.xs]
    eps = [api.asap_moe_mailbox_post(m, i, x, o, stream=s) for i, (x, o, s) in enumerate(zip(c.xs, outs, streams))]
    torch.cuda.synchronize()
    for i in range(n):
        api.asap_moe_mailbox_serve(m, i, eps[i])
    torch.cuda.synchronize()
    assert api.asap_moe_mailbox_rounds(m) == (n, [n] + [0] * (n - 1))
    for a, b in zip(c.ref, outs):
        assert same_bits(a, b)
    assert_clean(c.h)
    m.close()


@pytest.mark.parametrize("cfg", [DS, MX], ids=lambda c: c.name)
def test_randomised_posts_sizes_slots_and_streams(cfg):
    """120 posts of random sizes (0, 1, 31-33 around a chunk boundary, up to
    the slot's capacity) into random slots from three producer streams, each
    behind a random GPU sleep, each served at once from one of two server
    streams: every output bit-identical to asap_moe_layer."""
    c = Case.get(cfg)
    rng = np.random.default_rng(321)
    T = max(cfg.microbatches)
    m = api.asap_moe_mailbox_create(c.h, 5, T)
    prods = [torch.cuda.Stream() for _ in range(3)]
    servers = [torch.cuda.Stream() for _ in range(2)]
    inflight = []
    for it in range(120):
        s = int(rng.integers(0, 5))
        n = int(rng.choice([0, 1, 31, 32, 33, int(rng.integers(1, T + 1))]))
        x = inputs.make_tokens(cfg, n, 100 + it, DEV) if n else torch.empty((0, cfg.hidden), dtype=torch.bfloat16,
                                                                            device=DEV)
        ref = torch.empty_like(x)
        if n:
            api.asap_moe_layer(c.h, x, ref, api.workspace(c.h, n))
        out = torch.full_like(x, 3.0)
        p = prods[int(rng.integers(0, 3))]
        with torch.cuda.stream(p):
            torch.cuda._sleep(int(rng.integers(0, 100_000)))
        ep = api.asap_moe_mailbox_post(m, s, x, out, stream=p)
        api.asap_moe_mailbox_serve(m, s, ep, stream=servers[int(rng.integers(0, 2))])
        inflight.append((out, ref))
        if it % 40 == 39:
            torch.cuda.synchronize()
            assert all(same_bits(o, r) for o, r in inflight)
            inflight.clear()
    torch.cuda.synchronize()
    assert all(same_bits(o, r) for o, r in inflight)
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == 120 and sum(claimed) == 120
    assert_clean(c.h)
    m.close()


@pytest.mark.parametrize("cfg", [DS, F8], ids=lambda c: c.name)
def test_serve_many_closed_loop(cfg):
    """Each DP group posts its next micro-batch only once its previous one is
    served (its stream waits for it); one serve_many call per step names the
    step's posts.  Every round serves all of them, the outputs equal
    asap_moe_layer's bit for bit, and bad requests are refused."""
    c = Case.get(cfg)
    n = len(c.xs)
    m = api.asap_moe_mailbox_create(c.h, n, max(cfg.microbatches))
    prods = [torch.cuda.Stream() for _ in range(n)]
    server = torch.cuda.Stream()
    for step in range(3):
        outs = [torch.full_like(x, float(step + 2)) for x in c.xs]
        eps = []
        for i, (x, o, p) in enumerate(zip(c.xs, outs, prods)):
            if step:
                api.asap_moe_mailbox_wait(m, i, stream=p)
            eps.append(api.asap_moe_mailbox_post(m, i, x, o, stream=p))
        api.asap_moe_mailbox_serve_many(m, list(range(n)), eps, stream=server)
        for i, p in enumerate(prods):
            api.asap_moe_mailbox_wait(m, i, stream=p)
        torch.cuda.synchronize()
        for a, b in zip(c.ref, outs):
            assert same_bits(a, b)
    assert api.asap_moe_mailbox_rounds(m) == (3, [n, n, n])
    with pytest.raises(AsapError):
        api.asap_moe_mailbox_serve_many(m, [0, 0], [3, 3])          # a slot listed twice
    with pytest.raises(AsapError):
        api.asap_moe_mailbox_serve_many(m, [0], [4])                 # epoch 4 was never posted
    with pytest.raises(AsapError):
        api.asap_moe_mailbox_serve_many(m, [], [])                   # nothing to serve
    assert_clean(c.h)
    m.close()


def test_repost_keeps_the_previous_tensors_until_their_round_is_done():
    """The binding holds a post's tensors until its slot is posted again.  A
    repost drops the last reference to the previous x while the round that
    reads it may not have run yet (here it starts ~25 ms late); the memory
    must not go to another allocation on the main stream before that round
    is done, so the first post's output still equals asap_moe_layer's."""
    c = Case.get(DS)
    m = api.asap_moe_mailbox_create(c.h, 1, max(DS.microbatches))
    p = torch.cuda.Stream()
    server = torch.cuda.Stream()
    main = torch.cuda.current_stream()
    x0 = c.xs[0]
    o1 = torch.full_like(x0, 3.0)
    o2 = torch.full_like(x0, 4.0)
    tmp = x0.clone()
    p.wait_stream(main)
    ep1 = api.asap_moe_mailbox_post(m, 0, tmp, o1, stream=p)
    del tmp                                   # the mailbox holds the only reference now
    with torch.cuda.stream(server):
        torch.cuda._sleep(50_000_000)
    api.asap_moe_mailbox_serve(m, 0, ep1, stream=server)
    ep2 = api.asap_moe_mailbox_post(m, 0, x0, o2, stream=p)   # drops the previous x
    junk = torch.empty_like(x0)
    junk.fill_(-5.0)
    api.asap_moe_mailbox_serve(m, 0, ep2, stream=server)
    api.asap_moe_mailbox_wait(m, 0, stream=main)
    torch.cuda.synchronize()
    assert same_bits(c.ref[0], o1)
    assert same_bits(c.ref[0], o2)
    assert_clean(c.h)
    m.close()


def test_mailbox_output_against_oracle():
    """The chain to the oracle directly: one round serving three posts of the
    DeepSeek-V3-shaped layer, compared with the float64 layer on the tokens
    whose routing the float32 logits decide."""
    c = Case.get(DS)
    cfg = c.cfg
    m = api.asap_moe_mailbox_create(c.h, 3, max(cfg.microbatches))
    outs = [torch.empty_like(x) for x in c.xs[:3]]
    eps = [api.asap_moe_mailbox_post(m, i, c.xs[i], outs[i]) for i in range(3)]
    api.asap_moe_mailbox_serve(m, 2, eps[2])
    torch.cuda.synchronize()
    assert api.asap_moe_mailbox_rounds(m) == (1, [3])
    wf = {k: bf16_to_f64(c.w[k]) for k in ("router_w", "w_gate", "w_up", "w_down", "sh_gate", "sh_up", "sh_down")}
    ocfg = cfg.oracle_cfg()
    for x, o in zip(c.xs[:3], outs):
        xf = bf16_to_f64(x)
        r = oracle.moe_layer(xf, wf["router_w"], wf["w_gate"], wf["w_up"], wf["w_down"], ocfg,
                             shared=(wf["sh_gate"], wf["sh_up"], wf["sh_down"]))
        eps_l = oracle.logit_error_bound(xf, wf["router_w"])
        keep = np.array([oracle.token_decided(r["logits"][t], eps_l[t], ocfg) for t in range(x.shape[0])])
        compare_rows(bf16_to_f64(o)[keep], r["y"][keep])
    assert_clean(c.h)
    m.close()


def test_round_for_a_post_never_made_times_out_and_serves_the_rest():
    """A serve call for a post that nothing publishes (epoch 1 of an unused
    slot): the round's wait runs out after wait_ns, records status bit 128,
    and the round still serves the post that is ready."""
    c = Case.get(DS)
    m = api.asap_moe_mailbox_create(c.h, 2, max(DS.microbatches), wait_ns=20_000_000)
    out = torch.empty_like(c.xs[0])
    ep = api.asap_moe_mailbox_post(m, 0, c.xs[0], out)
    torch.cuda.synchronize()
    api.asap_moe_mailbox_serve(m, 1, 1)          # slot 1 is never posted
    torch.cuda.synchronize()
    assert same_bits(c.ref[0], out)
    assert api.asap_moe_mailbox_served(m, 0) == ep and api.asap_moe_mailbox_served(m, 1) == 0
    word = assert_clean(c.h, allowed=ST_MBOX_WAIT)
    assert word == ST_MBOX_WAIT
    # the mailbox is still usable: slot 0 again, then its own round
    api.asap_moe_mailbox_serve(m, 0, ep)
    out2 = torch.empty_like(c.xs[1])
    ep2 = api.asap_moe_mailbox_post(m, 0, c.xs[1], out2)
    api.asap_moe_mailbox_serve(m, 0, ep2)
    torch.cuda.synchronize()
    assert same_bits(c.ref[1], out2)
    assert api.asap_moe_mailbox_rounds(m) == (3, [1, 0, 1])
    assert_clean(c.h)
    m.close()


def test_host_side_rules():
    c = Case.get(DS)
    m = api.asap_moe_mailbox_create(c.h, 2, 1000)
    out = torch.empty_like(c.xs[0])
    ep = api.asap_moe_mailbox_post(m, 0, c.xs[0], out)
    with pytest.raises(AsapError, match="no serve call"):
        api.asap_moe_mailbox_post(m, 0, c.xs[0], out)          # backpressure: not served yet
    with pytest.raises(AsapError, match="no serve call"):
        api.asap_moe_mailbox_wait(m, 0)
    with pytest.raises(AsapError, match="slot outside"):
        api.asap_moe_mailbox_post(m, 2, c.xs[0], out)
    big = inputs.make_tokens(DS, 1001, 9, DEV)
    with pytest.raises(AsapError, match="slot_tokens"):
        api.asap_moe_mailbox_post(m, 1, big, torch.empty_like(big))
    api.asap_moe_mailbox_serve(m, 0, ep)
    api.asap_moe_mailbox_wait(m, 0)
    torch.cuda.synchronize()
    assert same_bits(c.ref[0], out)
    empty = torch.empty((0, DS.hidden), dtype=torch.bfloat16, device=DEV)
    ep0 = api.asap_moe_mailbox_post(m, 1, empty, empty)        # an empty post is served too
    api.asap_moe_mailbox_serve(m, 1, ep0)
    torch.cuda.synchronize()
    assert api.asap_moe_mailbox_served(m, 1) == ep0
    with pytest.raises(AsapError, match="n_slots"):
        api.asap_moe_mailbox_create(c.h, 65, 100)
    assert_clean(c.h)
    m.close()


def test_handle_outlives_its_mailboxes():
    """Destroying a handle while a mailbox created on it is open is refused
    (the mailbox uses the handle's weights and device); once the mailboxes
    are closed the handle is freed."""
    cfg = inputs.small_variant(DS, name="mbox_owner", microbatches=[64])
    h = api.asap_moe_create(cfg, inputs.make_weights(cfg, DEV), 64)
    m1 = api.asap_moe_mailbox_create(h, 1, 64)
    m2 = api.asap_moe_mailbox_create(h, 1, 64)
    with pytest.raises(AsapError, match="2 mailbox"):
        h.close()
    m1.close()
    with pytest.raises(AsapError, match="1 mailbox"):
        h.close()
    x = inputs.make_tokens(cfg, 64, 5, DEV)
    out = torch.empty_like(x)
    ref = torch.empty_like(x)
    ep = api.asap_moe_mailbox_post(m2, 0, x, out)              # the handle still works
    api.asap_moe_mailbox_serve(m2, 0, ep)
    api.asap_moe_layer(h, x, ref, api.workspace(h, 64))
    torch.cuda.synchronize()
    assert same_bits(ref, out)
    m2.close()
    h.close()
    assert h.ptr is None


def test_one_mailbox_serves_interleaved_layers():
    """Posts of two layers of one handle interleaved in the slots: each round
    claims only the ready posts of its own post's layer and runs that
    layer's weights; every output equals a single-layer handle's."""
    cfg = inputs.small_variant(DSV3, name="mbox_2layers", hidden=512, inter=256, shared_inter=256,
                               microbatches=[300, 77, 129, 200])
    ws = inputs.make_layer_weights(cfg, 2, DEV)
    h = api.asap_moe_create_layers(cfg, ws, 300)
    single = [api.asap_moe_create(inputs.layer_config(cfg, l), ws[l], 300) for l in range(2)]
    ids = [torch.tensor([l], dtype=torch.int32, device=DEV) for l in range(2)]
    layers = [0, 1, 0, 1]
    m = api.asap_moe_mailbox_create(h, 4, 300)
    xs = inputs.make_microbatches(cfg, DEV)
    outs = [torch.empty_like(x) for x in xs]
    eps = [api.asap_moe_mailbox_post(m, i, x, o, layer_id=ids[l])
           for i, (x, o, l) in enumerate(zip(xs, outs, layers))]
    torch.cuda.synchronize()
    for i in (1, 0, 3, 2):                  # a layer-1 post first
        api.asap_moe_mailbox_serve(m, i, eps[i])
    torch.cuda.synchronize()
    assert api.asap_moe_mailbox_rounds(m) == (4, [2, 2, 0, 0])
    for x, o, l in zip(xs, outs, layers):
        ref = torch.empty_like(x)
        api.asap_moe_layer(single[l], x, ref, api.workspace(single[l], x.shape[0]))
        torch.cuda.synchronize()
        assert same_bits(ref, o)
    assert_clean(h)
    m.close()
    h.close()
    for one in single:
        one.close()


def test_mailbox_on_a_layer_of_a_multi_layer_handle():
    cfg = inputs.small_variant(DSV3, name="mbox_layers", hidden=512, inter=256, shared_inter=256,
                               microbatches=[300, 77])
    ws = inputs.make_layer_weights(cfg, 2, DEV)
    h = api.asap_moe_create_layers(cfg, ws, 300)
    one = api.asap_moe_create(inputs.layer_config(cfg, 1), ws[1], 300)
    lid = torch.tensor([1], dtype=torch.int32, device=DEV)
    m = api.asap_moe_mailbox_create(h, 2, 300, layer_id=lid)
    xs = inputs.make_microbatches(cfg, DEV)
    outs = [torch.empty_like(x) for x in xs]
    eps = [api.asap_moe_mailbox_post(m, i, x, o) for i, (x, o) in enumerate(zip(xs, outs))]
    api.asap_moe_mailbox_serve(m, 0, eps[0])
    api.asap_moe_mailbox_serve(m, 1, eps[1])
    for x, o in zip(xs, outs):
        ref = torch.empty_like(x)
        api.asap_moe_layer(one, x, ref, api.workspace(one, x.shape[0]))
        torch.cuda.synchronize()
        assert same_bits(ref, o)
    assert_clean(h)
    m.close()
    h.close()
    one.close()


@pytest.mark.parametrize("cfg", [DSV3, STRESS, MIXTRAL], ids=lambda c: c.name)
def test_mailbox_full_size(cfg):
    """The bench's workloads at full size (DeepSeek-V3 4 x 4096; the stress
    workload's 8 ragged micro-batches of 362 to 8045 tokens with Zipf
    experts; Mixtral's 4 micro-batches), each posted from its own stream,
    every post served right after it on one MoE stream, twice (the second
    time the slots are reposted): every output bit-identical to
    asap_moe_layer on the same micro-batch."""
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, max(cfg.microbatches))
    del w
    torch.cuda.empty_cache()
    xs = inputs.make_microbatches(cfg, DEV)
    ref = []
    ws = api.workspace(h, max(cfg.microbatches))
    for x in xs:
        o = torch.empty_like(x)
        api.asap_moe_layer(h, x, o, ws)
        ref.append(o)
    torch.cuda.synchronize()
    del ws
    m = api.asap_moe_mailbox_create(h, len(xs), max(cfg.microbatches))
    producers = [torch.cuda.Stream() for _ in xs]
    server = torch.cuda.Stream()
    for rep in range(2):
        outs = [torch.full_like(x, 5.0) for x in xs]
        eps = [api.asap_moe_mailbox_post(m, i, x, o, stream=p)
               for i, (x, o, p) in enumerate(zip(xs, outs, producers))]
        for i, ep in enumerate(eps):
            api.asap_moe_mailbox_serve(m, i, ep, stream=server)
        torch.cuda.synchronize()
        for a, b in zip(ref, outs):
            assert same_bits(a, b)
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == 2 * len(xs) and sum(claimed) == 2 * len(xs)
    print(f"[{cfg.name} full size] posts per round: {claimed}")
    assert_clean(h)
    m.close()
    h.close()


def test_posts_and_rounds_from_host_threads():
    """One host thread per DP group posting on its own stream and a server
    thread serving each post as it learns of it (through a queue): the
    mailbox's host state is shared between threads behind its lock; every
    output still equals asap_moe_layer's."""
    import queue
    import threading
    c = Case.get(DS)
    n = len(c.xs)
    m = api.asap_moe_mailbox_create(c.h, n, max(DS.microbatches))
    outs = [[torch.full_like(x, 9.0) for x in c.xs] for _ in range(2)]
    q = queue.Queue()
    errors = []

    def producer(i):
        try:
            s = torch.cuda.Stream()
            for rep in range(2):
                if rep:
                    done[i].wait(timeout=30)
                    api.asap_moe_mailbox_wait(m, i, stream=s)
                q.put((i, api.asap_moe_mailbox_post(m, i, c.xs[i], outs[rep][i], stream=s)))
        except Exception as e:   # reported by the main thread
            errors.append(e)

    done = [threading.Event() for _ in range(n)]
    server = torch.cuda.Stream()
    threads = [threading.Thread(target=producer, args=(i,)) for i in range(n)]
    for t in threads:
        t.start()
    for _ in range(2 * n):
        i, ep = q.get(timeout=60)
        api.asap_moe_mailbox_serve(m, i, ep, stream=server)
        done[i].set()
    for t in threads:
        t.join(timeout=60)
    torch.cuda.synchronize()
    assert not errors, errors
    for rep in range(2):
        for a, b in zip(c.ref, outs[rep]):
            assert same_bits(a, b)
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == 2 * n and sum(claimed) == 2 * n
    assert_clean(c.h)
    m.close()


def test_mailbox_full_size_fp8():
    """The FP8 workload (8 x 4096 tokens, Zipf popularity) posted from eight
    streams, every post served right after it: each output bit-identical to
    asap_moe_layer's on the same micro-batch."""
    cfg = DSV3_FP8
    w = inputs.make_weights(cfg, DEV)
    h = api.asap_moe_create(cfg, w, max(cfg.microbatches))
    del w
    torch.cuda.empty_cache()
    xs = inputs.make_microbatches(cfg, DEV)
    ws = api.workspace(h, max(cfg.microbatches))
    ref = []
    for x in xs:
        o = torch.empty_like(x)
        api.asap_moe_layer(h, x, o, ws)
        ref.append(o)
    torch.cuda.synchronize()
    del ws
    m = api.asap_moe_mailbox_create(h, len(xs), max(cfg.microbatches))
    producers = [torch.cuda.Stream() for _ in xs]
    server = torch.cuda.Stream()
    outs = [torch.full_like(x, 5.0) for x in xs]
    eps = [api.asap_moe_mailbox_post(m, i, x, o, stream=p) for i, (x, o, p) in enumerate(zip(xs, outs, producers))]
    for i, ep in enumerate(eps):
        api.asap_moe_mailbox_serve(m, i, ep, stream=server)
    torch.cuda.synchronize()
    for a, b in zip(ref, outs):
        assert same_bits(a, b)
    rounds, claimed = api.asap_moe_mailbox_rounds(m)
    assert rounds == len(xs) and sum(claimed) == len(xs)
    print(f"[fp8 full size] posts per round: {claimed}")
    assert_clean(h)
    m.close()
    h.close()
