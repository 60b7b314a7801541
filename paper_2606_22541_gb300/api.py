"""Python binding of the C ABI, one function per entry point with the same name.

Tensors are torch CUDA tensors (the binding passes their device pointers);
``stream`` is a torch.cuda.Stream or None for the current stream.  Every step
of the layer runs in libasap_moe's kernels; nothing here computes.
"""
import ctypes
import threading

import torch

from . import _native
from ._native import AsapMoeConfig, AsapMoeWeights, check, lib
from .configs import GATING, DTYPE


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


# this thread's pending asap_moe_time_layer events (kept alive for the C side)
_timing = threading.local()


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def make_config(cfg, max_tokens):
    """C config from a configs.LayerConfig."""
    return AsapMoeConfig(hidden=cfg.hidden, n_experts=cfg.n_experts, top_k=cfg.top_k, inter=cfg.inter,
                         n_shared=cfg.n_shared, shared_inter=cfg.shared_inter, gating=GATING[cfg.gating],
                         n_groups=cfg.n_groups, topk_groups=cfg.topk_groups,
                         route_scale=float(cfg.route_scale), dtype=DTYPE[cfg.dtype],
                         max_tokens=int(max_tokens))


class Handle:
    """Owns an asap_moe_t; destroyed on close() or garbage collection."""

    def __init__(self, ptr, cfg, ccfg):
        self.ptr = ptr
        self.cfg = cfg
        self.ccfg = ccfg

    @property
    def max_tokens(self):
        return self.ccfg.max_tokens

    def close(self):
        """Frees the handle; raises AsapError (and keeps it) while a mailbox
        created on it is open."""
        if self.ptr:
            check("asap_moe_destroy", lib().asap_moe_destroy(self.ptr))
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def asap_moe_check_config(cfg, max_tokens=1):
    c = make_config(cfg, max_tokens)
    return lib().asap_moe_check_config(ctypes.byref(c))


def _weights_struct(weights, w):
    for name, _ in AsapMoeWeights._fields_:
        t = weights.get(name)
        setattr(w, name, None if t is None else t.data_ptr())


def asap_moe_create(cfg, weights, max_tokens):
    """weights: dict of CUDA tensors named like asap_moe_weights' fields."""
    c = make_config(cfg, max_tokens)
    w = AsapMoeWeights()
    _weights_struct(weights, w)
    out = ctypes.c_void_p()
    check("asap_moe_create", lib().asap_moe_create(ctypes.byref(c), ctypes.byref(w), ctypes.byref(out)))
    return Handle(out, cfg, c)


def asap_moe_create_layers(cfg, layers, max_tokens):
    """One handle over several layers of the same shape; layers: a list of
    weight dicts, one per layer (layer l = layers[l])."""
    c = make_config(cfg, max_tokens)
    ws = (AsapMoeWeights * len(layers))()
    for i, weights in enumerate(layers):
        _weights_struct(weights, ws[i])
    out = ctypes.c_void_p()
    check("asap_moe_create_layers", lib().asap_moe_create_layers(ctypes.byref(c), ws, len(layers), ctypes.byref(out)))
    return Handle(out, cfg, c)


def asap_moe_n_layers(h):
    out = ctypes.c_int32()
    check("asap_moe_n_layers", lib().asap_moe_n_layers(h.ptr, ctypes.byref(out)))
    return out.value


def asap_moe_destroy(h):
    h.close()


def asap_moe_workspace_size(cfg, n_tokens, max_tokens=None):
    c = make_config(cfg, max_tokens if max_tokens is not None else max(n_tokens, 1))
    out = ctypes.c_size_t()
    check("asap_moe_workspace_size", lib().asap_moe_workspace_size(ctypes.byref(c), int(n_tokens), ctypes.byref(out)))
    return out.value


def workspace(h, n_tokens, device="cuda"):
    """A workspace tensor large enough for one call with n_tokens tokens."""
    nbytes = asap_moe_workspace_size(h.cfg, n_tokens, h.max_tokens)
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)


def _ws(ws):
    return (_ptr(ws), ctypes.c_size_t(0 if ws is None else ws.numel() * ws.element_size()))


def asap_moe_router_logits(h, x, logits, ws, stream=None):
    p, n = _ws(ws)
    check("asap_moe_router_logits",
          lib().asap_moe_router_logits(h.ptr, _ptr(x), x.shape[0], _ptr(logits), p, n, _stream(stream)))


def asap_moe_route(h, x, idx, w, counts, offsets, ws, stream=None):
    p, n = _ws(ws)
    check("asap_moe_route", lib().asap_moe_route(h.ptr, _ptr(x), x.shape[0], _ptr(idx), _ptr(w), _ptr(counts),
                                                 _ptr(offsets), p, n, _stream(stream)))


def asap_moe_route_logits(h, logits, idx, w, counts, offsets, ws, stream=None):
    p, n = _ws(ws)
    check("asap_moe_route_logits",
          lib().asap_moe_route_logits(h.ptr, _ptr(logits), logits.shape[0], _ptr(idx), _ptr(w), _ptr(counts),
                                      _ptr(offsets), p, n, _stream(stream)))


def asap_moe_dispatch(h, x, idx, x_perm, perm_src, perm_dst, ws, stream=None, x_perm_scales=None):
    p, n = _ws(ws)
    check("asap_moe_dispatch",
          lib().asap_moe_dispatch(h.ptr, _ptr(x), x.shape[0], _ptr(idx), _ptr(x_perm), _ptr(x_perm_scales),
                                  _ptr(perm_src), _ptr(perm_dst), p, n, _stream(stream)))


def asap_moe_expert_ffn(h, x_perm, offsets, x, y_perm, y_shared, ws, stream=None, x_perm_scales=None):
    p, n = _ws(ws)
    check("asap_moe_expert_ffn",
          lib().asap_moe_expert_ffn(h.ptr, _ptr(x_perm), _ptr(x_perm_scales), _ptr(offsets), _ptr(x),
                                    x.shape[0], _ptr(y_perm), _ptr(y_shared), p, n, _stream(stream)))


def asap_moe_expert_gate_up(h, x_perm, offsets, x, h_perm, h_shared, stream=None, x_perm_scales=None, ws=None):
    """ws (optional): a workspace for x.shape[0] tokens; with it the GEMM claims
    its tiles dynamically."""
    p, nb = _ws(ws)
    check("asap_moe_expert_gate_up",
          lib().asap_moe_expert_gate_up(h.ptr, _ptr(x_perm), _ptr(x_perm_scales), _ptr(offsets), _ptr(x),
                                        x.shape[0], _ptr(h_perm), _ptr(h_shared), p, nb, _stream(stream)))


def asap_moe_expert_down(h, h_perm, offsets, h_shared, n, y_perm, y_shared, stream=None, h_perm_scales=None,
                         ws=None):
    p, nb = _ws(ws)
    check("asap_moe_expert_down",
          lib().asap_moe_expert_down(h.ptr, _ptr(h_perm), _ptr(h_perm_scales), _ptr(offsets), _ptr(h_shared),
                                     int(n), _ptr(y_perm), _ptr(y_shared), p, nb, _stream(stream)))


def asap_moe_combine(h, y_perm, y_shared, w, perm_dst, out, stream=None):
    check("asap_moe_combine", lib().asap_moe_combine(h.ptr, _ptr(y_perm), _ptr(y_shared), _ptr(w), _ptr(perm_dst),
                                                     out.shape[0], _ptr(out), _stream(stream)))


def asap_moe_layer(h, x, out, ws, stream=None):
    p, n = _ws(ws)
    try:
        check("asap_moe_layer", lib().asap_moe_layer(h.ptr, _ptr(x), x.shape[0], _ptr(out), p, n, _stream(stream)))
    finally:
        _timing.events = None   # the call has taken this thread's timing request


def asap_moe_layer_batched(h, xs, outs, ws, stream=None):
    """Serve several ready micro-batches in one pass (one grouped GEMM per
    weight matrix); outs[i] equals asap_moe_layer on xs[i] bit for bit."""
    cnt = len(xs)
    xa = (ctypes.c_void_p * cnt)(*[x.data_ptr() for x in xs])
    na = (ctypes.c_int32 * cnt)(*[x.shape[0] for x in xs])
    oa = (ctypes.c_void_p * cnt)(*[o.data_ptr() for o in outs])
    p, n = _ws(ws)
    check("asap_moe_layer_batched",
          lib().asap_moe_layer_batched(h.ptr, cnt, xa, na, oa, p, n, _stream(stream)))


def asap_moe_layer_dyn(h, layer_id, x, out, ws, stream=None):
    """asap_moe_layer for the layer whose id the kernels read from layer_id
    (a one-element int32 CUDA tensor) when they run."""
    p, n = _ws(ws)
    try:
        check("asap_moe_layer_dyn", lib().asap_moe_layer_dyn(h.ptr, _ptr(layer_id), _ptr(x), x.shape[0], _ptr(out), p,
                                                             n, _stream(stream)))
    finally:
        _timing.events = None   # the call has taken this thread's timing request


def asap_moe_layer_batched_dyn(h, layer_id, xs, outs, ws, stream=None):
    """asap_moe_layer_batched for micro-batches of the layer at layer_id."""
    cnt = len(xs)
    xa = (ctypes.c_void_p * cnt)(*[x.data_ptr() for x in xs])
    na = (ctypes.c_int32 * cnt)(*[x.shape[0] for x in xs])
    oa = (ctypes.c_void_p * cnt)(*[o.data_ptr() for o in outs])
    p, n = _ws(ws)
    check("asap_moe_layer_batched_dyn",
          lib().asap_moe_layer_batched_dyn(h.ptr, _ptr(layer_id), cnt, xa, na, oa, p, n, _stream(stream)))


def asap_moe_time_layer(events):
    """Events (torch.cuda.Event, enable_timing=True; up to 6) for this
    thread's next asap_moe_layer / _dyn call to record: before its first
    kernel and after route, dispatch, gate/up, down and combine."""
    events = list(events)
    for ev in events:
        if ev.cuda_event == 0:   # torch creates the CUDA event at its first record
            ev.record()
    arr = (ctypes.c_void_p * max(1, len(events)))(*[ev.cuda_event for ev in events])
    check("asap_moe_time_layer", lib().asap_moe_time_layer(len(events), arr))
    _timing.events = events     # alive until the layer call that records them returns


def asap_moe_route_noalloc(h, x, idx, w, counts, offsets, stream=None):
    """asap_moe_route with its scratch in the library's static device array
    (at most 4096 tokens; calls overlapping on the GPU race)."""
    check("asap_moe_route_noalloc",
          lib().asap_moe_route_noalloc(h.ptr, _ptr(x), x.shape[0], _ptr(idx), _ptr(w), _ptr(counts),
                                       _ptr(offsets), _stream(stream)))


class Mailbox:
    """Owns an asap_moe_mailbox_t (slots that DP-group streams post routed
    micro-batches into and that service rounds on the MoE stream claim on the
    device); destroyed on close() or garbage collection.  Keeps the tensors
    of every post alive until the mailbox is closed or the slot is reposted."""

    def __init__(self, ptr, handle, n_slots, slot_tokens):
        self.ptr = ptr
        self.handle = handle          # the weights must outlive the mailbox
        self.n_slots = n_slots
        self.slot_tokens = slot_tokens
        self._keep = {}

    def close(self):
        if self.ptr:
            lib().asap_moe_mailbox_destroy(self.ptr)
            self.ptr = None
            self._keep.clear()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def asap_moe_mailbox_create(h, n_slots, slot_tokens, layer_id=None, wait_ns=2_000_000_000):
    """A mailbox of n_slots slots of up to slot_tokens tokens on h (layer_id:
    None for layer 0, or a one-element int32 CUDA tensor)."""
    out = ctypes.c_void_p()
    check("asap_moe_mailbox_create",
          lib().asap_moe_mailbox_create(h.ptr, int(n_slots), int(slot_tokens), _ptr(layer_id), int(wait_ns),
                                        ctypes.byref(out)))
    m = Mailbox(out, h, n_slots, slot_tokens)
    m._layer = layer_id
    return m


def asap_moe_mailbox_post(m, slot, x, out, stream=None, layer_id=None):
    """Post x (n tokens) into slot; returns the post's epoch.  layer_id: None
    (the mailbox's default layer) or a one-element int32 CUDA tensor.  The
    mailbox keeps x, out and layer_id alive until the slot is posted again or
    the mailbox is closed."""
    s = torch.cuda.current_stream() if stream is None else stream
    ep = ctypes.c_uint64()
    check("asap_moe_mailbox_post",
          lib().asap_moe_mailbox_post(m.ptr, int(slot), _ptr(x), x.shape[0], _ptr(out), _ptr(layer_id),
                                      _stream(s), ctypes.byref(ep)))
    old = m._keep.get(int(slot))
    if old is not None:
        # The post just enqueued on s waits for the round that served the
        # slot's previous post, so once s reaches this point that round is
        # done with the previous tensors.  Recording s on them keeps the
        # caching allocator from handing their memory to another stream
        # before then, even when this reference was the last one.
        for t in old:
            if t is not None:
                t.record_stream(s)
    m._keep[int(slot)] = (x, out, layer_id)
    return ep.value


def asap_moe_mailbox_serve(m, slot, epoch, stream=None):
    try:
        check("asap_moe_mailbox_serve", lib().asap_moe_mailbox_serve(m.ptr, int(slot), int(epoch), _stream(stream)))
    finally:
        m._timing = None


def asap_moe_mailbox_serve_many(m, slots, epochs, stream=None):
    """One service round for the posts (slots[i], epochs[i]) already made."""
    n = len(slots)
    cs = (ctypes.c_int32 * n)(*[int(v) for v in slots])
    ce = (ctypes.c_uint64 * n)(*[int(v) for v in epochs])
    try:
        check("asap_moe_mailbox_serve_many", lib().asap_moe_mailbox_serve_many(m.ptr, n, cs, ce, _stream(stream)))
    finally:
        m._timing = None


def asap_moe_mailbox_wait(m, slot, stream=None):
    check("asap_moe_mailbox_wait", lib().asap_moe_mailbox_wait(m.ptr, int(slot), _stream(stream)))


def asap_moe_mailbox_served(m, slot):
    ep = ctypes.c_uint64()
    check("asap_moe_mailbox_served", lib().asap_moe_mailbox_served(m.ptr, int(slot), ctypes.byref(ep)))
    return ep.value


def asap_moe_mailbox_time_gemms(m, ev_before, ev_after):
    """torch.cuda.Event pair (enable_timing=True) recorded around the next
    serve call's GEMMs."""
    for ev in (ev_before, ev_after):
        if ev.cuda_event == 0:   # torch creates the CUDA event at its first record
            ev.record()
    check("asap_moe_mailbox_time_gemms",
          lib().asap_moe_mailbox_time_gemms(m.ptr, ctypes.c_void_p(ev_before.cuda_event),
                                            ctypes.c_void_p(ev_after.cuda_event)))
    m._timing = (ev_before, ev_after)   # alive until the serve call that records them returns


def asap_moe_mailbox_rounds(m, cap=4096):
    """(rounds run so far, list of the posts each round claimed); synchronises."""
    n = ctypes.c_int32()
    buf = (ctypes.c_int32 * cap)()
    check("asap_moe_mailbox_rounds", lib().asap_moe_mailbox_rounds(m.ptr, ctypes.byref(n), buf, cap))
    return n.value, list(buf[:min(cap, n.value)])


COMBINE_SEPARATE, COMBINE_FUSED = 0, 1


def asap_moe_set_combine(h, mode):
    """Where asap_moe_layer combines on a bf16 handle: COMBINE_SEPARATE (a
    kernel after the down GEMM, the default) or COMBINE_FUSED (inside the down
    GEMM); bit-identical outputs."""
    check("asap_moe_set_combine", lib().asap_moe_set_combine(h.ptr, int(mode)))


TILING_AUTO, TILING_SINGLE, TILING_PAIRED = 0, 1, 2


def asap_moe_set_tiling(h, mode):
    """Tile shape of the BF16 grouped expert GEMMs: TILING_AUTO, _SINGLE or
    _PAIRED (bit-identical results; only the speed differs)."""
    check("asap_moe_set_tiling", lib().asap_moe_set_tiling(h.ptr, int(mode)))


def asap_moe_status(h):
    """(code, raw status word); code is ASAP_OK or ASAP_ERR_DEVICE_STATUS."""
    word = ctypes.c_uint32()
    code = lib().asap_moe_status(h.ptr, ctypes.byref(word))
    return code, word.value


def asap_moe_last_error():
    return lib().asap_moe_last_error().decode(errors="replace")
