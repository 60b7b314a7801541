"""Cost of resolving the layer id on the host, against layer-oblivious calls
enqueued ahead of time (bubble-free kernel dispatching, Section 3.4.2).

    python -m paper_2606_22541_gb300.dispatch_bubble [--workload dsv3_bf16] [--layers 3]
        [--tokens 4096] [--microbatches 24]

A producer stream stands in for the attention DP groups: micro-batch i
arrives when a producer kernel has landed its hidden states and written its
layer id (drawn at random from the layers) into device memory, event a_i.
Arrivals are spaced wider than one MoE layer, so every arrival finds the MoE
stream idle and any dispatch delay lies on the critical path.  The MoE side
serves the arrivals in order in one of three modes:

  host    the host waits for a_i, reads the layer id back, then enqueues the
          layer's kernels (asap_moe_layer_dyn with a fixed id): what a kernel
          that takes its layer as a launch argument requires;
  ahead   every call is enqueued before the first arrival, behind a stream
          wait on a_i, with the id slot of micro-batch i: the kernels read the
          layer when they run (asap_moe_layer_dyn);
  graph   as ahead, but each call is one replay of a CUDA graph captured once
          per micro-batch buffer.

Per mode: latency from arrival to completion, and from arrival to the start
of the layer's first kernel (the bubble), mean over the micro-batches; plus
the host time to enqueue one call.  One JSON line per mode.
"""
import argparse
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="dsv3_bf16")
    ap.add_argument("--layers", type=int, default=3)
    ap.add_argument("--tokens", type=int, default=4096)
    ap.add_argument("--microbatches", type=int, default=24)
    ap.add_argument("--gap-ms", type=float, default=0.0, help="arrival spacing (0: 1.5 x one layer + 1 ms)")
    ap.add_argument("--seed", type=int, default=11)
    args = ap.parse_args()

    import numpy as np
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_22541_gb300 import api, inputs
    from paper_2606_22541_gb300.configs import CONFIGS

    cfg = CONFIGS[args.workload]
    dev = "cuda"
    n, M, NL = args.tokens, args.microbatches, args.layers
    ws_layers = inputs.make_layer_weights(cfg, NL, dev)
    h = api.asap_moe_create_layers(cfg, ws_layers, n)
    del ws_layers
    torch.cuda.empty_cache()
    order = np.random.default_rng(args.seed).integers(0, NL, M).astype(np.int32)
    fixed_ids = torch.arange(NL, dtype=torch.int32, device=dev)
    staged = [inputs.make_tokens(cfg, n, i % 4, dev) for i in range(4)]     # payloads the producer lands
    xs = [torch.empty_like(staged[0]) for _ in range(M)]
    outs = [torch.empty_like(staged[0]) for _ in range(M)]
    wss = [api.workspace(h, n) for _ in range(M)]
    sched = torch.tensor(order, device=dev)
    producer = torch.cuda.Stream()
    moe = torch.cuda.Stream()

    # one layer's time, for the arrival spacing
    slot = torch.zeros(1, dtype=torch.int32, device=dev)
    for _ in range(3):
        api.asap_moe_layer_dyn(h, slot, staged[0], outs[0], wss[0])
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    api.asap_moe_layer_dyn(h, slot, staged[0], outs[0], wss[0])
    e1.record()
    torch.cuda.synchronize()
    layer_ms = e0.elapsed_time(e1)
    gap_ms = args.gap_ms or (1.5 * layer_ms + 1.0)
    # torch.cuda._sleep counts SM cycles; calibrate them against events
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0.record()
    torch.cuda._sleep(10_000_000)
    c1.record()
    torch.cuda.synchronize()
    cycles_per_ms = 10_000_000 / c0.elapsed_time(c1)

    graphs = None

    def run(mode):
        nonlocal graphs
        slots = torch.full((M,), -1, dtype=torch.int32, device=dev)
        arrive = [torch.cuda.Event(enable_timing=True) for _ in range(M)]
        start = [torch.cuda.Event(enable_timing=True) for _ in range(M)]
        done = [torch.cuda.Event(enable_timing=True) for _ in range(M)]
        if mode == "graph" and graphs is None:
            graphs = []
            for i in range(M):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=moe):
                    api.asap_moe_layer_dyn(h, slots_g[i:i + 1], xs[i], outs[i], wss[i])
                graphs.append(g)
        slot_t = slots_g if mode == "graph" else slots
        torch.cuda.synchronize()
        # producer: arrivals every gap_ms, the first one after the host has had
        # time to enqueue everything
        with torch.cuda.stream(producer):
            torch.cuda._sleep(int(40 * cycles_per_ms))
            for i in range(M):
                torch.cuda._sleep(int(gap_ms * cycles_per_ms))
                xs[i].copy_(staged[i % 4])
                slot_t[i:i + 1].copy_(sched[i:i + 1])
                arrive[i].record(producer)
        t_enq = time.perf_counter()
        if mode == "host":
            n_enq = 0.0
            for i in range(M):
                arrive[i].synchronize()
                layer = int(slot_t[i].item())                 # the host resolves the layer
                t0 = time.perf_counter()
                start[i].record(moe)
                api.asap_moe_layer_dyn(h, fixed_ids[layer:layer + 1], xs[i], outs[i], wss[i], stream=moe)
                done[i].record(moe)
                n_enq += time.perf_counter() - t0
            enq_us = n_enq / M * 1e6
        else:
            for i in range(M):
                moe.wait_event(arrive[i])
                start[i].record(moe)
                if mode == "graph":
                    with torch.cuda.stream(moe):
                        graphs[i].replay()
                else:
                    api.asap_moe_layer_dyn(h, slot_t[i:i + 1], xs[i], outs[i], wss[i], stream=moe)
                done[i].record(moe)
            enq_us = (time.perf_counter() - t_enq) / M * 1e6
        torch.cuda.synchronize()
        lat = np.array([arrive[i].elapsed_time(done[i]) for i in range(M)])
        bub = np.array([arrive[i].elapsed_time(start[i]) for i in range(M)])
        # in host mode the start event is recorded by the host after the read
        # back, so it marks when the stream could first begin the layer
        res = [o.clone() for o in outs]
        return dict(latency_ms=float(lat.mean()), start_delay_us=float(bub.mean() * 1e3),
                    start_delay_max_us=float(bub.max() * 1e3), enqueue_us_per_call=enq_us), res

    slots_g = torch.full((M,), -1, dtype=torch.int32, device=dev)
    results = {}
    for mode in ("host", "ahead", "graph", "host", "ahead", "graph"):
        r, outs_mode = run(mode)
        results.setdefault(mode, []).append(r)
        if mode == "host":
            ref = outs_mode
        else:
            same = all(torch.equal(a.view(torch.int16), b.view(torch.int16)) for a, b in zip(ref, outs_mode))
            if not same:
                raise RuntimeError(f"{mode} outputs differ from the host-dispatched ones")
    code, word = api.asap_moe_status(h)
    if code != 0:
        raise RuntimeError(f"device status word {word:#x}")
    for mode, rs in results.items():
        r = rs[-1]
        print(json.dumps({"mode": mode, "workload": cfg.name, "layers": NL, "tokens": n, "microbatches": M,
                          "layer_ms": layer_ms, "gap_ms": gap_ms, **r}), flush=True)
    h.close()


if __name__ == "__main__":
    main()
