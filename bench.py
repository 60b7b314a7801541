#!/usr/bin/env python
"""Throughput of the expert-side MoE layer on one GB300 (and N replicas).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Workload (default): the DeepSeek-V3-shaped BF16 MoE layer of the paper's
evaluation model (ASAP Table 1 and Section 5.1: H = 7168, 256 routed experts
plus 1 shared, top-8; intermediate 2048), 16384 tokens per step as 4
micro-batches of 4096 tokens, each submitted through asap_moe_layer on its
own CUDA stream with no host barrier between them (Section 3.4.2).  Inputs
are seeded synthetic tensors; 22.6 GB of expert weights make every step's
working set far larger than the 129 MB L2.

One JSON line on rank 0: tokens/s over the timed steps, plus the roofline of
the dominant kernel (the gate/up grouped GEMM), per-kernel timings measured
with CUDA events on the stream each kernel runs on, the float64 oracle timed
on the host cores on a bounded sample, the end-to-end figure through host
buffers, and the SM clocks sampled during the timed region.

``--impl reference`` times the float64 oracle instead (host cores, bounded
sample per step) on the same workload and metric.
"""
import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "MoE-layer prefill tokens/s on 1 GB300; grouped-GEMM % of tensor peak"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="dsv3_bf16")
    ap.add_argument("--kernel-steps", type=int, default=3)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-mailbox", action="store_true", help="skip the mailbox (device-side ready set) leg")
    ap.add_argument("--no-extra-workloads", action="store_true",
                    help="skip the brief per-stream and aggregated timing of the other workloads")
    ap.add_argument("--mailbox-latest-first", action="store_true",
                    help="start each step's mailbox rounds from its last post instead of its first")
    ap.add_argument("--mailbox-closed-loop", action="store_true",
                    help="steps back to back, each DP-group stream posting its next micro-batch only once its "
                         "previous one has been served (its layer output is back)")
    ap.add_argument("--fused-combine", action="store_true",
                    help="asap_moe_layer combines inside the down GEMM (asap_moe_set_combine) instead of a kernel after it")
    ap.add_argument("--mailbox-serve-many", action="store_true",
                    help="one asap_moe_mailbox_serve_many call per step for the step's posts instead of one serve "
                         "call per post")
    ap.add_argument("--mailbox-depth", type=int, default=2,
                    help="mailbox slots per micro-batch stream: the posts a DP group may have in flight")
    ap.add_argument("--mailbox-back-to-back", action="store_true",
                    help="mailbox leg without a barrier between steps")
    ap.add_argument("--mailbox-priority", type=int, default=0,
                    help="1: the posting streams get the highest CUDA stream priority")
    ap.add_argument("--cpu-sample-tokens", type=int, default=12)
    ap.add_argument("--microbatches", default=None,
                    help="comma-separated micro-batch sizes overriding the workload's")
    ap.add_argument("--measure-fp8-peak", action="store_true",
                    help="print the dense e4m3 matmul peak (torch._scaled_mm 8192^3, best of 10) and exit")
    return ap.parse_args()


# ------------------------------------------------------------ distributed plumbing

class Dist:
    """Control plane of N independent replicas: barrier and max-reduce only."""

    def __init__(self):
        self.rank = int(os.environ.get("RANK", "0"))
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.local_rank = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            dist.init_process_group("gloo")
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, v):
        if not self.pg:
            return v
        import torch
        t = torch.tensor([float(v)], dtype=torch.float64)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(dict(sm=float(parts[1]), max=float(parts[2]), power=float(parts[3]),
                                 hw=parts[5], hwt=parts[6], swt=parts[7], swp=parts[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        load = [r for r in rows if r["power"] > 300.0] or rows
        reasons = set()
        for r in load:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("swp", "sw_power_cap")):
                if r[key].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in load), "sm_max_mhz": max(r["max"] for r in rows),
                "samples": len(rows), "samples_under_load": len(load),
                "power_w_max": max(r["power"] for r in rows), "reasons": sorted(reasons)}


# ------------------------------------------------------------ oracle baseline (host cores)

def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_inputs(cfg, x_tokens, device):
    """Raw bf16 bit patterns (host numpy) of everything the oracle reads for
    a few tokens: the tokens, the router, the shared expert and the routed
    experts those tokens select (found by a first, untimed oracle routing)."""
    import numpy as np
    import torch
    import oracle
    from paper_2606_22541_gb300 import inputs

    def bits(t):
        return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)

    xb = bits(x_tokens)
    wrb = bits(inputs.router_weights_bf16(cfg, device))
    idx, _ = oracle.route(oracle.router_logits(oracle.bf16_bits_to_f64(xb), oracle.bf16_bits_to_f64(wrb)),
                          cfg.oracle_cfg())
    experts = {int(e): tuple(bits(t) for t in inputs.expert_weights_bf16(cfg, int(e), device))
               for e in np.unique(idx)}
    shared = tuple(bits(t) for t in inputs.shared_weights_bf16(cfg, device)) if cfg.n_shared else None
    return dict(x=xb, router=wrb, experts=experts, shared=shared)


def oracle_run(cfg, inp):
    """The float64 oracle on prepared inputs: bf16 decode, routing over all
    experts, each token's routed experts (decoded one at a time) and the
    shared expert."""
    import oracle
    f64 = oracle.bf16_bits_to_f64
    xf = f64(inp["x"])
    L = oracle.router_logits(xf, f64(inp["router"]))
    idx, w = oracle.route(L, cfg.oracle_cfg())
    shared = tuple(f64(b) for b in inp["shared"]) if inp["shared"] is not None else None
    ex = inp["experts"]
    return oracle.moe_layer_tokens(xf, idx, w, lambda e: f64(ex[e][0]), lambda e: f64(ex[e][1]),
                                   lambda e: f64(ex[e][2]), shared)


def cpu_baseline(cfg, device, n_tokens):
    from paper_2606_22541_gb300 import inputs
    x = inputs.make_tokens(cfg, n_tokens, 0, device)
    inp = oracle_inputs(cfg, x, device)
    t0 = time.perf_counter()
    oracle_run(cfg, inp)
    dt = time.perf_counter() - t0
    return {"value": n_tokens / dt, "unit": "tokens/s", "cores": host_cores(), "kind": "oracle",
            "sample": f"{n_tokens} tokens of micro-batch 0: float64 routing over all {cfg.n_experts} experts, "
                      f"then each token's {cfg.top_k} routed experts and the shared expert, weights decoded "
                      f"from bf16 as the oracle reads them ({dt:.1f} s); numpy elementwise work on one thread, "
                      f"BLAS on up to {host_cores()} threads"}


# ------------------------------------------------------------ roofline evidence

def profile_traffic(name, source_files):
    """Per-launch DRAM bytes from a committed ncu summary, or None when the
    summary is missing or the kernel's sources changed since it was taken."""
    path = os.path.join(ROOT, "profiles", name)
    if not os.path.exists(path):
        return None, None
    text = open(path).read()
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    h = re.search(r"source_sha256:\s*([0-9a-f]+)", text)
    if not m or not h:
        return None, None
    if h.group(1) != sources_sha256(source_files):
        return None, "stale"
    return float(m.group(1)), os.path.relpath(path, ROOT)


def sources_sha256(files):
    d = hashlib.sha256()
    for f in files:
        d.update(open(os.path.join(ROOT, f), "rb").read())
    return d.hexdigest()


GEMM_SOURCES = ["paper_2606_22541_gb300/csrc/gemm_tc.cu", "paper_2606_22541_gb300/csrc/common.cuh",
                "paper_2606_22541_gb300/csrc/gemm_sched.cuh", "paper_2606_22541_gb300/csrc/gemm_config.h"]


def weight_gb(cfg):
    eb = 2 if cfg.dtype == "bf16" else 1
    return (cfg.n_experts * 3 * cfg.hidden * cfg.inter + cfg.n_shared * 3 * cfg.hidden * cfg.shared_inter) * eb / 1e9


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ------------------------------------------------------------ our arm

def run_ours(args, dist):
    import numpy as np
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_22541_gb300 import api, inputs
    from paper_2606_22541_gb300.configs import CONFIGS

    cfg = CONFIGS[args.workload]
    if args.microbatches:
        from paper_2606_22541_gb300.inputs import small_variant
        cfg = small_variant(cfg, microbatches=[int(v) for v in args.microbatches.split(",")])
    torch.cuda.set_device(dist.local_rank)
    dev = f"cuda:{dist.local_rank}"
    mbs = cfg.microbatches
    n_max = max(mbs)
    weights = inputs.make_weights(cfg, dev)
    h = api.asap_moe_create(cfg, weights, sum(mbs))   # sum: the batched call serves all at once
    del weights
    if args.fused_combine and cfg.dtype == "bf16":   # the fused combine is the bf16 down GEMM's
        api.asap_moe_set_combine(h, api.COMBINE_FUSED)
    torch.cuda.empty_cache()
    xs = inputs.make_microbatches(cfg, dev)
    outs = [torch.empty_like(x) for x in xs]
    wss = [api.workspace(h, x.shape[0], dev) for x in xs]
    streams = [torch.cuda.Stream(device=dev) for _ in xs]
    main = torch.cuda.current_stream()
    tokens_per_step = sum(mbs)

    nvtx = torch.cuda.nvtx.range  # named ranges for a trace of the run (no cost without a tracing tool)

    def step():
        ev = torch.cuda.Event()
        ev.record(main)
        for x, o, ws, s in zip(xs, outs, wss, streams):
            s.wait_event(ev)                       # device-side ordering only
            api.asap_moe_layer(h, x, o, ws, stream=s)
        for s in streams:
            main.wait_stream(s)

    with nvtx("warm-up steps"):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()
    dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(dist.local_rank)
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(main)
    with nvtx("timed steps"):
        for _ in range(args.steps):
            with nvtx("step"):
                step()
    t_end.record(main)
    torch.cuda.synchronize()
    dist.barrier()
    clk = clocks.stop()
    elapsed_ms = dist.max(t_start.elapsed_time(t_end))
    code, word = api.asap_moe_status(h)
    if code != 0:
        raise RuntimeError(f"device status word {word:#x} after the timed region")
    # route (one kernel for E = 256 with grouped sigmoid gating, else router,
    # gate and scan), dispatch, gate/up GEMM, down GEMM, combine (none when
    # the combine runs inside the down GEMM)
    fused = cfg.n_experts == 256 and cfg.gating == "sigmoid_grouped" and cfg.n_groups in (1, 2, 4, 8)
    launches_per_mb = (1 if fused else 3) + (3 if args.fused_combine and cfg.dtype == "bf16" else 4)
    result = {
        "metric": METRIC,
        "value": dist.world * tokens_per_step * args.steps / (elapsed_ms / 1e3),
        "unit": "tokens/s",
        "n_gpus": dist.world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": elapsed_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded normal inputs, random-init weights of the layer's shape)",
        "config": {"workload": f"{cfg.name}: MoE layer, H={cfg.hidden}, E={cfg.n_experts} routed + "
                               f"{cfg.n_shared} shared, I={cfg.inter}, top-{cfg.top_k}, {cfg.gating} gating"
                               + (f" ({cfg.n_groups} groups, top-{cfg.topk_groups})" if cfg.n_groups > 1 else "")
                               + f", {len(mbs)} micro-batches ({','.join(map(str, mbs))} tokens), one CUDA stream each",
                   "tokens_per_step": tokens_per_step, "microbatches": mbs,
                   "parallelism": f"replicas x{dist.world} (no data-path collective)",
                   "l2": f"inputs larger than L2: {weight_gb(cfg):.1f} GB of expert weights streamed every step",
                   **({"combine": "fused into the down GEMM"} if args.fused_combine and cfg.dtype == "bf16" else {})},
        "gpu_launches": launches_per_mb * len(mbs) * args.steps,
        "clocks": clk,
    }

    # ---------------- per-kernel timings, each on the stream it runs on
    with nvtx("per-kernel pass"):
        kern = kernel_pass(args, h, cfg, xs, dev)
    peaks, peaks_src = load_peaks()
    result["kernels"] = kern["table"]
    tensor_peak = None
    if cfg.dtype != "bf16":
        # e4m3 tensor peak: the measured bf16 figure times the nominal fp8/bf16 ratio (4.5 / 2.25)
        tensor_peak = 2.0 * peaks["bf16_tflops_sustained"]
        result["dtype"] = "e4m3 (fp32 accumulate, bf16 out)"
    result["roofline"] = roofline(kern, peaks, peaks_src, tensor_peak, cfg.name)
    gemm_flops = kern["gemm_flops"]
    gemm_ms = kern["gemm_ms"]
    result["grouped_gemm_tensor_frac"] = {
        "achieved_tflops": gemm_flops / (gemm_ms / 1e3) / 1e12,
        "of_burst_measured": gemm_flops / (gemm_ms / 1e3) / 1e12 / peaks["bf16_tflops"],
        "of_sustained_measured": gemm_flops / (gemm_ms / 1e3) / 1e12 / peaks["bf16_tflops_sustained"],
        "peaks": peaks_src,
        "note": "algorithmic FLOPs of both grouped GEMMs (routed + shared) over their event-timed durations"}

    # route, dispatch and combine of a micro-batch together (the HBM-bound
    # steps around the grouped GEMMs)
    small = [nm for nm in ("route", "dispatch", "combine") if nm in kern["table"]]
    sb = sum(kern["alg"][nm]["bytes"] for nm in small)
    sms = sum(kern["avg"][nm] for nm in small)
    result["route_dispatch_combine"] = {
        "alg_bytes": sb, "ms": sms, "gbs": sb / (sms / 1e3) / 1e9,
        "frac_of_measured_hbm": sb / (sms / 1e3) / 1e9 / peaks["hbm_gbs"],
        "note": "the three steps' algorithmic bytes over their summed event times in the per-kernel pass "
                "(events recorded by asap_moe_layer between its own steps)"}

    # ---------------- all micro-batches in one pass (one grouped GEMM per weight matrix)
    with nvtx("host-aggregated pass"):
        result["aggregated"] = aggregated_pass(args, h, cfg, xs, dev, peaks, tensor_peak, dist)

    # ---------------- the device decides the sets: mailbox posts and service rounds
    if not args.no_mailbox:
        with nvtx("mailbox pass"):
            result["mailbox"] = mailbox_pass(args, h, cfg, xs, dev, peaks, tensor_peak, kern, dist,
                                             latest_first=args.mailbox_latest_first,
                                             pipelined=args.mailbox_back_to_back or args.mailbox_closed_loop,
                                             closed_loop=args.mailbox_closed_loop,
                                             serve_many=args.mailbox_serve_many)
        # a serving loop: each DP group posts its next micro-batch once its
        # previous one is served, the server names each step's posts in one call
        if not (args.mailbox_closed_loop and args.mailbox_serve_many):
            with nvtx("mailbox serving-loop pass"):
                result["mailbox_serving_loop"] = mailbox_pass(args, h, cfg, xs, dev, peaks, tensor_peak, kern, dist,
                                                              pipelined=True, closed_loop=True, serve_many=True)

    # the same fraction where several micro-batches share the GEMMs: sets the
    # device chose (mailbox rounds) and sets the host chose (aggregated call)
    gtf = result["grouped_gemm_tensor_frac"]
    gtf["note"] += ("; per-stream launches (one micro-batch each) here, the mailbox rounds' and the "
                    "host-aggregated launches' in mailbox_* and aggregated_*")
    for leg in ("mailbox", "aggregated"):
        r = result.get(leg) or {}
        for k in ("of_burst_measured", "of_sustained_measured"):
            if "grouped_gemm_frac_" + k in r:
                gtf[f"{leg}_{k}"] = r["grouped_gemm_frac_" + k]

    # ---------------- per-micro-batch latency of the per-stream step
    with nvtx("latency pass"):
        result["latency"] = latency_pass(args, h, xs, outs, wss, streams, main)
    if cfg.zipf_s is not None:
        result["expert_popularity"] = popularity(h, cfg, xs, dev)

    # ---------------- end to end through host buffers
    with nvtx("end-to-end pass"):
        result["e2e"] = e2e_pass(args, h, cfg, xs, outs, wss, streams, main, dist)

    # ---------------- the other workloads, briefly (N = 1 only)
    if dist.world == 1 and not args.no_extra_workloads:
        h.close()
        del xs, outs, wss
        torch.cuda.empty_cache()
        result["other_workloads"] = {name: other_workload(args, name, dev)
                                     for name in ("mixtral", "dsv3_stress", "dsv3_fp8") if name != cfg.name}
        h = None

    # ---------------- float64 oracle on the host cores
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(cfg, dev, args.cpu_sample_tokens)
    else:
        result["cpu_baseline"] = None
    if h is not None:
        h.close()
    return result


def other_workload(args, name, dev):
    """Another configuration's per-stream step (every micro-batch through
    asap_moe_layer on its own stream; each step's streams wait for the
    previous step on the device, as in the headline) and its host-aggregated
    step (asap_moe_layer_batched), timed with CUDA events: W warm-up and
    K = max(3, steps // 2) timed steps each."""
    import torch
    from paper_2606_22541_gb300 import api, inputs
    from paper_2606_22541_gb300.configs import CONFIGS

    cfg = CONFIGS[name]
    mbs = cfg.microbatches
    w = inputs.make_weights(cfg, dev)
    h = api.asap_moe_create(cfg, w, sum(mbs))
    del w
    torch.cuda.empty_cache()
    xs = inputs.make_microbatches(cfg, dev)
    outs = [torch.empty_like(x) for x in xs]
    wss = [api.workspace(h, x.shape[0], dev) for x in xs]
    streams = [torch.cuda.Stream(device=dev) for _ in xs]
    main = torch.cuda.current_stream()
    steps = max(3, args.steps // 2)

    def per_stream():
        ev = torch.cuda.Event()
        ev.record(main)
        for x, o, ws, s in zip(xs, outs, wss, streams):
            s.wait_event(ev)
            api.asap_moe_layer(h, x, o, ws, stream=s)
        for s in streams:
            main.wait_stream(s)

    ws_all = api.workspace(h, sum(mbs), dev)

    def aggregated():
        api.asap_moe_layer_batched(h, xs, outs, ws_all)

    res = {}
    for key, fn in (("per_stream", per_stream), ("aggregated", aggregated)):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(main)
        for _ in range(steps):
            fn()
        b.record(main)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / steps
        res[key] = {"value": sum(mbs) / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms}
    code, word = api.asap_moe_status(h)
    h.close()
    if code != 0:
        raise RuntimeError(f"{name}: device status word {word:#x}")
    res.update({"microbatches": mbs, "dtype": cfg.dtype, "steps": steps,
                "note": "per-stream: one stream per micro-batch through asap_moe_layer; aggregated: "
                        "asap_moe_layer_batched over the step's micro-batches"})
    return res


def head_start(stream):
    """Holds the stream's device work for about 100 us (a device-side spin,
    no memory traffic) so that the host enqueues the calls that follow before
    the device reaches their first event: an event pair right after a host
    synchronize would otherwise time the host's launch of the call too."""
    import torch
    with torch.cuda.stream(stream):
        torch.cuda._sleep(200_000)


def kernel_pass(args, h, cfg, xs, dev):
    """The same work as the timed steps, one asap_moe_layer call after
    another on one stream, each recording CUDA events between its own steps
    (asap_moe_time_layer), so every kernel of the layer is timed where it
    runs, without overlap from the other micro-batches."""
    import numpy as np
    import torch
    from paper_2606_22541_gb300 import api

    n = max(x.shape[0] for x in xs)
    k, E, H, I, Is = cfg.top_k, cfg.n_experts, cfg.hidden, cfg.inter, cfg.shared_inter
    s = torch.cuda.current_stream()
    idx = torch.empty((n, k), dtype=torch.int32, device=dev)
    w = torch.empty((n, k), dtype=torch.float32, device=dev)
    counts = torch.empty(E, dtype=torch.int32, device=dev)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=dev)
    out = torch.empty((n, H), dtype=torch.bfloat16, device=dev)
    ws = api.workspace(h, n, dev)
    fp8 = cfg.dtype != "bf16"
    names = ["route", "dispatch", "gemm_gate_up_swiglu", "gemm_down", "combine"]
    if fp8:
        names = ["route", "dispatch", "expert_ffn_fp8", "combine"]
    times = {nm: [] for nm in names}
    active = []   # experts with tokens, per micro-batch (for the weight bytes)
    for x in xs:
        m = x.shape[0]
        api.asap_moe_route(h, x, idx[:m], w[:m], counts, offsets, ws, stream=s)
        torch.cuda.synchronize()
        active.append(int((counts > 0).sum().item()))
    for it in range(args.kernel_steps + 1):
        rec = []
        head_start(s)
        for x in xs:
            m = x.shape[0]
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
            api.asap_moe_time_layer(ev)
            api.asap_moe_layer(h, x, out[:m], ws, stream=s)
            rec.append(ev)
        torch.cuda.synchronize()
        if it == 0:
            continue   # warm-up round
        for ev in rec:
            d = [ev[j].elapsed_time(ev[j + 1]) for j in range(5)]   # route, dispatch, gate/up, down, combine
            for nm, v in zip(names, [d[0], d[1], d[2] + d[3], d[4]] if fp8 else d):
                times[nm].append(v)
    avg = {nm: sum(v) / len(v) for nm, v in times.items()}
    mins = {nm: min(v) for nm, v in times.items()}
    mean_active = sum(active) / len(active)
    wb = 2  # bf16 activations
    eb = 1 if fp8 else 2  # expert-weight element bytes

    def alg_of(m, act):
        """Algorithmic bytes / FLOPs of each step for one micro-batch of m
        tokens whose routing reaches ``act`` experts."""
        nk = m * k
        a = {
            # route: read x and the router weights, write idx, w, counts, offsets
            # (the logits between the router GEMM and the gate are not algorithmic)
            "route": dict(bytes=m * H * wb + E * H * wb + nk * 8 + (2 * E + 1) * 4, flops=2.0 * m * H * E),
            "dispatch": dict(bytes=m * H * wb + nk * H * wb + nk * 12, flops=0.0),
            "gemm_gate_up_swiglu": dict(
                bytes=act * 2 * I * H * eb + (2 * Is * H * eb if cfg.n_shared else 0)
                + nk * H * wb + (m * H * wb if cfg.n_shared else 0) + nk * I * wb + (m * Is * wb if cfg.n_shared else 0),
                flops=2.0 * nk * H * 2 * I + (2.0 * m * H * 2 * Is if cfg.n_shared else 0.0)),
            "gemm_down": dict(
                bytes=act * H * I * eb + (H * Is * eb if cfg.n_shared else 0)
                + nk * I * wb + (m * Is * wb if cfg.n_shared else 0) + nk * H * wb + (m * H * wb if cfg.n_shared else 0),
                flops=2.0 * nk * I * H + (2.0 * m * Is * H if cfg.n_shared else 0.0)),
            "combine": dict(bytes=nk * H * wb + (m * H * wb if cfg.n_shared else 0) + m * H * wb + nk * 8, flops=0.0),
        }
        if fp8:
            # e4m3 activations (x_perm, h) and bf16 outputs
            a["dispatch"] = dict(bytes=m * H * wb + nk * H + nk * (H // 128) * 4 + nk * 12, flops=0.0)
            a["expert_ffn_fp8"] = dict(
                bytes=act * 3 * I * H + (3 * Is * H if cfg.n_shared else 0) + nk * H + 2 * nk * I
                + (m * H * 2 + m * H + 2 * m * Is if cfg.n_shared else 0) + nk * H * 2 + (m * H * 2 if cfg.n_shared else 0),
                flops=a["gemm_gate_up_swiglu"]["flops"] + a["gemm_down"]["flops"])
        return a

    # per launch: the mean over the micro-batches (work and time alike), so
    # rates are total work over total time also when the sizes differ
    per_mb = [alg_of(x.shape[0], act) for x, act in zip(xs, active)]
    alg = {nm: dict(bytes=sum(a[nm]["bytes"] for a in per_mb) / len(per_mb),
                    flops=sum(a[nm]["flops"] for a in per_mb) / len(per_mb)) for nm in per_mb[0]}
    table = {}
    for nm in names:
        sec = avg[nm] / 1e3
        table[nm] = {"ms": avg[nm], "min_ms": mins[nm], "alg_bytes": alg[nm]["bytes"], "alg_flops": alg[nm]["flops"],
                     "gbs": alg[nm]["bytes"] / sec / 1e9, "tflops": alg[nm]["flops"] / sec / 1e12}
    total_ms = sum(avg.values())
    for nm in names:
        table[nm]["share"] = avg[nm] / total_ms
    gemm_flops = alg["gemm_gate_up_swiglu"]["flops"] + alg["gemm_down"]["flops"]
    gemm_ms = avg["expert_ffn_fp8"] if fp8 else avg["gemm_gate_up_swiglu"] + avg["gemm_down"]
    return {"table": table, "avg": avg, "alg": alg, "gemm_flops": gemm_flops, "gemm_ms": gemm_ms,
            "active_experts": mean_active, "serial_ms_per_microbatch": total_ms}


def roofline(kern, peaks, peaks_src, tensor_peak=None, workload=None):
    nm = max(kern["avg"], key=kern["avg"].get)
    a = kern["alg"][nm]
    sec = kern["avg"][nm] / 1e3
    tpk = tensor_peak or peaks["bf16_tflops_sustained"]
    t_hbm = a["bytes"] / (peaks["hbm_gbs"] * 1e9)
    t_tc = a["flops"] / (tpk * 1e12) if a["flops"] else 0.0
    # the committed capture covers the DeepSeek-V3 BF16 gate/up launch only
    traffic, src = (profile_traffic("gemm_gate_up_swiglu_dsv3.md", GEMM_SOURCES)
                    if workload == "dsv3_bf16" and nm == "gemm_gate_up_swiglu" else (None, None))
    if t_tc >= t_hbm:
        achieved = a["flops"] / sec / 1e12
        peak = tpk
        r = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak}
    else:
        achieved = a["bytes"] / sec / 1e9
        peak = peaks["hbm_gbs"]
        r = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak}
    r.update({"traffic": traffic, "kernel": nm, "alg_bytes_per_launch": a["bytes"],
              "alg_flops_per_launch": a["flops"], "avg_launch_ms": kern["avg"][nm],
              "peak_source": f"{peaks_src} ({'sustained bf16 tensor' if r['bound'] == 'tensor' else 'HBM copy'})",
              "hbm_frac_of_measured": a["bytes"] / sec / 1e9 / peaks["hbm_gbs"],
              "tensor_frac_of_sustained_measured": (a["flops"] / sec / 1e12 / tpk) if a["flops"] else None,
              "traffic_source": src})
    return r


def aggregated_pass(args, h, cfg, xs, dev, peaks, tensor_peak, dist):
    """The same micro-batches through asap_moe_layer_batched: each expert's
    weights stream once per step instead of once per micro-batch.  Also times
    the two grouped GEMMs on the combined segments (route + dispatch of the
    concatenated tokens, then the gate/up and down calls, events between)."""
    import torch
    from paper_2606_22541_gb300 import api

    n_all = sum(x.shape[0] for x in xs)
    ws = api.workspace(h, n_all, dev)
    outs = [torch.empty_like(x) for x in xs]
    s = torch.cuda.current_stream()
    for _ in range(args.warmup):
        api.asap_moe_layer_batched(h, xs, outs, ws)
    torch.cuda.synchronize()
    dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(s)
    for _ in range(args.steps):
        api.asap_moe_layer_batched(h, xs, outs, ws)
    b.record(s)
    torch.cuda.synchronize()
    ms = dist.max(a.elapsed_time(b)) / args.steps
    res = {"value": dist.world * n_all / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
           "note": "asap_moe_layer_batched over the step's micro-batches on one stream; outputs are bit-identical "
                   "to the per-micro-batch calls"}
    if cfg.dtype != "bf16":
        return res
    k, E, H, I, Is = cfg.top_k, cfg.n_experts, cfg.hidden, cfg.inter, cfg.shared_inter
    x = torch.cat(xs)
    idx = torch.empty((n_all, k), dtype=torch.int32, device=dev)
    w = torch.empty((n_all, k), dtype=torch.float32, device=dev)
    counts = torch.empty(E, dtype=torch.int32, device=dev)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=dev)
    api.asap_moe_route(h, x, idx, w, counts, offsets, ws)
    x_perm = torch.empty((n_all * k, H), dtype=torch.bfloat16, device=dev)
    ps = torch.empty(n_all * k, dtype=torch.int32, device=dev)
    pd = torch.empty((n_all, k), dtype=torch.int32, device=dev)
    api.asap_moe_dispatch(h, x, idx, x_perm, ps, pd, ws)
    hb = torch.empty((n_all * k, I), dtype=torch.bfloat16, device=dev)
    hsh = torch.empty((n_all, Is), dtype=torch.bfloat16, device=dev) if cfg.n_shared else None
    y = torch.empty_like(x_perm)
    ysh = torch.empty((n_all, H), dtype=torch.bfloat16, device=dev) if cfg.n_shared else None
    t1, t2 = [], []
    for it in range(args.kernel_steps + 1):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        head_start(s)
        e[0].record(s)
        api.asap_moe_expert_gate_up(h, x_perm, offsets, x, hb, hsh, ws=ws)
        e[1].record(s)
        api.asap_moe_expert_down(h, hb, offsets, hsh, n_all, y, ysh, ws=ws)
        e[2].record(s)
        torch.cuda.synchronize()
        if it:
            t1.append(e[0].elapsed_time(e[1]))
            t2.append(e[1].elapsed_time(e[2]))
    g1, g2 = sum(t1) / len(t1), sum(t2) / len(t2)
    nk = n_all * k
    flops = 2.0 * nk * H * 2 * I + 2.0 * nk * I * H + (6.0 * n_all * H * Is if cfg.n_shared else 0.0)
    tf = flops / ((g1 + g2) / 1e3) / 1e12
    active = int((counts > 0).sum().item())
    wbytes = active * 3 * H * I * 2 + (3 * H * Is * 2 if cfg.n_shared else 0)
    res.update({"gemm_gate_up_ms": g1, "gemm_down_ms": g2, "grouped_gemm_tflops": tf,
                "grouped_gemm_frac_of_burst_measured": tf / peaks["bf16_tflops"],
                "grouped_gemm_frac_of_sustained_measured": tf / peaks["bf16_tflops_sustained"],
                "weight_gb_per_step": wbytes / 1e9})
    return res


def mailbox_pass(args, h, cfg, xs, dev, peaks, tensor_peak, kern, dist, latest_first=False, pipelined=False,
                 closed_loop=False, serve_many=False):
    """The step's micro-batches posted into a mailbox, each from its own
    stream, and served by rounds on one MoE stream: the host serves every post
    right after making it (no host batching), and each round claims on the
    device every post published by the time it starts, serving all of them
    with one grouped GEMM pass.  Slots are double-buffered across steps.
    Outputs are bit-identical to asap_moe_layer's (tested).  Reports the
    step rate, how the device grouped the posts, and the grouped GEMMs'
    tensor fraction (algorithmic FLOPs of the step over the event-timed GEMMs
    of its rounds).  latest_first: the step's rounds are started from its
    last post backwards (a server that, knowing of several posts, starts the
    round from the newest; the device still claims whatever is published).
    closed_loop (with pipelined): a DP group's stream makes its next post only
    once its previous post has been served, as a prefill pipeline whose next
    step needs this layer's output would.
    pipelined: no barrier between steps: a step's posts wait only for the
    rounds that served their slots' previous posts (the post's own
    backpressure), so they are made while the previous step's rounds run, as
    in a serving loop where DP groups keep sending."""
    import torch
    from paper_2606_22541_gb300 import api

    n_mb = len(xs)
    depth = max(1, args.mailbox_depth)
    m = api.asap_moe_mailbox_create(h, depth * n_mb, max(x.shape[0] for x in xs))
    # --mailbox-priority: the DP groups' streams above the MoE stream
    hi = torch.cuda.Stream.priority_range()[1] if args.mailbox_priority else 0
    producers = [torch.cuda.Stream(priority=hi) for _ in xs]
    server = torch.cuda.Stream()
    main = torch.cuda.current_stream()
    outs = [[torch.empty_like(x) for x in xs] for _ in range(depth)]

    consumers = [torch.cuda.Stream() for _ in xs]

    def step(si, gemm_events=None, latency=None):
        b = si % depth
        ev = torch.cuda.Event(enable_timing=latency is not None)
        ev.record(main)
        eps = []
        for i, (x, p) in enumerate(zip(xs, producers)):
            if not pipelined:
                p.wait_event(ev)
            elif closed_loop and si > 0:
                api.asap_moe_mailbox_wait(m, ((si - 1) % depth) * n_mb + i, stream=p)
            eps.append(api.asap_moe_mailbox_post(m, b * n_mb + i, x, outs[b][i], stream=p))
        if serve_many:
            if gemm_events is not None:
                api.asap_moe_mailbox_time_gemms(m, *gemm_events[0])
            api.asap_moe_mailbox_serve_many(m, [b * n_mb + i for i in range(n_mb)], eps, stream=server)
        for r, i in enumerate(reversed(range(n_mb)) if latest_first else range(n_mb)):
            if serve_many:
                break
            if gemm_events is not None:
                api.asap_moe_mailbox_time_gemms(m, *gemm_events[r])
            api.asap_moe_mailbox_serve(m, b * n_mb + i, eps[i], stream=server)
        if latency is not None:
            # each post's completion as its DP group would see it: a stream of
            # its own waits for the post's round
            ends = []
            for i, c in enumerate(consumers):
                api.asap_moe_mailbox_wait(m, b * n_mb + i, stream=c)
                e = torch.cuda.Event(enable_timing=True)
                e.record(c)
                ends.append(e)
            latency.append((ev, ends))
        for i in range(n_mb):
            api.asap_moe_mailbox_wait(m, b * n_mb + i, stream=main)

    for si in range(args.warmup):
        step(si)
    torch.cuda.synchronize()
    r0, _ = api.asap_moe_mailbox_rounds(m)
    dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(main)
    for si in range(args.steps):
        step(args.warmup + si)
    b.record(main)
    torch.cuda.synchronize()
    ms = dist.max(a.elapsed_time(b)) / args.steps
    r1, claimed = api.asap_moe_mailbox_rounds(m)
    sizes = claimed[r0:r1]
    # the GEMMs of every round, timed with events on the MoE stream
    gemm_ms = []
    nonempty = []
    lat = []
    base = args.warmup + args.steps
    for si in range(args.kernel_steps):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_mb)]
        rb, _ = api.asap_moe_mailbox_rounds(m)
        # as in the timed steps, every post is enqueued before the device
        # reaches the step (a step right after a host synchronize would
        # otherwise route its first post before the host has made the others)
        head_start(main)
        step(base + si, evs, lat)
        torch.cuda.synchronize()
        ra, cl = api.asap_moe_mailbox_rounds(m)
        gemm_ms.append(sum(e0.elapsed_time(e1) for e0, e1 in (evs[:1] if serve_many else evs)))
        nonempty.append(sum(1 for c in cl[rb:ra] if c > 0))
    api.asap_moe_mailbox_rounds(m)
    code, word = api.asap_moe_status(h)
    m.close()
    if code != 0:
        raise RuntimeError(f"device status word {word:#x} after the mailbox leg")
    post_ms = [[e0.elapsed_time(e) for e in ends] for e0, ends in lat]
    post_lat = [sum(v[i] for v in post_ms) / len(post_ms) for i in range(n_mb)]
    flops = kern["gemm_flops"] * n_mb    # per micro-batch mean x micro-batches
    g = sum(gemm_ms) / len(gemm_ms)
    tf = flops / (g / 1e3) / 1e12
    tpk_burst = 2.0 * peaks["bf16_tflops"] if tensor_peak else peaks["bf16_tflops"]
    tpk_sus = tensor_peak or peaks["bf16_tflops_sustained"]
    hist = {}
    for c in sizes:
        hist[str(c)] = hist.get(str(c), 0) + 1
    n_tok = sum(x.shape[0] for x in xs)
    return {"value": dist.world * n_tok / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "rounds_per_step": (r1 - r0) / args.steps,
            "nonempty_rounds_per_step": sum(1 for c in sizes if c > 0) / args.steps,
            "posts_per_nonempty_round": (sum(sizes) / max(1, sum(1 for c in sizes if c > 0))),
            "round_sizes_histogram": hist,
            "grouped_gemm_ms_per_step": g, "grouped_gemm_tflops": tf,
            "grouped_gemm_frac_of_burst_measured": tf / tpk_burst,
            "grouped_gemm_frac_of_sustained_measured": tf / tpk_sus,
            "gemm_timing_nonempty_rounds_per_step": sum(nonempty) / len(nonempty),
            "post_latency_ms": post_lat,
            "post_latency_note": "in the GEMM-timing steps: step start (every DP-group stream waits on it) to "
                                 "each post's completion as seen by a stream of its own",
            "serve_order": ("one serve_many call per step" if serve_many else
                            "latest post first" if latest_first else "post order"),
            "steps": ("closed loop per DP group, no barrier between steps" if closed_loop else
                      "back to back, no barrier between steps" if pipelined else "one barrier per step"),
            "slots_per_stream": depth,
            "posting_stream_priority": "highest" if args.mailbox_priority else "default",
            "note": "asap_moe_mailbox_post from one stream per micro-batch, asap_moe_mailbox_serve for every post "
                    "right after it on one MoE stream; the rounds claim on the device whatever has been published"}


def latency_pass(args, h, xs, outs, wss, streams, main):
    """Per-micro-batch latency of the per-stream step: CUDA events from the
    step's first submission (every stream waits on it) to each micro-batch's
    completion on its own stream; the aggregate rate is the step's tokens
    over the span to the last completion."""
    import torch
    from paper_2606_22541_gb300 import api

    lat = [[] for _ in xs]
    spans = []
    for it in range(args.kernel_steps + 1):
        ev0 = torch.cuda.Event(enable_timing=True)
        ends = [torch.cuda.Event(enable_timing=True) for _ in xs]
        ev0.record(main)
        for x, o, ws, s, e in zip(xs, outs, wss, streams, ends):
            s.wait_event(ev0)
            api.asap_moe_layer(h, x, o, ws, stream=s)
            e.record(s)
        for s in streams:
            main.wait_stream(s)
        torch.cuda.synchronize()
        if it == 0:
            continue
        t = [ev0.elapsed_time(e) for e in ends]
        for i, v in enumerate(t):
            lat[i].append(v)
        spans.append(max(t))
    n_tok = sum(x.shape[0] for x in xs)
    span = sum(spans) / len(spans)
    return {"per_microbatch_ms": [sum(v) / len(v) for v in lat],
            "microbatch_tokens": [x.shape[0] for x in xs],
            "first_submit_to_last_complete_ms": span,
            "aggregate_tokens_per_s": n_tok / (span / 1e3),
            "note": "CUDA events: step start on the submitting stream -> each micro-batch's completion on its own "
                    "stream, mean over the kernel steps"}


def popularity(h, cfg, xs, dev):
    """Realised expert popularity of a Zipf-biased workload: each expert's
    share of the routed (token, slot) pairs over all micro-batches, ranked,
    beside the Zipf target p_r ~ r^-s; and the exponent fitted to the
    realised shares of ranks 2..64 by least squares in log-log."""
    import numpy as np
    import torch
    from paper_2606_22541_gb300 import api

    E, k = cfg.n_experts, cfg.top_k
    tot = np.zeros(E, np.int64)
    active = []
    for x in xs:
        n = x.shape[0]
        idx = torch.empty((n, k), dtype=torch.int32, device=dev)
        w = torch.empty((n, k), dtype=torch.float32, device=dev)
        counts = torch.empty(E, dtype=torch.int32, device=dev)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=dev)
        api.asap_moe_route(h, x, idx, w, counts, offsets, api.workspace(h, n, dev))
        c = counts.cpu().numpy().astype(np.int64)
        tot += c
        active.append(int((c > 0).sum()))
    share = np.sort(tot)[::-1] / tot.sum()
    r = np.arange(1, E + 1, dtype=np.float64)
    target = r ** -cfg.zipf_s
    target /= target.sum()
    sel = slice(1, 64)
    fit = -np.polyfit(np.log(r[sel]), np.log(np.maximum(share[sel], 1e-12)), 1)[0]
    return {"zipf_s": cfg.zipf_s, "realised_top8_share": [float(v) for v in share[:8]],
            "zipf_target_top8_share": [float(v) for v in target[:8]],
            "fitted_exponent_ranks_2_64": float(fit), "experts_with_tokens_total": int((tot > 0).sum()),
            "active_experts_per_microbatch": active,
            "note": "share of the routed (token, slot) pairs; with top-8 one expert holds at most 1/8"}


def e2e_pass(args, h, cfg, xs, outs, wss, streams, main, dist):
    """tokens/s through asap_moe_layer with the inputs in pinned host memory:
    every step copies each micro-batch host->device, runs the layer and copies
    the output back, all inside the timed region.  The copies run on their
    own streams with two device buffers per micro-batch, as a serving loop
    would: step s+1's uploads overlap step s's layers, and step s's downloads
    overlap step s+1's."""
    import torch
    from paper_2606_22541_gb300 import api

    hx = [x.cpu().pin_memory() for x in xs]
    ho = [torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs]
    dx = [[torch.empty_like(x) for x in xs] for _ in range(2)]
    do = [[torch.empty_like(o) for o in outs] for _ in range(2)]
    up = torch.cuda.Stream()
    down = torch.cuda.Stream()
    n_mb = len(xs)
    done = [[None] * n_mb for _ in range(2)]    # the layer that last used buffer b of micro-batch i
    fetched = [[None] * n_mb for _ in range(2)]  # the download that last read output buffer b

    def step(s):
        b = s % 2
        for i in range(n_mb):
            ev_in = torch.cuda.Event()
            with torch.cuda.stream(up):
                if done[b][i] is not None:
                    up.wait_event(done[b][i])   # the layer of step s-2 no longer reads dx[b][i]
                dx[b][i].copy_(hx[i], non_blocking=True)
                ev_in.record(up)
            st = streams[i]
            st.wait_event(ev_in)
            if fetched[b][i] is not None:
                st.wait_event(fetched[b][i])    # step s-2's output has been downloaded
            api.asap_moe_layer(h, dx[b][i], do[b][i], wss[i], stream=st)
            ev_done = torch.cuda.Event()
            ev_done.record(st)
            done[b][i] = ev_done
            ev_out = torch.cuda.Event()
            with torch.cuda.stream(down):
                down.wait_event(ev_done)
                ho[i].copy_(do[b][i], non_blocking=True)
                ev_out.record(down)
            fetched[b][i] = ev_out

    def drain():
        main.wait_stream(up)
        main.wait_stream(down)
        for st in streams:
            main.wait_stream(st)

    steps = max(3, args.steps // 2)
    for s in range(max(3, args.warmup)):
        step(s)
    drain()
    torch.cuda.synchronize()
    dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(main)
    for st in (up, down, *streams):
        st.wait_event(a)
    for s in range(steps):
        step(s)
    drain()
    b.record(main)
    torch.cuda.synchronize()
    ms = dist.max(a.elapsed_time(b))
    tokens = sum(x.shape[0] for x in xs)
    return {"value": dist.world * tokens * steps / (ms / 1e3), "unit": "tokens/s",
            "h2d_bytes_per_step": sum(x.numel() * x.element_size() for x in hx),
            "d2h_bytes_per_step": sum(o.numel() * o.element_size() for o in ho), "steps": steps,
            "note": "uploads and downloads on their own streams, double-buffered across steps"}


# ------------------------------------------------------------ reference arm (the oracle)

def run_reference(args, dist):
    import torch
    from paper_2606_22541_gb300 import inputs
    from paper_2606_22541_gb300.configs import CONFIGS

    cfg = CONFIGS[args.workload]
    dev = f"cuda:{dist.local_rank}" if torch.cuda.is_available() else "cpu"
    per_step = 1
    x = inputs.make_tokens(cfg, (args.warmup + args.steps) * per_step, 0, dev)
    dt = 0.0
    for i in range(args.warmup + args.steps):
        inp = oracle_inputs(cfg, x[i * per_step:(i + 1) * per_step], dev)   # input preparation, untimed
        t0 = time.perf_counter()
        oracle_run(cfg, inp)
        if i >= args.warmup:
            dt += time.perf_counter() - t0
    value = args.steps * per_step / dt
    sample = (f"{per_step} token per step of micro-batch 0 (float64 routing over all experts, its "
              f"{cfg.top_k} routed experts and the shared expert, weights decoded from bf16 per expert)")
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": dist.world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded normal inputs, random-init weights of the layer's shape)",
            "config": {"workload": cfg.name, "tokens_per_step": per_step},
            "cpu_baseline": {"kind": "oracle", "cores": host_cores(), "sample": sample, "value": value,
                             "unit": "tokens/s"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def measure_fp8_peak():
    """Dense e4m3 matmul throughput: torch._scaled_mm at 8192^3, best of 10."""
    import torch
    n = 8192
    a = torch.randn(n, n, device="cuda").to(torch.float8_e4m3fn)
    b = torch.randn(n, n, device="cuda").to(torch.float8_e4m3fn).t()
    one = torch.ones((), device="cuda")
    for _ in range(3):
        torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)
    best = 1e9
    for _ in range(10):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)
        e1.record()
        torch.cuda.synchronize()
        best = min(best, e0.elapsed_time(e1))
    return {"fp8_e4m3_tflops": 2.0 * n ** 3 / (best / 1e3) / 1e12, "ms": best, "n": n,
            "how": "torch._scaled_mm e4m3 x e4m3 -> bf16, 8192^3, best of 10, CUDA events"}


def main():
    args = parse_args()
    if args.measure_fp8_peak:
        print(json.dumps(measure_fp8_peak()), flush=True)
        return
    dist = Dist()
    if args.impl == "reference":
        if dist.rank == 0:
            print(json.dumps(run_reference(args, dist)), flush=True)
        dist.close()
        return
    res = run_ours(args, dist)
    if dist.rank == 0:
        print(json.dumps(res), flush=True)
    dist.close()


if __name__ == "__main__":
    main()
