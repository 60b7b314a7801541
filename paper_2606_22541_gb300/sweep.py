"""Latency of one MoE-layer call against its token count on one GB300.

    python -m paper_2606_22541_gb300.sweep [--workload dsv3_bf16] [--tokens 128,256,...]

ASAP motivates length-aware batching with this curve (Section 2.2.2): MoE
latency stays flat while the layer is bound by loading expert weights, then
grows linearly once the token count makes it compute-bound; the paper places
the knee near 2k tokens on its hardware.  This tool measures the same curve
for asap_moe_layer: per token count, the best and median of R timed calls
(CUDA events, inputs resident), tokens/s, the grouped-GEMM FLOP rate and the
rate at which the active experts' weights stream.  One JSON line per point.
"""
import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="dsv3_bf16")
    ap.add_argument("--tokens", default="128,256,512,1024,2048,4096,8192,16384,32768")
    ap.add_argument("--reps", type=int, default=10)
    args = ap.parse_args()

    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_22541_gb300 import api, inputs
    from paper_2606_22541_gb300.configs import CONFIGS

    cfg = CONFIGS[args.workload]
    sizes = [int(v) for v in args.tokens.split(",")]
    dev = "cuda"
    w = inputs.make_weights(cfg, dev)
    h = api.asap_moe_create(cfg, w, max(sizes))
    del w
    torch.cuda.empty_cache()
    eb = 2 if cfg.dtype == "bf16" else 1
    for n in sizes:
        x = inputs.make_tokens(cfg, n, 0, dev)
        out = torch.empty_like(x)
        ws = api.workspace(h, n)
        api.asap_moe_layer(h, x, out, ws)
        torch.cuda.synchronize()
        times = []
        for _ in range(args.reps):
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            api.asap_moe_layer(h, x, out, ws)
            b.record()
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b))
        times.sort()
        # active experts of this call (for the weight stream rate)
        idx = torch.empty((n, cfg.top_k), dtype=torch.int32, device=dev)
        wt = torch.empty((n, cfg.top_k), dtype=torch.float32, device=dev)
        counts = torch.empty(cfg.n_experts, dtype=torch.int32, device=dev)
        offs = torch.empty(cfg.n_experts + 1, dtype=torch.int32, device=dev)
        api.asap_moe_route(h, x, idx, wt, counts, offs, ws)
        active = int((counts > 0).sum().item())
        best = times[0]
        flops = n * cfg.flops_per_token()
        wbytes = (active * 3 * cfg.hidden * cfg.inter + cfg.n_shared * 3 * cfg.hidden * cfg.shared_inter) * eb
        print(json.dumps({"workload": cfg.name, "tokens": n, "best_ms": best, "median_ms": times[len(times) // 2],
                          "tokens_per_s": n / (best / 1e3), "gemm_tflops": flops / (best / 1e3) / 1e12,
                          "active_experts": active, "weight_gbs": wbytes / (best / 1e3) / 1e9}), flush=True)
        del x, out, ws
        torch.cuda.empty_cache()
    code, word = api.asap_moe_status(h)
    if code != 0:
        raise RuntimeError(f"device status word {word:#x}")
    h.close()


if __name__ == "__main__":
    main()
