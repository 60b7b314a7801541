"""Calibration of the Zipf logit-bias strength of the skewed workloads.

    python -m paper_2606_22541_gb300.zipf_calibrate [--workload dsv3_stress] [--betas 0.5,0.6,...]

For each strength beta the workload's router weights and micro-batches are
drawn as inputs.py draws them, every micro-batch is routed by the library
(asap_moe_route), and the realised shares of the routed (token, slot) pairs
are ranked.  Printed per beta: the exponent fitted to ranks 2..64 by least
squares in log-log (the target is the workload's zipf_s; rank 1 is left out
because top-k routing caps one expert at 1/k of the pairs), the top shares
and the experts that receive tokens.  The expert FFN is irrelevant to the
routing, so the handle is made with a narrow one.
"""
import argparse
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def realised_shares(cfg, device):
    from paper_2606_22541_gb300 import api, inputs
    narrow = inputs.small_variant(cfg, inter=128, shared_inter=128)
    h = api.asap_moe_create(narrow, inputs.make_weights(narrow, device), max(cfg.microbatches))
    E, k = cfg.n_experts, cfg.top_k
    tot = np.zeros(E, np.int64)
    for x in inputs.make_microbatches(cfg, device):
        n = x.shape[0]
        idx = torch.empty((n, k), dtype=torch.int32, device=device)
        w = torch.empty((n, k), dtype=torch.float32, device=device)
        counts = torch.empty(E, dtype=torch.int32, device=device)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=device)
        api.asap_moe_route(h, x, idx, w, counts, offsets, api.workspace(h, n, device))
        tot += counts.cpu().numpy().astype(np.int64)
    h.close()
    return np.sort(tot)[::-1] / tot.sum(), int((tot > 0).sum())


def fitted_exponent(share, lo=1, hi=64):
    r = np.arange(1, len(share) + 1, dtype=np.float64)
    return float(-np.polyfit(np.log(r[lo:hi]), np.log(np.maximum(share[lo:hi], 1e-12)), 1)[0])


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="dsv3_stress")
    ap.add_argument("--betas", default="0.5,0.6,0.63,0.7,0.8,1.0")
    args = ap.parse_args()
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_22541_gb300 import inputs
    from paper_2606_22541_gb300.configs import CONFIGS
    base = CONFIGS[args.workload]
    print(f"{args.workload}: target exponent {base.zipf_s}, {sum(base.microbatches)} tokens")
    for beta in (float(b) for b in args.betas.split(",")):
        share, active = realised_shares(inputs.small_variant(base, zipf_beta=beta), "cuda")
        print(f"beta {beta:.3f}: fitted exponent (ranks 2..64) {fitted_exponent(share):.3f}, "
              f"top shares {np.round(share[:4], 4).tolist()}, experts with tokens {active}")


if __name__ == "__main__":
    main()
