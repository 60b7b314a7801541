"""The five layer configurations the MoE layer is exercised on.

Shapes follow the model the paper evaluates (DeepSeek-V3.2: 256 routed experts
plus one shared expert, top-8, hidden 7168, 16-bit data; ASAP Table 1 and
Section 5.1) and two smaller families (a tiny correctness case and a
Mixtral-8x7B-shaped layer).  Micro-batches stand for token batches arriving
independently from attention DP groups (Section 3.3); each runs on its own CUDA
stream with no host barrier between them (Section 3.4.2).
"""
from dataclasses import dataclass, field, asdict
from typing import List, Optional

GATING = {"softmax": 0, "softmax_renorm": 1, "sigmoid_grouped": 2}
DTYPE = {"bf16": 0, "fp8_e4m3_block128": 1}


@dataclass(frozen=True)
class LayerConfig:
    name: str
    hidden: int            # H
    n_experts: int         # E routed experts
    top_k: int             # k
    inter: int             # I, routed expert intermediate
    n_shared: int          # 0 or 1
    shared_inter: int      # I_s
    gating: str
    n_groups: int = 1
    topk_groups: int = 1
    route_scale: float = 1.0
    dtype: str = "bf16"
    microbatches: List[int] = field(default_factory=list)
    zipf_s: Optional[float] = None   # expert-popularity skew of the inputs
    # strength of the Zipf logit bias: logit e carries zipf_beta * ln p_pi(e).
    # Calibrated so that the realised shares of the routed (token, slot) pairs
    # follow r^-zipf_s: the exponent fitted to ranks 2..64 of the stress
    # workload's routing on a GB300 is 1.069 at 0.60, 1.104 at 0.62, 1.119 at
    # 0.63 and 1.754 at 1.0 (python -m paper_2606_22541_gb300.zipf_calibrate);
    # the top ranks stay below Zipf's because top-8 routing caps one expert at
    # 1/8 of the pairs.
    zipf_beta: float = 0.62
    seed: int = 1000

    @property
    def n_tokens(self):
        return sum(self.microbatches)

    @property
    def max_microbatch(self):
        return max(self.microbatches) if self.microbatches else 0

    def oracle_cfg(self):
        """Plain mapping handed to the oracle."""
        return dict(n_experts=self.n_experts, top_k=self.top_k, gating=self.gating,
                    n_groups=self.n_groups, topk_groups=self.topk_groups,
                    route_scale=self.route_scale)

    def flops_per_token(self):
        """Multiply-adds x 2 of the expert FFNs (router excluded)."""
        return 6 * self.hidden * self.inter * self.top_k + 6 * self.hidden * self.shared_inter * self.n_shared

    def router_flops_per_token(self):
        return 2 * self.hidden * self.n_experts

    def as_dict(self):
        return asdict(self)


def _stress_lengths(seed, count=8, mu=7.5, sigma=1.0, lo=128, hi=16384):
    """The recipe of the stress workload's micro-batch lengths: round(lognormal
    (mu, sigma)) clipped to [lo, hi] from numpy's PCG64 stream.  numpy does
    not keep its lognormal stream stable across versions, so the workload uses
    the lengths this recipe gave once (STRESS_LENGTHS), not a fresh draw."""
    import numpy as np
    rng = np.random.Generator(np.random.PCG64(seed))
    v = np.round(rng.lognormal(mu, sigma, size=count)).astype(int)
    return [int(min(max(a, lo), hi)) for a in v]


# _stress_lengths(1003) with numpy 2.5
STRESS_LENGTHS = [4014, 1179, 8045, 5228, 362, 1108, 2591, 5185]


TINY = LayerConfig("tiny", hidden=256, n_experts=8, top_k=2, inter=128, n_shared=0,
                   shared_inter=0, gating="softmax", microbatches=[96, 160], seed=1000)
MIXTRAL = LayerConfig("mixtral", hidden=4096, n_experts=8, top_k=2, inter=14336, n_shared=0,
                      shared_inter=0, gating="softmax_renorm",
                      microbatches=[1024, 1536, 2048, 3584], seed=1001)
DSV3 = LayerConfig("dsv3_bf16", hidden=7168, n_experts=256, top_k=8, inter=2048, n_shared=1,
                   shared_inter=2048, gating="sigmoid_grouped", n_groups=8, topk_groups=4,
                   route_scale=2.5, microbatches=[4096] * 4, seed=1002)
STRESS = LayerConfig("dsv3_stress", hidden=7168, n_experts=256, top_k=8, inter=2048, n_shared=1,
                     shared_inter=2048, gating="sigmoid_grouped", n_groups=8, topk_groups=4,
                     route_scale=2.5, microbatches=list(STRESS_LENGTHS), zipf_s=1.1, seed=1003)
DSV3_FP8 = LayerConfig("dsv3_fp8", hidden=7168, n_experts=256, top_k=8, inter=2048, n_shared=1,
                       shared_inter=2048, gating="sigmoid_grouped", n_groups=8, topk_groups=4,
                       route_scale=2.5, dtype="fp8_e4m3_block128", microbatches=[4096] * 8,
                       zipf_s=1.1, seed=1004)

# Profiling case of the DeepSeek-V3 layer's grouped GEMMs: the same per-expert
# shape (M_e ~ 128 rows, K = 7168, N = 2 x 2048) with 32 experts, so one
# launch's weights (2.8 GB) exceed L2 while the device holds a few GB.
DSV3_E32 = LayerConfig("dsv3_e32_profile", hidden=7168, n_experts=32, top_k=8, inter=2048, n_shared=1,
                       shared_inter=2048, gating="sigmoid_grouped", n_groups=8, topk_groups=4,
                       route_scale=2.5, microbatches=[512], seed=1002)

DSV3_FP8_E32 = LayerConfig("dsv3_fp8_e32_profile", hidden=7168, n_experts=32, top_k=8, inter=2048, n_shared=1,
                           shared_inter=2048, gating="sigmoid_grouped", n_groups=8, topk_groups=4,
                           route_scale=2.5, dtype="fp8_e4m3_block128", microbatches=[512], seed=1004)

# Profiling case of the grouped GEMMs where they are bound by the tensor core:
# the DeepSeek-V3 expert shape with 32 experts and 4096 tokens, i.e. ~1024 rows
# per expert (the regime of several micro-batches aggregated into one GEMM);
# 2.8 GB of weights and ~0.9 GB of activations on the device.
DSV3_E32_COMPUTE = LayerConfig("dsv3_e32_compute_profile", hidden=7168, n_experts=32, top_k=8, inter=2048,
                               n_shared=1, shared_inter=2048, gating="sigmoid_grouped", n_groups=8,
                               topk_groups=4, route_scale=2.5, microbatches=[4096], seed=1005)

# Profiling case of route, dispatch and combine: the DeepSeek-V3 routing shape
# (H = 7168, 256 experts, top-8, grouped sigmoid, 4096 tokens), whose bytes do
# not depend on the expert FFN width, with a narrow FFN (I = 256) so the device
# holds 2.8 GB of weights.
DSV3_ROUTING = LayerConfig("dsv3_routing_profile", hidden=7168, n_experts=256, top_k=8, inter=256, n_shared=1,
                           shared_inter=256, gating="sigmoid_grouped", n_groups=8, topk_groups=4,
                           route_scale=2.5, microbatches=[4096], seed=1002)

CONFIGS = {c.name: c for c in (TINY, MIXTRAL, DSV3, STRESS, DSV3_FP8, DSV3_E32, DSV3_E32_COMPUTE, DSV3_FP8_E32,
                               DSV3_ROUTING)}
