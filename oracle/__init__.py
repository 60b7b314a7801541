"""Float64 CPU oracle of the expert-side MoE layer of ASAP's data-parallel
prefill path (top-k gating, per-expert counts and offsets, dispatch, grouped
SwiGLU expert FFN with a shared expert, weighted combine).

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and
bench.py's CPU-baseline leg (and its ``--impl reference`` arm) may import,
call or execute anything in this package.  It shares no code with the CUDA
path: it imports neither the package nor its input generators, and reads
nothing but the arrays it is handed.

Parity status: every function here is pinned by ``tests/test_oracle_pins.py``
against brute force, closed forms, library conversions or a hand-worked
example, except the numerics of the full layer beyond those special cases,
for which the paper prints no worked example (the fp64 definition is the
authority there).
"""
from .formats import bf16_bits_to_f64, e4m3_bits_to_f64, round_to_e4m3_sat, E4M3_MAX
from .gating import (router_logits, route, route_token_softmax,
                     route_token_sigmoid_grouped, logit_error_bound,
                     token_decided, token_feasible, sigmoid)
from .layer import (expert_counts, expert_offsets, permutation, dispatch, silu,
                    swiglu, expert_ffn, combine, moe_layer, moe_layer_tokens,
                    moe_layer_tokens_by_expert,
                    quantize_rows_e4m3, dequant_blocks, swiglu_fp8,
                    moe_layer_tokens_fp8, moe_layer_tokens_fp8_by_expert)
