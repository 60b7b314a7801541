"""Seeded synthetic inputs for the MoE layer (hidden states, router and expert
weights), shaped like the workloads of the paper's evaluation.

This module holds no arithmetic of the layer itself: it draws normal numbers,
rounds them to the storage formats (bf16 round-to-nearest-even, e4m3 with
block scales for the FP8 configuration) and lays them out.  Both the CUDA path
and the float64 oracle consume exactly the bytes produced here.

Recipe (every workload):
  x   ~ N(0, 1), rounded to bf16
  Wg, Wu ~ N(0, 1/sqrt(H)), Wd ~ N(0, 1/sqrt(I)) (std = 1/sqrt(fan_in)), bf16
  router Wr ~ N(0, 0.02) for the tiny layer, N(0, 1/sqrt(H)) otherwise
  shared expert like a routed one with I_s
  Zipf popularity (skewed workloads): channel 0 of every token is set to 1
  (the rest stays N(0, 1)) and router column 0 to beta (ln p_{pi(e)} - mean),
  p_r ~ r^-s, pi a seeded expert permutation, so logit e carries a bias
  beta ln p_{pi(e)}; beta = cfg.zipf_beta, calibrated on the realised expert
  shares (zipf_calibrate.py).
  FP8: weights drawn as above in fp32, then per 128 x 128 block
  s = amax/448, q = e4m3(w / s) (torch's round-to-nearest-even cast).
Seeds: torch generator on the target device, seed = cfg.seed * 1000 + tensor id.
"""
import numpy as np
import torch


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def randn_bf16(shape, std, seed, device):
    """N(0, std^2) rounded to bf16."""
    g = _gen(device, seed)
    t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(torch.bfloat16)


def _randn_f32(shape, std, seed, device):
    g = _gen(device, seed)
    t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    return t.mul_(std)


def expert_stack_bf16(E, rows, cols, std, seed, device):
    """[E, rows, cols] bf16, drawn one expert at a time (bounded fp32 temp)."""
    out = torch.empty((E, rows, cols), dtype=torch.bfloat16, device=device)
    for e in range(E):
        out[e] = randn_bf16((rows, cols), std, seed * 1000 + e, device)
    return out


def quantize_block128_e4m3(w):
    """fp32 [R, C] -> (e4m3 [R, C], fp32 scales [R/128, C/128]) with
    s = amax/448 per 128 x 128 block (1 for an all-zero block)."""
    R, C = w.shape
    b = w.reshape(R // 128, 128, C // 128, 128)
    amax = b.abs().amax(dim=(1, 3))
    s = torch.where(amax > 0, amax / 448.0, torch.ones_like(amax))
    q = (b / s[:, None, :, None]).clamp_(-448.0, 448.0).to(torch.float8_e4m3fn)
    return q.reshape(R, C), s.contiguous()


def expert_stack_fp8(E, rows, cols, std, seed, device):
    q = torch.empty((E, rows, cols), dtype=torch.float8_e4m3fn, device=device)
    s = torch.empty((E, rows // 128, cols // 128), dtype=torch.float32, device=device)
    for e in range(E):
        q[e], s[e] = quantize_block128_e4m3(_randn_f32((rows, cols), std, seed * 1000 + e, device))
    return q, s


def zipf_logit_bias(E, s, seed):
    """ln p_{pi(e)} - mean, p_r proportional to r^-s (r = 1..E)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    perm = rng.permutation(E)
    r = np.arange(1, E + 1, dtype=np.float64)
    lp = -s * np.log(r)
    lp -= np.log(np.exp(lp).sum())
    b = lp[perm]
    return b - b.mean()


def make_weights(cfg, device):
    """Router, routed-expert and shared-expert weights of one layer."""
    H, E, I, Is = cfg.hidden, cfg.n_experts, cfg.inter, cfg.shared_inter
    base = cfg.seed * 1000
    w = dict(router_w=router_weights_bf16(cfg, device), router_bias=None)
    if cfg.dtype == "bf16":
        w["w_gate"] = expert_stack_bf16(E, I, H, 1 / np.sqrt(H), base + 2, device)
        w["w_up"] = expert_stack_bf16(E, I, H, 1 / np.sqrt(H), base + 3, device)
        w["w_down"] = expert_stack_bf16(E, H, I, 1 / np.sqrt(I), base + 4, device)
        if cfg.n_shared:
            w["sh_gate"] = randn_bf16((Is, H), 1 / np.sqrt(H), base + 5, device)
            w["sh_up"] = randn_bf16((Is, H), 1 / np.sqrt(H), base + 6, device)
            w["sh_down"] = randn_bf16((H, Is), 1 / np.sqrt(Is), base + 7, device)
    else:
        w["w_gate"], w["s_gate"] = expert_stack_fp8(E, I, H, 1 / np.sqrt(H), base + 2, device)
        w["w_up"], w["s_up"] = expert_stack_fp8(E, I, H, 1 / np.sqrt(H), base + 3, device)
        w["w_down"], w["s_down"] = expert_stack_fp8(E, H, I, 1 / np.sqrt(I), base + 4, device)
        if cfg.n_shared:
            sg, ssg = expert_stack_fp8(1, Is, H, 1 / np.sqrt(H), base + 5, device)
            su, ssu = expert_stack_fp8(1, Is, H, 1 / np.sqrt(H), base + 6, device)
            sd, ssd = expert_stack_fp8(1, H, Is, 1 / np.sqrt(Is), base + 7, device)
            w.update(sh_gate=sg[0], sh_s_gate=ssg[0], sh_up=su[0], sh_s_up=ssu[0],
                     sh_down=sd[0], sh_s_down=ssd[0])
    return w


def layer_config(cfg, layer):
    """The configuration whose make_weights draws layer ``layer`` of a model
    with several MoE layers of cfg's shape (layer 0 is cfg itself)."""
    from dataclasses import replace
    return cfg if layer == 0 else replace(cfg, seed=cfg.seed + 7919 * layer)


def make_layer_weights(cfg, n_layers, device):
    """Weights of layers 0 .. n_layers-1, one make_weights dict per layer."""
    return [make_weights(layer_config(cfg, layer), device) for layer in range(n_layers)]


def expert_weights_bf16(cfg, e, device):
    """(Wg_e [I, H], Wu_e [I, H], Wd_e [H, I]) of one routed expert, the same
    values make_weights draws for it (bf16 configurations)."""
    H, I = cfg.hidden, cfg.inter
    base = cfg.seed * 1000
    return (randn_bf16((I, H), 1 / np.sqrt(H), (base + 2) * 1000 + e, device),
            randn_bf16((I, H), 1 / np.sqrt(H), (base + 3) * 1000 + e, device),
            randn_bf16((H, I), 1 / np.sqrt(I), (base + 4) * 1000 + e, device))


def router_weights_bf16(cfg, device):
    """The router weights make_weights draws (bf16 configurations)."""
    H, E = cfg.hidden, cfg.n_experts
    r_std = 0.02 if cfg.name == "tiny" else 1.0 / np.sqrt(H)
    wr = randn_bf16((E, H), r_std, cfg.seed * 1000 + 1, device)
    if cfg.zipf_s is not None:
        b = torch.tensor(cfg.zipf_beta * zipf_logit_bias(E, cfg.zipf_s, cfg.seed), dtype=torch.float32,
                         device=device)
        wr[:, 0] = b.to(torch.bfloat16)
    return wr


def shared_weights_bf16(cfg, device):
    H, Is = cfg.hidden, cfg.shared_inter
    base = cfg.seed * 1000
    return (randn_bf16((Is, H), 1 / np.sqrt(H), base + 5, device),
            randn_bf16((Is, H), 1 / np.sqrt(H), base + 6, device),
            randn_bf16((H, Is), 1 / np.sqrt(Is), base + 7, device))


def make_tokens(cfg, n, mb_index, device):
    """Hidden states of micro-batch ``mb_index`` ([n, H] bf16)."""
    x = randn_bf16((n, cfg.hidden), 1.0, cfg.seed * 1000 + 100 + mb_index, device)
    if cfg.zipf_s is not None:
        x[:, 0] = 1.0
    return x


def make_microbatches(cfg, device, lengths=None):
    """One hidden-state tensor per micro-batch of the configuration."""
    lengths = cfg.microbatches if lengths is None else lengths
    return [make_tokens(cfg, n, i, device) for i, n in enumerate(lengths)]


def small_variant(cfg, **changes):
    """A copy of a configuration with some fields changed (test shapes)."""
    from dataclasses import replace
    return replace(cfg, **changes)
