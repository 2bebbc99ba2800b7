"""Seeded synthetic inputs for the 1.5-SPSA parameter-space step.

This module only produces inputs: parameter-set shapes, initial weights, loss
triples and the quadratic test problem. It holds none of the method's
arithmetic, so both the CUDA path and the CPU oracle can be fed from it.

The parameter sets mirror the tensor shapes of the models the paper trains
(OPT-1.3B/13B/30B and Qwen3-8B, Sec. 5.1-5.2); no trained weights are used:
every weight is drawn from N(0, 0.02^2).
"""
from dataclasses import dataclass

import numpy as np

DT_F32, DT_BF16, DT_F16 = 0, 1, 2

# 64-bit step seed of step s: STEP_SEED_BASE + s.
STEP_SEED_BASE = 0x15E5A0000


def step_seed(s: int) -> int:
    return STEP_SEED_BASE + int(s)


@dataclass(frozen=True)
class ParamSet:
    name: str
    shapes: tuple          # tuple of (tensor name, numel)
    dtype: int             # DT_* of every tensor
    K: int                 # probes per step
    eps: float = 1e-3

    @property
    def numels(self):
        return [n for _, n in self.shapes]

    @property
    def d(self) -> int:
        return int(sum(self.numels))

    @property
    def bytes_per_elem(self) -> int:
        return 4 if self.dtype == DT_F32 else 2


def opt_shapes(n_layers, d_model, ffn, vocab=50272, positions=2050):
    """OPT decoder: token + learned position embeddings (tied output head),
    per layer q/k/v/out projections with biases, two LayerNorms (weight and
    bias), fc1/fc2 with biases; a final LayerNorm."""
    D, F = d_model, ffn
    s = [("embed_tokens", vocab * D), ("embed_positions", positions * D)]
    for i in range(n_layers):
        p = f"layers.{i}."
        for proj in ("q_proj", "k_proj", "v_proj", "out_proj"):
            s += [(p + proj + ".weight", D * D), (p + proj + ".bias", D)]
        s += [(p + "self_attn_layer_norm.weight", D), (p + "self_attn_layer_norm.bias", D)]
        s += [(p + "fc1.weight", F * D), (p + "fc1.bias", F)]
        s += [(p + "fc2.weight", D * F), (p + "fc2.bias", D)]
        s += [(p + "final_layer_norm.weight", D), (p + "final_layer_norm.bias", D)]
    s += [("final_layer_norm.weight", D), ("final_layer_norm.bias", D)]
    return tuple(s)


def qwen3_shapes(n_layers=36, hidden=4096, inter=12288, n_q=32, n_kv=8, head_dim=128, vocab=151936):
    """Qwen3 decoder: untied embedding and LM head, per layer q/k/v/o
    projections without bias, per-head q_norm/k_norm (QK-norm), SwiGLU
    gate/up/down, two RMSNorm weights; a final RMSNorm."""
    H, I = hidden, inter
    s = [("embed_tokens", vocab * H)]
    for i in range(n_layers):
        p = f"layers.{i}."
        s += [(p + "q_proj.weight", n_q * head_dim * H), (p + "k_proj.weight", n_kv * head_dim * H),
              (p + "v_proj.weight", n_kv * head_dim * H), (p + "o_proj.weight", H * n_q * head_dim),
              (p + "q_norm.weight", head_dim), (p + "k_norm.weight", head_dim),
              (p + "gate_proj.weight", I * H), (p + "up_proj.weight", I * H), (p + "down_proj.weight", H * I),
              (p + "input_layernorm.weight", H), (p + "post_attention_layernorm.weight", H)]
    s += [("norm.weight", H), ("lm_head.weight", vocab * H)]
    return tuple(s)


TINY = ParamSet("tiny-quadratic-fp32-d2^20", (("theta", 1 << 20),), DT_F32, K=8, eps=1e-3)
OPT_1_3B = ParamSet("opt-1.3b-shape-bf16", opt_shapes(24, 2048, 8192), DT_BF16, K=16)
QWEN3_8B = ParamSet("qwen3-8b-shape-bf16", qwen3_shapes(), DT_BF16, K=64)
OPT_13B = ParamSet("opt-13b-shape-bf16", opt_shapes(40, 5120, 20480), DT_BF16, K=128)
OPT_30B = ParamSet("opt-30b-shape-fp16", opt_shapes(48, 7168, 28672), DT_F16, K=256)

CONFIGS = {p.name: p for p in (TINY, OPT_1_3B, QWEN3_8B, OPT_13B, OPT_30B)}
BY_KEY = {"tiny": TINY, "opt-1.3b": OPT_1_3B, "qwen3-8b": QWEN3_8B, "opt-13b": OPT_13B, "opt-30b": OPT_30B}

# Small-workload constants.
TINY_LR = 1e-2
TINY_STEPS = 10


def tiny_theta(d=1 << 20) -> np.ndarray:
    """theta ~ N(0, 0.02^2), fp32, from numpy default_rng(0)."""
    return (np.random.default_rng(0).standard_normal(d) * 0.02).astype(np.float32)


def tiny_curvatures(d=1 << 20) -> np.ndarray:
    """a_i log-uniform in [1e-2, 1e2], fp32, from numpy default_rng(1)."""
    return (10.0 ** np.random.default_rng(1).uniform(-2.0, 2.0, d)).astype(np.float32)


def synthetic_losses(K: int, step: int) -> np.ndarray:
    """Seeded loss triples (K rows of L+, L-, L0) standing in for forward
    passes: one clean loss L0 ~ U(2, 3) per step; per probe a signal
    g ~ U(0, 0.05) and two independent noises h+, h- ~ U(0, 0.01);
    L+ = L0 + g + h+, L- = L0 - g + h-."""
    rng = np.random.default_rng(1000 + int(step))
    l0 = rng.uniform(2.0, 3.0)
    g = rng.uniform(0.0, 0.05, K)
    hp = rng.uniform(0.0, 0.01, K)
    hm = rng.uniform(0.0, 0.01, K)
    out = np.empty((K, 3), dtype=np.float64)
    out[:, 0] = l0 + g + hp
    out[:, 1] = l0 - g + hm
    out[:, 2] = l0
    return out


def random_storage(rng: np.random.Generator, n: int, dtype: int, scale=0.02) -> np.ndarray:
    """n weights ~ N(0, scale^2) as raw storage: float32, or the uint16 bit
    patterns of bf16 / fp16 (bf16 via truncation of an fp32 draw, fp16 via
    numpy's float16 cast; any bit pattern is a valid input)."""
    x = (rng.standard_normal(n) * scale).astype(np.float32)
    if dtype == DT_F32:
        return x
    if dtype == DT_F16:
        return x.astype(np.float16).view(np.uint16)
    return (x.view(np.uint32) >> 16).astype(np.uint16)


def torch_dtype(dtype: int):
    import torch
    return {DT_F32: torch.float32, DT_BF16: torch.bfloat16, DT_F16: torch.float16}[dtype]


def allocate_params(ps: ParamSet, device="cuda", seed_base=1234, view_offset=0):
    """Separate device tensors shaped like `ps`, each ~ N(0, 0.02^2) drawn on
    the device from its own torch generator (seed_base + tensor index). With
    view_offset > 0 every tensor is a view that many elements into its own
    allocation (off the 32-byte grid unless the offset is a multiple of 32
    bytes)."""
    import torch
    out = []
    tdt = torch_dtype(ps.dtype)
    for i, (_, n) in enumerate(ps.shapes):
        if view_offset:
            t = torch.empty(n + view_offset, dtype=tdt, device=device)[view_offset:]
        else:
            t = torch.empty(n, dtype=tdt, device=device)
        g = torch.Generator(device=device)
        g.manual_seed(seed_base + i)
        t.normal_(0.0, 0.02, generator=g)
        out.append(t)
    return out
