"""Seeded synthetic inputs shared by the oracle-based tests and the CUDA path.

This module only draws numbers and names tensors: it holds none of the method's
arithmetic (no LayerNorm, attention, MLP, loss or optimizer).  Both the fp64
oracle (through the tests) and the CUDA library receive exactly the arrays made
here.

Workload recipe (stands in for the OpenWebText pre-training corpus of Sec. 5.1):
  * token ids: one stream of B*(T+1) ids drawn uniformly over [0, V) by
    ``numpy.random.default_rng(seed)``; inputs are ``stream[:, :T]`` and
    targets ``stream[:, 1:]`` (next-token prediction);
  * weights: every matrix and embedding ~ N(0, 0.02) drawn in fp64 and rounded
    to fp32; the GPT-2-small shape additionally scales W_o and W_down by
    1/sqrt(2L); LayerNorm gamma = 1, beta = 0; every bias = 0.

The five named shapes are the decoder stacks the paper trains (GPT-2 sizes,
Sec. 5.1 and App. A) plus a tiny stack for fp32 debugging.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

VARIANTS = ("gpt", "fal", "falplus")
# The paper's comparison blocks (Sec. 5.1 baselines, App. D ablations).
COMPARISON_VARIANTS = ("parallel", "ablation1", "ablation2")
ALL_VARIANTS = VARIANTS + COMPARISON_VARIANTS


@dataclasses.dataclass(frozen=True)
class Shape:
    name: str
    layers: int
    d_model: int
    heads: int
    d_ff: int
    seq: int
    batch: int
    vocab: int
    precision: str  # "fp32" (debug path) or "bf16"
    scale_out_proj: bool = False
    kv_heads: int = 0  # key/value heads (GQA groups); 0 = one per query head (MHA)

    @property
    def head_dim(self) -> int:
        return self.d_model // self.heads

    @property
    def kv(self) -> int:
        return self.kv_heads or self.heads

    @property
    def d_qkv(self) -> int:
        """Width of the fused QKV projection: d_model query columns and kv * head_dim
        key and value columns each."""
        return self.d_model + 2 * self.kv * self.head_dim

    @property
    def tokens(self) -> int:
        return self.batch * self.seq

    def replace(self, **kw) -> "Shape":
        return dataclasses.replace(self, **kw)


SHAPES = {
    "tiny": Shape("tiny", 2, 64, 4, 256, 32, 2, 256, "fp32"),
    "gpt2_small": Shape("gpt2_small", 12, 768, 12, 3072, 1024, 8, 50257, "bf16", True),
    "gpt2_medium": Shape("gpt2_medium", 24, 1024, 16, 4096, 1024, 8, 50257, "bf16"),
    "gpt_1p3b": Shape("gpt_1p3b", 24, 2048, 16, 8192, 2048, 4, 50257, "bf16"),
    "gpt2_xl": Shape("gpt2_xl", 48, 1600, 25, 6400, 1024, 8, 50257, "bf16"),
}


def model_flops_per_step(s: Shape) -> float:
    """Algorithmic training FLOPs of one step (forward + backward, no recompute).

    6 * tokens * (per-layer matmul parameters + tied LM head) plus causal
    attention counted at half of the dense 12*T*d per token and layer.
    """
    bt, d, f, L = s.tokens, s.d_model, s.d_ff, s.layers
    return 6.0 * bt * (L * (4 * d * d + 2 * d * f) + d * s.vocab) + 6.0 * bt * L * s.seq * d


def param_specs(variant: str, s: Shape, reuse: int = 1, separate_ln2: bool = False):
    """Canonical list of (name, shape, decayed) for a variant and shape.

    Layers are numbered from 0 (the paper's block 1 is ``h0``).  Weight
    matrices are stored [out, in].  Weight decay applies to matrices and
    embeddings only.  ``reuse`` (FAL+ only) is the paper's index k >= 1 of the
    block whose attention output later blocks add; blocks after it carry their
    own LayerNorm ``lnF`` on it.  ``separate_ln2`` (FAL only) gives every block
    a LayerNorm ``ln2`` of its own for the MLP input.
    """
    if variant not in ALL_VARIANTS:
        raise ValueError(f"unknown variant {variant!r}")
    if reuse < 1 or (reuse != 1 and variant != "falplus") or (separate_ln2 and variant != "fal"):
        raise ValueError("reuse applies to FAL+ and separate_ln2 to FAL")
    d, f, V, T, L = s.d_model, s.d_ff, s.vocab, s.seq, s.layers
    dq = s.d_qkv
    specs = [("wte", (V, d), True), ("wpe", (T, d), True)]
    for i in range(L):
        p = f"h{i}."
        specs += [
            (p + "ln1.g", (d,), False), (p + "ln1.b", (d,), False),
            (p + "attn.w_qkv", (dq, d), True), (p + "attn.b_qkv", (dq,), False),
            (p + "attn.w_o", (d, d), True), (p + "attn.b_o", (d,), False),
        ]
        if variant in ("gpt", "falplus") or (variant == "ablation2" and i == 0) or separate_ln2:
            specs += [(p + "ln2.g", (d,), False), (p + "ln2.b", (d,), False)]
        if variant == "falplus" and i >= reuse:
            specs += [(p + "lnF.g", (d,), False), (p + "lnF.b", (d,), False)]
        if variant == "ablation1":
            specs += [(p + "lnA.g", (d,), False), (p + "lnA.b", (d,), False)]
        specs += [
            (p + "mlp.w_up", (f, d), True), (p + "mlp.b_up", (f,), False),
            (p + "mlp.w_down", (d, f), True), (p + "mlp.b_down", (d,), False),
        ]
    if variant == "fal":
        specs += [("lnF.g", (d,), False), ("lnF.b", (d,), False)]
    specs += [("lnf.g", (d,), False), ("lnf.b", (d,), False)]
    return specs


def init_params(variant: str, s: Shape, seed: int = 0, std: float = 0.02, **spec_kw):
    """Seeded N(0, std) weights (fp64 draw rounded to fp32), LN gamma=1/beta=0, zero biases."""
    rng = np.random.default_rng([seed, 1])
    out = {}
    for name, shape, _ in param_specs(variant, s, **spec_kw):
        leaf = name.rsplit(".", 1)[-1]
        if name in ("wte", "wpe") or leaf.startswith("w_"):
            sd = std
            if s.scale_out_proj and leaf in ("w_o", "w_down"):
                sd = std / math.sqrt(2 * s.layers)
            out[name] = (rng.standard_normal(shape) * sd).astype(np.float32)
        elif leaf == "g":
            out[name] = np.ones(shape, np.float32)
        else:
            out[name] = np.zeros(shape, np.float32)
    return out


def perturb_params(params, seed: int, scale: float = 0.05):
    """Add seeded noise to every LN gamma/beta and bias so that no term of the
    model is trivially zero (used by parity tests; weights stay as drawn)."""
    rng = np.random.default_rng([seed, 2])
    out = {}
    for name, a in params.items():
        leaf = name.rsplit(".", 1)[-1]
        if leaf in ("g", "b") or leaf.startswith("b_"):
            out[name] = (a.astype(np.float64) + rng.standard_normal(a.shape) * scale).astype(np.float32)
        else:
            out[name] = a
    return out


def make_tokens(s: Shape, seed: int = 0):
    """tokens, targets: int32 [B, T], from one uniform stream of B*(T+1) ids."""
    rng = np.random.default_rng([seed, 0])
    stream = rng.integers(0, s.vocab, size=(s.batch, s.seq + 1), dtype=np.int64).astype(np.int32)
    return np.ascontiguousarray(stream[:, :-1]), np.ascontiguousarray(stream[:, 1:])


def adamw_hparams():
    """AdamW settings: lr and weight decay from App. A (1e-4, 1e-3); betas and
    eps are the common defaults (the paper does not state them)."""
    return dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=1e-3)
