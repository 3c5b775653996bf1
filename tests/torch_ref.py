"""Independent fp64 CPU model built from torch.nn library layers (test helper only).

It composes F.layer_norm, F.linear, F.scaled_dot_product_attention, F.gelu and
F.cross_entropy according to the block equations (Eq. 1, Eq. 2, the FAL+
equation of App. D.1) and differentiates with autograd.  It shares no code with
the oracle and none with the CUDA library; tests use it to pin the oracle's
forward composition and its manual backward.
"""
from __future__ import annotations

import torch
import torch.nn.functional as Fn


def _ln(x, p, name):
    d = x.shape[-1]
    return Fn.layer_norm(x, (d,), p[name + ".g"], p[name + ".b"], eps=1e-5)


def _mha(x, p, i, H, G=None):
    B, T, d = x.shape
    G = G or H
    hd = d // H
    qkv = Fn.linear(x, p[f"h{i}.attn.w_qkv"], p[f"h{i}.attn.b_qkv"])
    q, k, v = qkv.split([d, G * hd, G * hd], dim=-1)
    sh = lambda t, n: t.reshape(B, T, n, hd).transpose(1, 2)
    # grouped-query attention: each key / value head serves H / G query heads
    rep = lambda t: sh(t, G).repeat_interleave(H // G, dim=1)
    o = Fn.scaled_dot_product_attention(sh(q, H), rep(k), rep(v), is_causal=True)
    o = o.transpose(1, 2).reshape(B, T, d)
    return Fn.linear(o, p[f"h{i}.attn.w_o"], p[f"h{i}.attn.b_o"])


def _mlp(x, p, i):
    h = Fn.linear(x, p[f"h{i}.mlp.w_up"], p[f"h{i}.mlp.b_up"])
    return Fn.linear(Fn.gelu(h, approximate="tanh"), p[f"h{i}.mlp.w_down"], p[f"h{i}.mlp.b_down"])


def model_loss(params, variant, heads, tokens, targets, layers, parallel=False, reuse=1, separate_ln2=False,
               kv_heads=None):
    """Mean next-token loss.  ``parallel=True`` builds the GPT-J style block
    X + MHA(LN1(X)) + MLP(LN1(X)) (no first-attention term), as does the
    variant "parallel"; "ablation1" / "ablation2" are App. D's ablations;
    ``reuse`` = k makes FAL+ add block k's attention; ``separate_ln2`` gives
    FAL's MLP input a LayerNorm of its own."""
    p = params
    tok = torch.as_tensor(tokens, dtype=torch.long)
    B, T = tok.shape
    X = Fn.embedding(tok, p["wte"]) + p["wpe"][:T][None]
    a1 = None
    for i in range(layers):
        n1 = _ln(X, p, f"h{i}.ln1")
        a = _mha(n1, p, i, heads, kv_heads)
        if i == reuse - 1:
            a1 = a
        if parallel or variant == "parallel" or (variant == "ablation2" and i >= 1):
            m = n1
        elif variant == "ablation1":
            m = n1 + _ln(a, p, f"h{i}.lnA")
        elif variant == "fal":
            m = (_ln(X, p, f"h{i}.ln2") if separate_ln2 else n1) + _ln(a1, p, "lnF")
        else:
            m = _ln(X + a, p, f"h{i}.ln2")
            if variant == "falplus" and i >= reuse:
                m = m + _ln(a1, p, f"h{i}.lnF")
        X = X + a + _mlp(m, p, i)
    xf = _ln(X, p, "lnf")
    logits = xf @ p["wte"].T
    return Fn.cross_entropy(logits.reshape(B * T, -1), torch.as_tensor(targets, dtype=torch.long).reshape(-1))


def loss_and_grads(params_np, variant, heads, tokens, targets, layers, parallel=False, **kw):
    p = {k: torch.tensor(v, dtype=torch.float64, requires_grad=True) for k, v in params_np.items()}
    loss = model_loss(p, variant, heads, tokens, targets, layers, parallel, **kw)
    loss.backward()
    return float(loss), {k: t.grad.numpy() if t.grad is not None else torch.zeros_like(t).numpy() for k, t in p.items()}
