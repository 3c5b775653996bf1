"""Plain fp64 CPU oracle for GPT (Pre-LN), FAL and FAL+ decoder stacks.

TEST INFRASTRUCTURE: only the tests, the package's smoke check and the
benchmark's CPU-baseline leg may import this module.  The CUDA library never
calls it and shares no code with it.

Everything is the literal definition of the paper's equations in float64 with
NumPy (matmul is the only library primitive used):

  * GPT / Pre-LN block, Eq. 1 (Sec. 2):
        X_{i+1} = X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i + MHA_i(LN(X_i))))
  * FAL block, Eq. 2 (Sec. 4.1), every block i including the first:
        X_{i+1} = X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i) + LN(MHA_1(LN(X_1))))
    with LN(X_i) the same LayerNorm output that feeds MHA_i, and one LayerNorm
    LN_F on the first attention output shared by all blocks (Sec. 4.1: the
    first attention output is normalised a single time).
  * FAL+ block (Sec. 5; App. D.1 equation): block 1 is the standard block;
    block i >= 2 feeds MLP_i(LN(X_i + MHA_i(LN(X_i))) + LN_{F,i}(MHA_1(LN(X_1))))
    with its own LayerNorm LN_{F,i} on the first attention output.
  * Grouped-query attention (App. E, GQA): with G key/value heads, query head
    h attends with the key and value head of its group h // (H / G); G = H is
    multi-head attention.  The fused QKV projection then has d_model query
    columns and G * head_dim key and value columns each.
  * GPT-2 conventions (the paper builds on GPT-2, Sec. 5.1): learned position
    embedding, tied LM head, final LayerNorm, biases on every linear map,
    tanh-approximated GELU, LayerNorm eps 1e-5 with the population variance,
    attention scale 1/sqrt(head_dim), causal mask (key j visible to query t
    iff j <= t), mean token cross-entropy.
  * AdamW (App. A: lr 1e-4, weight decay 1e-3) with bias correction and
    decoupled weight decay on matrices and embeddings; gradient clipping to a
    global L2 norm (App. A clips at 1).
  * The paper's comparison blocks:
      - Parallel (Sec. 5.1 baselines; GPT-J style): X_i + MHA_i(LN(X_i)) +
        MLP_i(LN(X_i)), one LayerNorm feeding both branches;
      - Ablation1 (App. D): X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i) +
        LN(MHA_i(LN(X_i)))), the FAL structure with the block's own attention
        and a LayerNorm LN_{A,i} of its own on it, every block;
      - Ablation2 (App. D): block 1 is the standard block (its printed
        equation drops a parenthesis, read like FAL+'s block 1), every later
        block is the Parallel block;
      - FAL+ reusing block k (App. D "Ablation with Other Layers"): blocks 1..k
        are standard, block i > k adds LN_{F,i}(MHA_k(LN(X_k))); k = 1 is FAL+;
      - FAL with a separate LayerNorm on X_i for the MLP input
        (``separate_ln2``): the other reading of Eq. 2's MLP input, kept here
        only to show that the reading matters.

Parameters are a dict name -> array (names from the shared synthetic-input
module); weight matrices are [out, in].  Parity pins for every function here
live in tests/test_oracle.py.
"""
from __future__ import annotations

import math

import numpy as np

LN_EPS = 1e-5
GELU_C = math.sqrt(2.0 / math.pi)
GELU_A = 0.044715


# ---------------------------------------------------------------- primitives
def layer_norm(x, gamma=None, beta=None, eps=LN_EPS):
    """LN over the last axis; gamma=None gives the bare normalisation."""
    mu = x.mean(-1, keepdims=True)
    var = ((x - mu) ** 2).mean(-1, keepdims=True)
    rstd = 1.0 / np.sqrt(var + eps)
    xhat = (x - mu) * rstd
    y = xhat if gamma is None else xhat * gamma + beta
    return y, (xhat, rstd)


def layer_norm_backward(dy, cache, gamma=None):
    """Returns dx, dgamma, dbeta for y = xhat*gamma + beta (rows = tokens)."""
    xhat, rstd = cache
    g = dy if gamma is None else dy * gamma
    dx = rstd * (g - g.mean(-1, keepdims=True) - xhat * (g * xhat).mean(-1, keepdims=True))
    dgamma = (dy * xhat).reshape(-1, xhat.shape[-1]).sum(0)
    dbeta = dy.reshape(-1, xhat.shape[-1]).sum(0)
    return dx, dgamma, dbeta


def gelu(x):
    return 0.5 * x * (1.0 + np.tanh(GELU_C * (x + GELU_A * x ** 3)))


def gelu_grad(x):
    t = np.tanh(GELU_C * (x + GELU_A * x ** 3))
    return 0.5 * (1.0 + t) + 0.5 * x * (1.0 - t * t) * GELU_C * (1.0 + 3.0 * GELU_A * x * x)


def causal_attention(q, k, v):
    """q, k, v: [B, H, T, hd].  Returns ctx [B, H, T, hd] and P [B, H, T, T]."""
    T, hd = q.shape[-2], q.shape[-1]
    s = q @ np.swapaxes(k, -1, -2) / math.sqrt(hd)
    future = np.triu(np.ones((T, T), dtype=bool), 1)  # key j > query t
    s = np.where(future, -np.inf, s)
    s = s - s.max(-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(-1, keepdims=True)
    return p @ v, p


def causal_attention_backward(dctx, q, k, v, p):
    hd = q.shape[-1]
    dv = np.swapaxes(p, -1, -2) @ dctx
    dp = dctx @ np.swapaxes(v, -1, -2)
    ds = p * (dp - (dp * p).sum(-1, keepdims=True))
    dq = ds @ k / math.sqrt(hd)
    dk = np.swapaxes(ds, -1, -2) @ q / math.sqrt(hd)
    return dq, dk, dv


def cross_entropy(logits, targets):
    """Mean over rows of logsumexp(logits) - logits[target]; also dlogits."""
    n = logits.shape[0]
    mx = logits.max(-1, keepdims=True)
    e = np.exp(logits - mx)
    z = e.sum(-1, keepdims=True)
    lse = (mx + np.log(z))[:, 0]
    loss = float(np.mean(lse - logits[np.arange(n), targets]))
    dlogits = e / z
    dlogits[np.arange(n), targets] -= 1.0
    return loss, dlogits / n


# ---------------------------------------------------------------- the model
VARIANTS = ("gpt", "fal", "falplus", "parallel", "ablation1", "ablation2")


class Config:
    def __init__(self, variant, layers, d_model, heads, d_ff, seq, batch, vocab, reuse=1, separate_ln2=False,
                 kv_heads=0):
        assert variant in VARIANTS
        assert d_model % heads == 0
        assert reuse >= 1 and (reuse == 1 or variant == "falplus")
        assert not separate_ln2 or variant == "fal"
        self.variant, self.layers, self.d_model, self.heads = variant, layers, d_model, heads
        self.d_ff, self.seq, self.batch, self.vocab = d_ff, seq, batch, vocab
        self.reuse, self.separate_ln2 = reuse, separate_ln2
        self.kv_heads = kv_heads or heads
        assert heads % self.kv_heads == 0

    @classmethod
    def from_shape(cls, variant, s, **kw):
        return cls(variant, s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch, s.vocab,
                   kv_heads=getattr(s, "kv_heads", 0), **kw)


def _split_heads(x, B, T, H):
    return x.reshape(B, T, H, -1).transpose(0, 2, 1, 3)


def _merge_heads(x):
    B, H, T, hd = x.shape
    return x.transpose(0, 2, 1, 3).reshape(B * T, H * hd)


def forward(params, cfg, tokens, targets, layers=None):
    """Loss and the saved activations of one training forward pass.

    ``layers`` limits the stack depth (None = cfg.layers)."""
    P = {k: np.asarray(v, dtype=np.float64) for k, v in params.items()}
    B, T = tokens.shape
    d, H = cfg.d_model, cfg.heads
    L = cfg.layers if layers is None else layers
    var = cfg.variant
    X = (P["wte"][tokens] + P["wpe"][:T][None]).reshape(B * T, d)
    cache = {"X": [X], "layers": []}
    a1 = None    # first attention output (FAL), or block k's (FAL+ reusing k)
    k_reuse = cfg.reuse - 1
    for i in range(L):
        w = lambda n: P[f"h{i}.{n}"]
        c = {}
        u, c["ln1"] = layer_norm(X, w("ln1.g"), w("ln1.b"))
        qkv = u @ w("attn.w_qkv").T + w("attn.b_qkv")
        nkv = cfg.kv_heads
        q = _split_heads(qkv[:, :d], B, T, H)
        k = _split_heads(qkv[:, d:d + nkv * (d // H)], B, T, nkv)
        v = _split_heads(qkv[:, d + nkv * (d // H):], B, T, nkv)
        # every query head uses the key / value head of its group
        o, p = causal_attention(q, np.repeat(k, H // nkv, axis=1), np.repeat(v, H // nkv, axis=1))
        ctx = _merge_heads(o)
        a = ctx @ w("attn.w_o").T + w("attn.b_o")
        if i == k_reuse:
            a1 = a
        if var == "fal":
            if i == 0:
                cache["F"], cache["lnF"] = layer_norm(a1, P["lnF.g"], P["lnF.b"])
            if cfg.separate_ln2:
                m, c["ln2"] = layer_norm(X, w("ln2.g"), w("ln2.b"))
                m = m + cache["F"]
            else:
                m = u + cache["F"]
        elif var == "parallel" or (var == "ablation2" and i >= 1):
            m = u
        elif var == "ablation1":
            fa, c["lnA"] = layer_norm(a, w("lnA.g"), w("lnA.b"))
            m = u + fa
        else:  # gpt, falplus, block 1 of ablation2
            Y = X + a
            m, c["ln2"] = layer_norm(Y, w("ln2.g"), w("ln2.b"))
            c["Y"] = Y
            if var == "falplus" and i > k_reuse:
                fa, c["lnF"] = layer_norm(a1, w("lnF.g"), w("lnF.b"))
                m = m + fa
        h = m @ w("mlp.w_up").T + w("mlp.b_up")
        g = gelu(h)
        mlp = g @ w("mlp.w_down").T + w("mlp.b_down")
        X = X + a + mlp
        c.update(u=u, qkv=qkv, q=q, k=k, v=v, p=p, ctx=ctx, a=a, m=m, h=h, g=g)
        cache["layers"].append(c)
        cache["X"].append(X)
    xf, cache["lnf"] = layer_norm(X, P["lnf.g"], P["lnf.b"])
    logits = xf @ P["wte"].T
    loss, dlogits = cross_entropy(logits, targets.reshape(-1))
    cache.update(xf=xf, logits=logits, dlogits=dlogits, a1=a1, tokens=tokens, B=B, T=T, L=L)
    return loss, cache


def backward(params, cfg, cache):
    """Gradients of the mean loss w.r.t. every parameter (manual chain rule)."""
    P = {k: np.asarray(v, dtype=np.float64) for k, v in params.items()}
    B, T, L = cache["B"], cache["T"], cache["L"]
    d, H, var = cfg.d_model, cfg.heads, cfg.variant
    G = {k: np.zeros_like(v) for k, v in P.items()}

    dlogits = cache["dlogits"]
    G["wte"] += dlogits.T @ cache["xf"]
    dxf = dlogits @ P["wte"]
    dX, G["lnf.g"], G["lnf.b"] = layer_norm_backward(dxf, cache["lnf"], P["lnf.g"])

    dF = np.zeros((B * T, d))   # FAL: gradient reaching F = LN_F(a_1)
    da1 = np.zeros((B * T, d))  # FAL+: gradient reaching a_1 (or a_k) through LN_{F,i}
    k_reuse = cfg.reuse - 1
    for i in reversed(range(L)):
        c = cache["layers"][i]
        w = lambda n: P[f"h{i}.{n}"]
        gn = lambda n: f"h{i}.{n}"
        # X_{i+1} = X_i + a + mlp
        dXi = dX.copy()
        da = dX.copy()
        G[gn("mlp.w_down")] = dX.T @ c["g"]
        G[gn("mlp.b_down")] = dX.sum(0)
        dh = (dX @ w("mlp.w_down")) * gelu_grad(c["h"])
        G[gn("mlp.w_up")] = dh.T @ c["m"]
        G[gn("mlp.b_up")] = dh.sum(0)
        dm = dh @ w("mlp.w_up")
        du = np.zeros((B * T, d))
        if var == "fal":
            if cfg.separate_ln2:
                dx2, G[gn("ln2.g")], G[gn("ln2.b")] = layer_norm_backward(dm, c["ln2"], w("ln2.g"))
                dXi += dx2
            else:
                du += dm
            dF += dm
        elif var == "parallel" or (var == "ablation2" and i >= 1):
            du += dm
        elif var == "ablation1":
            du += dm
            dfa, G[gn("lnA.g")], G[gn("lnA.b")] = layer_norm_backward(dm, c["lnA"], w("lnA.g"))
            da += dfa
        else:
            dY, G[gn("ln2.g")], G[gn("ln2.b")] = layer_norm_backward(dm, c["ln2"], w("ln2.g"))
            dXi += dY
            da += dY
            if var == "falplus" and i > k_reuse:
                dfa, G[gn("lnF.g")], G[gn("lnF.b")] = layer_norm_backward(dm, c["lnF"], w("lnF.g"))
                da1 += dfa
        if var == "fal" and i == 0:
            dfa, G["lnF.g"], G["lnF.b"] = layer_norm_backward(dF, cache["lnF"], P["lnF.g"])
            da += dfa
        if var == "falplus" and i == k_reuse:
            da += da1
        G[gn("attn.w_o")] = da.T @ c["ctx"]
        G[gn("attn.b_o")] = da.sum(0)
        dctx = _split_heads(da @ w("attn.w_o"), B, T, H)
        nkv = cfg.kv_heads
        dq, dk, dv = causal_attention_backward(dctx, c["q"], np.repeat(c["k"], H // nkv, axis=1),
                                               np.repeat(c["v"], H // nkv, axis=1), c["p"])
        # a key / value head's gradient sums over the query heads of its group
        dk = dk.reshape(B, nkv, H // nkv, T, -1).sum(2)
        dv = dv.reshape(B, nkv, H // nkv, T, -1).sum(2)
        dqkv = np.concatenate([_merge_heads(dq), _merge_heads(dk), _merge_heads(dv)], axis=1)
        G[gn("attn.w_qkv")] = dqkv.T @ c["u"]
        G[gn("attn.b_qkv")] = dqkv.sum(0)
        du += dqkv @ w("attn.w_qkv")
        dxl, G[gn("ln1.g")], G[gn("ln1.b")] = layer_norm_backward(du, c["ln1"], w("ln1.g"))
        dX = dXi + dxl
    tok = cache["tokens"].reshape(-1)
    np.add.at(G["wte"], tok, dX)
    G["wpe"][:T] += dX.reshape(B, T, d).sum(0)
    return G


def clip_grad_norm(grads, max_norm):
    """Gradient clipping by the global L2 norm over every tensor (App. A clips
    at 1.0): when the norm exceeds max_norm every gradient is scaled by
    max_norm / norm.  Returns the clipped gradients and the norm before
    clipping."""
    norm = math.sqrt(sum(float(np.sum(np.asarray(g, np.float64) ** 2)) for g in grads.values()))
    scale = max_norm / norm if norm > max_norm else 1.0
    return {k: np.asarray(g, np.float64) * scale for k, g in grads.items()}, norm


def adamw_step(params, grads, m, v, t, lr, beta1, beta2, eps, weight_decay, decayed):
    """One AdamW step (t counts from 1).  ``decayed``: set of names that get
    decoupled weight decay.  Returns new (params, m, v) dicts in fp64."""
    newp, newm, newv = {}, {}, {}
    for k in params:
        p = np.asarray(params[k], np.float64)
        g = np.asarray(grads[k], np.float64)
        mk = beta1 * np.asarray(m[k], np.float64) + (1 - beta1) * g
        vk = beta2 * np.asarray(v[k], np.float64) + (1 - beta2) * g * g
        mhat = mk / (1 - beta1 ** t)
        vhat = vk / (1 - beta2 ** t)
        wd = weight_decay if k in decayed else 0.0
        newp[k] = p - lr * (mhat / (np.sqrt(vhat) + eps) + wd * p)
        newm[k], newv[k] = mk, vk
    return newp, newm, newv


def loss_only(params, cfg, tokens, targets, layers=None):
    return forward(params, cfg, tokens, targets, layers)[0]
