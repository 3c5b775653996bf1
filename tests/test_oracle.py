"""Pins for the fp64 oracle against things other than itself.

* library routines: torch F.layer_norm, F.gelu(tanh), scaled_dot_product_attention,
  F.cross_entropy, nn.TransformerEncoderLayer (Pre-LN = GPT block, Eq. 1),
  torch.optim.AdamW;
* closed forms and special cases (LayerNorm moments, GELU odd-part identity,
  attention with T=1 or q=0, loss at uniform logits = ln V);
* central finite differences of the oracle's own forward (manual backward);
* a third, autograd implementation built from torch.nn.functional layers;
* the structural invariants the paper states: block 1's attention is shared by
  all variants, FAL's MLP input never depends on the block's own MHA (Sec. 4.2),
  FAL+ reduces to GPT when every LN_{F,i} is switched off, FAL reduces to the
  parallel block when LN_F is switched off.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

from oracle import fal_oracle as O
from paper_2510_14614_gb300 import synth
import torch_ref

torch.set_default_dtype(torch.float64)

TINY = synth.SHAPES["tiny"]


def _params(variant, s=TINY, seed=0, perturb=True):
    p = synth.init_params(variant, s, seed)
    return synth.perturb_params(p, seed) if perturb else p


def _union_params(s=TINY, seed=0):
    """One value per name across all variants, so shared weights are equal."""
    out = {}
    for v in synth.VARIANTS:
        for k, a in _params(v, s, seed).items():
            out.setdefault(k, a)
    return out


def _pick(union, variant, s=TINY):
    return {n: union[n] for n, _, _ in synth.param_specs(variant, s)}


# ------------------------------------------------------------------ primitives
def test_layer_norm_matches_library_and_moments():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((7, 48)) * 3 + 1
    g, b = rng.standard_normal(48), rng.standard_normal(48)
    y, (xhat, rstd) = O.layer_norm(x, g, b)
    ref = Fn.layer_norm(torch.tensor(x), (48,), torch.tensor(g), torch.tensor(b), eps=1e-5).numpy()
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(xhat.mean(-1), 0, atol=1e-12)
    # population variance with eps: var(xhat) = var / (var + eps)
    v = x.var(-1)
    np.testing.assert_allclose(xhat.var(-1), v / (v + 1e-5), rtol=1e-12)


def test_layer_norm_backward_matches_autograd():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((5, 32))
    g, b, dy = rng.standard_normal(32), rng.standard_normal(32), rng.standard_normal((5, 32))
    _, c = O.layer_norm(x, g, b)
    dx, dg, db = O.layer_norm_backward(dy, c, g)
    tx, tg, tb = (torch.tensor(a, requires_grad=True) for a in (x, g, b))
    Fn.layer_norm(tx, (32,), tg, tb, eps=1e-5).backward(torch.tensor(dy))
    for a, t in ((dx, tx), (dg, tg), (db, tb)):
        np.testing.assert_allclose(a, t.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_gelu_library_and_identities():
    x = np.linspace(-6, 6, 241)
    ref = Fn.gelu(torch.tensor(x), approximate="tanh").numpy()
    np.testing.assert_allclose(O.gelu(x), ref, rtol=1e-13, atol=1e-15)
    # gelu(x) - gelu(-x) = x exactly (0.5x(1+t) + 0.5x(1-t))
    np.testing.assert_allclose(O.gelu(x) - O.gelu(-x), x, atol=1e-14)
    assert O.gelu(np.array(0.0)) == 0.0
    tx = torch.tensor(x, requires_grad=True)
    Fn.gelu(tx, approximate="tanh").sum().backward()
    np.testing.assert_allclose(O.gelu_grad(x), tx.grad.numpy(), rtol=1e-12, atol=1e-14)


def test_attention_special_cases():
    rng = np.random.default_rng(3)
    q, k, v = (rng.standard_normal((2, 3, 1, 8)) for _ in range(3))
    ctx, _ = O.causal_attention(q, k, v)
    np.testing.assert_allclose(ctx, v, atol=1e-15)          # T = 1: ctx = v
    T = 9
    q = np.zeros((1, 2, T, 4))
    k, v = rng.standard_normal((1, 2, T, 4)), rng.standard_normal((1, 2, T, 4))
    ctx, _ = O.causal_attention(q, k, v)
    running_mean = np.cumsum(v, axis=2) / np.arange(1, T + 1)[None, None, :, None]
    np.testing.assert_allclose(ctx, running_mean, rtol=1e-13, atol=1e-14)


def test_attention_matches_sdpa_forward_and_backward():
    rng = np.random.default_rng(4)
    q, k, v, do = (rng.standard_normal((2, 3, 17, 8)) for _ in range(4))
    ctx, p = O.causal_attention(q, k, v)
    dq, dk, dv = O.causal_attention_backward(do, q, k, v, p)
    tq, tk, tv = (torch.tensor(a, requires_grad=True) for a in (q, k, v))
    o = Fn.scaled_dot_product_attention(tq, tk, tv, is_causal=True)
    o.backward(torch.tensor(do))
    np.testing.assert_allclose(ctx, o.detach().numpy(), rtol=1e-11, atol=1e-13)
    for a, t in ((dq, tq), (dk, tk), (dv, tv)):
        np.testing.assert_allclose(a, t.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_cross_entropy_library_and_uniform():
    rng = np.random.default_rng(5)
    logits, tgt = rng.standard_normal((11, 37)) * 2, rng.integers(0, 37, 11)
    loss, dl = O.cross_entropy(logits, tgt)
    tl = torch.tensor(logits, requires_grad=True)
    ref = Fn.cross_entropy(tl, torch.tensor(tgt))
    ref.backward()
    assert abs(loss - float(ref.detach())) < 1e-12
    np.testing.assert_allclose(dl, tl.grad.numpy(), rtol=1e-10, atol=1e-14)
    loss_u, _ = O.cross_entropy(np.full((4, 37), 0.3), tgt[:4])
    assert abs(loss_u - math.log(37)) < 1e-13


def test_adamw_matches_torch_optim():
    rng = np.random.default_rng(6)
    hp = synth.adamw_hparams()
    hp = dict(hp, lr=1e-2, weight_decay=0.1)  # large enough to see every term
    params = {"w": rng.standard_normal((4, 3)), "b": rng.standard_normal(3)}
    tw, tb = torch.tensor(params["w"], requires_grad=True), torch.tensor(params["b"], requires_grad=True)
    opt = torch.optim.AdamW([{"params": [tw], "weight_decay": hp["weight_decay"]},
                             {"params": [tb], "weight_decay": 0.0}],
                            lr=hp["lr"], betas=(hp["beta1"], hp["beta2"]), eps=hp["eps"])
    m = {k: np.zeros_like(a) for k, a in params.items()}
    v = {k: np.zeros_like(a) for k, a in params.items()}
    for t in range(1, 4):
        grads = {"w": rng.standard_normal((4, 3)), "b": rng.standard_normal(3)}
        tw.grad, tb.grad = torch.tensor(grads["w"]), torch.tensor(grads["b"])
        opt.step()
        params, m, v = O.adamw_step(params, grads, m, v, t, hp["lr"], hp["beta1"], hp["beta2"],
                                    hp["eps"], hp["weight_decay"], {"w"})
        np.testing.assert_allclose(params["w"], tw.detach().numpy(), rtol=1e-12, atol=1e-14)
        np.testing.assert_allclose(params["b"], tb.detach().numpy(), rtol=1e-12, atol=1e-14)


# ------------------------------------------------------------------ the blocks
def test_gpt_block_equals_torch_pre_ln_encoder_layer():
    """Eq. 1 is the Pre-LN block that nn.TransformerEncoderLayer(norm_first=True) computes."""
    s = TINY
    p = _params("gpt", s)
    tok, tgt = synth.make_tokens(s, 0)
    cfg = O.Config.from_shape("gpt", s)
    _, cache = O.forward(p, cfg, tok, tgt)
    d = s.d_model
    for i in range(s.layers):
        layer = torch.nn.TransformerEncoderLayer(
            d, s.heads, s.d_ff, dropout=0.0, activation=lambda x: Fn.gelu(x, approximate="tanh"),
            layer_norm_eps=1e-5, batch_first=True, norm_first=True, dtype=torch.float64)
        sd = {
            "self_attn.in_proj_weight": p[f"h{i}.attn.w_qkv"], "self_attn.in_proj_bias": p[f"h{i}.attn.b_qkv"],
            "self_attn.out_proj.weight": p[f"h{i}.attn.w_o"], "self_attn.out_proj.bias": p[f"h{i}.attn.b_o"],
            "linear1.weight": p[f"h{i}.mlp.w_up"], "linear1.bias": p[f"h{i}.mlp.b_up"],
            "linear2.weight": p[f"h{i}.mlp.w_down"], "linear2.bias": p[f"h{i}.mlp.b_down"],
            "norm1.weight": p[f"h{i}.ln1.g"], "norm1.bias": p[f"h{i}.ln1.b"],
            "norm2.weight": p[f"h{i}.ln2.g"], "norm2.bias": p[f"h{i}.ln2.b"],
        }
        layer.load_state_dict({k: torch.tensor(np.asarray(a, np.float64)) for k, a in sd.items()})
        layer.train()
        x = torch.tensor(cache["X"][i].reshape(s.batch, s.seq, d))
        mask = torch.nn.Transformer.generate_square_subsequent_mask(s.seq, dtype=torch.float64)
        y = layer(x, src_mask=mask, is_causal=True).detach().numpy().reshape(-1, d)
        np.testing.assert_allclose(cache["X"][i + 1], y, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("variant", synth.VARIANTS)
@pytest.mark.parametrize("layers", [2, 3])
def test_forward_and_backward_match_autograd_model(variant, layers):
    s = TINY.replace(layers=layers)
    p = _params(variant, s, seed=layers)
    tok, tgt = synth.make_tokens(s, 1)
    cfg = O.Config.from_shape(variant, s)
    loss, cache = O.forward(p, cfg, tok, tgt)
    grads = O.backward(p, cfg, cache)
    tloss, tgrads = torch_ref.loss_and_grads(p, variant, s.heads, tok, tgt, s.layers)
    assert abs(loss - tloss) < 1e-12
    for k in p:
        np.testing.assert_allclose(grads[k], tgrads[k], rtol=1e-9, atol=1e-13, err_msg=k)


@pytest.mark.parametrize("variant", synth.VARIANTS)
@pytest.mark.parametrize("layers", [2, 3])
def test_backward_matches_central_differences(variant, layers):
    """Directional derivative of the fp64 loss along a random unit direction per
    tensor, by central differences, against <grad, direction>."""
    s = TINY.replace(layers=layers)
    p = {k: a.astype(np.float64) for k, a in _params(variant, s, seed=10 + layers).items()}
    tok, tgt = synth.make_tokens(s, 2)
    cfg = O.Config.from_shape(variant, s)
    loss, cache = O.forward(p, cfg, tok, tgt)
    grads = O.backward(p, cfg, cache)
    rng = np.random.default_rng(7)
    h = 1e-5
    for k in p:
        direction = rng.standard_normal(p[k].shape)
        direction /= np.linalg.norm(direction)
        pp, pm = dict(p), dict(p)
        pp[k] = p[k] + h * direction
        pm[k] = p[k] - h * direction
        fd = (O.loss_only(pp, cfg, tok, tgt) - O.loss_only(pm, cfg, tok, tgt)) / (2 * h)
        an = float((grads[k] * direction).sum())
        scale = np.linalg.norm(grads[k])
        assert abs(fd - an) <= 1e-6 * scale + 1e-11, (k, fd, an, scale)


def test_loss_at_init_is_log_vocab():
    for v in synth.VARIANTS:
        p = _params(v, TINY, perturb=False)
        tok, tgt = synth.make_tokens(TINY, 0)
        loss, _ = O.forward(p, O.Config.from_shape(v, TINY), tok, tgt)
        assert abs(loss - math.log(TINY.vocab)) < 0.05, (v, loss)


def test_first_block_attention_shared_by_all_variants():
    """a_1 = MHA_1(LN(X_1)) is the same for GPT, FAL, FAL+; FAL+ block 1 is the
    standard block (App. D.1), so GPT and FAL+ agree through X_2; FAL's block 1
    differs only through its MLP input (Eq. 2 at i=1)."""
    u = _union_params()
    tok, tgt = synth.make_tokens(TINY, 0)
    caches = {}
    for v in synth.VARIANTS:
        _, caches[v] = O.forward(_pick(u, v), O.Config.from_shape(v, TINY), tok, tgt)
    for v in ("fal", "falplus"):
        np.testing.assert_array_equal(caches[v]["a1"], caches["gpt"]["a1"])
    np.testing.assert_array_equal(caches["falplus"]["X"][1], caches["gpt"]["X"][1])
    assert not np.allclose(caches["fal"]["X"][1], caches["gpt"]["X"][1])
    fal0, gpt0 = caches["fal"]["layers"][0], caches["gpt"]["layers"][0]
    np.testing.assert_array_equal(fal0["u"], gpt0["u"])
    np.testing.assert_array_equal(fal0["ctx"], gpt0["ctx"])


@pytest.mark.parametrize("block", [1, 2])
def test_fal_mlp_input_independent_of_own_attention(block):
    """Sec. 4.2: in FAL, MLP_i never reads MHA_i, so changing block i's attention
    weights (i >= 2) leaves its MLP input and hidden state unchanged, while in
    GPT it changes them."""
    s = TINY.replace(layers=3)
    tok, tgt = synth.make_tokens(s, 0)
    rng = np.random.default_rng(8)
    for variant, should_change in (("fal", False), ("gpt", True), ("falplus", True)):
        p = _params(variant, s)
        q = dict(p)
        for n in ("attn.w_qkv", "attn.b_qkv", "attn.w_o", "attn.b_o"):
            k = f"h{block}.{n}"
            q[k] = p[k] + rng.standard_normal(p[k].shape).astype(np.float32) * 0.1
        cfg = O.Config.from_shape(variant, s)
        _, c0 = O.forward(p, cfg, tok, tgt)
        _, c1 = O.forward(q, cfg, tok, tgt)
        m0, m1 = c0["layers"][block]["m"], c1["layers"][block]["m"]
        assert np.array_equal(m0, m1) != should_change, variant
        assert not np.allclose(c0["X"][block + 1], c1["X"][block + 1])


def test_fal_mlp_input_tracks_first_attention():
    """Changing the shared LN_F (the first-attention path) shifts block 1's MLP
    input by exactly that change and changes every later FAL MLP input."""
    s = TINY.replace(layers=3)
    tok, tgt = synth.make_tokens(s, 0)
    p = {k: a.astype(np.float64) for k, a in _params("fal", s).items()}
    q = dict(p, **{"lnF.b": p["lnF.b"] + 0.5})
    cfg = O.Config.from_shape("fal", s)
    _, c0 = O.forward(p, cfg, tok, tgt)
    _, c1 = O.forward(q, cfg, tok, tgt)
    np.testing.assert_allclose(c1["layers"][0]["m"] - c0["layers"][0]["m"], 0.5, rtol=1e-12)
    for i in range(1, s.layers):
        assert not np.allclose(c1["layers"][i]["m"], c0["layers"][i]["m"])


def test_falplus_with_zero_first_attention_ln_is_gpt():
    s = TINY.replace(layers=3)
    u = _union_params(s)
    pf = _pick(u, "falplus", s)
    for i in range(1, s.layers):
        pf[f"h{i}.lnF.g"] = np.zeros_like(pf[f"h{i}.lnF.g"])
        pf[f"h{i}.lnF.b"] = np.zeros_like(pf[f"h{i}.lnF.b"])
    pg = _pick(u, "gpt", s)
    tok, tgt = synth.make_tokens(s, 3)
    lf, cf = O.forward(pf, O.Config.from_shape("falplus", s), tok, tgt)
    lg, cg = O.forward(pg, O.Config.from_shape("gpt", s), tok, tgt)
    assert lf == lg
    gf = O.backward(pf, O.Config.from_shape("falplus", s), cf)
    gg = O.backward(pg, O.Config.from_shape("gpt", s), cg)
    for k in pg:
        np.testing.assert_allclose(gf[k], gg[k], rtol=1e-12, atol=1e-15, err_msg=k)


def test_fal_with_zero_first_attention_ln_is_parallel_block():
    """With LN_F switched off, Eq. 2 is X + MHA(LN(X)) + MLP(LN(X)): the parallel
    (GPT-J) block the paper compares against (Sec. 5.1)."""
    s = TINY.replace(layers=3)
    p = _params("fal", s)
    p["lnF.g"] = np.zeros_like(p["lnF.g"])
    p["lnF.b"] = np.zeros_like(p["lnF.b"])
    tok, tgt = synth.make_tokens(s, 4)
    loss, cache = O.forward(p, O.Config.from_shape("fal", s), tok, tgt)
    grads = O.backward(p, O.Config.from_shape("fal", s), cache)
    tl, tg = torch_ref.loss_and_grads({k: v for k, v in p.items() if not k.startswith("lnF")},
                                      "fal", s.heads, tok, tgt, s.layers, parallel=True)
    assert abs(loss - tl) < 1e-12
    for k, g in tg.items():
        np.testing.assert_allclose(grads[k], g, rtol=1e-9, atol=1e-13, err_msg=k)


# ------------------------------------------------------------------ comparison blocks
# (variant, oracle/spec options) for the paper's comparison blocks and readings
COMPARISONS = [("parallel", {}), ("ablation1", {}), ("ablation2", {}), ("falplus", {"reuse": 2}),
               ("falplus", {"reuse": 3}), ("fal", {"separate_ln2": True})]
CMP_IDS = [v + "".join(f"-{k}{int(x)}" for k, x in kw.items()) for v, kw in COMPARISONS]


def _cparams(variant, kw, s, seed):
    return synth.perturb_params(synth.init_params(variant, s, seed, **kw), seed)


@pytest.mark.parametrize("variant,kw", COMPARISONS, ids=CMP_IDS)
def test_comparison_blocks_match_autograd_model(variant, kw):
    s = TINY.replace(layers=3)
    p = _cparams(variant, kw, s, 21)
    tok, tgt = synth.make_tokens(s, 5)
    cfg = O.Config.from_shape(variant, s, **kw)
    loss, cache = O.forward(p, cfg, tok, tgt)
    grads = O.backward(p, cfg, cache)
    tloss, tgrads = torch_ref.loss_and_grads(p, variant, s.heads, tok, tgt, s.layers, **kw)
    assert abs(loss - tloss) < 1e-12
    assert set(grads) == set(p)
    for k in p:
        np.testing.assert_allclose(grads[k], tgrads[k], rtol=1e-9, atol=1e-13, err_msg=k)


@pytest.mark.parametrize("variant,kw", COMPARISONS, ids=CMP_IDS)
def test_comparison_blocks_backward_matches_central_differences(variant, kw):
    s = TINY.replace(layers=3)
    p = {k: a.astype(np.float64) for k, a in _cparams(variant, kw, s, 22).items()}
    tok, tgt = synth.make_tokens(s, 6)
    cfg = O.Config.from_shape(variant, s, **kw)
    _, cache = O.forward(p, cfg, tok, tgt)
    grads = O.backward(p, cfg, cache)
    rng = np.random.default_rng(23)
    h = 1e-5
    for k in p:
        direction = rng.standard_normal(p[k].shape)
        direction /= np.linalg.norm(direction)
        pp, pm = dict(p), dict(p)
        pp[k], pm[k] = p[k] + h * direction, p[k] - h * direction
        fd = (O.loss_only(pp, cfg, tok, tgt) - O.loss_only(pm, cfg, tok, tgt)) / (2 * h)
        an = float((grads[k] * direction).sum())
        assert abs(fd - an) <= 1e-6 * np.linalg.norm(grads[k]) + 1e-11, (k, fd, an)


def _run(variant, p, s, tok, tgt, **kw):
    cfg = O.Config.from_shape(variant, s, **kw)
    loss, cache = O.forward(p, cfg, tok, tgt)
    return loss, cache, O.backward(p, cfg, cache)


def test_ablation1_with_zero_own_attention_ln_is_parallel():
    """Ablation1 (App. D) adds LN_{A,i}(MHA_i) to the MLP input; with every
    LN_{A,i} switched off it is the Parallel block."""
    s = TINY.replace(layers=3)
    p = _cparams("ablation1", {}, s, 24)
    for i in range(s.layers):
        p[f"h{i}.lnA.g"] = np.zeros_like(p[f"h{i}.lnA.g"])
        p[f"h{i}.lnA.b"] = np.zeros_like(p[f"h{i}.lnA.b"])
    q = {k: v for k, v in p.items() if ".lnA." not in k}
    tok, tgt = synth.make_tokens(s, 7)
    la, _, ga = _run("ablation1", p, s, tok, tgt)
    lp, _, gp = _run("parallel", q, s, tok, tgt)
    assert la == lp
    for k in q:
        np.testing.assert_array_equal(ga[k], gp[k], err_msg=k)


def test_ablation1_mlp_input_follows_own_attention():
    """Unlike FAL, Ablation1's MLP input in block i reads MHA_i: changing block
    2's attention weights changes block 2's MLP input."""
    s = TINY.replace(layers=3)
    p = _cparams("ablation1", {}, s, 25)
    q = dict(p, **{"h1.attn.w_o": p["h1.attn.w_o"] * 1.5})
    tok, tgt = synth.make_tokens(s, 8)
    _, c0, _ = _run("ablation1", p, s, tok, tgt)
    _, c1, _ = _run("ablation1", q, s, tok, tgt)
    np.testing.assert_array_equal(c0["layers"][1]["u"], c1["layers"][1]["u"])
    assert not np.allclose(c0["layers"][1]["m"], c1["layers"][1]["m"])


def test_ablation2_first_block_is_gpt_later_blocks_are_parallel():
    """Ablation2 (App. D) keeps only block 1's MHA-MLP connection: its block 1
    is the GPT block and every later block the Parallel block."""
    s = TINY.replace(layers=3)
    p = _cparams("ablation2", {}, s, 26)
    tok, tgt = synth.make_tokens(s, 9)
    _, c, _ = _run("ablation2", p, s, tok, tgt)
    g1 = {k: v for k, v in p.items() if not k.startswith(("h1.", "h2."))}
    _, cg, _ = _run("gpt", g1, s.replace(layers=1), tok, tgt)
    np.testing.assert_array_equal(c["X"][1], cg["X"][1])
    for i in (1, 2):
        np.testing.assert_array_equal(c["layers"][i]["m"], c["layers"][i]["u"])


def test_falplus_reuse_first_block_is_falplus_and_earlier_blocks_are_gpt():
    """FAL+ reusing block k: k = 1 is FAL+; blocks 1..k are standard blocks
    (GPT through X_{k+1}); with every LN_{F,i} switched off it is GPT."""
    s = TINY.replace(layers=3)
    tok, tgt = synth.make_tokens(s, 10)
    p1 = _cparams("falplus", {}, s, 27)
    l_a, _, g_a = _run("falplus", p1, s, tok, tgt)
    l_b, _, g_b = _run("falplus", p1, s, tok, tgt, reuse=1)
    assert l_a == l_b
    p2 = _cparams("falplus", {"reuse": 2}, s, 27)
    _, c2, _ = _run("falplus", p2, s, tok, tgt, reuse=2)
    pg = {k: v for k, v in p2.items() if ".lnF." not in k}
    _, cg, gg = _run("gpt", pg, s, tok, tgt)
    np.testing.assert_array_equal(c2["X"][2], cg["X"][2])
    np.testing.assert_array_equal(c2["a1"], cg["layers"][1]["a"])
    assert not np.allclose(c2["X"][3], cg["X"][3])
    z = dict(p2, **{"h2.lnF.g": np.zeros_like(p2["h2.lnF.g"]), "h2.lnF.b": np.zeros_like(p2["h2.lnF.b"])})
    lz, _, gz = _run("falplus", z, s, tok, tgt, reuse=2)
    lg, _, _ = _run("gpt", pg, s, tok, tgt)
    assert lz == lg
    for k in pg:
        np.testing.assert_allclose(gz[k], gg[k], rtol=1e-12, atol=1e-15, err_msg=k)


def test_separate_ln2_reading_of_fal():
    """The other reading of Eq. 2's MLP input (a LayerNorm of its own on X_i)
    equals the adopted one when that LayerNorm has LN1's parameters, and
    differs from it otherwise: the reading is observable."""
    s = TINY.replace(layers=3)
    tok, tgt = synth.make_tokens(s, 11)
    p = _cparams("fal", {}, s, 28)
    q = dict(p)
    for i in range(s.layers):
        q[f"h{i}.ln2.g"], q[f"h{i}.ln2.b"] = p[f"h{i}.ln1.g"], p[f"h{i}.ln1.b"]
    l0, _, _ = _run("fal", p, s, tok, tgt)
    l1, _, g1 = _run("fal", q, s, tok, tgt, separate_ln2=True)
    assert abs(l0 - l1) < 1e-13
    r = dict(q, **{"h1.ln2.b": q["h1.ln2.b"] + 0.3})
    l2, _, _ = _run("fal", r, s, tok, tgt, separate_ln2=True)
    assert abs(l2 - l0) > 1e-6
    # with LN2 tied to LN1, LN1's gradient under the shared reading is the sum of both
    _, _, g0 = _run("fal", p, s, tok, tgt)
    for i in range(s.layers):
        np.testing.assert_allclose(g1[f"h{i}.ln1.g"] + g1[f"h{i}.ln2.g"], g0[f"h{i}.ln1.g"], rtol=1e-9, atol=1e-13)


@pytest.mark.parametrize("max_norm", [1.0, 1e-3, 1e6])
def test_clip_grad_norm_matches_torch(max_norm):
    rng = np.random.default_rng(29)
    grads = {"a": rng.standard_normal((5, 7)), "b": rng.standard_normal(11) * 3}
    clipped, norm = O.clip_grad_norm(grads, max_norm)
    ts = [torch.zeros(g.shape, requires_grad=True) for g in grads.values()]
    for t, g in zip(ts, grads.values()):
        t.grad = torch.tensor(g)
    tn = torch.nn.utils.clip_grad_norm_(ts, max_norm)
    assert abs(norm - float(tn)) < 1e-12 * norm
    for t, k in zip(ts, grads):
        # torch divides by norm + 1e-6; the clipping definition divides by the norm
        np.testing.assert_allclose(clipped[k], t.grad.numpy(), rtol=2e-6 / max(min(norm, max_norm), 1e-30) + 1e-14)
    if norm <= max_norm:
        for k in grads:
            np.testing.assert_array_equal(clipped[k], grads[k])
    else:
        total = math.sqrt(sum(float((c ** 2).sum()) for c in clipped.values()))
        assert abs(total - max_norm) < 1e-12 * max_norm


# ------------------------------------------------------------------ grouped-query attention
GQA = [("fal", 2), ("gpt", 2), ("falplus", 1), ("fal", 4)]  # (variant, key/value heads) with H = 4


@pytest.mark.parametrize("variant,kv", GQA)
def test_gqa_matches_autograd_model(variant, kv):
    """App. E: GQA with G key/value heads; the torch model repeats each
    key / value head over its H / G query heads and differentiates by autograd."""
    s = TINY.replace(layers=3, kv_heads=kv)
    p = synth.perturb_params(synth.init_params(variant, s, 31), 31)
    assert p["h0.attn.w_qkv"].shape == (s.d_model + 2 * kv * s.head_dim, s.d_model)
    tok, tgt = synth.make_tokens(s, 12)
    cfg = O.Config.from_shape(variant, s)
    loss, cache = O.forward(p, cfg, tok, tgt)
    grads = O.backward(p, cfg, cache)
    tloss, tgrads = torch_ref.loss_and_grads(p, variant, s.heads, tok, tgt, s.layers, kv_heads=kv)
    assert abs(loss - tloss) < 1e-12
    for k in p:
        np.testing.assert_allclose(grads[k], tgrads[k], rtol=1e-9, atol=1e-13, err_msg=k)


@pytest.mark.parametrize("variant,kv", GQA[:2])
def test_gqa_backward_matches_central_differences(variant, kv):
    s = TINY.replace(layers=2, kv_heads=kv)
    p = {k: a.astype(np.float64) for k, a in synth.perturb_params(synth.init_params(variant, s, 32), 32).items()}
    tok, tgt = synth.make_tokens(s, 13)
    cfg = O.Config.from_shape(variant, s)
    _, cache = O.forward(p, cfg, tok, tgt)
    grads = O.backward(p, cfg, cache)
    rng = np.random.default_rng(33)
    h = 1e-5
    for k in p:
        direction = rng.standard_normal(p[k].shape)
        direction /= np.linalg.norm(direction)
        pp, pm = dict(p), dict(p)
        pp[k], pm[k] = p[k] + h * direction, p[k] - h * direction
        fd = (O.loss_only(pp, cfg, tok, tgt) - O.loss_only(pm, cfg, tok, tgt)) / (2 * h)
        an = float((grads[k] * direction).sum())
        assert abs(fd - an) <= 1e-6 * np.linalg.norm(grads[k]) + 1e-11, (k, fd, an)


def test_gqa_with_one_group_per_head_is_mha_and_shared_kv_acts_as_copies():
    """G = H is multi-head attention (App. E); and a GQA model equals the MHA
    model whose key / value projections repeat the group's rows for each of
    its query heads."""
    s = TINY.replace(layers=2)
    p = _params("fal", s, seed=34)
    tok, tgt = synth.make_tokens(s, 14)
    l_mha, _ = O.forward(p, O.Config.from_shape("fal", s), tok, tgt)
    l_g, _ = O.forward(p, O.Config.from_shape("fal", s.replace(kv_heads=s.heads)), tok, tgt)
    assert l_mha == l_g
    sg = s.replace(kv_heads=2)
    pg = synth.perturb_params(synth.init_params("fal", sg, 35), 35)
    d, hd, H = s.d_model, s.head_dim, s.heads
    pm = dict(pg)
    for i in range(s.layers):
        w, b = pg[f"h{i}.attn.w_qkv"], pg[f"h{i}.attn.b_qkv"]
        kw, vw = w[d:d + 2 * hd], w[d + 2 * hd:]
        kb, vb = b[d:d + 2 * hd], b[d + 2 * hd:]
        rep = lambda a: np.concatenate([a[(h // (H // 2)) * hd:(h // (H // 2) + 1) * hd] for h in range(H)], axis=0)
        pm[f"h{i}.attn.w_qkv"] = np.concatenate([w[:d], rep(kw), rep(vw)], axis=0)
        pm[f"h{i}.attn.b_qkv"] = np.concatenate([b[:d], rep(kb), rep(vb)], axis=0)
    l1, _ = O.forward(pg, O.Config.from_shape("fal", sg), tok, tgt)
    l2, _ = O.forward(pm, O.Config.from_shape("fal", s), tok, tgt)
    assert abs(l1 - l2) < 1e-12
