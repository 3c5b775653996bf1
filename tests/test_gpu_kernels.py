"""Kernel-level parity on the GPU, through the C ABI (include/fal_kernels.h).

GEMM: the tcgen05/TMA kernel against an fp64 matmul of the same bf16-rounded
operands, for every operand layout the backward uses (K-major / MN-major for A
and B), tile-multiple and ragged M, N, K.  Attention: forward and backward
against the oracle's causal attention on the same bf16-rounded q, k, v.
"""
import numpy as np
import pytest

from helpers import bf16_round, rel_fro
from oracle import fal_oracle as O

pytestmark = pytest.mark.gpu


def _dev_bf16(a, ld_mult=8):
    import torch
    rows, cols = a.shape
    ld = (cols + ld_mult - 1) // ld_mult * ld_mult
    t = torch.zeros((rows, ld), dtype=torch.bfloat16)
    t[:, :cols] = torch.as_tensor(a, dtype=torch.float32).to(torch.bfloat16)
    return t.cuda()


SHAPES = [(128, 256, 64), (256, 512, 1024), (300, 520, 200), (1, 17, 8), (129, 257, 65), (640, 1000, 768),
          (2048, 2304, 512), (4000, 2304, 256)]  # the last two span more 256x256 tiles than there are CTA pairs


@pytest.mark.parametrize("engine", ["tcgen05", "tcgen05_pair"])
@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 0), (1, 1)])
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_gemm_tcgen05_matches_matmul(M, N, K, a_mn, b_mn, engine):
    import torch
    from paper_2510_14614_gb300 import fal
    rng = np.random.default_rng(M * 7 + N * 3 + K + 11 * a_mn + 13 * b_mn)
    A = rng.standard_normal((M, K))
    B = rng.standard_normal((N, K))
    bias = rng.standard_normal(N).astype(np.float32)
    ref = bf16_round(A) @ bf16_round(B).T + bias
    At = _dev_bf16(A.T if a_mn else A)
    Bt = _dev_bf16(B.T if b_mn else B)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    C = fal.gemm(At, Bt, M, N, K, a_mn_major=a_mn, b_mn_major=b_mn, bias=torch.as_tensor(bias).cuda(),
                 out_f32=True, engine=engine, err=err, ldc=(N + 7) // 8 * 8)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    got = C.cpu().numpy()
    # fp32 accumulation of exact bf16 products: only summation rounding remains
    assert rel_fro(got, ref) < 2e-6, rel_fro(got, ref)
    np.testing.assert_allclose(got, ref, rtol=1e-4, atol=1e-4 * np.sqrt(K))


@pytest.mark.parametrize("M,N,K", [(300, 520, 200), (128, 256, 64)])
def test_gemm_tcgen05_bf16_output_and_simt_engine(M, N, K):
    import torch
    from paper_2510_14614_gb300 import fal
    rng = np.random.default_rng(5)
    A, B = rng.standard_normal((M, K)), rng.standard_normal((N, K))
    ref = bf16_round(A) @ bf16_round(B).T
    At, Bt = _dev_bf16(A), _dev_bf16(B)
    Cb = fal.gemm(At, Bt, M, N, K, out_f32=False, engine="tcgen05", ldc=(N + 7) // 8 * 8).float().cpu().numpy()
    assert rel_fro(Cb, ref) < 5e-3
    np.testing.assert_array_equal(Cb, bf16_round(Cb))
    Cs = fal.gemm(At, Bt, M, N, K, out_f32=True, engine="simt", ldc=(N + 7) // 8 * 8).cpu().numpy()
    assert rel_fro(Cs, ref) < 2e-6
    # a bf16 output whose row pitch is not a multiple of 16 bytes cannot be a
    # TMA store target: the kernel falls back to per-thread stores
    ldc = (N + 3) // 4 * 4
    if ldc % 8 == 0:
        ldc += 4
    Cf = fal.gemm(At, Bt, M, N, K, out_f32=False, engine="tcgen05", ldc=ldc).float().cpu().numpy()
    np.testing.assert_array_equal(Cf, Cb)


@pytest.mark.parametrize("hd", [64, 128])
@pytest.mark.parametrize("B,T,H", [(2, 200, 2), (1, 64, 3), (1, 1, 1), (1, 130, 2)])
def test_attention_forward_backward_match_oracle(B, T, H, hd):
    import torch
    from paper_2510_14614_gb300 import fal
    rng = np.random.default_rng(B * 1000 + T * 10 + H + hd)
    d = H * hd
    qkv = bf16_round(rng.standard_normal((B * T, 3 * d)))
    dctx = bf16_round(rng.standard_normal((B * T, d)))
    qkv_t = torch.as_tensor(qkv, dtype=torch.float32).to(torch.bfloat16).cuda()
    dctx_t = torch.as_tensor(dctx, dtype=torch.float32).to(torch.bfloat16).cuda()
    ctx_t, lse_t = fal.attention_fwd(qkv_t, B, T, H, hd)
    dqkv_t = fal.attention_bwd(qkv_t, ctx_t, lse_t, dctx_t, B, T, H, hd)
    torch.cuda.synchronize()
    sp = lambda x: x.reshape(B, T, H, hd).transpose(0, 2, 1, 3)
    mg = lambda x: x.transpose(0, 2, 1, 3).reshape(B * T, d)
    q, k, v = (sp(t) for t in np.split(qkv, 3, axis=1))
    ctx, p = O.causal_attention(q, k, v)
    # the kernel's backward consumes the bf16 ctx it produced, as in training
    ctx_gpu = ctx_t.float().cpu().numpy()
    dq, dk, dv = O.causal_attention_backward(sp(dctx), q, k, v, p)
    assert rel_fro(ctx_gpu, mg(ctx)) < 1e-2
    s = np.einsum("bhtd,bhsd->bhts", q, k) / np.sqrt(hd)
    s = np.where(np.triu(np.ones((T, T), bool), 1), -np.inf, s)
    lse_ref = np.log2(np.exp(s - s.max(-1, keepdims=True)).sum(-1)) + s.max(-1) * np.log2(np.e)
    np.testing.assert_allclose(lse_t.cpu().numpy(), lse_ref, rtol=1e-3, atol=1e-3)
    dqkv = dqkv_t.float().cpu().numpy()
    for got, ref in ((dqkv[:, :d], mg(dq)), (dqkv[:, d:2 * d], mg(dk)), (dqkv[:, 2 * d:], mg(dv))):
        assert rel_fro(got, ref) < 1e-2, rel_fro(got, ref)


@pytest.mark.parametrize("hd", [64, 128])
def test_attention_backward_persistent_items_against_oracle(hd):
    """More work items than SMs (each CTA of the persistent backward runs
    several key-block and query-block items back to back), a last band of
    heads narrower than the others and a ragged sequence length: dQ, dK and dV
    against the oracle's causal attention backward."""
    import torch
    from paper_2510_14614_gb300 import fal
    B, T, H = 3, 700, 6  # 6 blocks of 128 rows per sequence, 18 heads: 216 items
    rng = np.random.default_rng(700 + hd)
    d = H * hd
    qkv = bf16_round(rng.standard_normal((B * T, 3 * d)))
    dctx = bf16_round(rng.standard_normal((B * T, d)))
    qkv_t = torch.as_tensor(qkv, dtype=torch.float32).to(torch.bfloat16).cuda()
    dctx_t = torch.as_tensor(dctx, dtype=torch.float32).to(torch.bfloat16).cuda()
    ctx_t, lse_t = fal.attention_fwd(qkv_t, B, T, H, hd)
    dqkv_t = fal.attention_bwd(qkv_t, ctx_t, lse_t, dctx_t, B, T, H, hd)
    dqkv_t2 = fal.attention_bwd(qkv_t, ctx_t, lse_t, dctx_t, B, T, H, hd)
    torch.cuda.synchronize()
    sp = lambda x: x.reshape(B, T, H, hd).transpose(0, 2, 1, 3)
    mg = lambda x: x.transpose(0, 2, 1, 3).reshape(B * T, d)
    q, k, v = (sp(t) for t in np.split(qkv, 3, axis=1))
    ctx, p = O.causal_attention(q, k, v)
    dq, dk, dv = O.causal_attention_backward(sp(dctx), q, k, v, p)
    dqkv = dqkv_t.float().cpu().numpy()
    for got, ref in ((dqkv[:, :d], mg(dq)), (dqkv[:, d:2 * d], mg(dk)), (dqkv[:, 2 * d:], mg(dv))):
        assert rel_fro(got, ref) < 1e-2, rel_fro(got, ref)
    # each item's sums run in a fixed order whichever CTA takes it: repeat calls agree bit for bit
    np.testing.assert_array_equal(dqkv, dqkv_t2.float().cpu().numpy())


def test_attention_backward_more_token_rows_than_a_grid_dimension():
    """B*T = 66560 token rows (above the 65535 limit of a grid's y and z
    dimensions) in short sequences: the kernel-level backward, including its
    D = rowsum(dO * O) pre-pass, against the oracle on every row."""
    import torch
    from paper_2510_14614_gb300 import fal
    B, T, H, hd = 520, 128, 1, 64
    rng = np.random.default_rng(65536)
    d = H * hd
    qkv = bf16_round(rng.standard_normal((B * T, 3 * d)))
    dctx = bf16_round(rng.standard_normal((B * T, d)))
    qkv_t = torch.as_tensor(qkv, dtype=torch.float32).to(torch.bfloat16).cuda()
    dctx_t = torch.as_tensor(dctx, dtype=torch.float32).to(torch.bfloat16).cuda()
    ctx_t, lse_t = fal.attention_fwd(qkv_t, B, T, H, hd)
    dqkv_t = fal.attention_bwd(qkv_t, ctx_t, lse_t, dctx_t, B, T, H, hd)
    torch.cuda.synchronize()
    sp = lambda x: x.reshape(B, T, H, hd).transpose(0, 2, 1, 3)
    mg = lambda x: x.transpose(0, 2, 1, 3).reshape(B * T, d)
    q, k, v = (sp(t) for t in np.split(qkv, 3, axis=1))
    ctx, p = O.causal_attention(q, k, v)
    dq, dk, dv = O.causal_attention_backward(sp(dctx), q, k, v, p)
    assert rel_fro(ctx_t.float().cpu().numpy(), mg(ctx)) < 1e-2
    dqkv = dqkv_t.float().cpu().numpy()
    for got, ref in ((dqkv[:, :d], mg(dq)), (dqkv[:, d:2 * d], mg(dk)), (dqkv[:, 2 * d:], mg(dv))):
        assert rel_fro(got, ref) < 1e-2, rel_fro(got, ref)
