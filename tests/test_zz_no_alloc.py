"""The allocation-free attention backward entry point.

fal_kernel_attention_bwd_noalloc serves callers that may not allocate device
memory (for example code whose device memory is owned by a host framework's
pool, where a cudaMalloc of its own is not allowed, or callers that cannot pass
a scratch buffer).  It takes its scratch from a fixed array inside libfal.so.
This checks, through the C ABI, that two calls in a row match the allocating
entry point on the same inputs (so nothing left in the shared array by the
first call leaks into the second), and that oversize problems are refused.
The file is named to be collected last.
"""
import ctypes

import numpy as np
import pytest

from helpers import rel_fro

pytestmark = pytest.mark.gpu

TOL = 1e-2  # the bf16 parity tolerance used by every attention test


def _inputs(seed, B, T, H, hd):
    import torch
    from paper_2510_14614_gb300 import fal
    g = torch.Generator().manual_seed(seed)
    d = H * hd
    qkv = torch.randn((B * T, 3 * d), generator=g).to(torch.bfloat16).cuda()
    dctx = torch.randn((B * T, d), generator=g).to(torch.bfloat16).cuda()
    ctx, lse = fal.attention_fwd(qkv, B, T, H, hd)
    return qkv, ctx, lse, dctx


def _noalloc(qkv, ctx, lse, dctx, B, T, H, hd):
    import torch
    from paper_2510_14614_gb300 import fal
    dqkv = torch.empty_like(qkv)
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    code = fal.lib().fal_kernel_attention_bwd_noalloc(B, T, H, hd, p(qkv), p(ctx), p(lse), p(dctx), p(dqkv), None)
    return code, dqkv


@pytest.mark.parametrize("B,T,H,hd", [(2, 200, 2, 64), (1, 130, 2, 128), (520, 128, 1, 64)])
def test_noalloc_matches_allocating_entry_point_twice(B, T, H, hd):
    import torch
    from paper_2510_14614_gb300 import fal
    for call, seed in enumerate((1, 2)):
        qkv, ctx, lse, dctx = _inputs(seed, B, T, H, hd)
        ref = fal.attention_bwd(qkv, ctx, lse, dctx, B, T, H, hd)
        code, got = _noalloc(qkv, ctx, lse, dctx, B, T, H, hd)
        torch.cuda.synchronize()
        assert code == fal.FAL_OK, (call, code)
        err = rel_fro(got.float().cpu().numpy(), ref.float().cpu().numpy())
        assert err <= TOL, (call, err)
        assert np.isfinite(got.float().cpu().numpy()).all()


def test_noalloc_rejects_problems_above_its_fixed_scratch():
    import torch
    from paper_2510_14614_gb300 import fal
    B, T, H, hd = 2, 65536, 64, 64  # D needs B*H*T = 8 Mi floats, twice the array
    dummy = torch.empty(16, dtype=torch.bfloat16, device="cuda")
    p = ctypes.c_void_p(dummy.data_ptr())
    code = fal.lib().fal_kernel_attention_bwd_noalloc(B, T, H, hd, p, p, p, p, p, None)
    assert code == fal.FAL_ERR_WORKSPACE
