"""Host-side checks of the C ABI (no GPU): the library builds, loads, exports
every entry point the public headers declare, and validates configurations
before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2510_14614_gb300 import fal, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = []
    for hdr in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not hdr.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", hdr)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(fal_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def libfal():
    from paper_2510_14614_gb300 import build
    build.build()
    return fal.lib()


def test_library_exports_every_declared_symbol(libfal):
    names = _declared_functions()
    assert len(names) >= 20, names
    missing = [n for n in names if not hasattr(libfal, n)]
    assert not missing, missing
    # the binding declares a signature for each of them
    assert set(names) <= set(fal._SIGS), set(names) - set(fal._SIGS)


def test_status_strings(libfal):
    for code in range(7):
        assert libfal.fal_status_string(code)
    assert libfal.fal_status_string(99) == b"unknown status"


def _ws(cfg):
    n = ctypes.c_size_t()
    return fal.lib().fal_workspace_size(ctypes.byref(cfg), ctypes.byref(n)), n.value


@pytest.mark.parametrize("bad", [
    dict(heads=5),                        # d % H != 0
    dict(d_model=96, heads=3),            # head_dim 32 not supported in bf16
    dict(layers=0), dict(vocab=1), dict(batch=0),
    dict(d_ff=100),                       # not a multiple of 8
    dict(d_model=8192, heads=64),         # wider than the LN kernels support
    dict(variant="falplus", reuse_layer=3),   # reuses a block the 2-layer stack does not have
    dict(reuse_layer=2),                  # reuse_layer applies to FAL+ only
    dict(clip_norm=-1.0),
    dict(head_chunk=100), dict(head_chunk=-64),   # chunk width must be a positive multiple of 64
    dict(variant="gpt", layers=-1),
])
def test_workspace_size_rejects_bad_configs(libfal, bad):
    base = dict(variant="fal", layers=2, d_model=128, heads=2, d_ff=512, seq=64, batch=2, vocab=1000)
    base.update(bad)
    rc, _ = _ws(fal.make_config(**base))
    assert rc == fal.FAL_ERR_ARG


def test_workspace_size_accepts_all_shapes(libfal):
    for name, s in synth.SHAPES.items():
        for v in synth.ALL_VARIANTS:
            cfg = fal.make_config(v, s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch, s.vocab,
                                  precision=s.precision)
            rc, n = _ws(cfg)
            assert rc == 0, (name, v)
            assert n > 0
    # the 1.3B stack fits one GB300 with room to spare (activations + optimizer state)
    s = synth.SHAPES["gpt_1p3b"]
    _, n = _ws(fal.make_config("fal", s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch, s.vocab))
    assert n < 120 * 2**30


def test_chunked_head_shrinks_the_workspace(libfal):
    """With head_chunk > 0 the workspace holds two [B*T, head_chunk] chunks
    and the per-slice statistics instead of two [B*T, vocab] logit arrays."""
    s = synth.SHAPES["gpt_1p3b"]
    args = ("fal", s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch, s.vocab)
    _, full = _ws(fal.make_config(*args))
    rc, chunked = _ws(fal.make_config(*args, head_chunk=8192))
    assert rc == 0
    bt, vp = s.batch * s.seq, (s.vocab + 63) // 64 * 64
    saved = 2 * bt * vp * 2 - (2 * bt * 8192 * 2 + bt * ((s.vocab + 127) // 128) * 8 + 2 * bt * 4)
    assert abs((full - chunked) - saved) <= 64 * 1024, (full - chunked, saved)
    assert full - chunked > 2**30


def test_null_arguments_are_rejected(libfal):
    assert libfal.fal_workspace_size(None, None) == fal.FAL_ERR_ARG
    out = ctypes.c_void_p()
    cfg = fal.make_config("gpt", 1, 128, 2, 512, 64, 1, 1000)
    assert libfal.fal_create(ctypes.byref(cfg), None, 0, None, None, ctypes.byref(out)) == fal.FAL_ERR_ARG
    assert libfal.fal_backward(None) == fal.FAL_ERR_ARG
    assert libfal.fal_step(None) == fal.FAL_ERR_ARG
    assert libfal.fal_last_error(None) == b"null handle"
