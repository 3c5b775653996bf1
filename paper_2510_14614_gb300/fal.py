"""ctypes binding of libfal.so (C ABI in include/fal.h and include/fal_kernels.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch supplies device memory (the workspace) and CUDA streams.
There is no fallback: if libfal.so is missing or a CUDA device is absent the
calls raise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libfal.so")

FAL_OK, FAL_ERR_ARG, FAL_ERR_STATE, FAL_ERR_WORKSPACE, FAL_ERR_CUDA, FAL_ERR_TIMEOUT, FAL_ERR_UNSUPPORTED = range(7)
VARIANT = {"gpt": 0, "fal": 1, "falplus": 2, "parallel": 3, "ablation1": 4, "ablation2": 5}
PRECISION = {"bf16": 0, "fp32": 1}
SCHEDULE = {"serial": 0, "two_stream": 1}
ENGINE = {"tcgen05": 0, "simt": 1, "tcgen05_pair": 2}


class FalConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("variant", "layers", "d_model", "heads", "d_ff", "seq", "batch", "vocab",
                                            "precision", "schedule")] + \
               [(n, ctypes.c_float) for n in ("lr", "beta1", "beta2", "eps", "weight_decay")] + \
               [("reuse_layer", ctypes.c_int), ("clip_norm", ctypes.c_float), ("kv_heads", ctypes.c_int),
                ("head_chunk", ctypes.c_int)]


class FalTensorInfo(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("offset", ctypes.c_size_t), ("numel", ctypes.c_size_t),
                ("ndim", ctypes.c_int), ("shape", ctypes.c_int * 2), ("decayed", ctypes.c_int)]


class FalProfile(ctypes.Structure):
    _fields_ = [("gemm_ms", ctypes.c_double), ("gemm_flops", ctypes.c_double), ("gemm_launches", ctypes.c_longlong),
                ("attn_ms", ctypes.c_double), ("attn_flops", ctypes.c_double), ("attn_launches", ctypes.c_longlong)]


class FalLaunchRecord(ctypes.Structure):
    _fields_ = [("start_ms", ctypes.c_double), ("end_ms", ctypes.c_double), ("flops", ctypes.c_double),
                ("kind", ctypes.c_int), ("stream", ctypes.c_int), ("label", ctypes.c_char * 48)]


class FalError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{msg} (status {code})")
        self.code = code


_lib = None

_SIGS = {
    "fal_workspace_size": (ctypes.c_int, [ctypes.POINTER(FalConfig), ctypes.POINTER(ctypes.c_size_t)]),
    "fal_create": (ctypes.c_int, [ctypes.POINTER(FalConfig), ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p,
                                  ctypes.c_void_p, ctypes.POINTER(ctypes.c_void_p)]),
    "fal_destroy": (None, [ctypes.c_void_p]),
    "fal_forward": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(ctypes.c_float)]),
    "fal_backward": (ctypes.c_int, [ctypes.c_void_p]),
    "fal_prefill": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "fal_step": (ctypes.c_int, [ctypes.c_void_p]),
    "fal_train_step": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(ctypes.c_float)]),
    "fal_sync": (ctypes.c_int, [ctypes.c_void_p]),
    "fal_get_grad_norm": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_float)]),
    "fal_get_loss": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_float)]),
    "fal_param_count": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_size_t)]),
    "fal_param_info": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.POINTER(FalTensorInfo)]),
    "fal_set_params": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t]),
    "fal_get_params": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t]),
    "fal_get_grads": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t]),
    "fal_get_opt_state": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                         ctypes.POINTER(ctypes.c_longlong)]),
    "fal_set_opt_state": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                         ctypes.c_longlong]),
    "fal_get_tap": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_char_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t]),
    "fal_profile_enable": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int]),
    "fal_profile_read": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(FalProfile)]),
    "fal_profile_timeline": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(FalLaunchRecord), ctypes.c_int,
                                            ctypes.POINTER(ctypes.c_int)]),
    "fal_launch_count": (ctypes.c_longlong, []),
    "fal_debug_layernorm_stall": (ctypes.c_int, [ctypes.c_int, ctypes.c_longlong]),
    "fal_last_error": (ctypes.c_char_p, [ctypes.c_void_p]),
    "fal_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "fal_kernel_gemm": (ctypes.c_int, [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_long,
                                       ctypes.c_int, ctypes.c_void_p, ctypes.c_long, ctypes.c_int, ctypes.c_int,
                                       ctypes.c_void_p, ctypes.c_void_p, ctypes.c_long, ctypes.c_int, ctypes.c_int,
                                       ctypes.c_void_p, ctypes.c_void_p]),
    "fal_kernel_attention_fwd": (ctypes.c_int, [ctypes.c_int] * 4 + [ctypes.c_void_p] * 4),
    "fal_kernel_attention_bwd_scratch": (ctypes.c_size_t, [ctypes.c_int] * 4),
    "fal_kernel_attention_bwd": (ctypes.c_int, [ctypes.c_int] * 4 + [ctypes.c_void_p] * 7),
    "fal_kernel_attention_bwd_noalloc": (ctypes.c_int, [ctypes.c_int] * 4 + [ctypes.c_void_p] * 6),
}


def lib():
    """Loads libfal.so (building it first if absent).  Raises on failure."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            from . import build as _build
            _build.build()
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _lib = L
    return _lib


def _check(code, handle=None, what=""):
    if code != FAL_OK:
        L = lib()
        msg = L.fal_last_error(handle).decode() if handle else ""
        raise FalError(code, f"{what}: {L.fal_status_string(code).decode()} {msg}".strip())


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def _stream_ptr(s):
    return ctypes.c_void_p(s.cuda_stream if s is not None else 0)


def make_config(variant, layers, d_model, heads, d_ff, seq, batch, vocab, precision="bf16", schedule="serial",
                lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=1e-3, reuse_layer=1, clip_norm=0.0,
                kv_heads=0, head_chunk=0):
    return FalConfig(VARIANT[variant], layers, d_model, heads, d_ff, seq, batch, vocab, PRECISION[precision],
                     SCHEDULE[schedule], lr, beta1, beta2, eps, weight_decay, reuse_layer, clip_norm, kv_heads,
                     head_chunk)


def workspace_size(cfg: FalConfig) -> int:
    n = ctypes.c_size_t()
    _check(lib().fal_workspace_size(ctypes.byref(cfg), ctypes.byref(n)), what="fal_workspace_size")
    return n.value


class Model:
    """One decoder stack living in a torch-allocated device workspace."""

    def __init__(self, cfg: FalConfig, device="cuda", stream_main=None, stream_side=None):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.device = torch.device(device)
        nbytes = workspace_size(cfg)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        self.stream_main = stream_main if stream_main is not None else torch.cuda.Stream(self.device)
        self.stream_side = stream_side if stream_side is not None else torch.cuda.Stream(self.device)
        h = ctypes.c_void_p()
        _check(lib().fal_create(ctypes.byref(cfg), _ptr(self.workspace), nbytes, _stream_ptr(self.stream_main),
                                _stream_ptr(self.stream_side), ctypes.byref(h)), what="fal_create")
        self.h = h
        nt, ne = ctypes.c_int(), ctypes.c_size_t()
        _check(lib().fal_param_count(h, ctypes.byref(nt), ctypes.byref(ne)), h, "fal_param_count")
        self.n_params = ne.value
        self.tensors = []
        for i in range(nt.value):
            info = FalTensorInfo()
            _check(lib().fal_param_info(h, i, ctypes.byref(info)), h, "fal_param_info")
            shape = (info.shape[0], info.shape[1]) if info.ndim == 2 else (info.shape[0],)
            self.tensors.append((info.name.decode(), info.offset, info.numel, shape, bool(info.decayed)))
        self._tok = None

    def close(self):
        if getattr(self, "h", None):
            lib().fal_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------- parameters
    def flatten(self, params: dict) -> np.ndarray:
        flat = np.zeros(self.n_params, np.float32)
        for name, off, n, shape, _ in self.tensors:
            a = np.asarray(params[name], np.float32)
            if a.shape != shape:
                raise ValueError(f"{name}: shape {a.shape} != {shape}")
            flat[off:off + n] = a.reshape(-1)
        return flat

    def unflatten(self, flat: np.ndarray) -> dict:
        return {name: flat[off:off + n].reshape(shape).copy() for name, off, n, shape, _ in self.tensors}

    def set_params(self, params):
        """params: dict name -> array, or a flat float32 torch tensor (device or host)."""
        if isinstance(params, dict):
            flat = self.torch.from_numpy(self.flatten(params)).to(self.device)
        else:
            flat = params
        assert flat.numel() == self.n_params and flat.dtype == self.torch.float32
        _check(lib().fal_set_params(self.h, _ptr(flat), self.n_params), self.h, "fal_set_params")

    def _flat(self, fn):
        out = np.empty(self.n_params, np.float32)
        _check(fn(self.h, out.ctypes.data_as(ctypes.c_void_p), self.n_params), self.h, "copy")
        return out

    def params(self):
        return self.unflatten(self._flat(lib().fal_get_params))

    def grads(self):
        return self.unflatten(self._flat(lib().fal_get_grads))

    def opt_state(self):
        """(m, v, step): AdamW moments as dicts name -> array, and the steps taken."""
        m = np.empty(self.n_params, np.float32)
        v = np.empty(self.n_params, np.float32)
        step = ctypes.c_longlong()
        _check(lib().fal_get_opt_state(self.h, m.ctypes.data_as(ctypes.c_void_p), v.ctypes.data_as(ctypes.c_void_p),
                                       self.n_params, ctypes.byref(step)), self.h, "fal_get_opt_state")
        return self.unflatten(m), self.unflatten(v), step.value

    def set_opt_state(self, m: dict, v: dict, step: int):
        fm, fv = self.flatten(m), self.flatten(v)
        _check(lib().fal_set_opt_state(self.h, fm.ctypes.data_as(ctypes.c_void_p), fv.ctypes.data_as(ctypes.c_void_p),
                                       self.n_params, int(step)), self.h, "fal_set_opt_state")

    # ------------------------------------------------------------- training
    def _tokens(self, tokens, targets):
        """Accepts numpy arrays (host) or int32 torch tensors (device or pinned host)."""
        keep = []
        ptrs = []
        for a in (tokens, targets):
            if isinstance(a, np.ndarray):
                a = np.ascontiguousarray(a, dtype=np.int32)
                keep.append(a)
                ptrs.append(a.ctypes.data_as(ctypes.c_void_p))
            else:
                assert a.dtype == self.torch.int32 and a.is_contiguous()
                keep.append(a)
                ptrs.append(_ptr(a))
        self._tok = keep
        return ptrs

    def forward(self, tokens, targets, sync=True):
        t, g = self._tokens(tokens, targets)
        loss = ctypes.c_float()
        _check(lib().fal_forward(self.h, t, g, ctypes.byref(loss) if sync else None), self.h, "fal_forward")
        return loss.value if sync else None

    def prefill(self, tokens, sync=True):
        """Forward-only pass; returns the fp32 logits [B, V] of every sequence's
        last position (sync=True), or None with the work left queued."""
        t, _ = self._tokens(tokens, tokens)
        if not sync:
            _check(lib().fal_prefill(self.h, t, None), self.h, "fal_prefill")
            return None
        out = np.empty((self.cfg.batch, self.cfg.vocab), np.float32)
        _check(lib().fal_prefill(self.h, t, out.ctypes.data_as(ctypes.c_void_p)), self.h, "fal_prefill")
        return out

    def backward(self):
        _check(lib().fal_backward(self.h), self.h, "fal_backward")

    def step(self):
        _check(lib().fal_step(self.h), self.h, "fal_step")

    def train_step(self, tokens, targets, sync=True):
        t, g = self._tokens(tokens, targets)
        loss = ctypes.c_float()
        _check(lib().fal_train_step(self.h, t, g, ctypes.byref(loss) if sync else None), self.h, "fal_train_step")
        return loss.value if sync else None

    def sync(self):
        _check(lib().fal_sync(self.h), self.h, "fal_sync")

    def grad_norm(self):
        v = ctypes.c_float()
        _check(lib().fal_get_grad_norm(self.h, ctypes.byref(v)), self.h, "fal_get_grad_norm")
        return v.value

    def loss(self):
        v = ctypes.c_float()
        _check(lib().fal_get_loss(self.h, ctypes.byref(v)), self.h, "fal_get_loss")
        return v.value

    def profile_enable(self, on=True, every_launch=False):
        level = (2 if every_launch else 1) if on else 0
        _check(lib().fal_profile_enable(self.h, level), self.h, "fal_profile_enable")

    def profile_timeline(self, cap=100000):
        """Per-launch records since the last profile_read(): dicts with start/end ms, kind, stream, label."""
        arr = (FalLaunchRecord * cap)()
        n = ctypes.c_int(0)
        _check(lib().fal_profile_timeline(self.h, arr, cap, ctypes.byref(n)), self.h, "fal_profile_timeline")
        return [{"start_ms": r.start_ms, "end_ms": r.end_ms, "flops": r.flops, "kind": r.kind, "stream": r.stream,
                 "label": r.label.decode()} for r in arr[:n.value]]

    def profile_read(self):
        p = FalProfile()
        _check(lib().fal_profile_read(self.h, ctypes.byref(p)), self.h, "fal_profile_read")
        return {k: getattr(p, k) for k, _ in FalProfile._fields_}

    def tap(self, name, layer=0):
        c = self.cfg
        bt = c.batch * c.seq
        kv = c.kv_heads or c.heads
        dq = c.d_model + 2 * kv * (c.d_model // c.heads)
        cols = {"qkv": dq, "h": c.d_ff, "g": c.d_ff, "logits": c.vocab}.get(name, c.d_model)
        out = np.empty((bt, cols), np.float32)
        _check(lib().fal_get_tap(self.h, name.encode(), layer, out.ctypes.data_as(ctypes.c_void_p), out.size),
               self.h, f"fal_get_tap({name})")
        return out


def launch_count() -> int:
    """Kernels launched by libfal in this process."""
    return int(lib().fal_launch_count())


# ----------------------------------------------------------------- kernel API
def gemm(A, B, M, N, K, a_mn_major=False, b_mn_major=False, bias=None, out_f32=True, engine="tcgen05", err=None,
         stream=None, ldc=None):
    """C = A(m,k) B(n,k) (+bias) with the library's GEMM (torch tensors in, torch tensor out)."""
    import torch
    lda = A.shape[-1]
    ldb = B.shape[-1]
    ldc = ldc or N
    C = torch.empty((M, ldc), dtype=torch.float32 if out_f32 else torch.bfloat16, device=A.device)
    in_f32 = 1 if A.dtype == torch.float32 else 0
    code = lib().fal_kernel_gemm(M, N, K, _ptr(A), lda, int(a_mn_major), _ptr(B), ldb, int(b_mn_major), in_f32,
                                 _ptr(bias) if bias is not None else None, _ptr(C), ldc, int(out_f32), ENGINE[engine],
                                 _ptr(err) if err is not None else None, _stream_ptr(stream))
    _check(code, what="fal_kernel_gemm")
    return C[:, :N]


def attention_fwd(qkv, B, T, H, hd, stream=None):
    import torch
    ctx = torch.empty((B * T, H * hd), dtype=torch.bfloat16, device=qkv.device)
    lse = torch.empty((B, H, T), dtype=torch.float32, device=qkv.device)
    _check(lib().fal_kernel_attention_fwd(B, T, H, hd, _ptr(qkv), _ptr(ctx), _ptr(lse), _stream_ptr(stream)),
           what="fal_kernel_attention_fwd")
    return ctx, lse


def attention_bwd(qkv, ctx, lse, dctx, B, T, H, hd, stream=None):
    import torch
    dqkv = torch.empty_like(qkv)
    n = lib().fal_kernel_attention_bwd_scratch(B, T, H, hd)
    scratch = torch.empty(n, dtype=torch.float32, device=qkv.device)
    _check(lib().fal_kernel_attention_bwd(B, T, H, hd, _ptr(qkv), _ptr(ctx), _ptr(lse), _ptr(dctx), _ptr(dqkv),
                                          _ptr(scratch), _stream_ptr(stream)), what="fal_kernel_attention_bwd")
    return dqkv
