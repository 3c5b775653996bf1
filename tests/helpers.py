"""Shared helpers for GPU parity tests (no method arithmetic here)."""
import numpy as np


def rel_fro(got, ref):
    """Per-tensor relative Frobenius error ||got - ref|| / ||ref||."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.linalg.norm(ref)
    return float(np.linalg.norm(got - ref) / den) if den > 0 else float(np.linalg.norm(got))


def bf16_round(a):
    """Round-to-nearest-even to bfloat16, returned as float64."""
    import torch
    return torch.as_tensor(np.asarray(a, np.float32)).to(torch.bfloat16).to(torch.float64).numpy()


def padded(rows, cols, mult=8):
    return rows, (cols + mult - 1) // mult * mult
