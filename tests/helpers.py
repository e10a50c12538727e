"""Shared comparison helpers for the parity tests (no method arithmetic)."""
import numpy as np
import torch


def f64(t):
    """Exact fp64 numpy copy of a tensor's stored values."""
    return t.detach().to("cpu", torch.float64).numpy()


def rel_frob(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def cos(a, b):
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    return float(a @ b / max(np.linalg.norm(a) * np.linalg.norm(b), 1e-300))
