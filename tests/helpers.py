"""Shared helpers for the parity tests: seeded inputs go to both the CUDA path (through the
C ABI) and the CPU oracle; nothing here computes the method itself."""
from __future__ import annotations

import numpy as np

from workload import synth


def rel_fro(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


def f16_round(x: np.ndarray) -> np.ndarray:
    """Values of x rounded to IEEE half (as float64)."""
    return np.ascontiguousarray(x, np.float32).astype(np.float16).astype(np.float64)


def to_gpu(x, dtype=None):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def np_of(t):
    import torch
    if t.dtype in (torch.bfloat16, torch.float16):
        t = t.float()
    return t.detach().cpu().numpy()


def dense_blocks(dims, n=None, seed=0, **kw):
    return [synth.block_weights(dims, i, seed=seed, **kw) for i in range(n if n is not None else dims.n_layers)]
