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


def rowblock_err(got, ref, rows: int = 64) -> float:
    """Worst element-wise error of a row block relative to that block's largest reference value:
    max over blocks of max|got - ref| / max|ref|, blocks of `rows` consecutive rows (the
    kernels' tile height).  A wrong ragged tile or sequence boundary that touches a few rows
    shows here even when a norm over thousands of rows hides it."""
    a = np.asarray(got, np.float64).reshape(np.shape(got)[0], -1)
    b = np.asarray(ref, np.float64).reshape(a.shape)
    worst = 0.0
    for r0 in range(0, a.shape[0], rows):
        d = np.abs(a[r0:r0 + rows] - b[r0:r0 + rows]).max()
        worst = max(worst, float(d / max(np.abs(b[r0:r0 + rows]).max(), 1e-30)))
    return worst
