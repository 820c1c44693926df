"""AdamW update of the LoRA weights in plain numpy fp64 — TEST INFRASTRUCTURE ONLY.

Section 4 ("Utility Comparison") trains every model with the AdamW optimizer; Section 3
("Runtime implementation") keeps only the LoRA weights, their gradients and the optimizer
states, and accumulates gradients over the samples of a batch.  The paper gives no formula, so
this follows the published AdamW algorithm (Adam with decoupled weight decay): at step t >= 1,

    g   = grad_scale * grad                     (1 / #micro-batches for an accumulated sum)
    m   = beta1 * m + (1 - beta1) * g
    v   = beta2 * v + (1 - beta2) * g^2
    m^  = m / (1 - beta1^t),   v^ = v / (1 - beta2^t)
    p   = p - lr * (m^ / (sqrt(v^) + eps) + weight_decay * p)

Parity unpinned parts: none (pinned against closed forms and torch.optim.AdamW in tests).
"""
from __future__ import annotations

import dataclasses

import numpy as np


@dataclasses.dataclass(frozen=True)
class AdamWConfig:
    lr: float = 1e-3
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8
    weight_decay: float = 0.01
    grad_scale: float = 1.0


def adamw_step(p, g, m, v, t: int, cfg: AdamWConfig):
    """One AdamW update at step t (1-based).  Returns new (p, m, v) as float64 arrays."""
    p = np.asarray(p, np.float64)
    g = np.asarray(g, np.float64) * cfg.grad_scale
    m = cfg.beta1 * np.asarray(m, np.float64) + (1.0 - cfg.beta1) * g
    v = cfg.beta2 * np.asarray(v, np.float64) + (1.0 - cfg.beta2) * g * g
    m_hat = m / (1.0 - cfg.beta1 ** t)
    v_hat = v / (1.0 - cfg.beta2 ** t)
    p = p - cfg.lr * (m_hat / (np.sqrt(v_hat) + cfg.eps) + cfg.weight_decay * p)
    return p, m, v
