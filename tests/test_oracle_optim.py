"""Pins of the oracle's AdamW update (Section 4 trains with AdamW): closed forms of the first
step, the weight-decay-only case, and torch.optim.AdamW in float64 over several steps."""
import numpy as np
import pytest

from oracle.optim import AdamWConfig, adamw_step


def test_first_step_closed_form():
    """t = 1 from zero moments: m^ = g and v^ = g^2, so p1 = p0 (1 - lr wd) - lr g / (|g| + eps)."""
    rng = np.random.default_rng(0)
    p0, g = rng.standard_normal(1000), rng.standard_normal(1000)
    cfg = AdamWConfig(lr=3e-3, weight_decay=0.1, eps=1e-6)
    p1, m1, v1 = adamw_step(p0, g, np.zeros(1000), np.zeros(1000), 1, cfg)
    np.testing.assert_allclose(p1, p0 * (1 - cfg.lr * cfg.weight_decay) - cfg.lr * g / (np.abs(g) + cfg.eps),
                               rtol=1e-13, atol=1e-16)
    np.testing.assert_allclose(m1, (1 - cfg.beta1) * g, rtol=1e-15)
    np.testing.assert_allclose(v1, (1 - cfg.beta2) * g * g, rtol=1e-15)


def test_zero_gradient_is_pure_decay():
    p0 = np.linspace(-1, 1, 11)
    cfg = AdamWConfig(lr=0.1, weight_decay=0.5)
    p1, m1, v1 = adamw_step(p0, np.zeros(11), np.zeros(11), np.zeros(11), 3, cfg)
    np.testing.assert_array_equal(m1, 0.0)
    np.testing.assert_array_equal(v1, 0.0)
    np.testing.assert_allclose(p1, p0 * (1 - 0.05), rtol=1e-15)


def test_grad_scale_equals_averaged_gradient():
    rng = np.random.default_rng(1)
    p0, g = rng.standard_normal(64), rng.standard_normal(64)
    m0, v0 = rng.standard_normal(64) * 0.1, rng.random(64) * 0.1
    a = adamw_step(p0, 4 * g, m0, v0, 5, AdamWConfig(grad_scale=0.25))
    b = adamw_step(p0, g, m0, v0, 5, AdamWConfig())
    for x, y in zip(a, b):
        np.testing.assert_allclose(x, y, rtol=1e-14)


def test_matches_torch_adamw_float64():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(2)
    p = rng.standard_normal((16, 24))
    cfg = AdamWConfig(lr=2e-2, beta1=0.8, beta2=0.95, eps=1e-7, weight_decay=0.05)
    tp = torch.nn.Parameter(torch.from_numpy(p.copy()))
    opt = torch.optim.AdamW([tp], lr=cfg.lr, betas=(cfg.beta1, cfg.beta2), eps=cfg.eps,
                            weight_decay=cfg.weight_decay)
    m, v = np.zeros_like(p), np.zeros_like(p)
    for t in range(1, 6):
        g = rng.standard_normal(p.shape)
        tp.grad = torch.from_numpy(g.copy())
        opt.step()
        p, m, v = adamw_step(p, g, m, v, t, cfg)
        np.testing.assert_allclose(p, tp.detach().numpy(), rtol=1e-12, atol=1e-14)
