"""AdamW (Section 4 trains every model with AdamW) through the C ABI against the oracle, and a
multi-step LoRA fine-tuning loop (mebp_lora_step + mebp_adamw_step) followed step by step
against the oracle's Algorithm 1 + AdamW trajectory."""
import numpy as np
import pytest

from oracle import model as OM
from oracle.optim import AdamWConfig, adamw_step
from workload import synth

from .helpers import dense_blocks, np_of, rel_fro, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, DeviceBlock, DeviceModel, LoraSet, PackedLinear, compress  # noqa: E402


@pytest.fixture(scope="module")
def ctx():
    c = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=64, max_seq=64)
    yield c
    c.close()


def _cfg_pair(**kw):
    o = AdamWConfig(**kw)
    return o, M.adamw_cfg(o.lr, o.beta1, o.beta2, o.eps, o.weight_decay, o.grad_scale)


@pytest.mark.parametrize("n", [1, 7, 1001, 1 << 20])
def test_adamw_matches_oracle_over_steps(ctx, n):
    """fp32 kernel vs fp64 oracle over four steps.  Where beta1 m and (1 - beta1) g nearly cancel,
    fp32 keeps only an absolute accuracy of a few ulps of the summed terms, so each element's bound
    is 1e-5 relative plus 2e-7 times the sum of |g| (|g|^2 for v) it has seen."""
    rng = np.random.default_rng(n)
    oc, gc = _cfg_pair(lr=5e-3, beta1=0.85, beta2=0.99, eps=1e-6, weight_decay=0.02, grad_scale=0.5)
    p = rng.standard_normal(n).astype(np.float32)
    pg, mg, vg = to_gpu(p), torch.zeros(n, device="cuda"), torch.zeros(n, device="cuda")
    po, mo, vo = p.astype(np.float64), np.zeros(n), np.zeros(n)
    sum_g, sum_g2 = np.zeros(n), np.zeros(n)
    steps = 4
    for t in range(1, steps + 1):
        g = (rng.standard_normal(n) * 10.0 ** rng.uniform(-3, 1, n)).astype(np.float32)
        M.mebp_adamw_step(ctx.handle, pg, to_gpu(g), mg, vg, gc, t)
        po, mo, vo = adamw_step(po, g, mo, vo, t, oc)
        sum_g += np.abs(g.astype(np.float64)) * oc.grad_scale
        sum_g2 += (g.astype(np.float64) * oc.grad_scale) ** 2
    ctx.sync()
    assert np.all(np.abs(np_of(mg) - mo) <= 1e-5 * np.abs(mo) + 2e-7 * sum_g)
    assert np.all(np.abs(np_of(vg) - vo) <= 1e-5 * np.abs(vo) + 2e-7 * sum_g2)
    # the parameter moves by ~lr per step: compare the movement, not just the value
    move_g, move_o = np_of(pg).astype(np.float64) - p, po - p
    assert np.all(np.abs(move_g - move_o) <= 1e-4 * np.abs(move_o) + steps * oc.lr * 1e-4)


def test_adamw_rejects_bad_arguments(ctx):
    x = torch.zeros(64, device="cuda")
    cfg = M.adamw_cfg()
    for bad in (dict(step=0), dict(params=x[1:])):
        kw = dict(params=x, step=1)
        kw.update(bad)
        with pytest.raises(M.MebpError) as ei:
            M.mebp_adamw_step(ctx.handle, kw["params"], x, x.clone(), x.clone(), cfg, kw["step"])
        assert ei.value.code == M.ERR_INVALID_ARG
    with pytest.raises(M.MebpError):
        M.mebp_adamw_step(ctx.handle, x, x, x.clone(), x.clone(), M.adamw_cfg(beta1=1.0), 1)


def _small():
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=512, n_layers=3, vocab=2048,
                      batch=2, seq=64, rank=8, alpha=16.0)
    return dims, dense_blocks(dims), *synth.embedding(dims), [synth.lora_weights(dims, i) for i in range(dims.n_layers)]


def test_training_loop_follows_oracle_trajectory():
    """Three fine-tuning steps on one batch: the loss at every step within 1e-3 of the oracle's
    (it depends on every updated weight), and the total movement of every LoRA tensor within
    0.1 relative Frobenius of the oracle's.  Adam moves each coordinate by about lr whatever the
    gradient's size, so a coordinate whose gradient lies within the GPU path's gradient error
    (2e-2 relative Frobenius at most, about 0.3 % here) of zero may move either way; the movement
    bound allows for those coordinates."""
    dims, blocks, E, gf, loras = _small()
    ids = synth.token_ids(dims)
    oc, gc = _cfg_pair(lr=2e-3, weight_decay=0.01)  # a step flips coordinates with |g| near 0: keep lr small
    ctx = Context(dims)
    dblocks = [DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()}) for W in blocks]
    model = DeviceModel(dblocks, PackedLinear(*compress(ctx, to_gpu(E))), to_gpu(gf))
    ls = LoraSet(loras)
    idg = to_gpu(ids)
    loss = torch.zeros(1, device="cuda")
    pm = OM.PackedModel.compress(blocks, E, gf)
    lo = [OM.lora64(L) for L in loras]
    mo = [{n: (np.zeros_like(A), np.zeros_like(B)) for n, (A, B) in L.items()} for L in lo]
    vo = [{n: (np.zeros_like(A), np.zeros_like(B)) for n, (A, B) in L.items()} for L in lo]
    for t in range(1, 4):
        M.mebp_lora_step(ctx.handle, model.struct(), ls.lora_array(), idg, loss, ls.grads_array())
        ls.adamw(ctx, gc)
        ctx.sync()
        loss_o, go = OM.mebp_backpropagation(pm, lo, ids, dims)
        assert abs(loss.item() - loss_o) < 1e-3, (t, loss.item(), loss_o)
        for i in range(dims.n_layers):
            for n in lo[i]:
                new = []
                for j in range(2):
                    p, m, v = adamw_step(lo[i][n][j], go[i][n][j], mo[i][n][j], vo[i][n][j], t, oc)
                    new.append((p, m, v))
                lo[i][n] = (new[0][0], new[1][0])
                mo[i][n] = (new[0][1], new[1][1])
                vo[i][n] = (new[0][2], new[1][2])
    for i in range(dims.n_layers):
        for n, (A0, B0) in loras[i].items():
            a, b = ls.lora[i][n]
            assert rel_fro(np_of(a) - A0, lo[i][n][0] - A0) < 0.1, (i, n, "A")
            assert rel_fro(np_of(b) - B0, lo[i][n][1] - B0) < 0.1, (i, n, "B")


def test_training_loop_reduces_loss_on_a_fixed_batch():
    dims, blocks, E, gf, loras = _small()
    ctx = Context(dims)
    dblocks = [DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()}) for W in blocks]
    model = DeviceModel(dblocks, PackedLinear(*compress(ctx, to_gpu(E))), to_gpu(gf))
    ls = LoraSet(loras)
    idg = to_gpu(synth.token_ids(dims))
    loss = torch.zeros(1, device="cuda")
    hist = []
    for _ in range(20):
        M.mebp_lora_step(ctx.handle, model.struct(), ls.lora_array(), idg, loss, ls.grads_array())
        ls.adamw(ctx, M.adamw_cfg(lr=1e-2, weight_decay=0.0))
        ctx.sync()
        hist.append(loss.item())
    assert hist[-1] < hist[0] - 0.5, hist
    assert all(np.isfinite(hist))
