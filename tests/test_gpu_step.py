"""Algorithm 1 end to end (mebp_lora_step) against the oracle on the full
Qwen2.5-0.5B-shaped model (24 blocks, vocab 151936, batch 1 x seq 512), plus the
pinned-host checkpoint path, determinism and gradient accumulation."""
import numpy as np
import pytest

from oracle import model as OM
from workload import synth

from .helpers import dense_blocks, np_of, rel_fro, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, DeviceBlock, DeviceModel, LoraSet, PackedLinear, compress  # noqa: E402


def build(dims, blocks, E, gf, spill=False):
    ctx = Context(dims, spill=spill)
    dblocks = [DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()}) for W in blocks]
    model = DeviceModel(dblocks, PackedLinear(*compress(ctx, to_gpu(E))), to_gpu(gf))
    return ctx, model


def step(ctx, model, ls, ids, accumulate=False):
    loss = torch.zeros(1, device="cuda")
    M.mebp_lora_step(ctx.handle, model.struct(), ls.lora_array(), ids, loss, ls.grads_array(), accumulate)
    ctx.sync()
    return float(loss.item())


@pytest.mark.slow
def test_full_qwen05b_step_matches_oracle():
    dims = synth.preset(1)
    blocks = dense_blocks(dims)
    E, gf = synth.embedding(dims)
    loras = [synth.lora_weights(dims, i) for i in range(dims.n_layers)]
    ids = synth.token_ids(dims)
    ctx, model = build(dims, blocks, E, gf)
    ls = LoraSet(loras)
    loss = step(ctx, model, ls, to_gpu(ids))
    pm = OM.PackedModel.compress(blocks, E, gf)
    lo, go = OM.mebp_backpropagation(pm, loras, ids, dims)
    assert abs(loss - lo) < 1e-3, (loss, lo)
    worst = 0.0
    for i in range(dims.n_layers):
        for n, (dA, dB) in go[i].items():
            a, b = ls.grads[i][n]
            ea, eb = rel_fro(np_of(a), dA), rel_fro(np_of(b), dB)
            worst = max(worst, ea, eb)
            assert ea < 2e-2 and eb < 2e-2, (i, n, ea, eb)
    print("worst relative Frobenius error of a LoRA gradient:", worst)


def _small():
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=512, n_layers=4, vocab=2048,
                      batch=2, seq=96, rank=8, alpha=16.0)
    blocks = dense_blocks(dims)
    E, gf = synth.embedding(dims)
    loras = [synth.lora_weights(dims, i) for i in range(dims.n_layers)]
    return dims, blocks, E, gf, loras, synth.token_ids(dims)


def test_step_at_2048_tokens_matches_oracle():
    """The large-token path of the step: from 2048 tokens the gate|up GEMM applies the gated
    activation in its epilogue (and skips storing gate and up for blocks that are recomputed
    before their backward), the fused GEMMs use two accumulators and the LoRA-gradient
    reductions run on the tensor cores; four blocks, rank 16 on all seven linears."""
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=512, n_layers=4, vocab=2048,
                      batch=2, seq=1024, rank=16, alpha=32.0, targets=synth.TARGETS)
    blocks = dense_blocks(dims)
    E, gf = synth.embedding(dims)
    loras = [synth.lora_weights(dims, i) for i in range(dims.n_layers)]
    ids = synth.token_ids(dims)
    ctx, model = build(dims, blocks, E, gf)
    ls = LoraSet(loras)
    loss = step(ctx, model, ls, to_gpu(ids))
    lo, go = OM.mebp_backpropagation(OM.PackedModel.compress(blocks, E, gf), loras, ids, dims)
    assert abs(loss - lo) < 1e-3, (loss, lo)
    for i in range(dims.n_layers):
        for n, (dA, dB) in go[i].items():
            a, b = ls.grads[i][n]
            assert rel_fro(np_of(a), dA) < 2e-2 and rel_fro(np_of(b), dB) < 2e-2, (i, n)


def test_small_model_step_matches_oracle():
    dims, blocks, E, gf, loras, ids = _small()
    ctx, model = build(dims, blocks, E, gf)
    ls = LoraSet(loras)
    loss = step(ctx, model, ls, to_gpu(ids))
    lo, go = OM.mebp_backpropagation(OM.PackedModel.compress(blocks, E, gf), loras, ids, dims)
    assert abs(loss - lo) < 1e-3
    for i in range(dims.n_layers):
        for n, (dA, dB) in go[i].items():
            a, b = ls.grads[i][n]
            assert rel_fro(np_of(a), dA) < 2e-2 and rel_fro(np_of(b), dB) < 2e-2, (i, n)


def test_spill_to_host_is_bit_identical_and_deterministic():
    dims, blocks, E, gf, loras, ids = _small()
    idg = to_gpu(ids)
    res = []
    for spill in (False, True, True):
        ctx, model = build(dims, blocks, E, gf, spill=spill)
        ls = LoraSet(loras)
        loss = step(ctx, model, ls, idg)
        res.append((loss, [{n: (np_of(a), np_of(b)) for n, (a, b) in g.items()} for g in ls.grads]))
        ctx.close()
    for other in res[1:]:
        assert other[0] == res[0][0]
        for g0, g1 in zip(res[0][1], other[1]):
            for n in g0:
                np.testing.assert_array_equal(g0[n][0], g1[n][0])
                np.testing.assert_array_equal(g0[n][1], g1[n][1])


def test_step_gradient_accumulation_doubles():
    dims, blocks, E, gf, loras, ids = _small()
    ctx, model = build(dims, blocks, E, gf)
    ls = LoraSet(loras)
    idg = to_gpu(ids)
    step(ctx, model, ls, idg)
    once = [{n: (a.clone(), b.clone()) for n, (a, b) in g.items()} for g in ls.grads]
    step(ctx, model, ls, idg, accumulate=True)
    for g0, g1 in zip(once, ls.grads):
        for n in g0:
            assert torch.equal(2 * g0[n][0], g1[n][0]) and torch.equal(2 * g0[n][1], g1[n][1])


@pytest.mark.parametrize("spill", [False, True])
def test_graph_replay_is_bit_identical_to_eager(spill):
    """On a non-default stream the step is run eagerly once, captured on the second call and
    replayed afterwards; every call must give the eager result bit for bit."""
    dims, blocks, E, gf, loras, ids = _small()
    idg = to_gpu(ids)
    ctx, model = build(dims, blocks, E, gf, spill=spill)
    ls = LoraSet(loras)
    mstruct = model.struct()
    loss = torch.zeros(1, device="cuda")
    s = torch.cuda.Stream()
    results = []
    with torch.cuda.stream(s):
        for _ in range(4):
            n0 = M.mebp_kernel_launches()
            M.mebp_lora_step(ctx.handle, mstruct, ls.lora_array(), idg, loss, ls.grads_array())
            ctx.sync()
            results.append((float(loss.item()), [{n: (a.clone(), b.clone()) for n, (a, b) in g.items()}
                                                 for g in ls.grads], M.mebp_kernel_launches() - n0))
    M.mebp_enable_graphs(ctx.handle, False)
    with torch.cuda.stream(s):
        M.mebp_lora_step(ctx.handle, mstruct, ls.lora_array(), idg, loss, ls.grads_array())
        ctx.sync()
    ref = (float(loss.item()), ls.grads)
    for lo, gr, launches in results:
        assert lo == ref[0]
        assert launches == results[0][2]          # a replay counts the kernels it runs
        for g0, g1 in zip(gr, ref[1]):
            for n in g0:
                assert torch.equal(g0[n][0], g1[n][0]) and torch.equal(g0[n][1], g1[n][1])
