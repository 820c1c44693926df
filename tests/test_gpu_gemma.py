"""Gemma3 block options on the CUDA path against the oracle: QK-norm before RoPE, the sandwich
norms around attention and the MLP, the sqrt(D) embedding scale, and sliding-window local layers
with their own RoPE base.  Blocks are checked layer by layer (a local and a global layer, windows
narrower and wider than a 64-key tile, head dims 64 / 128 / 256, both attention-backward launch
modes), then Algorithm 1 end to end on a small model with a local/global layer pattern."""
import math

import numpy as np
import pytest

from oracle import model as OM
from oracle import quant
from workload import synth

from .helpers import dense_blocks, np_of, rel_fro, rowblock_err, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import (Context, DeviceBlock, DeviceModel, LoraSet, PackedLinear,  # noqa: E402
                                          compress)

TOL = 2e-2  # relative Frobenius error (fp16 operands, fp32 accumulate), as for the plain block
ELEM_TOL = 2e-2  # element-wise, per 64-row block relative to the block's largest value (as for the plain block)


def oracle_dense(W):
    out = {n: quant.dequant(*quant.compress(W[n])) for n in OM.LINEARS}
    for n in OM.NORMS:
        if n in W:
            out[n] = W[n].astype(np.float64)
    return out


def run_block(dims, layer):
    W = synth.block_weights(dims, layer, norm_jitter=0.1)
    L = synth.lora_weights(dims, layer)
    x = synth.hidden_input(dims)
    G = synth.upstream_grad(dims)
    ctx = Context(dims)
    blk = DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()})
    ls = LoraSet([L])
    xg, Gg = to_gpu(x), to_gpu(G)
    y = torch.empty_like(xg)
    dx = torch.empty_like(xg)
    M.mebp_block_recompute_fwd(ctx.handle, layer, blk.struct(), ls.layer(0), xg, y, dims.batch, dims.seq, False)
    M.mebp_block_bwd(ctx.handle, layer, blk.struct(), ls.layer(0), xg, Gg, dx, ls.layer_grads(0), dims.batch,
                     dims.seq)
    ctx.sync()
    Wd = oracle_dense(W)
    Lo = OM.lora64(L)
    xo = x.astype(np.float64)
    yo, _ = OM.block_forward(xo, Wd, Lo, dims, layer=layer)
    _, dxo, go = OM.block_objective(xo, Wd, Lo, G.astype(np.float64), dims, layer=layer)
    assert rel_fro(np_of(y) - xo, yo - xo) < TOL
    assert rel_fro(np_of(dx), dxo) < TOL, rel_fro(np_of(dx), dxo)
    ey, ed = rowblock_err(np_of(y) - xo, yo - xo), rowblock_err(np_of(dx), dxo)
    print(f"element-wise row-block error: y - x {ey:.2e}, dx {ed:.2e}")
    assert ey < ELEM_TOL and ed < ELEM_TOL, (ey, ed)
    for n, (dA, dB) in go.items():
        a, b = ls.grads[0][n]
        assert rel_fro(np_of(b), dB) < TOL, (n, "dB", rel_fro(np_of(b), dB))
        if np.linalg.norm(dA) > 0:
            assert rel_fro(np_of(a), dA) < TOL, (n, "dA", rel_fro(np_of(a), dA))
    return np_of(y), yo


CASES = [
    # window narrower than a key tile, three kv heads sharing nothing, GeGLU
    dict(hidden=192, n_heads=3, n_kv_heads=3, head_dim=64, intermediate=320, batch=2, seq=150, window=17, every=2),
    # window across tiles, grouped-query attention (2 query heads per kv head)
    dict(hidden=256, n_heads=4, n_kv_heads=2, head_dim=128, intermediate=512, batch=2, seq=200, window=70, every=3),
    # Gemma3-1B-like heads (hd 256, one kv head for four query heads)
    dict(hidden=512, n_heads=4, n_kv_heads=1, head_dim=256, intermediate=768, batch=1, seq=300, window=128, every=6),
]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("where", ["local", "global"])
def test_gemma_block_matches_oracle(case, where):
    c = dict(case)
    window, every = c.pop("window"), c.pop("every")
    dims = synth.tiny(n_layers=every, vocab=0, act="gelu_tanh", rank=16, alpha=32.0, targets=synth.TARGETS,
                      gemma_norms=True, sliding_window=window, global_every=every, rope_theta_local=1e4, **c)
    layer = 0 if where == "local" else every - 1
    assert dims.layer_is_local(layer) == (where == "local")
    run_block(dims, layer)


@pytest.mark.parametrize("hd,kv,batch,seq,window", [
    (128, 4, 5, 1024, 200),   # 320 key-block x kv-head items: the two-launch attention backward
    (256, 2, 8, 640, 100),    # head_dim 256 with > 2 waves: the single-buffered forward
])
def test_gemma_block_large_attention_grids_match_oracle(hd, kv, batch, seq, window):
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=kv, head_dim=hd, intermediate=256, n_layers=2, vocab=0,
                      act="gelu_tanh", batch=batch, seq=seq, rank=8, alpha=16.0, targets=("q", "k", "v", "o"),
                      gemma_norms=True, sliding_window=window, global_every=2)
    run_block(dims, 0)


def test_window_covering_the_sequence_equals_global_attention():
    """With the same RoPE base, a local layer whose window spans the sequence is the global layer."""
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=256, n_layers=2, vocab=0,
                      act="gelu_tanh", batch=2, seq=90, rank=8, alpha=16.0, gemma_norms=True, sliding_window=90,
                      global_every=2, rope_theta_local=1e6)
    W = synth.block_weights(dims, 0, norm_jitter=0.1)
    L = synth.lora_weights(dims, 0)
    x = to_gpu(synth.hidden_input(dims))
    ctx = Context(dims)
    blk = DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()})
    ls = LoraSet([L])
    ys = []
    for layer in (0, 1):
        y = torch.empty_like(x)
        M.mebp_block_recompute_fwd(ctx.handle, layer, blk.struct(), ls.layer(0), x, y, dims.batch, dims.seq, False)
        ys.append(y)
    ctx.sync()
    assert torch.equal(ys[0], ys[1])


def test_gemma_embedding_scale():
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=256, n_layers=1, vocab=512,
                      batch=2, seq=33, gemma_norms=True)
    E, _ = synth.embedding(dims)
    ctx = Context(dims)
    pE = PackedLinear(*compress(ctx, to_gpu(E)))
    ids = synth.token_ids(dims)
    x0 = torch.empty(ids.size, dims.hidden, device="cuda")
    M.mebp_embed(ctx.handle, pE.struct(), to_gpu(ids.reshape(-1)), x0)
    ctx.sync()
    ref = quant.dequant_rows(*quant.compress(E), ids.reshape(-1)) * np.float32(math.sqrt(dims.hidden))
    np.testing.assert_array_equal(np_of(x0), ref.astype(np.float32))


def test_gemma_model_step_matches_oracle():
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=512, n_layers=4, vocab=2048,
                      act="gelu_tanh", batch=2, seq=160, rank=8, alpha=16.0, targets=synth.TARGETS,
                      gemma_norms=True, sliding_window=48, global_every=3, rope_theta_local=1e4)
    blocks = dense_blocks(dims, norm_jitter=0.1)
    E, gf = synth.embedding(dims)
    loras = [synth.lora_weights(dims, i) for i in range(dims.n_layers)]
    ids = synth.token_ids(dims)
    ctx = Context(dims)
    dblocks = [DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()}) for W in blocks]
    model = DeviceModel(dblocks, PackedLinear(*compress(ctx, to_gpu(E))), to_gpu(gf))
    ls = LoraSet(loras)
    loss = torch.zeros(1, device="cuda")
    M.mebp_lora_step(ctx.handle, model.struct(), ls.lora_array(), to_gpu(ids), loss, ls.grads_array(), False)
    ctx.sync()
    lo, go = OM.mebp_backpropagation(OM.PackedModel.compress(blocks, E, gf), loras, ids, dims)
    assert abs(float(loss.item()) - lo) < 1e-3, (float(loss.item()), lo)
    for i in range(dims.n_layers):
        for n, (dA, dB) in go[i].items():
            a, b = ls.grads[i][n]
            assert rel_fro(np_of(a), dA) < TOL and rel_fro(np_of(b), dB) < TOL, (i, n)
