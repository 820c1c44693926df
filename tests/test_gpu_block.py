"""Block-level parity (forward_i / backward_i of Algorithm 1) of the CUDA path against the
oracle: the single Qwen2.5-0.5B-shaped block (batch 1 x seq 128, objective sum(G*y)) and
smaller blocks covering head dims 128 / 256, grouped-query attention, GeGLU, every LoRA
target, ranks 8-32 and sequence lengths that leave ragged tiles."""
import numpy as np
import pytest

from oracle import model as OM
from oracle import quant
from workload import synth

from .helpers import np_of, rel_fro, rowblock_err, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, DeviceBlock, LoraSet  # noqa: E402

TOL = 2e-2  # relative Frobenius error of gradients (stated bound; fp16 operands, fp32 accumulate)
# Element-wise bound on the activations y - x and dE/dx, per 64-row block relative to the block's
# largest value.  Every GEMM operand is rounded to fp16 (relative 2^-11); a block chains about six
# contractions plus softmax and norms, so elements carry errors of a few 1e-3 of the block's scale.
ELEM_TOL = 2e-2


def oracle_dense(W):
    """The oracle's own decode of the oracle's own compression of W."""
    out = {n: quant.dequant(*quant.compress(W[n])) for n in OM.LINEARS}
    out["norm1"] = W["norm1"].astype(np.float64)
    out["norm2"] = W["norm2"].astype(np.float64)
    return out


def run_block(dims, jitter=0.0, zero_b=False, x_scale=1.0):
    W = synth.block_weights(dims, 0, norm_jitter=jitter)
    L = synth.lora_weights(dims, 0, zero_b=zero_b)
    x = synth.hidden_input(dims) * np.float32(x_scale)
    G = synth.upstream_grad(dims)
    ctx = Context(dims)
    blk = DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()})
    ls = LoraSet([L])
    xg, Gg = to_gpu(x), to_gpu(G)
    y = torch.empty_like(xg)
    dx = torch.empty_like(xg)
    M.mebp_block_recompute_fwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, y, dims.batch, dims.seq, False)
    M.mebp_block_bwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, Gg, dx, ls.layer_grads(0), dims.batch, dims.seq)
    ctx.sync()
    gpu = dict(y=np_of(y), dx=np_of(dx), grads={n: (np_of(a), np_of(b)) for n, (a, b) in ls.grads[0].items()})
    # oracle
    Wd = oracle_dense(W)
    Lo = OM.lora64(L)
    xo = x.astype(np.float64)
    yo, _ = OM.block_forward(xo, Wd, Lo, dims)
    _, dxo, go = OM.block_objective(xo, Wd, Lo, G.astype(np.float64), dims)
    ref = dict(y=yo, dx=dxo, grads=go, x=xo)
    return gpu, ref, (ctx, blk, ls, xg, Gg)


def check(gpu, ref, tol=TOL, elem_tol=ELEM_TOL):
    assert rel_fro(gpu["y"] - ref["x"], ref["y"] - ref["x"]) < tol
    assert rel_fro(gpu["dx"], ref["dx"]) < tol
    ey = rowblock_err(gpu["y"] - ref["x"], ref["y"] - ref["x"])
    ed = rowblock_err(gpu["dx"], ref["dx"])
    print(f"element-wise row-block error: y - x {ey:.2e}, dx {ed:.2e}")
    assert ey < elem_tol, ey
    assert ed < elem_tol, ed
    for n, (dA, dB) in ref["grads"].items():
        ga, gb = gpu["grads"][n]
        assert rel_fro(gb, dB) < tol, (n, "dB", rel_fro(gb, dB))
        if np.linalg.norm(dA) > 0:
            assert rel_fro(ga, dA) < tol, (n, "dA", rel_fro(ga, dA))


def test_qwen05b_block_matches_oracle():
    gpu, ref, _ = run_block(synth.preset(0))
    check(gpu, ref)


@pytest.mark.parametrize("kw", [
    dict(hidden=256, n_heads=4, n_kv_heads=2, head_dim=128, intermediate=512, act="silu", batch=2, seq=80,
         rank=16, alpha=32.0, targets=synth.TARGETS),
    dict(hidden=512, n_heads=2, n_kv_heads=1, head_dim=256, intermediate=768, act="gelu_tanh", batch=1, seq=200,
         rank=32, alpha=64.0, targets=synth.TARGETS),
    dict(hidden=192, n_heads=3, n_kv_heads=3, head_dim=64, intermediate=320, act="gelu_tanh", batch=3, seq=33,
         rank=8, alpha=16.0, targets=("q", "v", "up", "down")),
])
def test_block_variants_match_oracle(kw):
    dims = synth.tiny(n_layers=1, vocab=0, **kw)
    gpu, ref, _ = run_block(dims, jitter=0.1)
    check(gpu, ref)


@pytest.mark.parametrize("kw", [
    # enough 128-row tiles for the tcgen05 attention kernels (forward and backward), ragged ends
    dict(hidden=256, n_heads=8, n_kv_heads=8, head_dim=64, intermediate=256, act="silu", batch=10, seq=200,
         rank=8, alpha=16.0, targets=("q", "k", "v", "o")),
    dict(hidden=256, n_heads=8, n_kv_heads=4, head_dim=128, intermediate=256, act="gelu_tanh", batch=20, seq=250,
         rank=16, alpha=32.0, targets=synth.TARGETS),
    dict(hidden=512, n_heads=4, n_kv_heads=2, head_dim=256, intermediate=256, act="silu", batch=20, seq=140,
         rank=8, alpha=16.0, targets=("q", "k", "v", "o")),
])
def test_block_on_tensor_core_attention_matches_oracle(kw):
    dims = synth.tiny(n_layers=1, vocab=0, **kw)
    gpu, ref, _ = run_block(dims, jitter=0.1)
    check(gpu, ref)


def test_lora_b_zero_block_equals_base_block_and_da_is_zero():
    dims = synth.preset(0)
    gpu, ref, (ctx, blk, ls, xg, Gg) = run_block(dims, zero_b=True)
    for n, (dA, dB) in gpu["grads"].items():
        assert np.all(dA == 0), n
        assert np.any(dB != 0), n
    # base block (no LoRA targets) is bit-identical to LoRA with B = 0
    base = dims.with_(targets=())
    ctx0 = Context(base)
    W = synth.block_weights(dims, 0)
    blk0 = DeviceBlock(ctx0, {k: to_gpu(v) for k, v in W.items()})
    y0 = torch.empty_like(xg)
    M.mebp_block_recompute_fwd(ctx0.handle, 0, blk0.struct(), M.Lora(), xg, y0, dims.batch, dims.seq, False)
    ctx0.sync()
    np.testing.assert_array_equal(np_of(y0), gpu["y"])


def test_saved_intermediates_give_the_same_backward_as_recompute():
    dims = synth.preset(0)
    gpu, _, (ctx, blk, ls, xg, Gg) = run_block(dims)
    y = torch.empty_like(xg)
    dx = torch.empty_like(xg)
    M.mebp_block_recompute_fwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, y, dims.batch, dims.seq, True)
    M.mebp_block_bwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, Gg, dx, ls.layer_grads(0), dims.batch, dims.seq)
    ctx.sync()
    np.testing.assert_array_equal(np_of(dx), gpu["dx"])
    for n, (a, b) in ls.grads[0].items():
        np.testing.assert_array_equal(np_of(a), gpu["grads"][n][0])
        np.testing.assert_array_equal(np_of(b), gpu["grads"][n][1])


@pytest.mark.parametrize("tokens,act", [(512, "silu"), (1024, "gelu_tanh"), (2048, "silu")])
def test_gated_activation_in_the_gemm_epilogue_is_bit_identical(tokens, act):
    """Without save_for_bwd the gate|up GEMM applies the gated activation in its epilogue and
    stores m alone (one-accumulator tiles below 2048 tokens, two from 2048); with it, gate and up
    are stored for the backward and, below 2048 tokens, a separate kernel computes m.  Both round
    gate and up to fp16 first, so the block outputs agree bit for bit."""
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=2560, act=act, n_layers=1,
                      vocab=0, batch=1, seq=tokens, rank=16)
    W = synth.block_weights(dims, 0)
    L = synth.lora_weights(dims, 0)
    ctx = Context(dims)
    blk = DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()})
    ls = LoraSet([L])
    xg = to_gpu(synth.hidden_input(dims))
    y0, y1 = torch.empty_like(xg), torch.empty_like(xg)
    M.mebp_block_recompute_fwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, y0, 1, tokens, False)
    M.mebp_block_recompute_fwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, y1, 1, tokens, True)
    ctx.sync()
    assert torch.isfinite(y0).all()
    assert torch.equal(y0, y1)
    ctx.close()


def test_gradient_accumulation_adds():
    dims = synth.preset(0)
    gpu, _, (ctx, blk, ls, xg, Gg) = run_block(dims)
    dx = torch.empty_like(xg)
    M.mebp_block_bwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, Gg, dx, ls.layer_grads(0), dims.batch, dims.seq,
                     accumulate=True)
    ctx.sync()
    for n, (a, b) in ls.grads[0].items():
        np.testing.assert_array_equal(np_of(a), 2 * gpu["grads"][n][0])
        np.testing.assert_array_equal(np_of(b), 2 * gpu["grads"][n][1])
