"""Parity at the workloads' full sizes, in the launch configuration the benchmark times,
on outputs the oracle can compute one sample at a time:

* fused GEMMs at M = 16384 (Gemma3-4B-shaped projections): sampled rows;
* one decoder block of the Gemma3-1B / Qwen2.5-1.5B / Gemma3-4B-shaped models run over the
  full batch, with the upstream gradient non-zero on the first and the last sequence only —
  sequences do not interact, so y of every sequence equals the oracle's block run on that
  sequence alone (element-wise), dE/dx of the two graded sequences equals the oracle's, dE/dx
  of the others is zero, and every LoRA gradient is the sum over the two graded sequences;
* the LM head over the full vocabulary: per-token loss and dE/dh on sampled tokens.
"""
import numpy as np
import pytest

from oracle import model as OM
from oracle import quant
from workload import synth

from .helpers import f16_round, np_of, rel_fro, rowblock_err, to_gpu
from .test_gpu_block import ELEM_TOL, oracle_dense

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, DeviceBlock, LoraSet, PackedLinear, compress  # noqa: E402


@pytest.mark.parametrize("name,N,K", [("qkv", 4096, 2560), ("o", 2560, 2048), ("gate_up", 20480, 2560),
                                      ("down", 2560, 10240)])
def test_gemm_rows_at_full_size(name, N, K):
    Mr = 16384
    rng = np.random.default_rng(N + K)
    W = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    qo, so = quant.compress(W)
    Wh = quant.f16_bits_to_f64(quant.dequant_f16_bits(qo, so))
    ctx = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=64, max_seq=64)
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    X = torch.randn(Mr, K, device="cuda").to(torch.float16)
    dY = torch.randn(Mr, N, device="cuda").to(torch.float16)
    Y = torch.empty(Mr, N, device="cuda")
    dX = torch.empty(Mr, K, device="cuda")
    M.mebp_linear_fwd(ctx.handle, X, Wp, y_f32=Y)
    M.mebp_linear_dx(ctx.handle, dY, Wp, dx=dX)
    ctx.sync()
    rows = np.sort(rng.choice(Mr, 24, replace=False))
    rows[-1] = Mr - 1
    Xr = np_of(X[rows]).astype(np.float64)
    dYr = np_of(dY[rows]).astype(np.float64)
    ref_y = Xr @ Wh.T
    ref_dx = dYr @ Wh
    # fp32 accumulation over the reduction: the bound grows with sqrt(reduction length)
    assert np.abs(np_of(Y[rows]) - ref_y).max() <= 2e-5 * max(1.0, np.sqrt(K / 2560)) * np.abs(ref_y).max()
    assert np.abs(np_of(dX[rows]) - ref_dx).max() <= 2e-5 * max(1.0, np.sqrt(N / 2560)) * np.abs(ref_dx).max()


@pytest.mark.parametrize("cfg", [2, 3, 4])
def test_block_at_full_batch_against_per_sequence_oracle(cfg):
    dims = synth.preset(cfg)
    W = synth.block_weights(dims, 0)
    L = synth.lora_weights(dims, 0)
    x = synth.hidden_input(dims)
    G = synth.upstream_grad(dims)
    S, B = dims.seq, dims.batch
    graded = sorted({0, B - 1})               # the first and the last sequence carry gradient
    for b in range(B):
        if b not in graded:
            G[b * S:(b + 1) * S] = 0.0
    ctx = Context(dims)
    blk = DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()})
    ls = LoraSet([L])
    xg, Gg = to_gpu(x), to_gpu(G)
    y = torch.empty_like(xg)
    dx = torch.empty_like(xg)
    M.mebp_block_recompute_fwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, y, B, S, False)
    M.mebp_block_bwd(ctx.handle, 0, blk.struct(), ls.layer(0), xg, Gg, dx, ls.layer_grads(0), B, S)
    ctx.sync()
    y_np, dx_np = np_of(y), np_of(dx)
    d1 = dims.with_(batch=1)
    Wd = oracle_dense(W)
    Lo = OM.lora64(L)
    # sequences do not interact: the oracle runs each one alone
    for b in range(B):
        rows = slice(b * S, (b + 1) * S)
        xb = x[rows].astype(np.float64)
        if b in graded:
            continue
        yo, _ = OM.block_forward(xb, Wd, Lo, d1)
        e = rowblock_err(y_np[rows] - xb, yo - xb)
        assert e < ELEM_TOL, (b, "y", e)
        assert float(np.abs(dx_np[rows]).max()) == 0.0, b
    grads = {}
    for b in graded:
        rows = slice(b * S, (b + 1) * S)
        xb = x[rows].astype(np.float64)
        yo, _ = OM.block_forward(xb, Wd, Lo, d1)
        _, dxo, go = OM.block_objective(xb, Wd, Lo, G[rows].astype(np.float64), d1)
        ey, ed = rowblock_err(y_np[rows] - xb, yo - xb), rowblock_err(dx_np[rows], dxo)
        print(f"sequence {b}: element-wise row-block error y - x {ey:.2e}, dx {ed:.2e}")
        assert rel_fro(y_np[rows] - xb, yo - xb) < 2e-2
        assert rel_fro(dx_np[rows], dxo) < 2e-2
        assert ey < ELEM_TOL and ed < ELEM_TOL, (b, ey, ed)
        for n, (dA, dB) in go.items():
            pa, pb = grads.get(n, (0.0, 0.0))
            grads[n] = (pa + dA, pb + dB)
    # LoRA gradients of the batch = the sum over the graded sequences
    for n, (dA, dB) in grads.items():
        a, b = ls.grads[0][n]
        assert rel_fro(np_of(a), dA) < 2e-2, (n, "dA", rel_fro(np_of(a), dA))
        assert rel_fro(np_of(b), dB) < 2e-2, (n, "dB", rel_fro(np_of(b), dB))


@pytest.mark.parametrize("cfg", [1, 4])
def test_lmhead_full_vocab_sampled_tokens(cfg):
    dims = synth.preset(cfg)
    T = dims.tokens
    E, gf = synth.embedding(dims)
    rng = np.random.default_rng(cfg)
    h = rng.standard_normal((T, dims.hidden)).astype(np.float32)
    tg = synth.token_ids(dims)
    tgt = OM.next_token_targets(tg).astype(np.int32)
    ctx = Context(dims)
    Ep = PackedLinear(*compress(ctx, to_gpu(E)))
    loss = torch.zeros(1, device="cuda")
    dh = torch.empty((T, dims.hidden), device="cuda")
    tok = torch.empty(T, device="cuda")
    M.mebp_lmhead_ce_fwd_bwd(ctx.handle, Ep.struct(), to_gpu(gf), to_gpu(h), to_gpu(tgt), loss, dh, tok)
    ctx.sync()
    n_valid = int((tgt >= 0).sum())
    tok_np = np_of(tok)
    assert abs(loss.item() - tok_np.sum() / n_valid) < 1e-4
    rows = np.sort(rng.choice(T, 24, replace=False))
    rows[-1] = dims.seq - 1                   # an ignored position
    Ed = quant.dequant(*quant.compress(E))
    hr = h[rows].astype(np.float64)
    # oracle on the sampled rows alone, rescaled from its own valid count to the full one
    _, dho, toko = OM.lm_head_ce(hr, gf.astype(np.float64), Ed, tgt[rows], dims.eps, want_token_loss=True)
    n_rows = int((tgt[rows] >= 0).sum())
    dho *= n_rows / n_valid
    np.testing.assert_allclose(tok_np[rows], toko, atol=2e-3)
    assert rel_fro(np_of(dh[rows]), dho) < 2e-2
