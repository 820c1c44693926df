"""LM head + cross-entropy parity (final RMSNorm, tied 4-bit embedding, mean next-token
loss, chunked over the vocabulary) against the oracle's full-logit definition."""
import numpy as np
import pytest

from oracle import model as OM
from oracle import quant
from workload import synth

from .helpers import np_of, rel_fro, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, PackedLinear, compress  # noqa: E402


def run(dims, T, chunk, ignore_every=7, h_scale=1.0, seed=0):
    E, gf = synth.embedding(dims, norm_jitter=0.1)
    rng = np.random.default_rng(seed)
    h = (rng.standard_normal((T, dims.hidden)) * h_scale).astype(np.float32)
    tg = rng.integers(0, dims.vocab, T).astype(np.int32)
    tg[::ignore_every] = -1
    ctx = Context(dims, max_tokens=T, vocab_chunk=chunk)
    Ep = PackedLinear(*compress(ctx, to_gpu(E)))
    loss = torch.zeros(1, device="cuda")
    dh = torch.empty((T, dims.hidden), device="cuda")
    tok = torch.empty(T, device="cuda")
    M.mebp_lmhead_ce_fwd_bwd(ctx.handle, Ep.struct(), to_gpu(gf), to_gpu(h), to_gpu(tg), loss, dh, tok)
    ctx.sync()
    Ed = quant.dequant(*quant.compress(E))
    lo, dho, toko = OM.lm_head_ce(h.astype(np.float64), gf.astype(np.float64), Ed, tg, dims.eps, want_token_loss=True)
    return float(loss.item()), np_of(dh), np_of(tok), lo, dho, toko, tg


@pytest.mark.parametrize("V,chunk,T", [(1088, 256, 100), (1088, 0, 100), (4096, 1024, 300), (64, 256, 5)])
def test_lmhead_matches_oracle(V, chunk, T):
    dims = synth.tiny(hidden=128, head_dim=64, vocab=V)
    loss, dh, tok, lo, dho, toko, tg = run(dims, T, chunk)
    assert abs(loss - lo) < 1e-3
    np.testing.assert_allclose(tok, toko, atol=2e-3)
    assert np.all(tok[tg < 0] == 0)
    assert rel_fro(dh, dho) < 2e-2
    assert np.all(dh[tg < 0] == 0)


def test_lmhead_chunking_does_not_change_the_result_beyond_rounding():
    dims = synth.tiny(hidden=128, head_dim=64, vocab=4096)
    a = run(dims, 300, 256)
    b = run(dims, 300, 4096)
    assert abs(a[0] - b[0]) < 1e-5
    assert rel_fro(a[1], b[1]) < 1e-3


def test_lmhead_uniform_logits_give_log_v():
    dims = synth.tiny(hidden=64, head_dim=64, vocab=512)
    T = 40
    ctx = Context(dims, max_tokens=T)
    Ep = PackedLinear(*compress(ctx, torch.zeros((512, 64), device="cuda")))
    loss = torch.zeros(1, device="cuda")
    dh = torch.empty((T, 64), device="cuda")
    h = torch.randn((T, 64), device="cuda")
    tg = torch.randint(0, 512, (T,), dtype=torch.int32, device="cuda")
    M.mebp_lmhead_ce_fwd_bwd(ctx.handle, Ep.struct(), torch.ones(64, device="cuda"), h, tg, loss, dh)
    ctx.sync()
    assert abs(loss.item() - np.log(512)) < 1e-5
    assert float(dh.abs().max()) == 0.0
