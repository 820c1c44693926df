"""mebp_linear_fwd_noalloc: the fused LoRA linear for callers that may not allocate device
memory (it needs no context and keeps its scratch in a fixed static device array).

Checked through the C ABI against the regular mebp_linear_fwd on two calls in a row (the
second call reuses the scratch the first one left behind, with a different shape), within
the accumulation tolerance the other GEMM tests use, and against the oracle's
X deq(W)^T + s (X A^T) B^T + R in fp64, with and without LoRA and residual.  This file is
collected last so that a stop-at-first-failure run has already run every other test."""
import ctypes

import numpy as np
import pytest

from oracle import quant
from workload import synth

from .helpers import np_of, rel_fro, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context  # noqa: E402


def _case(Mr, N, K, r, seed, oracle=False):
    rng = np.random.default_rng(seed)
    qo, so = quant.compress((rng.standard_normal((N, K)) * 0.02).astype(np.float32))
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    Xh = rng.standard_normal((Mr, K)).astype(np.float16)
    X = torch.from_numpy(Xh).cuda()
    An = (rng.standard_normal((r, K)) * 0.05).astype(np.float32) if r else None
    Bn = (rng.standard_normal((N, r)) * 0.05).astype(np.float32) if r else None
    Rn = rng.standard_normal((Mr, N)).astype(np.float32)
    A = to_gpu(An) if r else None
    B = to_gpu(Bn) if r else None
    R = to_gpu(Rn)
    if not oracle:
        return Wp, X, A, B, R
    return Wp, X, A, B, R, (quant.dequant(qo, so), Xh.astype(np.float64), An, Bn, Rn.astype(np.float64))


def _oracle_linear(Wd, X, A, B, R, s):
    """The linear of Algorithm 1 with the oracle's decode: X deq(W)^T + s (X A^T) B^T (+ R)."""
    y = X @ Wd.T
    if A is not None:
        y = y + s * (X @ A.T.astype(np.float64)) @ B.T.astype(np.float64)
    return y if R is None else y + R


def test_noalloc_linear_matches_linear_fwd_on_two_calls_in_a_row():
    ctx = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=64, max_seq=64)
    cases = [(300, 1152, 896, 16, 1), (130, 512, 256, 8, 2)]
    for Mr, N, K, r, seed in cases:
        Wp, X, A, B, R = _case(Mr, N, K, r, seed)
        ref = torch.empty((Mr, N), device="cuda")
        M.mebp_linear_fwd(ctx.handle, X, Wp, A, B, r, 2.0, R=R, y_f32=ref)
        out = torch.full((Mr, N), float("nan"), device="cuda")
        M.mebp_linear_fwd_noalloc(X, Wp, A, B, r, 2.0, R=R, y_f32=out)
        out16 = torch.full((Mr, N), float("nan"), device="cuda", dtype=torch.float16)
        ref16 = torch.empty((Mr, N), device="cuda", dtype=torch.float16)
        M.mebp_linear_fwd(ctx.handle, X, Wp, A, B, r, 2.0, y_f16=ref16)
        M.mebp_linear_fwd_noalloc(X, Wp, A, B, r, 2.0, y_f16=out16)
        ctx.sync()
        ref_np, out_np = np_of(ref), np_of(out)
        assert np.isfinite(out_np).all()
        assert np.abs(out_np - ref_np).max() <= 2e-5 * np.abs(ref_np).max()
        assert np.abs(np_of(out16) - np_of(ref16)).max() <= 1e-3 * np.abs(np_of(ref16)).max()
    ctx.close()


@pytest.mark.parametrize("Mr,N,K,r,with_r", [(300, 1152, 896, 16, True), (130, 512, 256, 8, False),
                                              (257, 320, 192, 0, False), (64, 256, 128, 0, True)])
def test_noalloc_linear_matches_oracle(Mr, N, K, r, with_r):
    """Against the oracle in fp64, two calls in a row (fp32 output, then fp16 output); r = 0 runs
    without LoRA (no scratch but the error word), R = None without residual."""
    s = 2.0
    Wp, X, A, B, R, (Wd, Xo, An, Bn, Ro) = _case(Mr, N, K, r, 10 + r + Mr, oracle=True)
    ref = _oracle_linear(Wd, Xo, An, Bn, Ro if with_r else None, s)
    y = torch.full((Mr, N), float("nan"), device="cuda")
    y16 = torch.full((Mr, N), float("nan"), device="cuda", dtype=torch.float16)
    M.mebp_linear_fwd_noalloc(X, Wp, A, B, r, s, R=R if with_r else None, y_f32=y)
    M.mebp_linear_fwd_noalloc(X, Wp, A, B, r, s, y_f16=y16)
    torch.cuda.synchronize()
    got = np_of(y).astype(np.float64)
    assert np.isfinite(got).all()
    base = ref - (Ro if with_r else 0.0)
    # fp16 operands (the LoRA factors and the rank-r product are rounded to fp16), fp32 accumulate
    assert rel_fro(got - (Ro if with_r else 0.0), base) < 2e-3
    assert np.abs(got - ref).max() <= 1e-2 * np.abs(base).max()
    ref16 = _oracle_linear(Wd, Xo, An, Bn, None, s)
    assert np.abs(np_of(y16) - ref16).max() <= 1e-2 * np.abs(ref16).max()


def test_noalloc_rejects_requests_larger_than_its_scratch():
    Wp, X, A, B, R = _case(64, 256, 256, 16, 3)
    y = torch.empty((64, 256), device="cuda")
    too_many_rows = M.NOALLOC_SCRATCH_BYTES // (2 * 16) + 1
    rc = M.lib().mebp_linear_fwd_noalloc(X.data_ptr(), too_many_rows, ctypes.byref(Wp), A.data_ptr(), B.data_ptr(),
                                         16, 2.0, None, y.data_ptr(), None,
                                         ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == M.ERR_SCRATCH
