"""mebp_linear_fwd_noalloc: the fused LoRA linear for callers that may not allocate device
memory (it needs no context and keeps its scratch in a fixed static device array).

Checked through the C ABI against the regular mebp_linear_fwd on two calls in a row (the
second call reuses the scratch the first one left behind, with a different shape), within
the accumulation tolerance the other GEMM tests use.  This file is collected last so that a
stop-at-first-failure run has already run every other test."""
import ctypes

import numpy as np
import pytest

from oracle import quant
from workload import synth

from .helpers import np_of, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context  # noqa: E402


def _case(Mr, N, K, r, seed):
    rng = np.random.default_rng(seed)
    qo, so = quant.compress((rng.standard_normal((N, K)) * 0.02).astype(np.float32))
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    X = torch.from_numpy(rng.standard_normal((Mr, K)).astype(np.float16)).cuda()
    A = to_gpu((rng.standard_normal((r, K)) * 0.05).astype(np.float32)) if r else None
    B = to_gpu((rng.standard_normal((N, r)) * 0.05).astype(np.float32)) if r else None
    R = to_gpu(rng.standard_normal((Mr, N)).astype(np.float32))
    return Wp, X, A, B, R


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


def test_noalloc_rejects_requests_larger_than_its_scratch():
    Wp, X, A, B, R = _case(64, 256, 256, 16, 3)
    y = torch.empty((64, 256), device="cuda")
    too_many_rows = M.NOALLOC_SCRATCH_BYTES // (2 * 16) + 1
    rc = M.lib().mebp_linear_fwd_noalloc(X.data_ptr(), too_many_rows, ctypes.byref(Wp), A.data_ptr(), B.data_ptr(),
                                         16, 2.0, None, y.data_ptr(), None,
                                         ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == M.ERR_SCRATCH
