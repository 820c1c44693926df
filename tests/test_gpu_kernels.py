"""Kernel-level parity of the CUDA path (through the C ABI) against the CPU oracle:
compression and decode bit-exact, embedding gather exact, and the fused dequant-GEMMs
(forward and transposed) against fp64 references built from the oracle's decode."""
import numpy as np
import pytest

from oracle import quant
from workload import synth

from .helpers import f16_round, np_of, rel_fro, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, compress  # noqa: E402


@pytest.fixture(scope="module")
def ctx():
    c = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=4096, max_seq=64)
    yield c
    c.close()


def _w(rows, cols, seed, std=0.02):
    W = (np.random.default_rng(seed).standard_normal((rows, cols)) * std).astype(np.float32)
    W[min(3, rows - 1), 64:128 if cols >= 128 else 64] *= 500.0  # a loud group
    if rows > 5:
        W[5, :64] = 0.0                                            # an all-zero group
    return W


@pytest.mark.parametrize("rows,cols", [(1, 64), (7, 192), (256, 896), (1152, 896), (333, 4864)])
def test_compress_bit_exact(ctx, rows, cols):
    W = _w(rows, cols, rows + cols)
    q, s = compress(ctx, to_gpu(W))
    ctx.sync()
    qo, so = quant.compress(W)
    np.testing.assert_array_equal(np_of(q), qo)
    np.testing.assert_array_equal(s.cpu().numpy().view(np.uint16), so.view(np.uint16))


def test_decode_bit_exact(ctx):
    W = _w(320, 1024, 5, std=0.3)
    qo, so = quant.compress(W)
    out = torch.empty((320, 1024), dtype=torch.int16, device="cuda")
    M.mebp_decode_weights(ctx.handle, M.packed(to_gpu(qo), to_gpu(so)), out)
    ctx.sync()
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint16), quant.dequant_f16_bits(qo, so))


def test_embedding_gather_exact(ctx):
    V, D = 1000, 256
    E = _w(V, D, 9, std=0.5)
    qo, so = quant.compress(E)
    ids = np.random.default_rng(1).integers(0, V, 777).astype(np.int32)
    x0 = torch.empty((777, D), dtype=torch.float32, device="cuda")
    M.mebp_embed(ctx.handle, M.packed(to_gpu(qo), to_gpu(so)), to_gpu(ids), x0)
    ctx.sync()
    np.testing.assert_array_equal(np_of(x0).astype(np.float64), quant.dequant_rows(qo, so, ids))


def test_embedding_bad_id_flags_device_error(ctx):
    V, D = 128, 64
    qo, so = quant.compress(_w(V, D, 3))
    ids = to_gpu(np.array([1, 2, V + 5], np.int32))
    x0 = torch.full((3, D), 7.0, device="cuda")
    M.mebp_embed(ctx.handle, M.packed(to_gpu(qo), to_gpu(so)), ids, x0)
    with pytest.raises(M.MebpError) as ei:
        ctx.sync()
    assert ei.value.code == M.ERR_DEVICE
    assert (x0[2] == 0).all()
    ctx.sync()  # the error word was cleared


# (M, N, K): ragged tiles, a single tile, split-K (small grids), two-accumulator tiles (M >= 2048, or
# a large N: 152 256-column tiles x 2 row tiles), and a transposed pass with a 608-tile split reduction
SHAPES = [(200, 320, 192), (128, 256, 64), (1, 64, 64), (300, 1152, 896), (513, 512, 1024), (512, 896, 4864),
          (2048, 256, 128), (2304 + 77, 576, 640), (300, 38912, 128)]


def _x(M_, K, seed, scale=1.0):
    x = (np.random.default_rng(seed).standard_normal((M_, K)) * scale).astype(np.float32)
    return f16_round(x)


@pytest.mark.parametrize("Mr,N,K", SHAPES)
def test_linear_fwd_matches_exact_operand_product(ctx, Mr, N, K):
    """No LoRA: Y must equal X_f16 . fp16(deq(W))^T up to fp32 accumulation."""
    W = _w(N, K, N + K)
    qo, so = quant.compress(W)
    X = _x(Mr, K, 1)
    ref = X @ quant.f16_bits_to_f64(quant.dequant_f16_bits(qo, so)).T
    Xg = to_gpu(X.astype(np.float32)).to(torch.float16)
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    y = torch.empty((Mr, N), dtype=torch.float32, device="cuda")
    yb = torch.empty((Mr, N), dtype=torch.float16, device="cuda")
    M.mebp_linear_fwd(ctx.handle, Xg, Wp, y_f32=y)
    M.mebp_linear_fwd(ctx.handle, Xg, Wp, y_f16=yb)
    ctx.sync()
    scale = np.abs(ref).max()
    assert np.abs(np_of(y) - ref).max() <= 2e-5 * scale + 1e-6
    assert np.abs(np_of(yb) - ref).max() <= 1e-3 * scale + 1e-6


@pytest.mark.parametrize("Mr,N,K", SHAPES)
def test_linear_dx_matches_exact_operand_product(ctx, Mr, N, K):
    """No LoRA: dX = dY_f16 . fp16(deq(W)) up to fp32 accumulation (W is [N, K])."""
    W = _w(N, K, N + 2 * K)
    qo, so = quant.compress(W)
    dY = _x(Mr, N, 2)
    ref = dY @ quant.f16_bits_to_f64(quant.dequant_f16_bits(qo, so))
    dx = torch.empty((Mr, K), dtype=torch.float32, device="cuda")
    M.mebp_linear_dx(ctx.handle, to_gpu(dY.astype(np.float32)).to(torch.float16), M.packed(to_gpu(qo), to_gpu(so)),
                     dx=dx)
    ctx.sync()
    assert np.abs(np_of(dx) - ref).max() <= 2e-5 * np.abs(ref).max() + 1e-6


@pytest.mark.parametrize("r,Mr,N,K", [(r, *shape) for r in (8, 16, 32)
                                      for shape in ((200, 320, 192), (300, 1152, 896), (2304 + 77, 576, 640))]
                         + [(16, 4096 + 77, 1152, 1536)]   # > 152 tiles: persistent CTAs run several
                         # above 1024 tokens the rank-r products run on the tcgen05 kernel
                         # (one rank block of 16 or 32 columns, K split over a cluster or not)
                         + [(r, 2500, 640, 1024) for r in (8, 24, 32)] + [(32, 16384 + 5, 256, 2560)])
def test_linear_with_lora_against_oracle(ctx, r, Mr, N, K):
    """Y = X deq(W)^T + s (X A^T) B^T (+R) and dX = dY deq(W) + s (dY B) A against fp64."""
    s = 2.0
    rng = np.random.default_rng(r)
    W = _w(N, K, 11)
    qo, so = quant.compress(W)
    Wd = quant.dequant(qo, so)
    A = (rng.standard_normal((r, K)) * 0.05).astype(np.float32)
    B = (rng.standard_normal((N, r)) * 0.05).astype(np.float32)
    X = _x(Mr, K, 3)
    R = rng.standard_normal((Mr, N)).astype(np.float32)
    ref = X @ Wd.T + s * (X @ A.T.astype(np.float64)) @ B.T.astype(np.float64) + R
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    y = torch.empty((Mr, N), dtype=torch.float32, device="cuda")
    Ag, Bg = to_gpu(A), to_gpu(B)
    M.mebp_linear_fwd(ctx.handle, to_gpu(X.astype(np.float32)).to(torch.float16), Wp, Ag, Bg, r, s, R=to_gpu(R), y_f32=y)
    dY = _x(Mr, N, 4)
    ref_dx = dY @ Wd + s * (dY @ B.astype(np.float64)) @ A.astype(np.float64)
    dx = torch.empty((Mr, K), dtype=torch.float32, device="cuda")
    M.mebp_linear_dx(ctx.handle, to_gpu(dY.astype(np.float32)).to(torch.float16), Wp, Ag, Bg, r, s, dx=dx)
    ctx.sync()
    assert rel_fro(np_of(y) - R, ref - R) < 2e-3
    assert rel_fro(np_of(dx), ref_dx) < 2e-3
    # the LoRA term itself is carried (not just the base product)
    base = X @ Wd.T
    lora_term = ref - R - base
    got_term = np_of(y).astype(np.float64) - R - base
    assert rel_fro(got_term, lora_term) < 1e-2


# K split through memory.  A context sized for the Qwen2.5-0.5B-shaped step (512 tokens) holds
# fp32 partial-tile scratch (its gate|up dX and LM-head dH passes want it); a GEMM with few output
# tiles over a long K then runs as tiles x splits CTAs not bound to clusters, and a second launch
# sums the partials in split order.  (trans, M, N, K) in GEMM terms: an M x N output over K; the
# comments give the plan (accumulators per CTA, splits).
KSPLIT = [(True, 512, 896, 9728),     # the gate|up dX shape: one accumulator, 9 splits
          (True, 300, 640, 8256),     # ragged rows, 129 K steps
          (False, 200, 576, 16384),   # forward: one accumulator, 25 splits
          (True, 512, 896, 32768)]    # two accumulators, 19 splits (152 CTAs)


@pytest.fixture(scope="module")
def kctx():
    c = Context(synth.preset(1), max_tokens=512, max_seq=512)
    yield c
    c.close()


@pytest.mark.parametrize("trans,Mr,N,K", KSPLIT)
def test_ksplit_through_memory_matches_exact_operand_product(kctx, trans, Mr, N, K):
    """No LoRA: the split GEMM equals the operand product up to fp32 accumulation (fp32 and, in
    the forward, fp16 outputs and a residual), is deterministic, and ran as two launches."""
    rng = np.random.default_rng(K + Mr)
    W = _w(K, N, 31) if trans else _w(N, K, 31)        # dX = dY W with W [K_gemm, N_gemm]
    qo, so = quant.compress(W)
    Wd = quant.f16_bits_to_f64(quant.dequant_f16_bits(qo, so))
    X = _x(Mr, K, 7)
    ref = X @ Wd if trans else X @ Wd.T
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    Xg = to_gpu(X.astype(np.float32)).to(torch.float16)
    y = torch.empty((Mr, N), dtype=torch.float32, device="cuda")
    y2 = torch.empty_like(y)
    run = (lambda out: M.mebp_linear_dx(kctx.handle, Xg, Wp, dx=out)) if trans else \
        (lambda out: M.mebp_linear_fwd(kctx.handle, Xg, Wp, y_f32=out))
    n0 = M.mebp_kernel_launches()
    run(y)
    assert M.mebp_kernel_launches() - n0 == 2          # the GEMM and the split sum
    run(y2)
    kctx.sync()
    scale = np.abs(ref).max()
    assert np.abs(np_of(y) - ref).max() <= 2e-5 * scale + 1e-6
    assert torch.equal(y, y2)
    if not trans:
        R = rng.standard_normal((Mr, N)).astype(np.float32)
        yr = torch.empty_like(y)
        yb = torch.empty((Mr, N), dtype=torch.float16, device="cuda")
        M.mebp_linear_fwd(kctx.handle, Xg, Wp, R=to_gpu(R), y_f32=yr)
        M.mebp_linear_fwd(kctx.handle, Xg, Wp, y_f16=yb)
        kctx.sync()
        assert np.abs(np_of(yr) - (ref + R)).max() <= 2e-5 * (scale + np.abs(R).max()) + 1e-6
        assert np.abs(np_of(yb) - ref).max() <= 1e-3 * scale + 1e-6


@pytest.mark.parametrize("trans", [False, True])
def test_ksplit_through_memory_with_lora_against_oracle(kctx, trans):
    """The LoRA block rides with the last split: Y = X deq(W)^T + s (X A^T) B^T + R and
    dX = dY deq(W) + s (dY B) A against fp64 at split shapes."""
    s, r = 2.0, 16
    rng = np.random.default_rng(5)
    Mr, Nl, Kl = (300, 9728, 896) if trans else (300, 576, 16384)   # the layer's W is [Nl, Kl]
    qo, so = quant.compress(_w(Nl, Kl, 12))
    Wd = quant.dequant(qo, so)
    A = (rng.standard_normal((r, Kl)) * 0.05).astype(np.float32)
    B = (rng.standard_normal((Nl, r)) * 0.05).astype(np.float32)
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    Ag, Bg = to_gpu(A), to_gpu(B)
    if trans:
        dY = _x(Mr, Nl, 8)
        ref = dY @ Wd + s * (dY @ B.astype(np.float64)) @ A.astype(np.float64)
        out = torch.empty((Mr, Kl), dtype=torch.float32, device="cuda")
        M.mebp_linear_dx(kctx.handle, to_gpu(dY.astype(np.float32)).to(torch.float16), Wp, Ag, Bg, r, s, dx=out)
        kctx.sync()
        assert rel_fro(np_of(out), ref) < 2e-3
    else:
        X = _x(Mr, Kl, 9)
        R = rng.standard_normal((Mr, Nl)).astype(np.float32)
        ref = X @ Wd.T + s * (X @ A.T.astype(np.float64)) @ B.T.astype(np.float64) + R
        out = torch.empty((Mr, Nl), dtype=torch.float32, device="cuda")
        M.mebp_linear_fwd(kctx.handle, to_gpu(X.astype(np.float32)).to(torch.float16), Wp, Ag, Bg, r, s,
                          R=to_gpu(R), y_f32=out)
        kctx.sync()
        assert rel_fro(np_of(out) - R, ref - R) < 2e-3
        base = X @ Wd.T
        assert rel_fro(np_of(out).astype(np.float64) - R - base, ref - R - base) < 1e-2


def test_lora_b_zero_is_bit_identical_to_base(ctx):
    Mr, N, K, r = 257, 512, 384, 16
    W = _w(N, K, 21)
    qo, so = quant.compress(W)
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    X = to_gpu(_x(Mr, K, 5).astype(np.float32)).to(torch.float16)
    A = to_gpu((np.random.default_rng(0).standard_normal((r, K)) * 0.1).astype(np.float32))
    B0 = torch.zeros((N, r), device="cuda")
    y0 = torch.empty((Mr, N), device="cuda")
    y1 = torch.empty((Mr, N), device="cuda")
    M.mebp_linear_fwd(ctx.handle, X, Wp, y_f32=y0)
    M.mebp_linear_fwd(ctx.handle, X, Wp, A, B0, r, 2.0, y_f32=y1)
    dY = to_gpu(_x(Mr, N, 6).astype(np.float32)).to(torch.float16)
    d0 = torch.empty((Mr, K), device="cuda")
    d1 = torch.empty((Mr, K), device="cuda")
    M.mebp_linear_dx(ctx.handle, dY, Wp, dx=d0)
    M.mebp_linear_dx(ctx.handle, dY, Wp, A, B0, r, 2.0, dx=d1)
    ctx.sync()
    assert torch.equal(y0, y1)
    assert torch.equal(d0, d1)


def test_linear_rejects_bad_shapes(ctx):
    q = torch.zeros((64, 48), dtype=torch.uint8, device="cuda")   # cols = 96: not a multiple of 64
    s = torch.zeros((1, 64), dtype=torch.float16, device="cuda")
    X = torch.zeros((4, 96), dtype=torch.float16, device="cuda")
    y = torch.empty((4, 64), device="cuda")
    with pytest.raises(M.MebpError) as ei:
        M.mebp_linear_fwd(ctx.handle, X, M.packed(q, s), y_f32=y)
    assert ei.value.code == M.ERR_INVALID_ARG


def test_linear_rejects_misaligned_outputs_and_residual(ctx):
    """y and R are stored / read as 16-byte vectors: views off a 16-byte boundary are refused on
    the host with MEBP_ERR_INVALID_ARG (nothing is launched)."""
    Mr, N, K = 4, 64, 64
    qo, so = quant.compress(_w(N, K, 1))
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    X = torch.zeros((Mr, K), dtype=torch.float16, device="cuda")
    buf = torch.zeros(Mr * N + 4, device="cuda")
    off = buf[2:2 + Mr * N].view(Mr, N)          # 8 bytes past a 16-byte boundary
    good = torch.zeros((Mr, N), device="cuda")
    buf16 = torch.zeros(Mr * N + 8, dtype=torch.float16, device="cuda")
    off16 = buf16[4:4 + Mr * N].view(Mr, N)
    for kw in (dict(y_f32=off), dict(y_f16=off16), dict(y_f32=good, R=off)):
        with pytest.raises(M.MebpError) as ei:
            M.mebp_linear_fwd(ctx.handle, X, Wp, **kw)
        assert ei.value.code == M.ERR_INVALID_ARG
    with pytest.raises(M.MebpError) as ei:
        M.mebp_linear_dx(ctx.handle, torch.zeros((Mr, N), dtype=torch.float16, device="cuda"), Wp, dx=off)
    assert ei.value.code == M.ERR_INVALID_ARG
    ctx.sync()


def test_fp16_overflow_is_reported_not_silent(ctx):
    """A GEMM output stored as fp16 that leaves the fp16 range (|y| > 65504) sets MEBP_ERR_NONFINITE,
    reported by mebp_sync; the fp32 output of the same product is fine, and the error word is
    cleared afterwards (inputs chosen on the host so that |y| ~ 1e5: only an inf is produced)."""
    Mr, N, K = 64, 128, 256
    W = np.full((N, K), 0.25, np.float32)
    qo, so = quant.compress(W)
    Wp = M.packed(to_gpu(qo), to_gpu(so))
    X = torch.full((Mr, K), 2000.0, device="cuda", dtype=torch.float16)   # y = 256 * 2000 * 0.25 = 128000
    y32 = torch.empty((Mr, N), device="cuda")
    M.mebp_linear_fwd(ctx.handle, X, Wp, y_f32=y32)
    ctx.sync()
    assert float(y32.max()) == pytest.approx(128000.0, rel=1e-3)
    y16 = torch.empty((Mr, N), device="cuda", dtype=torch.float16)
    M.mebp_linear_fwd(ctx.handle, X, Wp, y_f16=y16)
    with pytest.raises(M.MebpError) as ei:
        ctx.sync()
    assert ei.value.code == M.ERR_NONFINITE
    X.fill_(1.0)
    M.mebp_linear_fwd(ctx.handle, X, Wp, y_f16=y16)
    ctx.sync()                                     # the error word was cleared; in range now
    assert torch.isfinite(y16.float()).all()


def test_gated_mlp_overflow_is_reported():
    """The gated-MLP product m = act(g) u is stored as fp16: a block whose gate / up outputs are
    large enough that m leaves the fp16 range reports MEBP_ERR_NONFINITE at mebp_sync."""
    from paper_2510_03425_gb300.model import DeviceBlock, LoraSet
    dims = synth.tiny(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=256, n_layers=1, vocab=0,
                      batch=1, seq=64, rank=8, alpha=16.0, targets=())
    W = synth.block_weights(dims, 0)
    W["gate"] = np.full_like(W["gate"], 0.06)      # b = norm(h1) * 24 ~ 24, so g = u ~ 0.06 * 256 * 24 = 369
    W["up"] = np.full_like(W["up"], 0.06)          # and m = silu(g) u ~ 1.4e5 > 65504 (g, u themselves fit)
    W["norm2"] = np.full_like(W["norm2"], 24.0)
    c = Context(dims)
    blk = DeviceBlock(c, {k: to_gpu(v) for k, v in W.items()})
    x = to_gpu(np.ones((dims.tokens, dims.hidden), np.float32))
    y = torch.empty_like(x)
    M.mebp_block_recompute_fwd(c.handle, 0, blk.struct(), LoraSet([{}]).layer(0), x, y, 1, dims.seq, False)
    with pytest.raises(M.MebpError) as ei:
        c.sync()
    assert ei.value.code == M.ERR_NONFINITE
    c.close()
