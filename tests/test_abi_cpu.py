"""Host-side checks of the C ABI (no GPU needed): the library loads, exports every
function include/mebp.h declares, and rejects bad configurations before touching CUDA."""
import ctypes
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2510_03425_gb300", "libmebp.so")


@pytest.fixture(scope="module")
def binding():
    if not os.path.exists(LIB):
        from paper_2510_03425_gb300 import build
        build.build()
    from paper_2510_03425_gb300 import mebp
    return mebp


def test_library_exports_every_declared_function(binding):
    names = binding.header_functions()
    assert len(names) >= 14
    lib = ctypes.CDLL(LIB)
    for n in names:
        assert hasattr(lib, n), n
    # the five calls of the boundary
    for n in ("mebp_compress_weights", "mebp_block_recompute_fwd", "mebp_block_bwd", "mebp_lmhead_ce_fwd_bwd",
              "mebp_lora_step"):
        assert n in names


def test_binding_wraps_every_declared_function(binding):
    for n in binding.header_functions():
        assert callable(getattr(binding, n)), n


def _cfg(binding, **kw):
    from workload import synth
    c = binding.model_cfg(synth.preset(1))
    for k, v in kw.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("field,value,code", [
    ("hidden", 900, 1),            # not a multiple of 64
    ("n_kv_heads", 3, 1),          # H % KV != 0
    ("head_dim", 96, 5),           # unsupported head dim
    ("lora_rank", 40, 1),          # rank > 32
    ("lora_rank", 12, 5),          # rank not a multiple of 8
    ("vocab_chunk", 100, 1),       # chunk not a multiple of 256
    ("max_tokens", 0, 1),
    ("act", 7, 1),
    ("sliding_window", -1, 1),     # negative window
])
def test_ctx_create_rejects_bad_configs_without_a_gpu(binding, field, value, code):
    cfg = _cfg(binding, **{field: value})
    out = ctypes.c_void_p()
    rc = binding.lib().mebp_ctx_create(ctypes.byref(cfg), 0, ctypes.byref(out))
    assert rc == code
    assert not out.value


def test_ctx_create_rejects_a_window_without_global_layers_or_local_base(binding):
    for kw in (dict(sliding_window=128, global_every=0), dict(sliding_window=128, rope_theta_local=0.0)):
        cfg = _cfg(binding, **kw)
        out = ctypes.c_void_p()
        assert binding.lib().mebp_ctx_create(ctypes.byref(cfg), 0, ctypes.byref(out)) == 1
        assert not out.value


def test_model_cfg_carries_the_gemma3_options(binding):
    from workload import synth
    d = synth.preset(2).with_(gemma_norms=True, sliding_window=512, global_every=6, rope_theta_local=1e4)
    c = binding.model_cfg(d)
    assert (c.gemma_norms, c.sliding_window, c.global_every, c.rope_theta_local) == (1, 512, 6, 1e4)
    assert binding.model_cfg(synth.preset(2)).gemma_norms == 0


def test_null_context_is_rejected(binding):
    lib = binding.lib()
    assert lib.mebp_sync(None, None) == binding.ERR_INVALID_ARG
    assert lib.mebp_lora_step(None, None, None, None, 1, 1, None, None, 0, None) == binding.ERR_INVALID_ARG
    assert lib.mebp_last_error(None) == b"NULL context"


@pytest.mark.parametrize("which", ["X", "qpack", "scales", "y_f32", "y_f16", "R"])
def test_noalloc_rejects_misaligned_pointers_before_touching_cuda(binding, which):
    """The fused GEMM reads X and the weights by TMA and stores y / reads R as 16-byte vectors:
    a pointer off a 16-byte boundary is refused on the host, before any CUDA call (the
    addresses below are never dereferenced)."""
    ptrs = dict(X=0x10000, qpack=0x20000, scales=0x30000, y_f32=0x40000, y_f16=None, R=0x50000)
    if which == "y_f16":
        ptrs["y_f32"] = None
        ptrs["y_f16"] = 0x40000
    ptrs[which] += 8
    W = binding.Packed(ptrs["qpack"], ptrs["scales"], 64, 128)
    rc = binding.lib().mebp_linear_fwd_noalloc(ptrs["X"], 16, ctypes.byref(W), None, None, 0, 1.0, ptrs["R"],
                                                ptrs["y_f32"], ptrs["y_f16"], None)
    assert rc == binding.ERR_INVALID_ARG
