"""ctypes binding of ``libmebp.so`` (include/mebp.h).

Argument marshalling only: every function here has the name of the C entry point it
calls, takes torch tensors (device memory) or plain numbers, passes raw pointers and the
current CUDA stream, and raises ``MebpError`` on a non-zero status.  All compute runs in
the library's CUDA kernels; there is no CPU fallback — if the library is missing the
import of this module fails loudly.
"""
from __future__ import annotations

import ctypes
import os
import re
from ctypes import POINTER, c_char_p, c_float, c_int, c_int32, c_int64, c_uint32, c_void_p

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmebp.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "mebp.h")

OK, ERR_INVALID_ARG, ERR_CUDA, ERR_OOM, ERR_TIMEOUT, ERR_UNSUPPORTED, ERR_DEVICE, ERR_SCRATCH, ERR_NONFINITE = range(9)
NOALLOC_SCRATCH_BYTES = 8 << 20
T_Q, T_K, T_V, T_O, T_GATE, T_UP, T_DOWN = range(7)
WS_NAMES = ("checkpoints", "forward_sets", "backward", "attention_split", "lm_head", "lora_shadows", "other",
            "host_checkpoints")
TARGET_NAMES = ("q", "k", "v", "o", "gate", "up", "down")
ACT = {"silu": 0, "gelu_tanh": 1}


class MebpError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"mebp error {code}: {msg}")
        self.code = code


class ModelCfg(ctypes.Structure):
    _fields_ = [("hidden", c_int32), ("n_heads", c_int32), ("n_kv_heads", c_int32), ("head_dim", c_int32),
                ("intermediate", c_int32), ("vocab", c_int32), ("n_layers", c_int32), ("act", c_int32),
                ("rope_theta", c_float), ("rms_eps", c_float), ("lora_rank", c_int32), ("lora_scale", c_float),
                ("lora_targets", c_uint32), ("max_tokens", c_int32), ("max_seq", c_int32),
                ("spill_ckpts", c_int32), ("vocab_chunk", c_int32), ("gemma_norms", c_int32),
                ("sliding_window", c_int32), ("global_every", c_int32), ("rope_theta_local", c_float),
                ("min_memory", c_int32)]


class Packed(ctypes.Structure):
    _fields_ = [("qpack", c_void_p), ("scales", c_void_p), ("rows", c_int64), ("cols", c_int64)]


class BlockWeights(ctypes.Structure):
    _fields_ = [("qkv", Packed), ("o", Packed), ("gate_up", Packed), ("down", Packed),
                ("norm1", c_void_p), ("norm2", c_void_p), ("q_norm", c_void_p), ("k_norm", c_void_p),
                ("post_attn_norm", c_void_p), ("post_ffn_norm", c_void_p)]


class Lora(ctypes.Structure):
    _fields_ = [("A", c_void_p * 7), ("B", c_void_p * 7)]


class LoraGrads(ctypes.Structure):
    _fields_ = [("dA", c_void_p * 7), ("dB", c_void_p * 7)]


class Profile(ctypes.Structure):
    _fields_ = [("gemm_launches", c_int64), ("gemm_ms", ctypes.c_double), ("gemm_flops", ctypes.c_double),
                ("fwd_ms", ctypes.c_double), ("fwd_flops", ctypes.c_double),
                ("dx_ms", ctypes.c_double), ("dx_flops", ctypes.c_double), ("gemm_busy_ms", ctypes.c_double),
                ("gemm_bytes", ctypes.c_double)]


class KernelStat(ctypes.Structure):
    _fields_ = [("name", c_char_p), ("launches", c_int64), ("ms", ctypes.c_double), ("bytes", ctypes.c_double),
                ("flops", ctypes.c_double)]


class AdamWCfg(ctypes.Structure):
    _fields_ = [("lr", c_float), ("beta1", c_float), ("beta2", c_float), ("eps", c_float),
                ("weight_decay", c_float), ("grad_scale", c_float)]


class ModelWeights(ctypes.Structure):
    _fields_ = [("embed", Packed), ("final_norm", c_void_p), ("blocks", POINTER(BlockWeights))]


_SIGS = {
    "mebp_ctx_create": (c_int, [POINTER(ModelCfg), c_int, POINTER(c_void_p)]),
    "mebp_ctx_destroy": (None, [c_void_p]),
    "mebp_last_error": (c_char_p, [c_void_p]),
    "mebp_sync": (c_int, [c_void_p, c_void_p]),
    "mebp_workspace_bytes": (c_int64, [c_void_p]),
    "mebp_workspace_breakdown": (c_int, [c_void_p, POINTER(c_int64), POINTER(c_int)]),
    "mebp_compress_weights": (c_int, [c_void_p, c_void_p, c_int64, c_int64, c_int, c_void_p, c_void_p, c_void_p]),
    "mebp_decode_weights": (c_int, [c_void_p, POINTER(Packed), c_void_p, c_void_p]),
    "mebp_embed": (c_int, [c_void_p, POINTER(Packed), c_void_p, c_int64, c_void_p, c_void_p]),
    "mebp_linear_fwd": (c_int, [c_void_p, c_void_p, c_int64, POINTER(Packed), c_void_p, c_void_p, c_int, c_float,
                                c_void_p, c_void_p, c_void_p, c_void_p]),
    "mebp_linear_dx": (c_int, [c_void_p, c_void_p, c_int64, POINTER(Packed), c_void_p, c_void_p, c_int, c_float,
                               c_void_p, c_void_p, c_void_p]),
    "mebp_block_recompute_fwd": (c_int, [c_void_p, c_int, POINTER(BlockWeights), POINTER(Lora), c_void_p, c_void_p,
                                         c_int, c_int, c_int, c_void_p]),
    "mebp_block_bwd": (c_int, [c_void_p, c_int, POINTER(BlockWeights), POINTER(Lora), c_void_p, c_void_p, c_void_p,
                               POINTER(LoraGrads), c_int, c_int, c_int, c_void_p]),
    "mebp_lmhead_ce_fwd_bwd": (c_int, [c_void_p, POINTER(Packed), c_void_p, c_void_p, c_void_p, c_int64, c_void_p,
                                       c_void_p, c_void_p, c_void_p]),
    "mebp_linear_fwd_noalloc": (c_int, [c_void_p, c_int64, POINTER(Packed), c_void_p, c_void_p, c_int, c_float,
                                        c_void_p, c_void_p, c_void_p, c_void_p]),
    "mebp_kernel_launches": (c_int64, []),
    "mebp_enable_graphs": (c_int, [c_void_p, c_int]),
    "mebp_profile_begin": (c_int, [c_void_p]),
    "mebp_profile_end": (c_int, [c_void_p, POINTER(Profile)]),
    "mebp_profile_kernels": (c_int, [c_void_p, POINTER(KernelStat), c_int, POINTER(c_int)]),
    "mebp_lora_step": (c_int, [c_void_p, POINTER(ModelWeights), POINTER(Lora), c_void_p, c_int, c_int, c_void_p,
                               POINTER(LoraGrads), c_int, c_void_p]),
    "mebp_adamw_step": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_int64, POINTER(AdamWCfg), c_int64,
                                c_void_p]),
}


def header_functions(path: str = HEADER):
    """Names of the functions include/mebp.h declares."""
    with open(path) as f:
        txt = f.read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\*\s]+?\b(mebp_\w+)\s*\(", txt, flags=re.M)))


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = load_library()


def lib() -> ctypes.CDLL:
    return _lib


# ----------------------------------------------------------------------------- helpers
def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream=None):
    if stream is not None:
        return c_void_p(stream if isinstance(stream, int) else stream.cuda_stream)
    import torch
    return c_void_p(torch.cuda.current_stream().cuda_stream)


def _check(ctx, rc: int):
    if rc != OK:
        msg = _lib.mebp_last_error(ctx)
        raise MebpError(rc, msg.decode() if msg else "")


def packed(qpack, scales) -> Packed:
    """Descriptor of a compressed weight; it keeps the two tensors alive while it exists."""
    rows = qpack.shape[0]
    cols = qpack.shape[1] * 2
    p = Packed(_ptr(qpack), _ptr(scales), rows, cols)
    p._keep = (qpack, scales)
    return p


def lora_struct(tensors: dict) -> Lora:
    """tensors: {target name: (A, B)} of fp32 device tensors."""
    L = Lora()
    for i, n in enumerate(TARGET_NAMES):
        if n in tensors:
            L.A[i] = _ptr(tensors[n][0])
            L.B[i] = _ptr(tensors[n][1])
    return L


def grads_struct(tensors: dict) -> LoraGrads:
    G = LoraGrads()
    for i, n in enumerate(TARGET_NAMES):
        if n in tensors:
            G.dA[i] = _ptr(tensors[n][0])
            G.dB[i] = _ptr(tensors[n][1])
    return G


def model_cfg(dims, max_tokens=None, max_seq=None, spill=None, vocab_chunk=0, min_memory=False) -> ModelCfg:
    """ModelCfg from a ``workload.ModelDims``-like object."""
    mask = sum(1 << TARGET_NAMES.index(t) for t in dims.targets)
    return ModelCfg(dims.hidden, dims.n_heads, dims.n_kv_heads, dims.head_dim, dims.intermediate, dims.vocab,
                    dims.n_layers, ACT[dims.act], dims.rope_theta, dims.eps, dims.rank, dims.alpha / dims.rank,
                    mask, max_tokens or dims.batch * dims.seq, max_seq or dims.seq,
                    int(dims.spill if spill is None else spill), vocab_chunk,
                    int(getattr(dims, "gemma_norms", False)), int(getattr(dims, "sliding_window", 0)),
                    int(getattr(dims, "global_every", 1)), float(getattr(dims, "rope_theta_local", 1e4)),
                    int(min_memory))


# ----------------------------------------------------------------------------- C entry points
def mebp_ctx_create(cfg: ModelCfg, device: int = 0) -> c_void_p:
    out = c_void_p()
    rc = _lib.mebp_ctx_create(ctypes.byref(cfg), device, ctypes.byref(out))
    if rc != OK:
        raise MebpError(rc, "context creation failed")
    return out


def mebp_ctx_destroy(ctx):
    _lib.mebp_ctx_destroy(ctx)


def mebp_last_error(ctx) -> str:
    return _lib.mebp_last_error(ctx).decode()


def mebp_sync(ctx, stream=None):
    _check(ctx, _lib.mebp_sync(ctx, _stream(stream)))


def mebp_workspace_bytes(ctx) -> int:
    return _lib.mebp_workspace_bytes(ctx)


def mebp_workspace_breakdown(ctx) -> tuple:
    """({purpose: bytes} in the order of WS_NAMES, number of intermediate sets)."""
    arr = (c_int64 * len(WS_NAMES))()
    n = c_int()
    _check(ctx, _lib.mebp_workspace_breakdown(ctx, arr, ctypes.byref(n)))
    return dict(zip(WS_NAMES, list(arr))), n.value


def mebp_compress_weights(ctx, W, qpack, scales, group: int = 64, stream=None):
    rows, cols = W.shape
    _check(ctx, _lib.mebp_compress_weights(ctx, _ptr(W), rows, cols, group, _ptr(qpack), _ptr(scales),
                                           _stream(stream)))


def mebp_decode_weights(ctx, w: Packed, out, stream=None):
    _check(ctx, _lib.mebp_decode_weights(ctx, ctypes.byref(w), _ptr(out), _stream(stream)))


def mebp_embed(ctx, E: Packed, ids, x0, stream=None):
    _check(ctx, _lib.mebp_embed(ctx, ctypes.byref(E), _ptr(ids), ids.numel(), _ptr(x0), _stream(stream)))


def mebp_linear_fwd(ctx, X, W: Packed, A=None, B=None, r=0, s=1.0, R=None, y_f32=None, y_f16=None, stream=None):
    _check(ctx, _lib.mebp_linear_fwd(ctx, _ptr(X), X.shape[0], ctypes.byref(W), _ptr(A), _ptr(B), r, s, _ptr(R),
                                     _ptr(y_f32), _ptr(y_f16), _stream(stream)))


def mebp_linear_dx(ctx, dY, W: Packed, A=None, B=None, r=0, s=1.0, R=None, dx=None, stream=None):
    _check(ctx, _lib.mebp_linear_dx(ctx, _ptr(dY), dY.shape[0], ctypes.byref(W), _ptr(A), _ptr(B), r, s, _ptr(R),
                                    _ptr(dx), _stream(stream)))


def mebp_block_recompute_fwd(ctx, layer: int, w: BlockWeights, lora: Lora, x, y, batch: int, seq: int,
                             save_for_bwd: bool = False, stream=None):
    _check(ctx, _lib.mebp_block_recompute_fwd(ctx, layer, ctypes.byref(w), ctypes.byref(lora), _ptr(x), _ptr(y),
                                              batch, seq, int(save_for_bwd), _stream(stream)))


def mebp_block_bwd(ctx, layer: int, w: BlockWeights, lora: Lora, x, dy, dx, grads: LoraGrads, batch: int, seq: int,
                   accumulate: bool = False, stream=None):
    _check(ctx, _lib.mebp_block_bwd(ctx, layer, ctypes.byref(w), ctypes.byref(lora), _ptr(x), _ptr(dy), _ptr(dx),
                                    ctypes.byref(grads), batch, seq, int(accumulate), _stream(stream)))


def mebp_lmhead_ce_fwd_bwd(ctx, E: Packed, final_norm, h, targets, loss, dh, token_loss=None, stream=None):
    _check(ctx, _lib.mebp_lmhead_ce_fwd_bwd(ctx, ctypes.byref(E), _ptr(final_norm), _ptr(h), _ptr(targets),
                                            targets.numel(), _ptr(loss), _ptr(dh), _ptr(token_loss),
                                            _stream(stream)))


def mebp_lora_step(ctx, model: ModelWeights, lora_array, ids, loss, grads_array, accumulate: bool = False,
                   stream=None):
    """lora_array / grads_array: ctypes arrays (Lora * L, LoraGrads * L)."""
    B, S = ids.shape
    _check(ctx, _lib.mebp_lora_step(ctx, ctypes.byref(model), lora_array, _ptr(ids), B, S, _ptr(loss), grads_array,
                                    int(accumulate), _stream(stream)))


def adamw_cfg(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01, grad_scale=1.0) -> AdamWCfg:
    return AdamWCfg(lr, beta1, beta2, eps, weight_decay, grad_scale)


def mebp_adamw_step(ctx, params, grads, m, v, cfg: AdamWCfg, step: int, stream=None):
    """In-place AdamW update of flat fp32 buffers (params, m, v written; grads read)."""
    _check(ctx, _lib.mebp_adamw_step(ctx, _ptr(params), _ptr(grads), _ptr(m), _ptr(v), params.numel(),
                                     ctypes.byref(cfg), int(step), _stream(stream)))


def mebp_kernel_launches() -> int:
    return _lib.mebp_kernel_launches()


def mebp_profile_begin(ctx):
    _check(ctx, _lib.mebp_profile_begin(ctx))


def mebp_profile_end(ctx) -> Profile:
    p = Profile()
    _check(ctx, _lib.mebp_profile_end(ctx, ctypes.byref(p)))
    return p


def mebp_profile_kernels(ctx) -> dict:
    """{kind: {"launches", "ms", "bytes", "flops"}} of the last profiled interval (kinds with launches)."""
    arr = (KernelStat * 64)()
    n = c_int()
    _check(ctx, _lib.mebp_profile_kernels(ctx, arr, 64, ctypes.byref(n)))
    return {arr[i].name.decode(): {"launches": arr[i].launches, "ms": arr[i].ms, "bytes": arr[i].bytes,
                                   "flops": arr[i].flops} for i in range(min(n.value, 64)) if arr[i].launches}


def mebp_enable_graphs(ctx, on: bool = True):
    _check(ctx, _lib.mebp_enable_graphs(ctx, int(on)))


def mebp_linear_fwd_noalloc(X, W: Packed, A=None, B=None, r=0, s=1.0, R=None, y_f32=None, y_f16=None, stream=None):
    """mebp_linear_fwd without a context or any device allocation (fixed static scratch)."""
    rc = _lib.mebp_linear_fwd_noalloc(_ptr(X), X.shape[0], ctypes.byref(W), _ptr(A), _ptr(B), r, s, _ptr(R),
                                      _ptr(y_f32), _ptr(y_f16), _stream(stream))
    if rc != OK:
        raise MebpError(rc, "mebp_linear_fwd_noalloc failed")
