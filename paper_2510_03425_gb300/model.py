"""Device-side model state for the C ABI: compressed base weights, LoRA masters and
gradient buffers held as torch tensors, plus the ctypes descriptors that point at them.

torch only owns the memory here; compression runs in ``mebp_compress_weights``.
"""
from __future__ import annotations

import ctypes
from typing import Dict, List, Sequence, Tuple

import torch

from . import mebp as M

LINEARS = ("q", "k", "v", "o", "gate", "up", "down")


class Context:
    """Owns one ``mebp_ctx``."""

    def __init__(self, dims, device: int = 0, max_tokens=None, max_seq=None, spill=None, vocab_chunk=0,
                 min_memory=False):
        self.dims = dims
        self.cfg = M.model_cfg(dims, max_tokens=max_tokens, max_seq=max_seq, spill=spill, vocab_chunk=vocab_chunk,
                               min_memory=min_memory)
        self.handle = M.mebp_ctx_create(self.cfg, device)

    def close(self):
        if self.handle:
            M.mebp_ctx_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def sync(self, stream=None):
        M.mebp_sync(self.handle, stream)


def compress(ctx: Context, W: torch.Tensor) -> Tuple[torch.Tensor, torch.Tensor]:
    """4-bit group-64 compression of a dense fp32 device matrix (kernel: mebp_compress_weights)."""
    W = W.contiguous().float()
    rows, cols = W.shape
    q = torch.empty((rows, cols // 2), dtype=torch.uint8, device=W.device)
    s = torch.empty((cols // 64, rows), dtype=torch.float16, device=W.device)
    M.mebp_compress_weights(ctx.handle, W, q, s)
    return q, s


class PackedLinear:
    def __init__(self, qpack: torch.Tensor, scales: torch.Tensor):
        self.qpack, self.scales = qpack, scales

    def struct(self) -> M.Packed:
        return M.packed(self.qpack, self.scales)


class DeviceBlock:
    def __init__(self, ctx: Context, W: Dict[str, torch.Tensor]):
        """W: dense fp32 device tensors q, k, v, o, gate, up, down ([N, K]) and norm1, norm2; for
        the Gemma3 block also q_norm, k_norm ([head_dim]) and post_attn_norm, post_ffn_norm."""
        self.qkv = PackedLinear(*compress(ctx, torch.cat([W["q"], W["k"], W["v"]], 0)))
        self.o = PackedLinear(*compress(ctx, W["o"]))
        self.gate_up = PackedLinear(*compress(ctx, torch.cat([W["gate"], W["up"]], 0)))
        self.down = PackedLinear(*compress(ctx, W["down"]))
        self.norms = {n: W[n].contiguous().float() for n in
                      ("norm1", "norm2", "q_norm", "k_norm", "post_attn_norm", "post_ffn_norm") if n in W}
        self.norm1 = self.norms["norm1"]
        self.norm2 = self.norms["norm2"]

    def struct(self) -> M.BlockWeights:
        opt = [self.norms[n].data_ptr() if n in self.norms else None
               for n in ("q_norm", "k_norm", "post_attn_norm", "post_ffn_norm")]
        return M.BlockWeights(self.qkv.struct(), self.o.struct(), self.gate_up.struct(), self.down.struct(),
                              self.norm1.data_ptr(), self.norm2.data_ptr(), *opt)


class DeviceModel:
    def __init__(self, blocks: Sequence[DeviceBlock], embed: PackedLinear | None, final_norm: torch.Tensor | None):
        self.blocks = list(blocks)
        self.embed = embed
        self.final_norm = final_norm
        self._arr = (M.BlockWeights * len(self.blocks))(*[b.struct() for b in self.blocks])

    def struct(self) -> M.ModelWeights:
        return M.ModelWeights(self.embed.struct(), self.final_norm.data_ptr(),
                              ctypes.cast(self._arr, ctypes.POINTER(M.BlockWeights)))


def to_device(x, device="cuda") -> torch.Tensor:
    if isinstance(x, torch.Tensor):
        return x.to(device=device, dtype=torch.float32).contiguous()
    return torch.from_numpy(x).to(device=device, dtype=torch.float32).contiguous()


class LoraSet:
    """LoRA masters and gradients of every layer: lora[l][name] = (A [r, K], B [N, r]).

    All masters live in one flat fp32 buffer and all gradients in another (each tensor a view,
    16-byte aligned), so the optimizer updates every LoRA weight in one pass."""

    def __init__(self, layers: List[Dict[str, Tuple]], device="cuda"):
        import numpy as np
        sizes = []
        for L in layers:
            for n, (A, B) in L.items():
                sizes += [int(np.prod(A.shape)), int(np.prod(B.shape))]
        offs, n = [], 0
        for sz in sizes:
            offs.append(n)
            n += (sz + 3) // 4 * 4
        self.n = n
        self.params = torch.zeros(n, dtype=torch.float32, device=device)
        self.grad_flat = torch.zeros(n, dtype=torch.float32, device=device)
        self.lora, self.grads, k = [], [], 0
        for L in layers:
            lw, lg = {}, {}
            for name, (A, B) in L.items():
                views = []
                for src in (A, B):
                    sz, o = int(np.prod(src.shape)), offs[k]
                    p = self.params[o:o + sz].view(*src.shape)
                    p.copy_(to_device(src, device))
                    views.append((p, self.grad_flat[o:o + sz].view(*src.shape)))
                    k += 1
                lw[name] = (views[0][0], views[1][0])
                lg[name] = (views[0][1], views[1][1])
            self.lora.append(lw)
            self.grads.append(lg)
        self._la = (M.Lora * len(self.lora))(*[M.lora_struct(L) for L in self.lora])
        self._ga = (M.LoraGrads * len(self.grads))(*[M.grads_struct(G) for G in self.grads])
        self.m = self.v = None
        self.t = 0

    def adamw(self, ctx, cfg=None, stream=None):
        """One AdamW update of every LoRA weight from the current gradients (mebp_adamw_step)."""
        if self.m is None:
            self.m = torch.zeros_like(self.params)
            self.v = torch.zeros_like(self.params)
        self.t += 1
        M.mebp_adamw_step(ctx.handle, self.params, self.grad_flat, self.m, self.v, cfg or M.adamw_cfg(), self.t,
                          stream)

    def lora_array(self):
        return self._la

    def grads_array(self):
        return self._ga

    def layer(self, i) -> M.Lora:
        return self._la[i]

    def layer_grads(self, i) -> M.LoraGrads:
        return self._ga[i]
