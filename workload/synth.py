"""Model presets and seeded generators for synthetic MeBP workloads.

The paper (Section 4) trains Qwen2.5 and Gemma3 models on WikiText-2; neither
the data nor the checkpoints are available, so every input here is synthetic
with the shapes and value distributions of those workloads:

* base weights ~ N(0, 0.02^2) (compressed to 4-bit afterwards by whoever uses them),
* LoRA A, B ~ N(0, 0.01^2),
* RMSNorm gains = 1 (or 1 + N(0, 0.1^2) when ``norm_jitter`` is set),
* hidden-state inputs ~ N(0, 1), upstream gradients ~ N(0, 1),
* token ids uniform in [0, V).

Seeds: 0 base weights, 1 LoRA, 2 inputs / ids, 3 upstream gradient.  Each
draw uses numpy's PCG64 keyed by (seed, layer, tensor index) so any single
tensor can be regenerated on its own.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Tuple

import numpy as np

# LoRA target names in the order used everywhere (bit i of a target mask).
TARGETS = ("q", "k", "v", "o", "gate", "up", "down")


@dataclasses.dataclass(frozen=True)
class ModelDims:
    name: str
    hidden: int          # D
    n_heads: int         # H
    n_kv_heads: int      # KV
    head_dim: int        # hd
    intermediate: int    # I
    act: str             # "silu" | "gelu_tanh"
    n_layers: int        # L
    vocab: int           # V (0: single block, no LM head)
    batch: int           # B
    seq: int             # S
    rank: int            # r
    alpha: float         # LoRA alpha; scale s = alpha / r
    targets: Tuple[str, ...]
    rope_theta: float = 1e6
    eps: float = 1e-6
    spill: bool = False  # activation checkpoints in pinned host memory
    # Gemma3 block fidelity (off for the benchmark presets): QK-norm, sandwich norms and the
    # sqrt(D) embedding scale; sliding-window attention on local layers (window > 0), every
    # global_every-th layer global, local layers with their own RoPE base.
    gemma_norms: bool = False
    sliding_window: int = 0
    global_every: int = 6
    rope_theta_local: float = 1e4

    def layer_is_local(self, layer: int) -> bool:
        return self.sliding_window > 0 and (layer + 1) % self.global_every != 0

    @property
    def tokens(self) -> int:
        return self.batch * self.seq

    @property
    def lora_scale(self) -> float:
        return self.alpha / self.rank

    @property
    def target_mask(self) -> int:
        return sum(1 << TARGETS.index(t) for t in self.targets)

    def with_(self, **kw) -> "ModelDims":
        return dataclasses.replace(self, **kw)


_ALL7 = TARGETS
PRESETS: Dict[int, ModelDims] = {
    # Qwen2.5-0.5B-shaped single block, batch 1 x seq 128, objective sum(G * y).
    0: ModelDims("qwen2.5-0.5b-block", 896, 14, 2, 64, 4864, "silu", 1, 0, 1, 128,
                 8, 16.0, ("q", "k", "v", "o")),
    # Full Qwen2.5-0.5B-shaped model, batch 1 x seq 512.
    1: ModelDims("qwen2.5-0.5b", 896, 14, 2, 64, 4864, "silu", 24, 151936, 1, 512,
                 8, 16.0, ("q", "k", "v", "o")),
    # Gemma3-1B-shaped model (plain pre-norm block with GeGLU), batch 1 x seq 1024.
    2: ModelDims("gemma3-1b", 1152, 4, 1, 256, 6912, "gelu_tanh", 26, 262144, 1, 1024,
                 16, 32.0, ("q", "k", "v", "o", "up", "down")),
    # Qwen2.5-1.5B-shaped model, batch 4 x seq 1024, checkpoints spilled to host.
    3: ModelDims("qwen2.5-1.5b", 1536, 12, 2, 128, 8960, "silu", 28, 151936, 4, 1024,
                 16, 32.0, _ALL7, spill=True),
    # Gemma3-4B-shaped model, batch 8 x seq 2048.
    4: ModelDims("gemma3-4b", 2560, 8, 4, 256, 10240, "gelu_tanh", 34, 262144, 8, 2048,
                 32, 64.0, _ALL7),
}


def preset(i: int) -> ModelDims:
    return PRESETS[i]


def tiny(**kw) -> ModelDims:
    """A small model for oracle self-tests (finite differences etc.)."""
    base = dict(name="tiny", hidden=64, n_heads=2, n_kv_heads=1, head_dim=32,
                intermediate=128, act="silu", n_layers=2, vocab=97, batch=2, seq=8,
                rank=8, alpha=16.0, targets=_ALL7)
    base.update(kw)
    return ModelDims(**base)


def linear_shapes(d: ModelDims) -> Dict[str, Tuple[int, int]]:
    """(N_out, K_in) of every linear layer of one block."""
    D, H, KV, hd, I = d.hidden, d.n_heads, d.n_kv_heads, d.head_dim, d.intermediate
    return {"q": (H * hd, D), "k": (KV * hd, D), "v": (KV * hd, D), "o": (D, H * hd),
            "gate": (I, D), "up": (I, D), "down": (D, I)}


def _rng(seed: int, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *key])))


def _normal(seed: int, key, shape, std: float) -> np.ndarray:
    g = _rng(seed, *key)
    return (g.standard_normal(size=shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def block_weights(d: ModelDims, layer: int, seed: int = 0, norm_jitter: float = 0.0,
                  std: float = 0.02) -> Dict[str, np.ndarray]:
    """Dense fp32 base weights of block ``layer``: W[name] is [N_out, K_in] (PyTorch Linear layout)."""
    out = {}
    for i, (name, shp) in enumerate(linear_shapes(d).items()):
        out[name] = _normal(seed, (layer, i), shp, std)
    names = ("norm1", "norm2") + (("post_attn_norm", "post_ffn_norm") if d.gemma_norms else ())
    for j, name in enumerate(names):
        g = np.ones(d.hidden, np.float32)
        if norm_jitter:
            g += _normal(seed, (layer, 100 + j), (d.hidden,), norm_jitter)
        out[name] = g
    if d.gemma_norms:
        for j, name in enumerate(("q_norm", "k_norm")):
            g = np.ones(d.head_dim, np.float32)
            if norm_jitter:
                g += _normal(seed, (layer, 110 + j), (d.head_dim,), norm_jitter)
            out[name] = g
    return out


def embedding(d: ModelDims, seed: int = 0, std: float = 0.02, norm_jitter: float = 0.0, rows: int = 0):
    """Tied embedding / LM-head matrix E [V, D] and the final RMSNorm gain [D]; rows > 0 draws only
    the first `rows` rows (the same values as E[:rows])."""
    E = _normal(seed, (10_000, 0), (rows if rows > 0 else d.vocab, d.hidden), std)
    g = np.ones(d.hidden, np.float32)
    if norm_jitter:
        g += _normal(seed, (10_000, 1), (d.hidden,), norm_jitter)
    return E, g


def lora_weights(d: ModelDims, layer: int, seed: int = 1, std: float = 0.01,
                 zero_b: bool = False) -> Dict[str, Tuple[np.ndarray, np.ndarray]]:
    """LoRA (A [r, K_in], B [N_out, r]) for every targeted linear of block ``layer``."""
    out = {}
    shapes = linear_shapes(d)
    for i, name in enumerate(TARGETS):
        if name not in d.targets:
            continue
        N, K = shapes[name]
        A = _normal(seed, (layer, 2 * i), (d.rank, K), std)
        B = np.zeros((N, d.rank), np.float32) if zero_b else _normal(seed, (layer, 2 * i + 1), (N, d.rank), std)
        out[name] = (A, B)
    return out


def hidden_input(d: ModelDims, seed: int = 2) -> np.ndarray:
    """Block input hidden states x [B*S, D] ~ N(0, 1)."""
    return _normal(seed, (0,), (d.tokens, d.hidden), 1.0)


def token_ids(d: ModelDims, seed: int = 2) -> np.ndarray:
    """Token ids [B, S] uniform in [0, V)."""
    return _rng(seed, 1).integers(0, d.vocab, size=(d.batch, d.seq), dtype=np.int64).astype(np.int32)


def upstream_grad(d: ModelDims, seed: int = 3) -> np.ndarray:
    """Upstream gradient G = dE/dy [B*S, D] ~ N(0, 1) for the single-block objective E = sum(G * y)."""
    return _normal(seed, (0,), (d.tokens, d.hidden), 1.0)


# ----------------------------------------------------------------------------- device-side draws
# Large presets (billions of weights) are drawn directly on the GPU with torch's seeded
# Philox generator: same distributions, a different (but equally seeded) stream from the
# numpy draws above.  Used by the benchmark; parity tests use the numpy draws.

def _torch_normal(shape, std, seed, key, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(np.random.SeedSequence([seed, *key]).generate_state(1, np.uint64)[0] & 0x7FFFFFFFFFFFFFFF))
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32) * std


def torch_block_weights(d: ModelDims, layer: int, seed: int = 0, device="cuda", std: float = 0.02):
    import torch
    out = {name: _torch_normal(shp, std, seed, (layer, i), device) for i, (name, shp) in enumerate(linear_shapes(d).items())}
    for name in ("norm1", "norm2") + (("post_attn_norm", "post_ffn_norm") if d.gemma_norms else ()):
        out[name] = torch.ones(d.hidden, device=device)
    if d.gemma_norms:
        out["q_norm"] = torch.ones(d.head_dim, device=device)
        out["k_norm"] = torch.ones(d.head_dim, device=device)
    return out


def torch_embedding(d: ModelDims, seed: int = 0, device="cuda", std: float = 0.02):
    import torch
    return _torch_normal((d.vocab, d.hidden), std, seed, (10_000, 0), device), torch.ones(d.hidden, device=device)
