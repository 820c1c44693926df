"""MeBP training step in plain numpy fp64 — TEST INFRASTRUCTURE ONLY.

What it follows:

* Section 3, "Gradient checkpointing compilation": the model is split into
  blocks ``y = F_i(x, w)``; each block's backward graph ``B_i(x, dE/dy, w)``
  returns ``(dE/dx, dE/dw)`` and is the VJP of the scalar
  ``s = sum(dE/dy * y)`` (the upstream gradient is held constant).
* Algorithm 1 (``Backpropagation``): a forward loop that stores only
  block-boundary checkpoints, then a reverse loop that, for each block,
  decompresses its weights, recomputes the block from its stored *input*
  checkpoint and applies the VJP.  Only LoRA gradients are returned; the
  compressed base weights are frozen.
* Section 3, "Base model weights compression": every base matrix, the tied
  embedding included, is used as ``deq = q * s`` (see ``quant``) and is
  decompressed only when its block runs.
* Section 4 ("Performance Comparison"): checkpoints at every transformer layer,
  the final linear layer and the cross-entropy layer — here the final RMSNorm,
  tied LM head and mean next-token cross-entropy form the last subgraph.

The block itself is the pre-norm decoder block of the Qwen2.5 / Gemma3 models
the paper evaluates (the paper does not spell it out; the readings are):
RMSNorm -> q,k,v projections (+LoRA) -> half-split RoPE on q,k -> causal
grouped-query attention -> o projection (+LoRA) + residual -> RMSNorm ->
act(gate) * up (+LoRA) -> down projection (+LoRA) + residual, with
act = SiLU (Qwen) or tanh-approximated GELU (Gemma).  No biases, eps = 1e-6,
RoPE theta = 1e6, LoRA ``Y = X W^T + s (X A^T) B^T`` with ``s = alpha / r``.

With ``dims.gemma_norms`` the block follows the Gemma3 architecture of the paper's Gemma models:
per-head RMSNorm of q and k (gains q_norm, k_norm) before RoPE, RMSNorm of the attention output
and of the MLP output before each residual add (gains post_attn_norm, post_ffn_norm; the
pre-norms stay norm1 / norm2), and input embeddings scaled by sqrt(D).  With
``dims.sliding_window = W > 0`` every layer except each ``global_every``-th is local: position i
attends to j with 0 <= i - j < W, and its RoPE base is ``rope_theta_local``.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Tuple

import numpy as np

from . import quant

LINEARS = ("q", "k", "v", "o", "gate", "up", "down")
NORMS = ("norm1", "norm2", "q_norm", "k_norm", "post_attn_norm", "post_ffn_norm")


# ----------------------------------------------------------------------------- basic ops

def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float):
    """y = x / sqrt(mean(x^2) + eps) * g over the last axis; returns (y, r) with r = 1/sqrt(.)."""
    r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    return x * r * g, r


def rmsnorm_vjp(dy: np.ndarray, x: np.ndarray, g: np.ndarray, r: np.ndarray) -> np.ndarray:
    """dx = r (g*dy) - x r^3 / D * sum(g*dy*x)."""
    D = x.shape[-1]
    gd = g * dy
    return r * gd - x * (r ** 3) * np.sum(gd * x, axis=-1, keepdims=True) / D


def silu(x):
    return x / (1.0 + np.exp(-x))


def silu_grad(x):
    sg = 1.0 / (1.0 + np.exp(-x))
    return sg * (1.0 + x * (1.0 - sg))


_GC = math.sqrt(2.0 / math.pi)


def gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(_GC * (x + 0.044715 * x ** 3)))


def gelu_tanh_grad(x):
    th = np.tanh(_GC * (x + 0.044715 * x ** 3))
    return 0.5 * (1.0 + th) + 0.5 * x * (1.0 - th * th) * _GC * (1.0 + 3 * 0.044715 * x * x)


ACT = {"silu": (silu, silu_grad), "gelu_tanh": (gelu_tanh, gelu_tanh_grad)}


def rope_angles(seq: int, hd: int, theta: float) -> np.ndarray:
    """angle[p, j] = p * theta^(-2j/hd) for positions p < seq and j < hd/2."""
    j = np.arange(hd // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * j / hd)
    return np.arange(seq, dtype=np.float64)[:, None] * inv_freq[None, :]


def rope(x: np.ndarray, ang: np.ndarray, inverse: bool = False) -> np.ndarray:
    """Half-split rotation of x [T, nh, hd] by ang [T, hd/2]: (x1, x2) -> (x1 c - x2 s, x2 c + x1 s).

    ``inverse`` rotates by -angle, which is both the inverse and the transpose
    (hence the VJP) of the rotation.
    """
    h = x.shape[-1] // 2
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    if inverse:
        s = -s
    x1, x2 = x[..., :h], x[..., h:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def attention(q, k, v, batch: int, seq: int, window: int = 0):
    """Causal grouped-query attention.  q [T, H, hd], k/v [T, KV, hd], T = batch*seq.

    Query head h reads key/value head h // (H/KV); scores are scaled by 1/sqrt(hd)
    and position i attends to positions j <= i of its own sequence (and, with a
    sliding window W > 0, only to i - j < W).
    Returns o [T, H, hd], lse [batch, H, seq], P (list per (b, h)) for the VJP.
    """
    T, H, hd = q.shape
    KV = k.shape[1]
    grp = H // KV
    scale = 1.0 / math.sqrt(hd)
    causal = np.tril(np.ones((seq, seq), dtype=bool))
    if window > 0:
        causal &= np.triu(np.ones((seq, seq), dtype=bool), -(window - 1))
    o = np.zeros_like(q)
    lse = np.zeros((batch, H, seq))
    probs = {}
    for b in range(batch):
        sl = slice(b * seq, (b + 1) * seq)
        for h in range(H):
            kh = h // grp
            Sc = (q[sl, h] @ k[sl, kh].T) * scale
            Sc = np.where(causal, Sc, -np.inf)
            m = Sc.max(axis=1, keepdims=True)
            E = np.exp(Sc - m)
            l = E.sum(axis=1, keepdims=True)
            P = E / l
            o[sl, h] = P @ v[sl, kh]
            lse[b, h] = (m + np.log(l))[:, 0]
            probs[(b, h)] = P
    return o, lse, probs


def attention_vjp(do, q, k, v, probs, batch: int, seq: int):
    """VJP of ``attention``: dP = dO V^T, dS = P * (dP - rowsum(P * dP)),
    dQ = dS K / sqrt(hd), dK = dS^T Q / sqrt(hd), dV = P^T dO; dK, dV summed over
    the query heads sharing a key/value head."""
    T, H, hd = q.shape
    KV = k.shape[1]
    grp = H // KV
    scale = 1.0 / math.sqrt(hd)
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for b in range(batch):
        sl = slice(b * seq, (b + 1) * seq)
        for h in range(H):
            kh = h // grp
            P = probs[(b, h)]
            dP = do[sl, h] @ v[sl, kh].T
            dS = P * (dP - np.sum(P * dP, axis=1, keepdims=True))
            dq[sl, h] = (dS @ k[sl, kh]) * scale
            dk[sl, kh] += (dS.T @ q[sl, h]) * scale
            dv[sl, kh] += P.T @ do[sl, h]
    return dq, dk, dv


# ----------------------------------------------------------------------------- LoRA linear

def linear(X, W, lora: Optional[Tuple[np.ndarray, np.ndarray]], s: float):
    """Y = X W^T (+ s (X A^T) B^T); returns (Y, U) with U = X A^T (None without LoRA)."""
    Y = X @ W.T
    if lora is None:
        return Y, None
    A, B = lora
    U = X @ A.T
    return Y + s * (U @ B.T), U


def linear_vjp(dY, X, U, W, lora, s: float, need_dx: bool = True):
    """dX = dY W + s (dY B) A; dB = s dY^T U; dA = (s dY B)^T X.  Base W gets no gradient (frozen)."""
    dX = dY @ W if need_dx else None
    if lora is None:
        return dX, None
    A, B = lora
    dU = s * (dY @ B)
    if need_dx:
        dX = dX + dU @ A
    dB = s * (dY.T @ U)
    dA = dU.T @ X
    return dX, (dA, dB)


# ----------------------------------------------------------------------------- the block

def block_forward(x, W: Dict[str, np.ndarray], lora: Dict[str, Tuple], dims, save: bool = False, layer: int = 0):
    """One pre-norm decoder block y = F(x, w).  x [T, D] float64; W holds dense
    (already decompressed) matrices W[name] [N_out, K_in] and norm gains.  ``layer``
    selects local or global attention when dims.sliding_window > 0.
    Returns y, and the saved intermediates when ``save``."""
    D, H, KV, hd = dims.hidden, dims.n_heads, dims.n_kv_heads, dims.head_dim
    T = x.shape[0]
    s = dims.lora_scale
    act, _ = ACT[dims.act]
    gemma = getattr(dims, "gemma_norms", False)
    local = dims.layer_is_local(layer) if hasattr(dims, "layer_is_local") else False
    theta = dims.rope_theta_local if local else dims.rope_theta
    window = dims.sliding_window if local else 0
    pos_ang = rope_angles(dims.seq, hd, theta)[np.arange(T) % dims.seq]

    a, r1 = rmsnorm(x, W["norm1"], dims.eps)
    q, Uq = linear(a, W["q"], lora.get("q"), s)
    k, Uk = linear(a, W["k"], lora.get("k"), s)
    v, Uv = linear(a, W["v"], lora.get("v"), s)
    q_raw, k_raw = q.reshape(T, H, hd), k.reshape(T, KV, hd)
    rq = rk = None
    if gemma:  # QK-norm: per-head RMSNorm before the rotation
        qn, rq = rmsnorm(q_raw, W["q_norm"], dims.eps)
        kn, rk = rmsnorm(k_raw, W["k_norm"], dims.eps)
    else:
        qn, kn = q_raw, k_raw
    q = rope(qn, pos_ang)
    k = rope(kn, pos_ang)
    v = v.reshape(T, KV, hd)
    o, lse, probs = attention(q, k, v, dims.batch, dims.seq, window)
    o2 = o.reshape(T, H * hd)
    ao, Uo = linear(o2, W["o"], lora.get("o"), s)
    rpa = None
    if gemma:  # sandwich norm on the attention output
        aon, rpa = rmsnorm(ao, W["post_attn_norm"], dims.eps)
    else:
        aon = ao
    h1 = x + aon
    b, r2 = rmsnorm(h1, W["norm2"], dims.eps)
    g, Ug = linear(b, W["gate"], lora.get("gate"), s)
    u, Uu = linear(b, W["up"], lora.get("up"), s)
    m = act(g) * u
    dn, Ud = linear(m, W["down"], lora.get("down"), s)
    rpf = None
    if gemma:  # sandwich norm on the MLP output
        dnn, rpf = rmsnorm(dn, W["post_ffn_norm"], dims.eps)
    else:
        dnn = dn
    y = h1 + dnn
    if not save:
        return y, None
    cache = dict(x=x, a=a, r1=r1, q=q, k=k, v=v, o=o, lse=lse, probs=probs, o2=o2, h1=h1,
                 b=b, r2=r2, g=g, u=u, m=m, U=dict(q=Uq, k=Uk, v=Uv, o=Uo, gate=Ug, up=Uu, down=Ud),
                 ang=pos_ang, gemma=gemma, q_raw=q_raw, k_raw=k_raw, rq=rq, rk=rk, ao=ao, rpa=rpa, dn=dn, rpf=rpf)
    return y, cache


def block_backward(dy, cache, W, lora, dims, need_dx: bool = True):
    """Block VJP B(x, dE/dy, w) -> (dE/dx, {name: (dA, dB)})."""
    H, KV, hd = dims.n_heads, dims.n_kv_heads, dims.head_dim
    T = dy.shape[0]
    s = dims.lora_scale
    act, act_grad = ACT[dims.act]
    c = cache
    grads = {}
    U = c["U"]

    def lin_bwd(name, dY, X, need=True):
        dX, gr = linear_vjp(dY, X, U[name], W[name], lora.get(name), s, need_dx=need)
        if gr is not None:
            grads[name] = gr
        return dX

    # y = h1 + [norm_pf](down(m))
    ddn = rmsnorm_vjp(dy, c["dn"], W["post_ffn_norm"], c["rpf"]) if c["gemma"] else dy
    dm = lin_bwd("down", ddn, c["m"])
    ag = act(c["g"])
    dg = dm * c["u"] * act_grad(c["g"])
    du = dm * ag
    db = lin_bwd("gate", dg, c["b"]) + lin_bwd("up", du, c["b"])
    dh1 = dy + rmsnorm_vjp(db, c["h1"], W["norm2"], c["r2"])
    # h1 = x + [norm_pa](o_proj(attn))
    dao = rmsnorm_vjp(dh1, c["ao"], W["post_attn_norm"], c["rpa"]) if c["gemma"] else dh1
    do2 = lin_bwd("o", dao, c["o2"])
    dq, dk, dv = attention_vjp(do2.reshape(T, H, hd), c["q"], c["k"], c["v"], c["probs"],
                               dims.batch, dims.seq)
    dq = rope(dq, c["ang"], inverse=True)
    dk = rope(dk, c["ang"], inverse=True)
    if c["gemma"]:
        dq = rmsnorm_vjp(dq, c["q_raw"], W["q_norm"], c["rq"])
        dk = rmsnorm_vjp(dk, c["k_raw"], W["k_norm"], c["rk"])
    dq = dq.reshape(T, H * hd)
    dk = dk.reshape(T, KV * hd)
    dv = dv.reshape(T, KV * hd)
    da_q = lin_bwd("q", dq, c["a"], need_dx)
    da_k = lin_bwd("k", dk, c["a"], need_dx)
    da_v = lin_bwd("v", dv, c["a"], need_dx)
    if not need_dx:
        return None, grads
    da = da_q + da_k + da_v
    dx = dh1 + rmsnorm_vjp(da, c["x"], W["norm1"], c["r1"])
    return dx, grads


def block_objective(x, W, lora, G, dims, layer: int = 0):
    """Single-block objective E = sum(G * y) (the scalar of Section 3 with dE/dy = G).
    Returns E, dE/dx and the LoRA gradients, through one checkpointed recompute + backward."""
    y, _ = block_forward(x, W, lora, dims, layer=layer)                 # forward pass: only the output is kept
    E = float(np.sum(G * y))
    _, cache = block_forward(x, W, lora, dims, save=True, layer=layer)  # recompute from the stored input
    dx, grads = block_backward(G, cache, W, lora, dims)
    return E, dx, grads


# ----------------------------------------------------------------------------- LM head + CE

def next_token_targets(ids: np.ndarray) -> np.ndarray:
    """targets[b, s] = ids[b, s+1] for s < S-1, and -1 (ignored) at the last position."""
    t = np.full_like(ids, -1)
    t[:, :-1] = ids[:, 1:]
    return t.reshape(-1)


def lm_head_ce(h, g_f, E_deq, targets, eps: float, row_block: int = 256, want_token_loss=False):
    """Final RMSNorm, tied LM head z = hf E^T and mean cross-entropy over valid targets.

    loss = mean_t [logsumexp(z_t) - z_t[y_t]];  dz = (softmax(z_t) - onehot(y_t)) / N_valid.
    Returns loss, dE/dh (and the per-token loss terms).  Tokens are processed in
    independent row blocks only to bound memory; each row's arithmetic is the
    plain definition.
    """
    hf, r = rmsnorm(h, g_f, eps)
    T = h.shape[0]
    valid = targets >= 0
    n_valid = int(valid.sum())
    dhf = np.zeros_like(hf)
    tok_loss = np.zeros(T)
    for t0 in range(0, T, row_block):
        sl = slice(t0, min(T, t0 + row_block))
        z = hf[sl] @ E_deq.T
        m = z.max(axis=1, keepdims=True)
        lse = m[:, 0] + np.log(np.exp(z - m).sum(axis=1))
        tg = targets[sl]
        ok = tg >= 0
        rows = np.nonzero(ok)[0]
        zt = np.zeros(len(tg))
        zt[rows] = z[rows, tg[rows]]
        tok_loss[sl] = np.where(ok, lse - zt, 0.0)
        dz = np.exp(z - lse[:, None])
        dz[rows, tg[rows]] -= 1.0
        dz *= (ok / max(n_valid, 1))[:, None]
        dhf[sl] = dz @ E_deq
    loss = float(tok_loss.sum() / max(n_valid, 1))
    dh = rmsnorm_vjp(dhf, h, g_f, r)
    if want_token_loss:
        return loss, dh, tok_loss
    return loss, dh


# ----------------------------------------------------------------------------- Algorithm 1

class PackedModel:
    """Compressed base weights of a whole model (InitializeModel keeps only these).

    blocks[i][name] = (qpack, scales) for the seven linears, plus dense fp32 norm
    gains; embed = (qpack, scales) of the tied [V, D] matrix; final_norm = gain.
    """

    def __init__(self, blocks, embed, final_norm):
        self.blocks = blocks
        self.embed = embed
        self.final_norm = final_norm

    @classmethod
    def compress(cls, dense_blocks, E=None, g_f=None):
        blocks = []
        for Wb in dense_blocks:
            pb = {n: quant.compress(Wb[n]) for n in LINEARS}
            for nm in NORMS:
                if nm in Wb:
                    pb[nm] = np.asarray(Wb[nm], np.float64)
            blocks.append(pb)
        embed = quant.compress(E) if E is not None else None
        return cls(blocks, embed, None if g_f is None else np.asarray(g_f, np.float64))

    def decompress_block(self, i: int) -> Dict[str, np.ndarray]:
        """LazyLoadAndDecompressWeights(i): dense float64 matrices of block i."""
        pb = self.blocks[i]
        W = {n: quant.dequant(*pb[n]) for n in LINEARS}
        for nm in NORMS:
            if nm in pb:
                W[nm] = pb[nm]
        return W


def embed_tokens(model: PackedModel, ids: np.ndarray, dims=None) -> np.ndarray:
    """x0[t] = deq(E)[id_t] (the embedding is compressed like every base matrix), times sqrt(D)
    for the Gemma3 block."""
    x0 = quant.dequant_rows(*model.embed, ids.reshape(-1))
    if dims is not None and getattr(dims, "gemma_norms", False):
        x0 = x0 * math.sqrt(dims.hidden)
    return x0


def lora64(lora_layer):
    return {n: (np.asarray(A, np.float64), np.asarray(B, np.float64)) for n, (A, B) in lora_layer.items()}


def mebp_backpropagation(model: PackedModel, lora: List[Dict], ids: np.ndarray, dims,
                         want_trace: bool = False):
    """Algorithm 1, Backpropagation(x): returns (loss, lora_grads[layer][name] = (dA, dB)).

    The backward graph of block i consumes the checkpoint that is block i's
    *input* (ckpts_{i-1}); Section 3 defines B_i(x, dE/dy, w) with x the block
    input, so that is the reading taken for the index of the checkpoint loaded
    in the backward loop.
    """
    n = len(model.blocks)
    targets = next_token_targets(ids)
    ckpts = {0: embed_tokens(model, ids, dims)}           # ckpts_storage <- {x}
    for i in range(1, n + 1):                             # forward loop, checkpoints only
        W = model.decompress_block(i - 1)
        ckpts[i], _ = block_forward(ckpts[i - 1], W, lora64(lora[i - 1]), dims, layer=i - 1)
    E_deq = quant.dequant(*model.embed)                   # final linear layer (tied embedding)
    loss, g, tok = lm_head_ce(ckpts[n], model.final_norm, E_deq, targets, dims.eps, want_token_loss=True)
    del E_deq
    trace = {"ckpts": dict(ckpts), "dh": g.copy(), "tok_loss": tok, "dys": {}} if want_trace else None
    grads: List[Optional[Dict]] = [None] * n
    del ckpts[n]
    for i in range(n, 0, -1):                             # backward loop, reverse order
        W = model.decompress_block(i - 1)
        lw = lora64(lora[i - 1])
        _, cache = block_forward(ckpts[i - 1], W, lw, dims, save=True, layer=i - 1)   # recompute block i
        if want_trace:
            trace["dys"][i] = g.copy()
        g, grads[i - 1] = block_backward(g, cache, W, lw, dims, need_dx=(i > 1))
        del ckpts[i - 1]                                  # the checkpoint is removed once used
    if want_trace:
        return loss, grads, trace
    return loss, grads


def full_backpropagation(model: PackedModel, lora: List[Dict], ids: np.ndarray, dims):
    """Reference without checkpointing: one forward that keeps every intermediate
    of every block, then the backward from those stored intermediates."""
    n = len(model.blocks)
    targets = next_token_targets(ids)
    x = embed_tokens(model, ids, dims)
    caches, Ws = [], []
    for i in range(n):
        W = model.decompress_block(i)
        x, cache = block_forward(x, W, lora64(lora[i]), dims, save=True, layer=i)
        caches.append(cache)
        Ws.append(W)
    E_deq = quant.dequant(*model.embed)
    loss, g = lm_head_ce(x, model.final_norm, E_deq, targets, dims.eps)
    grads = [None] * n
    for i in range(n - 1, -1, -1):
        g, grads[i] = block_backward(g, caches[i], Ws[i], lora64(lora[i]), dims, need_dx=(i > 0))
    return loss, grads


def lora_param_count(dims) -> int:
    """Trainable parameters: sum over layers and targeted linears of r * (K_in + N_out)."""
    D, H, KV, hd, I = dims.hidden, dims.n_heads, dims.n_kv_heads, dims.head_dim, dims.intermediate
    shapes = {"q": (H * hd, D), "k": (KV * hd, D), "v": (KV * hd, D), "o": (D, H * hd),
              "gate": (I, D), "up": (I, D), "down": (D, I)}
    return dims.n_layers * sum(dims.rank * (shapes[t][0] + shapes[t][1]) for t in dims.targets)
