"""Pins of the oracle's Gemma3 block options (QK-norm, sandwich norms, sqrt(D) embedding scale,
sliding-window local layers): finite differences of the block and of Algorithm 1's loss,
checkpointed == non-checkpointed, brute-force windowed attention, and special cases that
reduce to known results (zero post-norm gains give the identity block, a window as long as the
sequence is plain causal attention, a window of one returns v, unit QK-norm gains give unit-RMS
heads)."""
import math

import numpy as np

from oracle import model as M
from workload import synth


def _dims(**kw):
    base = dict(act="gelu_tanh", n_heads=4, n_kv_heads=2, head_dim=16, hidden=32, intermediate=48, batch=2, seq=7,
                rank=3, alpha=6.0, gemma_norms=True, sliding_window=3, global_every=2, rope_theta_local=1e4)
    base.update(kw)
    return synth.tiny(**base)


def _dense(dims, layer):
    W = synth.block_weights(dims, layer, norm_jitter=0.1, std=0.2)
    return {k: v.astype(np.float64) for k, v in W.items()}


def test_layer_pattern():
    d = _dims(global_every=3)
    assert [d.layer_is_local(i) for i in range(6)] == [True, True, False, True, True, False]
    assert not any(_dims(sliding_window=0).layer_is_local(i) for i in range(4))


def test_gemma_block_vjp_matches_central_differences_local_and_global():
    dims = _dims()
    rng = np.random.default_rng(1)
    W = _dense(dims, 0)
    L = M.lora64(synth.lora_weights(dims, 0, std=0.1))
    x = rng.standard_normal((dims.tokens, dims.hidden))
    G = rng.standard_normal((dims.tokens, dims.hidden))
    h = 1e-6
    for layer in (0, 1):  # local (window 3, theta 1e4) and global
        assert dims.layer_is_local(layer) == (layer == 0)

        def E(xx, LL):
            return float(np.sum(G * M.block_forward(xx, W, LL, dims, layer=layer)[0]))

        _, dx, grads = M.block_objective(x, W, L, G, dims, layer=layer)
        for (i, j) in [(0, 0), (6, 31), (13, 5), (9, 17)]:
            xp, xm = x.copy(), x.copy()
            xp[i, j] += h
            xm[i, j] -= h
            fd = (E(xp, L) - E(xm, L)) / (2 * h)
            assert abs(fd - dx[i, j]) <= 1e-6 * max(1.0, abs(dx[i, j])), (layer, i, j, fd, dx[i, j])
        for name in synth.TARGETS:
            for which in (0, 1):
                arr = L[name][which]
                for idx in [(0, 0), (arr.shape[0] - 1, arr.shape[1] - 1)]:
                    Lp = {k: (a.copy(), b.copy()) for k, (a, b) in L.items()}
                    Lm = {k: (a.copy(), b.copy()) for k, (a, b) in L.items()}
                    Lp[name][which][idx] += h
                    Lm[name][which][idx] -= h
                    fd = (E(x, Lp) - E(x, Lm)) / (2 * h)
                    an = grads[name][which][idx]
                    assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (layer, name, which, idx, fd, an)


def test_zero_post_norm_gains_make_the_block_the_identity():
    dims = _dims()
    W = _dense(dims, 0)
    W["post_attn_norm"] = np.zeros(dims.hidden)
    W["post_ffn_norm"] = np.zeros(dims.hidden)
    x = np.random.default_rng(2).standard_normal((dims.tokens, dims.hidden))
    y, _ = M.block_forward(x, W, M.lora64(synth.lora_weights(dims, 0, std=0.1)), dims)
    np.testing.assert_array_equal(y, x)


def test_sliding_window_attention_special_cases_and_brute_force():
    rng = np.random.default_rng(3)
    S, H, KV, hd = 9, 4, 2, 5
    q = rng.standard_normal((S, H, hd))
    k = rng.standard_normal((S, KV, hd))
    v = rng.standard_normal((S, KV, hd))
    o_full, lse_full, _ = M.attention(q, k, v, 1, S)
    o_s, lse_s, _ = M.attention(q, k, v, 1, S, window=S)
    np.testing.assert_array_equal(o_s, o_full)        # a window as long as the sequence: plain causal
    np.testing.assert_array_equal(lse_s, lse_full)
    o1, _, _ = M.attention(q, k, v, 1, S, window=1)   # only itself: o = v of the head's group
    np.testing.assert_allclose(o1, v[:, [0, 0, 1, 1]], rtol=0, atol=1e-15)
    W = 4
    o, lse, _ = M.attention(q, k, v, 1, S, window=W)
    for h in range(H):
        kh = h * KV // H
        for i in range(S):
            js = [j for j in range(S) if j <= i and i - j < W]
            sc = [sum(q[i, h, d] * k[j, kh, d] for d in range(hd)) / math.sqrt(hd) for j in js]
            mx = max(sc)
            w = [math.exp(s_ - mx) for s_ in sc]
            ref = [sum(wj * v[j, kh, d] for wj, j in zip(w, js)) / sum(w) for d in range(hd)]
            np.testing.assert_allclose(o[i, h], ref, rtol=1e-12)
            assert abs(lse[0, h, i] - (mx + math.log(sum(w)))) < 1e-12


def test_unit_qk_norm_gains_give_unit_rms_heads():
    dims = _dims(sliding_window=0)
    W = {k: v.astype(np.float64) for k, v in synth.block_weights(dims, 0, std=0.2).items()}  # unit gains
    x = np.random.default_rng(4).standard_normal((dims.tokens, dims.hidden))
    _, c = M.block_forward(x, W, {}, dims, save=True)
    # rotation preserves the norm, so the stored (rotated) heads keep RMS sqrt(1 - eps r^2) ~ 1
    for t in (c["q"], c["k"]):
        rms = np.sqrt(np.mean(t * t, axis=-1))
        np.testing.assert_allclose(rms, 1.0, atol=1e-5)


def test_embedding_scale():
    dims = _dims(n_layers=1, vocab=37, hidden=64, intermediate=128)
    E, gf = synth.embedding(dims, std=0.5)
    pm = M.PackedModel.compress([synth.block_weights(dims, 0)], E, gf)
    ids = synth.token_ids(dims)
    plain = M.embed_tokens(pm, ids)
    np.testing.assert_allclose(M.embed_tokens(pm, ids, dims), plain * math.sqrt(dims.hidden), rtol=1e-15)


def test_gemma_algorithm1_checkpointed_exact_and_loss_finite_differences():
    dims = _dims(n_layers=3, vocab=31, global_every=3, hidden=64, intermediate=128)
    blocks = [synth.block_weights(dims, i, norm_jitter=0.1, std=0.2) for i in range(dims.n_layers)]
    E, gf = synth.embedding(dims, std=0.5, norm_jitter=0.1)
    pm = M.PackedModel.compress(blocks, E, gf)
    lora = [synth.lora_weights(dims, i, std=0.1) for i in range(dims.n_layers)]
    ids = synth.token_ids(dims)
    loss1, g1 = M.mebp_backpropagation(pm, lora, ids, dims)
    loss2, g2 = M.full_backpropagation(pm, lora, ids, dims)
    assert loss1 == loss2
    for a, b in zip(g1, g2):
        for n in a:
            np.testing.assert_array_equal(a[n][0], b[n][0])
            np.testing.assert_array_equal(a[n][1], b[n][1])
    h = 1e-6
    for layer, name, which, idx in [(0, "q", 0, (1, 3)), (2, "k", 1, (5, 2)), (1, "down", 0, (0, 40))]:
        lp = [{k: (a.astype(np.float64).copy(), b.astype(np.float64).copy()) for k, (a, b) in L.items()} for L in lora]
        lm = [{k: (a.astype(np.float64).copy(), b.astype(np.float64).copy()) for k, (a, b) in L.items()} for L in lora]
        lp[layer][name][which][idx] += h
        lm[layer][name][which][idx] -= h
        fd = (M.mebp_backpropagation(pm, lp, ids, dims)[0] - M.mebp_backpropagation(pm, lm, ids, dims)[0]) / (2 * h)
        an = g1[layer][name][which][idx]
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (layer, name, fd, an)


def test_local_rope_base_applies_to_local_layers_only():
    x = np.random.default_rng(5).standard_normal((14, 32))
    same = _dims(sliding_window=7, rope_theta_local=1e6)            # window >= seq, same base
    W = _dense(same, 0)
    y_loc, _ = M.block_forward(x, W, {}, same, layer=0)
    y_glb, _ = M.block_forward(x, W, {}, same, layer=1)
    np.testing.assert_array_equal(y_loc, y_glb)
    other = _dims(sliding_window=7, rope_theta_local=1e3)
    assert np.abs(M.block_forward(x, W, {}, other, layer=0)[0] - y_loc).max() > 1e-3
    np.testing.assert_array_equal(M.block_forward(x, W, {}, other, layer=1)[0], y_glb)
