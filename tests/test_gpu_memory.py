"""The memory claim of Section 3 ("Runtime implementation"): besides the compressed weights, the
checkpoints and the LoRA state, a step holds the intermediates of one subgraph at a time.

Checked on the CUDA path's own accounting (mebp_workspace_breakdown) and on the device:
* the workspace grows with the number of blocks only by the checkpoints and the per-block LoRA
  operand copies (intermediates are sized for one block, never for L);
* with min_memory the context holds exactly one set of block intermediates (half of the default
  two-set workspace for them) and the step's results are bit-identical to the default's;
* a step allocates no device memory (free memory before and after steps is unchanged);
* the whole device footprint is within weights + checkpoints + one block's working set + the
  LM-head workspace + LoRA state, the working set bounded per token from the block's shapes.
"""
import numpy as np
import pytest

from workload import synth

from .helpers import dense_blocks, to_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2510_03425_gb300 import mebp as M  # noqa: E402
from paper_2510_03425_gb300.model import Context, DeviceBlock, DeviceModel, LoraSet, PackedLinear, compress  # noqa: E402


def _dims(n_layers, **kw):
    base = dict(hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, intermediate=512, n_layers=n_layers, vocab=2048,
                batch=2, seq=96, rank=8, alpha=16.0)
    base.update(kw)
    return synth.tiny(**base)


def _shadow_bytes_per_layer(d):
    """fp16 LoRA operand copies of one block: A_cat [kxp, K], B_cat and B_cat^T [N, kxp] per fused linear."""
    D, I, hd = d.hidden, d.intermediate, d.head_dim
    lins = {"qkv": (("q", "k", "v"), (d.n_heads + 2 * d.n_kv_heads) * hd, D), "o": (("o",), D, d.n_heads * hd),
            "gu": (("gate", "up"), 2 * I, D), "down": (("down",), D, I)}
    tot = 0
    for tg, N, K in lins.values():
        kx = d.rank * sum(t in d.targets for t in tg)
        kxp = (kx + 15) // 16 * 16
        tot += 2 * (kxp * K + 2 * N * kxp)
    return tot


def test_workspace_grows_with_depth_only_by_checkpoints_and_lora_copies():
    d4, d8 = _dims(4), _dims(8)
    c4, c8 = Context(d4), Context(d8)
    b4, n4 = M.mebp_workspace_breakdown(c4.handle)
    b8, n8 = M.mebp_workspace_breakdown(c8.handle)
    T, D = d4.tokens, d4.hidden
    assert n4 == n8 == 2
    assert b8["checkpoints"] - b4["checkpoints"] == 4 * T * D * 4          # four more fp32 [T, D] slots
    assert b8["lora_shadows"] - b4["lora_shadows"] == 4 * _shadow_bytes_per_layer(d4)
    for k in ("forward_sets", "backward", "attention_split", "lm_head", "other"):
        assert b8[k] == b4[k], k
    assert M.mebp_workspace_bytes(c8.handle) == sum(v for k, v in b8.items() if k != "host_checkpoints")
    c4.close()
    c8.close()


def _model(d):
    blocks = dense_blocks(d)
    E, gf = synth.embedding(d)
    loras = [synth.lora_weights(d, i) for i in range(d.n_layers)]
    return blocks, E, gf, loras, synth.token_ids(d)


def _step(ctx, blocks, E, gf, loras, ids, n=1, stream=None):
    model = DeviceModel([DeviceBlock(ctx, {k: to_gpu(v) for k, v in W.items()}) for W in blocks],
                        PackedLinear(*compress(ctx, to_gpu(E))), to_gpu(gf))
    ls = LoraSet(loras)
    loss = torch.zeros(1, device="cuda")
    ms, idg = model.struct(), to_gpu(ids)
    ctx.sync()
    for _ in range(n):
        M.mebp_lora_step(ctx.handle, ms, ls.lora_array(), idg, loss, ls.grads_array(), False, stream)
    ctx.sync(stream)
    return model, ls, float(loss.item())


def test_min_memory_holds_one_set_and_gives_identical_results():
    d = _dims(4)
    data = _model(d)
    c2, c1 = Context(d), Context(d, min_memory=True)
    b2, n2 = M.mebp_workspace_breakdown(c2.handle)
    b1, n1 = M.mebp_workspace_breakdown(c1.handle)
    assert (n2, n1) == (2, 1)
    assert b2["forward_sets"] == 2 * b1["forward_sets"]
    _, ls2, l2 = _step(c2, *data)
    _, ls1, l1 = _step(c1, *data)
    assert l1 == l2
    for g1, g2 in zip(ls1.grads, ls2.grads):
        for n in g1:
            assert torch.equal(g1[n][0], g2[n][0]) and torch.equal(g1[n][1], g2[n][1]), n
    c2.close()
    c1.close()


@pytest.mark.parametrize("min_memory", [False, True])
def test_step_allocates_nothing_and_fits_the_bound(min_memory):
    d = _dims(6)
    blocks, E, gf, loras, ids = _model(d)
    torch.cuda.synchronize()
    free_before_ctx, _ = torch.cuda.mem_get_info()
    reserved_before = torch.cuda.memory_reserved()
    ctx = Context(d, min_memory=min_memory)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        model, ls, _ = _step(ctx, blocks, E, gf, loras, ids, n=3, stream=s)  # eager, capture, replay
        idg = to_gpu(ids)
        loss = torch.zeros(1, device="cuda")
        ms = model.struct()
        M.mebp_lora_step(ctx.handle, ms, ls.lora_array(), idg, loss, ls.grads_array(), False, s)  # eager (new key)
        M.mebp_lora_step(ctx.handle, ms, ls.lora_array(), idg, loss, ls.grads_array(), False, s)  # capture
        ctx.sync(s)
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        alloc0 = torch.cuda.memory_allocated()
        for _ in range(3):
            M.mebp_lora_step(ctx.handle, ms, ls.lora_array(), idg, loss, ls.grads_array(), False, s)
        ctx.sync(s)
        free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0                                   # no device allocation inside a step
    assert torch.cuda.memory_allocated() == alloc0
    # the bound: weights + checkpoints + one block's working set + LM-head workspace + LoRA state
    T, D, I, H, KV, hd = d.tokens, d.hidden, d.intermediate, d.n_heads, d.n_kv_heads, d.head_dim
    nqkv, na = (H + 2 * KV) * hd, H * hd
    # per token, every activation of one block's forward (fp16 GEMM operands, fp32 residual
    # stream and statistics) and of its backward (their gradients), each at most twice
    act_tok = 2 * (2 * D + nqkv + na + 3 * I) + 4 * (2 * D + H + 2) + 2 * 64
    sets = 1 if min_memory else 2
    block_ws = T * (sets * act_tok + 2 * act_tok)
    br, _ = M.mebp_workspace_breakdown(ctx.handle)
    lora_state = 8 * ls.n + br["lora_shadows"]
    weights = sum(t.numel() * t.element_size() for b in model.blocks for lin in (b.qkv, b.o, b.gate_up, b.down)
                  for t in (lin.qpack, lin.scales)) + model.embed.qpack.numel() + 2 * model.embed.scales.numel()
    # "other": RoPE tables, device scalars and the split-K scratch of the LoRA-gradient reductions
    # (a backward working buffer sized, like the rest, for one block at T tokens)
    assert br["other"] <= T * 4 * 2 * (2 * I + nqkv) + (1 << 20), br["other"]
    bound = (weights + br["checkpoints"] + block_ws + br["lm_head"] + br["attention_split"] + br["other"] + lora_state
             + (1 << 20))
    ws = M.mebp_workspace_bytes(ctx.handle)
    assert br["forward_sets"] + br["backward"] <= block_ws, (br["forward_sets"], br["backward"], block_ws)
    assert ws + weights + 8 * ls.n <= bound
    # and the device agrees with the accounting: besides torch's tensors, the device memory taken
    # since before the context is its workspace plus what the driver holds for the library's code
    # (loaded on first launch), the captured graph and allocator rounding
    used_by_ctx = (free_before_ctx - free0) - (torch.cuda.memory_reserved() - reserved_before)
    assert used_by_ctx <= ws + (256 << 20), (used_by_ctx, ws)
    ctx.close()
