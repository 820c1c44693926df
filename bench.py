"""Benchmark of one MeBP LoRA training step (Algorithm 1) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config C] [--impl gb300|reference]

A step = embed -> checkpointed forward loop over all blocks -> LM-head cross-entropy
(forward + backward, vocabulary-chunked) -> reverse loop of block recompute + backward,
producing the loss and every LoRA gradient (mebp_lora_step).  The default workload is the
full Qwen2.5-0.5B-shaped model (24 blocks, vocab 151936, batch 1 x seq 512, LoRA r8 on
q/k/v/o, 4-bit group-64 base weights).  Prints one JSON line (rank 0).

--impl reference times the CPU oracle (plain numpy fp64) on the host cores, on a bounded
sample of the same workload (one block's forward + recompute + backward and an LM-head
token sample), extrapolated to the step.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from workload import synth  # noqa: E402

METRIC = "train tokens/s per LoRA step (1 GB300); fused dequant-GEMM % of BF16 tensor peak"


def workload_name(d) -> str:
    return (f"{d.name}: {d.n_layers} blocks (D {d.hidden}, H {d.n_heads}/KV {d.n_kv_heads}, hd {d.head_dim}, "
            f"I {d.intermediate}, {d.act}), vocab {d.vocab}, batch {d.batch} x seq {d.seq}, "
            f"LoRA r{d.rank} on {'/'.join(d.targets)}, 4-bit g64 fp16-scale base weights"
            + (", checkpoints spilled to pinned host" if d.spill else "")
            + (f", Gemma3 block (QK-norm, sandwich norms, sqrt(D) embedding, window {d.sliding_window} on "
               f"{d.global_every - 1} of every {d.global_every} layers, local RoPE base {d.rope_theta_local:g})"
               if d.gemma_norms else ""))


def gemma3_extras(d):
    """The Gemma-shaped workload with the Gemma3 block options on: QK-norm, sandwich norms,
    sqrt(D) embedding scale, five local layers (window 512 for the 1B shape, 1024 for the 4B
    shape, RoPE base 1e4) per global layer."""
    return d.with_(gemma_norms=True, sliding_window=512 if d.hidden < 2048 else 1024, global_every=6,
                   rope_theta_local=1e4)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ----------------------------------------------------------------------------- CPU oracle sample
def oracle_sample(d, lm_tokens: int = 32):
    """Time the oracle on one block (forward, recompute, backward) and an LM-head token
    sample; return (tokens/s extrapolated to the whole step, description)."""
    from oracle import model as OM
    from oracle import quant

    W = synth.block_weights(d, 0)
    L = OM.lora64(synth.lora_weights(d, 0))
    x = synth.hidden_input(d).astype(np.float64)
    G = synth.upstream_grad(d).astype(np.float64)
    t0 = time.perf_counter()
    pm = OM.PackedModel.compress([W])
    Wd = pm.decompress_block(0)
    OM.block_objective(x, Wd, L, G, d)
    t_block = time.perf_counter() - t0
    t_lm = 0.0
    if d.vocab:
        E, gf = synth.embedding(d)
        qE = quant.compress(E)
        t1 = time.perf_counter()
        Ed = quant.dequant(*qE)
        t_deq = time.perf_counter() - t1
        h = x[:lm_tokens]
        tg = synth.token_ids(d).reshape(-1)[:lm_tokens].astype(np.int64)
        t2 = time.perf_counter()
        OM.lm_head_ce(h, gf.astype(np.float64), Ed, tg, d.eps)
        t_lm = t_deq + (time.perf_counter() - t2) * d.tokens / lm_tokens
    t_step = d.n_layers * t_block + t_lm
    desc = (f"oracle (numpy fp64) on 1 of {d.n_layers} blocks at the full {d.tokens} tokens (compress + decompress + "
            f"forward + recompute + backward) and the LM head on {lm_tokens} of {d.tokens} tokens, extrapolated "
            f"linearly to the step")
    return d.tokens / t_step, desc


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.p = None
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                       "-i", str(gpu_index), "-lms", "100"], stdout=subprocess.PIPE,
                                      stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
            out, _ = self.p.communicate()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- GPU arm
def build_model(ctx, d, device):
    import torch

    from paper_2510_03425_gb300.model import DeviceBlock, DeviceModel, PackedLinear, compress
    big = d.n_layers * d.hidden * d.intermediate > 2e8
    blocks = []
    for i in range(d.n_layers):
        if big:
            W = synth.torch_block_weights(d, i, device=device)
        else:
            W = {k: torch.from_numpy(v).to(device) for k, v in synth.block_weights(d, i).items()}
        blocks.append(DeviceBlock(ctx, W))
        del W
    if big:
        E, gf = synth.torch_embedding(d, device=device)
    else:
        En, gfn = synth.embedding(d)
        E, gf = torch.from_numpy(En).to(device), torch.from_numpy(gfn).to(device)
    emb = PackedLinear(*compress(ctx, E))
    del E
    torch.cuda.empty_cache()
    return DeviceModel(blocks, emb, gf)


def run_gpu(args, d, rank, world, local_rank):
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context, LoraSet

    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    ctx = Context(d, device=local_rank)
    model = build_model(ctx, d, device)
    ls = LoraSet([synth.lora_weights(d, i) for i in range(d.n_layers)], device=device)
    ids_host = torch.from_numpy(synth.token_ids(d, seed=2 + rank)).pin_memory()
    ids = ids_host.to(device)
    loss = torch.zeros(1, device=device)
    loss_host = torch.zeros(1).pin_memory()
    mstruct = model.struct()
    # a dedicated stream: mebp_lora_step replays a captured CUDA graph on non-default streams
    st = torch.cuda.Stream(device)
    torch.cuda.set_stream(st)

    def step():
        M.mebp_lora_step(ctx.handle, mstruct, ls.lora_array(), ids, loss, ls.grads_array(), False, st)

    gpu_index = local_rank
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis and vis.split(",")[local_rank].strip().isdigit():
        gpu_index = int(vis.split(",")[local_rank])
    clocks = ClockSampler(gpu_index)
    for _ in range(args.warmup):
        step()
    ctx.sync()
    # ---- timed region: K steps, inputs resident in HBM
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    n0 = M.mebp_kernel_launches()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(args.steps):
        step()
    e1.record(st)
    torch.cuda.synchronize()
    launches = M.mebp_kernel_launches() - n0
    if dist:
        dist.barrier()
    clk = clocks.stop()
    ctx.sync()
    t = e0.elapsed_time(e1) / 1e3
    if dist:
        tt = torch.tensor([t], device=device)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        t = float(tt.item())
    value = world * d.tokens * args.steps / t

    # ---- GEMM roofline: CUDA events around every fused dequant-GEMM launch of K more steps
    M.mebp_profile_begin(ctx.handle)
    for _ in range(args.steps):
        step()
    prof = M.mebp_profile_end(ctx.handle)

    # ---- end to end through the public API: ids host->device, step, loss device->host
    ctx.sync()
    h2d = ids_host.numel() * ids_host.element_size()
    d2h = loss.numel() * loss.element_size()
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2.record(st)
    for _ in range(args.steps):
        ids.copy_(ids_host, non_blocking=True)
        step()
        loss_host.copy_(loss, non_blocking=True)
    e3.record(st)
    torch.cuda.synchronize()
    te = e2.elapsed_time(e3) / 1e3
    if dist:
        tt = torch.tensor([te], device=device)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        te = float(tt.item())
    ctx.sync()

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return None
    pk, src = peaks()
    long_step = t / args.steps > 1.0
    peak = pk["bf16_tflops_sustained"] if long_step else pk["bf16_tflops"]
    achieved = prof.gemm_flops / (prof.gemm_ms / 1e3) / 1e12 if prof.gemm_ms > 0 else None
    weights_mb = sum(b.qkv.qpack.numel() + b.o.qpack.numel() + b.gate_up.qpack.numel() + b.down.qpack.numel()
                     for b in model.blocks) / 2**20 * (1 + 1 / 16)
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * t / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": workload_name(d), "config_index": args.config, "global_batch": world * d.batch,
                   "seq_len": d.seq, "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "l2": f"inputs larger than L2: {weights_mb:.0f} MB of packed block weights plus the "
                         f"{d.vocab}x{d.hidden} packed LM head are streamed every step"},
        "roofline": {"kernel": "dequant_gemm_kernel (fused 4-bit dequant GEMM, tcgen05)", "bound": "tensor",
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": (achieved / peak) if achieved else None, "traffic": None,
                     "peak_source": f"{src} {'sustained' if long_step else 'burst'} dense bf16 GEMM rate "
                                    "(MEASURED_PEAKS.json); fp16 and bf16 share the kind::f16 rate (nominal ratio 1)",
                     "launches_per_step": prof.gemm_launches / args.steps,
                     "share_of_step": (prof.gemm_ms / 1e3) / t if t > 0 else None,
                     "fwd_tflops": prof.fwd_flops / max(prof.fwd_ms, 1e-9) / 1e9,
                     "dx_tflops": prof.dx_flops / max(prof.dx_ms, 1e-9) / 1e9},
        "e2e": {"value": world * d.tokens * args.steps / te, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches),
        "clocks": clk,
    }
    ctx.close()
    if dist:
        dist.destroy_process_group()
    return out


def lora_params(d) -> int:
    """Trainable LoRA parameters: r * (K_in + N_out) per targeted linear and layer."""
    shapes = synth.linear_shapes(d)
    return d.n_layers * sum(d.rank * (shapes[t][0] + shapes[t][1]) for t in d.targets)


def adamw_bench(config: int = 4, reps: int = 20, warmup: int = 3):
    """The AdamW update (mebp_adamw_step) alone over the flat LoRA buffer of a workload: reads
    p, g, m, v and writes p, m, v, 28 bytes per parameter; HBM-bound."""
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context
    d = synth.preset(config)
    n = lora_params(d)
    ctx = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=64, max_seq=64)
    g = torch.Generator(device="cuda")
    g.manual_seed(11)
    p = torch.randn(n, device="cuda", generator=g)
    gr = torch.randn(n, device="cuda", generator=g)
    m, v = torch.zeros(n, device="cuda"), torch.zeros(n, device="cuda")
    cfg = M.adamw_cfg(lr=1e-4)
    for t in range(1, warmup + 1):
        M.mebp_adamw_step(ctx.handle, p, gr, m, v, cfg, t)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for t in range(warmup + 1, warmup + reps + 1):
        M.mebp_adamw_step(ctx.handle, p, gr, m, v, cfg, t)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    ctx.sync()
    ctx.close()
    pk, src = peaks()
    gbs = 28.0 * n / (ms / 1e3) / 1e9
    return {"workload": f"AdamW over the {n} LoRA parameters of {d.name} (r{d.rank} on {'/'.join(d.targets)}), "
                        f"flat fp32 buffers ({28.0 * n / 1e9:.2f} GB per update, larger than L2)",
            "bound": "hbm", "us": 1e3 * ms, "achieved": gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": gbs / pk["hbm_gbs"], "peak_source": f"{src} copy bandwidth"}


def _time_ms(f, reps: int, warmup: int = 3) -> float:
    import torch
    for _ in range(warmup):
        f()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        f()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def table2(reps: int = 10):
    """Analogues of the paper's Table 2 (share of each pass spent on weight decompression) and
    Table 3 (sequence-length sweep) on GB300.

    Per projection GEMM of a workload: t_fused (this library: decode inside the GEMM mainloop),
    t_dense (cuBLAS fp16 GEMM on weights decoded beforehand: a dense model with no compression)
    and t_decode (the standalone decode of the whole matrix: the paper's decompress-then-compute
    design pays t_decode + t_dense).  Reported per pass: the fused path's overhead over the dense
    GEMM, (t_fused - t_dense) / t_fused, and the decompression share of decompress-then-compute,
    t_decode / (t_decode + t_dense) -- the quantity Table 2 reports for the iPhone."""
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context, LoraSet, compress
    torch.backends.cuda.matmul.allow_fp16_reduced_precision_reduction = False
    out = {"decompression": {}, "seq_sweep": {}}
    ctx = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=64, max_seq=64)
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    for cfg_i in (1, 4):
        d = synth.preset(cfg_i)
        Mr = d.tokens
        shapes = synth.linear_shapes(d)
        mats = {"qkv": (shapes["q"][0] + 2 * shapes["k"][0], d.hidden), "o": shapes["o"],
                "gate_up": (2 * d.intermediate, d.hidden), "down": shapes["down"]}
        rows, tot = {}, {"fused_fwd": 0.0, "dense_fwd": 0.0, "fused_dx": 0.0, "dense_dx": 0.0, "decode": 0.0}
        for name, (N, K) in mats.items():
            W = torch.randn(N, K, device="cuda", generator=g) * 0.02
            q, sc = compress(ctx, W)
            del W
            Wp = M.packed(q, sc)
            Wd = torch.empty((N, K), dtype=torch.int16, device="cuda")
            X = torch.randn(Mr, K, device="cuda", generator=g).half()
            dY = torch.randn(Mr, N, device="cuda", generator=g).half()
            Y = torch.empty(Mr, N, device="cuda", dtype=torch.float16)
            dX = torch.empty(Mr, K, device="cuda")
            t_dec = _time_ms(lambda: M.mebp_decode_weights(ctx.handle, Wp, Wd), reps)
            Wh = Wd.view(torch.float16)
            t_ff = _time_ms(lambda: M.mebp_linear_fwd(ctx.handle, X, Wp, y_f16=Y), reps)
            t_fd = _time_ms(lambda: M.mebp_linear_dx(ctx.handle, dY, Wp, dx=dX), reps)
            t_df = _time_ms(lambda: torch.matmul(X, Wh.t(), out=Y), reps)
            dXh = torch.empty(Mr, K, device="cuda", dtype=torch.float16)
            t_dd = _time_ms(lambda: torch.matmul(dY, Wh, out=dXh), reps)
            rows[name] = {"N": N, "K": K, "fused_fwd_us": 1e3 * t_ff, "dense_fwd_us": 1e3 * t_df,
                          "fused_dx_us": 1e3 * t_fd, "dense_dx_us": 1e3 * t_dd, "decode_us": 1e3 * t_dec}
            for k, v in (("fused_fwd", t_ff), ("dense_fwd", t_df), ("fused_dx", t_fd), ("dense_dx", t_dd),
                         ("decode", t_dec)):
                tot[k] += v
            del q, sc, Wp, Wd, X, dY, Y, dX, dXh
        out["decompression"][d.name] = {
            "M": Mr, "per_gemm": rows,
            "fused_over_dense_fwd": (tot["fused_fwd"] - tot["dense_fwd"]) / tot["fused_fwd"],
            "fused_over_dense_dx": (tot["fused_dx"] - tot["dense_dx"]) / tot["fused_dx"],
            "decode_share_separate_fwd": tot["decode"] / (tot["decode"] + tot["dense_fwd"]),
            "decode_share_separate_dx": tot["decode"] / (tot["decode"] + tot["dense_dx"]),
        }
        torch.cuda.empty_cache()
    ctx.close()
    # Table 3 analogue: Qwen2.5-1.5B shape, batch 1, the paper's sequence lengths
    base = synth.preset(3).with_(batch=1, spill=False)
    for S in (128, 256, 512, 1024):
        d = base.with_(seq=S)
        c2 = Context(d)
        model = build_model(c2, d, torch.device("cuda"))
        ls = LoraSet([synth.lora_weights(d, i) for i in range(d.n_layers)])
        ids = torch.from_numpy(synth.token_ids(d)).cuda()
        loss = torch.zeros(1, device="cuda")
        st = torch.cuda.Stream()
        ms = model.struct()

        def step():
            M.mebp_lora_step(c2.handle, ms, ls.lora_array(), ids, loss, ls.grads_array(), False, st)
        with torch.cuda.stream(st):
            t = _time_ms(step, reps)
        wb = sum(b.qkv.qpack.numel() + b.o.qpack.numel() + b.gate_up.qpack.numel() + b.down.qpack.numel()
                 for b in model.blocks) * (1 + 1 / 16) + model.embed.qpack.numel() * (1 + 1 / 16)
        out["seq_sweep"][S] = {"ms_per_step": t, "tokens_per_s": S / (t / 1e3),
                               "workspace_mb": M.mebp_workspace_bytes(c2.handle) / 2**20,
                               "packed_weights_mb": wb / 2**20, "lora_and_grads_mb": 2 * 4 * ls.n / 2**20}
        c2.close()
        del model, ls
        torch.cuda.empty_cache()
    return out


def launch_list_step(args, d):
    """Warm-up steps, then one step run eagerly (no graph replay) inside an NVTX range, so a
    profiler can list exactly the kernels of one step."""
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context, LoraSet
    device = torch.device("cuda", 0)
    ctx = Context(d, device=0)
    model = build_model(ctx, d, device)
    ls = LoraSet([synth.lora_weights(d, i) for i in range(d.n_layers)], device=device)
    ids = torch.from_numpy(synth.token_ids(d)).to(device)
    loss = torch.zeros(1, device=device)
    mstruct = model.struct()
    st = torch.cuda.Stream(device)
    torch.cuda.set_stream(st)
    for _ in range(args.warmup):
        M.mebp_lora_step(ctx.handle, mstruct, ls.lora_array(), ids, loss, ls.grads_array(), False, st)
    ctx.sync()
    M.mebp_enable_graphs(ctx.handle, False)
    n0 = M.mebp_kernel_launches()
    torch.cuda.nvtx.range_push("mebp_step")
    M.mebp_lora_step(ctx.handle, mstruct, ls.lora_array(), ids, loss, ls.grads_array(), False, st)
    torch.cuda.nvtx.range_pop()
    ctx.sync()
    print(json.dumps({"launch_list_step": workload_name(d), "kernels": M.mebp_kernel_launches() - n0,
                      "loss": float(loss.item())}), flush=True)
    ctx.close()


def gemm_bench(config: int, m_tokens=None, reps: int = 10, warmup: int = 3, shapes_only=None):
    """The fused dequant-GEMMs alone (forward Y = X deq(W)^T and transposed dX = dY deq(W)) at
    the four projection shapes of a workload, M = its token count.  Returns a dict."""
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context, compress
    d = synth.preset(config)
    Mr = m_tokens or d.tokens
    shapes = synth.linear_shapes(d)
    mats = {"qkv": (shapes["q"][0] + 2 * shapes["k"][0], d.hidden), "o": shapes["o"],
            "gate_up": (2 * d.intermediate, d.hidden), "down": shapes["down"]}
    if shapes_only:
        mats = {k: v for k, v in mats.items() if k in shapes_only}
    ctx = Context(synth.tiny(vocab=0, head_dim=64), max_tokens=64, max_seq=64)
    g = torch.Generator(device="cuda")
    g.manual_seed(7)
    res, tot_flops, tot_ms = {}, 0.0, 0.0
    for name, (N, K) in mats.items():
        W = torch.randn(N, K, device="cuda", generator=g) * 0.02
        q, sc = compress(ctx, W)
        del W
        Wp = M.packed(q, sc)
        X = torch.randn(Mr, K, device="cuda", generator=g).half()
        Y = torch.empty(Mr, N, device="cuda", dtype=torch.float16)
        dY = torch.randn(Mr, N, device="cuda", generator=g).half()
        dX = torch.empty(Mr, K, device="cuda")
        for mode in ("fwd", "dx"):
            def f():
                if mode == "fwd":
                    M.mebp_linear_fwd(ctx.handle, X, Wp, y_f16=Y)
                else:
                    M.mebp_linear_dx(ctx.handle, dY, Wp, dx=dX)
            for _ in range(warmup):
                f()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                f()
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / reps
            fl = 2.0 * Mr * N * K
            res[f"{name}_{mode}"] = {"M": Mr, "N": N if mode == "fwd" else K, "K": K if mode == "fwd" else N,
                                     "us": 1e3 * ms, "tflops": fl / ms / 1e9}
            tot_flops += fl
            tot_ms += ms
        del X, Y, dY, dX, q, sc, Wp
    ctx.sync()
    ctx.close()
    pk, src = peaks()
    tf = tot_flops / tot_ms / 1e9
    return {"workload": f"projection GEMMs of {d.name}, M = {Mr} tokens, 4-bit g64 weights, fp16 operands",
            "tflops": tf, "peak": pk["bf16_tflops"], "frac": tf / pk["bf16_tflops"],
            "peak_source": f"{src} burst dense bf16 GEMM rate (fp16 shares it)", "per_gemm": res}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=150)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", type=int, default=1, help="workload preset 0..4 (default 1)")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--gemm-bench", action="store_true",
                    help="time only the fused dequant-GEMMs at the config's projection shapes")
    ap.add_argument("--gemm-m", type=int, default=None, help="token count M for --gemm-bench")
    ap.add_argument("--gemm-shapes", default=None, help="comma list of qkv,o,gate_up,down for --gemm-bench")
    ap.add_argument("--table2", action="store_true",
                    help="decompression-overhead (Table 2) and sequence-length (Table 3) analogues")
    ap.add_argument("--gemma3", action="store_true",
                    help="Gemma-shaped configs (2, 4) with the Gemma3 block options on")
    ap.add_argument("--launch-list", action="store_true",
                    help="no timing: after the warm-up run one eager step inside the NVTX range "
                         "'mebp_step' (for ncu --nvtx --nvtx-include mebp_step/)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    d = synth.preset(args.config)
    if args.gemma3:
        if d.act != "gelu_tanh":
            ap.error("--gemma3 applies to the Gemma-shaped configs 2 and 4")
        d = gemma3_extras(d)

    if args.gemm_bench:
        out = gemm_bench(args.config, args.gemm_m, reps=args.steps, warmup=args.warmup,
                         shapes_only=args.gemm_shapes.split(",") if args.gemm_shapes else None)
        print(json.dumps(out), flush=True)
        return

    if args.launch_list:
        launch_list_step(args, d)
        return
    if args.table2:
        print(json.dumps(table2()), flush=True)
        return

    if args.impl == "reference":
        if rank != 0:
            return
        cores = os.cpu_count()
        vals = []
        for i in range(args.warmup + args.steps):
            v, desc = oracle_sample(d)
            if i >= args.warmup:
                vals.append(v)
        v = statistics.mean(vals)
        print(json.dumps({
            "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * d.tokens / v, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": workload_name(d), "config_index": args.config, "global_batch": d.batch,
                       "seq_len": d.seq, "parallelism": "host cores"},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": desc},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }), flush=True)
        return

    out = run_gpu(args, d, rank, world, local_rank)
    if out is None:
        return
    if world == 1:
        # second half of the metric: the fused dequant-GEMM alone at the largest workload's shapes
        out["fused_gemm_isolated"] = gemm_bench(4)
        out["adamw_isolated"] = adamw_bench(4)
    if world == 1 and not args.no_cpu_baseline:
        v, desc = oracle_sample(d)
        out["cpu_baseline"] = {"value": v, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                               "sample": desc}
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
