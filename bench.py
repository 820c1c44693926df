"""Benchmark of one MeBP LoRA training step (Algorithm 1) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config C] [--impl gb300|reference]
                    [--per-block] [--min-memory] [--gemm-bench] [--table2] [--launch-list]

A step = embed -> checkpointed forward loop over all blocks -> LM-head cross-entropy
(forward + backward, vocabulary-chunked) -> reverse loop of block recompute + backward,
producing the loss and every LoRA gradient (mebp_lora_step).  The default workload is the
largest preset, the Gemma3-4B-shaped model (34 blocks, vocab 262144, batch 8 x seq 2048, LoRA
r32 on all seven linears, 4-bit group-64 base weights).  Prints one JSON line (rank 0).

--impl reference times the CPU oracle (plain numpy fp64) on the host cores, each step one
bounded sample of the same workload (one block's forward + recompute + backward on part of a
sequence and an LM-head sample), extrapolated to the step.
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
def blas_threads() -> int:
    """Threads the oracle's numpy BLAS uses (threadpoolctl when present, else the environment or
    the core count)."""
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 0) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(k, "").isdigit():
            return int(os.environ[k])
    return os.cpu_count() or 1


class OracleSample:
    """The oracle (numpy fp64) on a bounded sample of one training step, extrapolated to the step.

    Sample: block 0 decompressed (LazyLoadAndDecompressWeights), its forward, then the recompute +
    backward (block_objective) on the first `block_tokens` tokens of one sequence; and the LM head
    (final norm + logits + CE + dE/dh) on `lm_tokens` tokens against a `lm_rows`-row slice of the
    decompressed vocabulary.  Extrapolation is linear in what each part scales with: a block's
    decompression x 2 L (forward and recompute), its forward + backward x L x tokens / block_tokens,
    the embedding's decompression x V / lm_rows, the LM head x tokens / lm_tokens x V / lm_rows.
    Attention's quadratic term is extrapolated
    linearly too, which slightly flatters the CPU.  Compression (done once when a model is loaded)
    is outside the timed sample.  full=True times the whole Algorithm 1 step instead (--cpu-full-step;
    about 40 s on 8 cores for the Qwen2.5-0.5B shape, hours for the larger ones)."""

    def __init__(self, d, block_tokens: int = 256, lm_tokens: int = 32, lm_rows: int = 16384, full: bool = False):
        from oracle import model as OM
        from oracle import quant
        self.d = d
        self.OM = OM
        self.full = full and d.vocab > 0
        if self.full:
            self.blocks = [synth.block_weights(d, i) for i in range(d.n_layers)]
            self.E, self.gf = synth.embedding(d)
            self.pm = OM.PackedModel.compress(self.blocks, self.E, self.gf)
            self.loras = [synth.lora_weights(d, i) for i in range(d.n_layers)]
            self.ids = synth.token_ids(d)
            self.desc = (f"oracle (numpy fp64) full Algorithm 1 step: {d.n_layers} blocks, {d.tokens} tokens, "
                         f"vocab {d.vocab} (no extrapolation)")
            return
        bt = min(block_tokens, d.seq)
        self.bt = bt
        d1 = d.with_(batch=1, seq=bt)
        self.d1 = d1
        self.pm = OM.PackedModel.compress([synth.block_weights(d, 0)])
        self.L = OM.lora64(synth.lora_weights(d, 0))
        self.x = synth.hidden_input(d)[:bt].astype(np.float64)
        self.G = synth.upstream_grad(d)[:bt].astype(np.float64)
        self.lm = None
        if d.vocab:
            rows = min(lm_rows, d.vocab)
            E, gf = synth.embedding(d, rows=rows)
            self.qE = quant.compress(E)
            self.gf = gf.astype(np.float64)
            rng = np.random.default_rng(3)
            self.h = rng.standard_normal((lm_tokens, d.hidden))
            self.tg = rng.integers(0, rows, lm_tokens).astype(np.int64)
            self.lm = (rows, lm_tokens)
        rows = self.lm[0] if self.lm else 0
        self.desc = (f"oracle (numpy fp64): block 0 decompressed (x{2 * d.n_layers}: every block, forward and "
                     f"recompute) and its forward + recompute + backward on {bt} of the {d.seq} tokens of one "
                     f"sequence (x{d.n_layers} blocks x{d.tokens // bt}); the embedding's first {rows} rows "
                     f"decompressed (x{d.vocab / max(1, rows):.0f}) and the LM head (final norm, logits, CE, dE/dh) "
                     f"on {lm_tokens} tokens against them (x{d.tokens // lm_tokens} x{d.vocab / max(1, rows):.0f}); "
                     f"extrapolated linearly to the step")

    def run(self):
        """Returns (seconds the sample took, seconds of the whole step it stands for)."""
        OM, d = self.OM, self.d
        if self.full:
            t0 = time.perf_counter()
            OM.mebp_backpropagation(self.pm, self.loras, self.ids, d)
            t = time.perf_counter() - t0
            return t, t
        from oracle import quant
        t0 = time.perf_counter()
        Wd = self.pm.decompress_block(0)            # once per block and pass: x L x 2 (forward, recompute)
        t1 = time.perf_counter()
        OM.block_forward(self.x, Wd, self.L, self.d1)
        OM.block_objective(self.x, Wd, self.L, self.G, self.d1)  # per token: x L x tokens / bt
        t2 = time.perf_counter()
        t_dec, t_blk = t1 - t0, t2 - t1
        t_dec_e = t_ce = 0.0
        if self.lm:
            t3 = time.perf_counter()
            Ed = quant.dequant(*self.qE)            # once per step: x V / rows
            t4 = time.perf_counter()
            OM.lm_head_ce(self.h, self.gf, Ed, self.tg, d.eps)  # per token and row: x tokens / lm_tokens x V / rows
            t5 = time.perf_counter()
            t_dec_e, t_ce = t4 - t3, t5 - t4
        sample = t_dec + t_blk + t_dec_e + t_ce
        full = d.n_layers * (2 * t_dec + t_blk * d.tokens / self.bt)
        if self.lm:
            vr = d.vocab / self.lm[0]
            full += t_dec_e * vr + t_ce * (d.tokens / self.lm[1]) * vr
        return sample, full


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


GEMM_SOURCES = ("gemm.cu", "gemm_s.cu", "dequant.cuh", "common.cuh")
TRAFFIC_PROFILE = os.path.join(ROOT, "profiles", "dequant_gemm_gemma4b_step_traffic.md")


def gemm_sources_sha() -> str:
    import hashlib
    h = hashlib.sha256()
    for f in GEMM_SOURCES:
        with open(os.path.join(ROOT, "paper_2510_03425_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def gemm_traffic(config: int):
    """DRAM bytes per fused-GEMM launch of one step from the committed ncu summary, or None when
    the summary is for another workload or the kernel sources changed since it was taken."""
    import re
    try:
        with open(TRAFFIC_PROFILE) as f:
            txt = f.read()
    except OSError:
        return None, "no ncu summary"
    kv = dict(re.findall(r"^([a-z0-9_]+):\s*(\S+)\s*$", txt, flags=re.M))
    if kv.get("workload_config") != str(config):
        return None, "ncu summary is for another workload"
    if kv.get("kernel_sources_sha256") != gemm_sources_sha():
        return None, "kernel changed since the ncu capture"
    return float(kv["traffic_per_launch_bytes"]), os.path.relpath(TRAFFIC_PROFILE, ROOT)


def make_step(M, ctx, mstruct, ls, ids, loss, st):
    def step():
        M.mebp_lora_step(ctx.handle, mstruct, ls.lora_array(), ids, loss, ls.grads_array(), False, st)
    return step


def time_steps(step, n, st):
    import torch
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(n):
        step()
    e1.record(st)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / 1e3


def model_bytes(model, ls):
    pw = sum(t.numel() * t.element_size() for b in model.blocks for lin in (b.qkv, b.o, b.gate_up, b.down)
             for t in (lin.qpack, lin.scales))
    pw += model.embed.qpack.numel() + model.embed.scales.numel() * 2
    return pw, 2 * 4 * ls.n  # packed weights (+ scales); LoRA masters + gradients (fp32)


def max_over_ranks(x: float, dist, device=None) -> float:
    """The largest of every rank's x (a job's time is its slowest rank's); x itself when there is
    no process group.  NCCL reduces a device tensor, gloo a host one."""
    if dist is None:
        return x
    import torch
    dev = device if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank: int, steps: int, world: int, seconds: float) -> float:
    """Whole-job throughput: the tokens every rank processed over the slowest rank's time."""
    return world * tokens_per_rank * steps / seconds


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
    ctx = Context(d, device=local_rank, min_memory=args.min_memory)
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
    step = make_step(M, ctx, mstruct, ls, ids, loss, st)

    gpu_index = local_rank
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis and vis.split(",")[local_rank].strip().isdigit():
        gpu_index = int(vis.split(",")[local_rank])
    torch.cuda.reset_peak_memory_stats(device)
    for _ in range(args.warmup):
        step()
    ctx.sync()
    free0, total = torch.cuda.mem_get_info(device)
    # ---- timed region: K steps, inputs resident in HBM
    clocks = ClockSampler(gpu_index)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    n0 = M.mebp_kernel_launches()
    t = time_steps(step, args.steps, st)
    launches = M.mebp_kernel_launches() - n0
    if dist:
        dist.barrier()
    clk = clocks.stop()
    ctx.sync()
    free1, _ = torch.cuda.mem_get_info(device)
    t = max_over_ranks(t, dist, device)
    value = job_tokens_per_s(d.tokens, args.steps, world, t)

    # ---- per-kernel CUDA events over K more steps (run eagerly: the events order each launch on
    # its stream), the fused GEMMs' union of busy intervals, and the step's wall time meanwhile
    kp = max(3, args.steps // 4)
    M.mebp_profile_begin(ctx.handle)
    t_prof = time_steps(step, kp, st)
    prof = M.mebp_profile_end(ctx.handle)
    kstats = M.mebp_profile_kernels(ctx.handle)

    # ---- end to end through the public API: ids host->device, step, loss device->host
    ctx.sync()
    h2d = ids_host.numel() * ids_host.element_size()
    d2h = loss.numel() * loss.element_size()

    def e2e_step():
        ids.copy_(ids_host, non_blocking=True)
        step()
        loss_host.copy_(loss, non_blocking=True)
    te = max_over_ranks(time_steps(e2e_step, args.steps, st), dist, device)
    ctx.sync()
    peak_torch = torch.cuda.max_memory_allocated(device)
    ws = M.mebp_workspace_bytes(ctx.handle)
    breakdown, nsets = M.mebp_workspace_breakdown(ctx.handle)
    pw_bytes, lora_bytes = model_bytes(model, ls)

    mm = None
    kstats_serial, kp_serial = None, 0
    if rank == 0 and world == 1 and not args.min_memory and args.compare_min_memory:
        # the paper's bound: one set of block intermediates (no recompute / backward overlap)
        c2 = Context(d, device=local_rank, min_memory=True)
        step2 = make_step(M, c2, mstruct, ls, ids, loss, st)
        for _ in range(3):
            step2()
        c2.sync()
        n2 = max(3, args.steps // 2)
        t2 = time_steps(step2, n2, st)
        c2.sync()
        ws2 = M.mebp_workspace_bytes(c2.handle)
        mm = {"workspace_bytes": ws2, "peak_device_bytes": peak_torch + ws2,
              "workspace": M.mebp_workspace_breakdown(c2.handle)[0], "ms_per_step": 1e3 * t2 / n2,
              "tokens_per_s": d.tokens * n2 / t2, "slowdown": (t2 / n2) / (t / args.steps)}
        # one stream, nothing concurrent: per-kernel event times free of interference
        kp_serial = 3
        M.mebp_profile_begin(c2.handle)
        time_steps(step2, kp_serial, st)
        M.mebp_profile_end(c2.handle)
        kstats_serial = M.mebp_profile_kernels(c2.handle)
        c2.close()

    if rank != 0:
        ctx.close()
        if dist:
            dist.destroy_process_group()
        return None
    pk, src = peaks()
    sustained = t > 1.0  # the GEMMs run inside a seconds-long loop of steps
    peak = pk["bf16_tflops_sustained"] if sustained else pk["bf16_tflops"]
    achieved = prof.gemm_flops / (prof.gemm_ms / 1e3) / 1e12 if prof.gemm_ms > 0 else None
    busy_share = (prof.gemm_busy_ms / 1e3) / t_prof if t_prof > 0 else None
    assert busy_share is None or busy_share <= 1.0 + 1e-6, busy_share
    traffic, traffic_src = gemm_traffic(args.config) if not (args.gemma3 or args.min_memory) else (None, "n/a")
    ks_src, ks_n = (kstats_serial, kp_serial) if kstats_serial else (kstats, kp)
    tot_ms = sum(v["ms"] for v in ks_src.values()) or 1.0
    kernels = {"how": ("CUDA events around every launch of " + str(ks_n) + " eager steps on one stream "
                       "(min_memory context: nothing runs concurrently); bytes and flops algorithmic"
                       if kstats_serial else
                       "CUDA events around every launch of " + str(ks_n) + " eager steps (three streams: launches "
                       "overlap, times include interference)")}
    for name, v in sorted(ks_src.items(), key=lambda kv: -kv[1]["ms"]):
        e = {"launches_per_step": v["launches"] / ks_n, "ms_per_step": v["ms"] / ks_n,
             "share_of_kernel_time": v["ms"] / tot_ms}
        if v["bytes"] and v["ms"]:
            e["gbs"] = v["bytes"] / (v["ms"] / 1e3) / 1e9
            e["hbm_frac"] = e["gbs"] / pk["hbm_gbs"]
        if v["flops"] and v["ms"]:
            e["tflops"] = v["flops"] / (v["ms"] / 1e3) / 1e12
        kernels[name] = e
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * t / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": workload_name(d), "config_index": args.config, "global_batch": world * d.batch,
                   "seq_len": d.seq, "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "l2": f"inputs larger than L2: {pw_bytes / 2**20:.0f} MB of packed weights are streamed every "
                         "step (no flush needed)"},
        "roofline": {"kernel": "dequant_gemm_kernel (fused 4-bit dequant GEMM, tcgen05), every launch of the step",
                     "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": (achieved / peak) if achieved else None, "traffic": traffic,
                     "algorithmic_bytes": prof.gemm_bytes / max(prof.gemm_launches, 1),
                     "traffic_source": traffic_src,
                     "peak_source": f"{src} {'sustained' if sustained else 'burst'} dense bf16 GEMM rate "
                                    "(MEASURED_PEAKS.json); fp16 and bf16 share the kind::f16 rate (nominal ratio 1)",
                     "how": f"CUDA events on the launching stream around every fused-GEMM launch of {kp} eager "
                            "steps; achieved = sum of algorithmic flops / sum of launch durations",
                     "launches_per_step": prof.gemm_launches / kp,
                     "busy_share_of_step": busy_share,
                     "fwd_tflops": prof.fwd_flops / max(prof.fwd_ms, 1e-9) / 1e9,
                     "dx_tflops": prof.dx_flops / max(prof.dx_ms, 1e-9) / 1e9},
        "kernels": kernels,
        "memory": {"peak_device_bytes": peak_torch + ws, "torch_peak_allocated_bytes": peak_torch,
                   "library_workspace_bytes": ws, "workspace": breakdown, "intermediate_sets": nsets,
                   "packed_weights_bytes": pw_bytes, "lora_masters_and_grads_bytes": lora_bytes,
                   "device_used_bytes": total - free0,
                   "step_allocates_nothing": free0 == free1,
                   **({"min_memory": mm} if mm else {})},
        "e2e": {"value": job_tokens_per_s(d.tokens, args.steps, world, te), "unit": "tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches),
        "clocks": clk,
    }
    ctx.close()
    if dist:
        dist.destroy_process_group()
    return out


def per_block(args, d, reps: int = 3):
    """Analogue of the paper's Fig. 2 (per-layer time and memory): one eager step through the
    public entry points, phase by phase (embedding, forward_i of every block, the LM head + CE,
    backward_i of every block in reverse), each phase bracketed by CUDA events on the stream and
    an NVTX range (emb, f_i, lm, b_i).  Memory per phase is the working set the phase touches
    beyond the resident weights, LoRA state and checkpoints, from the workspace breakdown."""
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context, LoraSet
    device = torch.device("cuda", 0)
    ctx = Context(d, device=0)
    model = build_model(ctx, d, device)
    ls = LoraSet([synth.lora_weights(d, i) for i in range(d.n_layers)], device=device)
    ids = torch.from_numpy(synth.token_ids(d)).to(device)
    tg = torch.cat([ids[:, 1:], torch.full((d.batch, 1), -1, dtype=ids.dtype, device=device)], 1).reshape(-1)
    T, D, L = d.tokens, d.hidden, d.n_layers
    ck = torch.empty((L + 1, T, D), device=device)
    dy = torch.empty((T, D), device=device)
    dx = torch.empty((T, D), device=device)
    loss = torch.zeros(1, device=device)
    st = torch.cuda.Stream(device)
    torch.cuda.set_stream(st)
    E = model.embed.struct()
    blk = [b.struct() for b in model.blocks]
    lor = [ls.layer(i) for i in range(L)]
    grd = [ls.layer_grads(i) for i in range(L)]
    names = ["emb"] + [f"f_{i}" for i in range(L)] + ["lm"] + [f"b_{i}" for i in reversed(range(L))]
    times = {n: [] for n in names}
    for rep in range(reps + 1):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)]
        k = 0
        ev[0].record(st)

        def mark(name):
            nonlocal k
            torch.cuda.nvtx.range_pop()
            k += 1
            ev[k].record(st)
        torch.cuda.nvtx.range_push("emb")
        M.mebp_embed(ctx.handle, E, ids.reshape(-1), ck[0], stream=st)
        mark("emb")
        for i in range(L):
            torch.cuda.nvtx.range_push(f"f_{i}")
            M.mebp_block_recompute_fwd(ctx.handle, i, blk[i], lor[i], ck[i], ck[i + 1], d.batch, d.seq, False, st)
            mark(f"f_{i}")
        torch.cuda.nvtx.range_push("lm")
        M.mebp_lmhead_ce_fwd_bwd(ctx.handle, E, model.final_norm, ck[L], tg, loss, dy, stream=st)
        mark("lm")
        for i in reversed(range(L)):
            torch.cuda.nvtx.range_push(f"b_{i}")
            M.mebp_block_bwd(ctx.handle, i, blk[i], lor[i], ck[i], dy, dx, grd[i], d.batch, d.seq, False, st)
            mark(f"b_{i}")
            dy, dx = dx, dy
        torch.cuda.synchronize()
        ctx.sync(st)
        if rep == 0:
            continue  # warm-up
        for j, n in enumerate(names):
            times[n].append(ev[j].elapsed_time(ev[j + 1]))
    br, nsets = M.mebp_workspace_breakdown(ctx.handle)
    act = T * D * 4
    fwd_set = br["forward_sets"] / nsets
    mem = {"emb": act, "lm": br["lm_head"] + 2 * act}
    for i in range(L):
        mem[f"f_{i}"] = fwd_set + 2 * act
        mem[f"b_{i}"] = fwd_set + br["backward"] + br["attention_split"] + 3 * act
    pw, lb = model_bytes(model, ls)
    ms = {n: statistics.median(v) for n, v in times.items()}
    f_mean = statistics.mean(ms[f"f_{i}"] for i in range(L))
    b_mean = statistics.mean(ms[f"b_{i}"] for i in range(L))
    out = {"per_block": workload_name(d), "reps": reps, "ms": ms, "working_set_bytes": mem,
           "resident_bytes": {"packed_weights": pw, "lora_masters_and_grads": lb,
                              "checkpoints": br["checkpoints"], "lora_shadows": br["lora_shadows"]},
           "summary": {"forward_block_ms": f_mean, "backward_block_ms": b_mean,
                       "backward_over_forward_time": b_mean / f_mean,
                       "backward_over_forward_memory": mem["b_0"] / mem["f_0"],
                       "lm_head_ms": ms["lm"], "lm_head_over_backward_block": ms["lm"] / b_mean,
                       "lm_head_working_set_over_backward_block": mem["lm"] / mem["b_0"],
                       "step_ms": sum(ms.values())}}
    ctx.close()
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


def block_only(args, d):
    """One decoder block of the workload (its dims and token count, one layer, no LM head):
    warm-up, then one eager forward_i + backward_i through the public entry points inside the
    NVTX range 'mebp_block'.  A few GB on the device at the Gemma3-4B shape, for full-set
    profiler captures of single kernels at the workload's size."""
    import torch

    from paper_2510_03425_gb300 import mebp as M
    from paper_2510_03425_gb300.model import Context, DeviceBlock, LoraSet
    d1 = d.with_(n_layers=1, vocab=0)
    device = torch.device("cuda", 0)
    ctx = Context(d1, device=0)
    W = synth.torch_block_weights(d1, 0, device=device)
    blk = DeviceBlock(ctx, W)
    del W
    ls = LoraSet([synth.lora_weights(d1, 0)], device=device)
    g = torch.Generator(device=device)
    g.manual_seed(2)
    x = torch.randn(d1.tokens, d1.hidden, device=device, generator=g)
    dy = torch.randn(d1.tokens, d1.hidden, device=device, generator=g)
    y, dx = torch.empty_like(x), torch.empty_like(x)
    st = torch.cuda.Stream(device)
    torch.cuda.set_stream(st)
    bw = blk.struct()

    def run():
        M.mebp_block_recompute_fwd(ctx.handle, 0, bw, ls.layer(0), x, y, d1.batch, d1.seq, False, st)
        M.mebp_block_bwd(ctx.handle, 0, bw, ls.layer(0), x, dy, dx, ls.layer_grads(0), d1.batch, d1.seq, False, st)
    for _ in range(args.warmup):
        run()
    ctx.sync(st)
    n0 = M.mebp_kernel_launches()
    torch.cuda.nvtx.range_push("mebp_block")
    run()
    torch.cuda.nvtx.range_pop()
    ctx.sync(st)
    print(json.dumps({"block_only": workload_name(d1), "kernels": M.mebp_kernel_launches() - n0}), flush=True)
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
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", type=int, default=4,
                    help="workload preset 0..4 (default 4: the Gemma3-4B-shaped full step, the largest)")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-full-step", action="store_true",
                    help="the CPU oracle times the whole step instead of a bounded sample (small configs only)")
    ap.add_argument("--no-extras", action="store_true",
                    help="only the step measurement (no isolated GEMM / AdamW figures, no min-memory comparison)")
    ap.add_argument("--min-memory", action="store_true",
                    help="run the step with one set of block intermediates (the paper's memory bound)")
    ap.add_argument("--gemm-bench", action="store_true",
                    help="time only the fused dequant-GEMMs at the config's projection shapes")
    ap.add_argument("--gemm-m", type=int, default=None, help="token count M for --gemm-bench")
    ap.add_argument("--gemm-shapes", default=None, help="comma list of qkv,o,gate_up,down for --gemm-bench")
    ap.add_argument("--table2", action="store_true",
                    help="decompression-overhead (Table 2) and sequence-length (Table 3) analogues")
    ap.add_argument("--per-block", action="store_true",
                    help="Fig. 2 analogue: per-phase time (CUDA events, NVTX emb / f_i / lm / b_i) and memory")
    ap.add_argument("--gemma3", action="store_true",
                    help="Gemma-shaped configs (2, 4) with the Gemma3 block options on")
    ap.add_argument("--block-only", action="store_true",
                    help="no timing: one decoder block of the workload (one layer, no LM head) run eagerly inside "
                         "the NVTX range 'mebp_block' after the warm-up (for single-kernel profiler captures)")
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
    args.compare_min_memory = not args.no_extras

    if args.gemm_bench:
        out = gemm_bench(args.config, args.gemm_m, reps=args.steps, warmup=args.warmup,
                         shapes_only=args.gemm_shapes.split(",") if args.gemm_shapes else None)
        print(json.dumps(out), flush=True)
        return

    if args.launch_list:
        launch_list_step(args, d)
        return
    if args.block_only:
        block_only(args, d)
        return
    if args.table2:
        print(json.dumps(table2()), flush=True)
        return
    if args.per_block:
        print(json.dumps(per_block(args, d)), flush=True)
        return

    if d.vocab == 0:  # a single block without a vocabulary: parity workload of the GPU tests
        raise SystemExit(f"preset {args.config} ({workload_name(d)}) has no vocabulary and no training step to "
                         "time: it is the single-block parity case of tests/test_gpu_block.py (--block-only and "
                         "--gemm-bench take it)")

    if args.impl == "reference":
        # the CPU oracle as it stands, on the host cores: each step one bounded sample of the
        # workload, its throughput extrapolated to the whole step (see OracleSample)
        if rank != 0:
            return
        smp = OracleSample(d, full=args.cpu_full_step)
        samples, fulls = [], []
        for i in range(args.warmup + args.steps):
            ts, tf = smp.run()
            if i >= args.warmup:
                samples.append(ts)
                fulls.append(tf)
        tf = statistics.mean(fulls)
        v = d.tokens / tf
        cores = blas_threads()
        print(json.dumps({
            "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(samples),
            "extrapolated_ms_per_full_step": 1e3 * tf, "extrapolated": not smp.full,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": workload_name(d), "config_index": args.config, "global_batch": d.batch,
                       "seq_len": d.seq, "parallelism": "single GPU",
                       "l2": "n/a (host cores; each step is one bounded sample of the workload)"},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": smp.desc},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }), flush=True)
        return

    out = run_gpu(args, d, rank, world, local_rank)
    if out is None:
        return
    if world == 1 and not args.no_extras:
        # second half of the metric: the fused dequant-GEMM alone at the largest workload's shapes
        out["fused_gemm_isolated"] = gemm_bench(4)
        out["adamw_isolated"] = adamw_bench(4)
    if world == 1 and not args.no_cpu_baseline:
        smp = OracleSample(d, full=args.cpu_full_step)
        ts, tf = smp.run()
        out["cpu_baseline"] = {"value": d.tokens / tf, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle",
                               "sample": smp.desc, "sample_seconds": ts, "extrapolated": not smp.full}
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
