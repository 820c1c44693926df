"""Source check of the programmatic-dependent-launch ordering the kernels rely on (no GPU).

A kernel may start once every CTA of its predecessor has triggered (griddepcontrol.launch_dependents).
Data a kernel reads before its own wait is only guaranteed complete if it was written before the
nearest preceding kernel that waits before it triggers.  The library keeps that simple: every
kernel waits before it triggers except the fused GEMMs, whose early reads are the packed weights
(never written inside a call).  A kernel added to the early set breaks that argument, so this
test pins the set, and checks that the tcgen05 attention kernels (whose operands come from the
kernel right before) issue no load before their wait."""
import glob
import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2510_03425_gb300", "csrc")

EARLY_TRIGGER = {"dequant_gemm_kernel", "dequant_gemm_narrow"}


def _bodies(src, pattern):
    out = []
    for m in re.finditer(pattern, src):
        i = src.index("{", m.end())
        depth, j = 0, i
        while True:
            if src[j] == "{":
                depth += 1
            elif src[j] == "}":
                depth -= 1
                if depth == 0:
                    break
            j += 1
        out.append((m.group(1), src[i:j]))
    return out


def _kernels():
    """(file, kernel name, body) of every __global__ function in the CUDA sources, with calls to
    the file's __device__ *_body functions replaced by those functions' bodies."""
    out = []
    for f in sorted(glob.glob(os.path.join(CSRC, "*.cu"))):
        src = open(f).read()
        helpers = dict(_bodies(src, r"__device__\s+__forceinline__\s+void\s+(\w+_body)\s*\("))
        for name, body in _bodies(src, r"__global__\s+void\s+(?:__launch_bounds__\([^)]*\)\s*)?(\w+)\s*\("):
            for h, hb in helpers.items():
                body = re.sub(h + r"\s*<[^;]*;", lambda _m, hb=hb: hb, body)
            out.append((os.path.basename(f), name, body))
    return out


def test_kernels_are_found():
    names = {k for _, k, _ in _kernels()}
    assert {"dvec_kernel", "fwd_tc_kernel", "dkdv_tc_kernel", "dq_tc_kernel", "bwd_split_tc_kernel",
            "rmsnorm_fwd_kernel", "skinny_slab_kernel", "skinny_tc_kernel"} <= names
    assert EARLY_TRIGGER <= names


def test_only_the_listed_kernels_trigger_before_they_wait():
    early = set()
    for f, name, body in _kernels():
        w, launch = body.find("griddep_wait()"), body.find("griddep_launch()")
        assert launch >= 0, f"{f}:{name} never triggers its dependents"
        if w < 0 or launch < w:
            early.add(name)
    assert early == EARLY_TRIGGER, early ^ EARLY_TRIGGER


def test_tensor_core_attention_loads_nothing_before_its_wait():
    """q, k, v (RoPE right before), dO and dvec (the kernel right before) are read only after the
    kernel's griddep_wait: before it, only barrier set-up and the TMEM allocation."""
    for f, name, body in _kernels():
        if name not in ("fwd_tc_kernel", "dkdv_tc_kernel", "dq_tc_kernel", "bwd_split_tc_kernel", "skinny_tc_kernel"):
            continue
        pre = body[:body.index("griddep_wait()")]
        for token in ("tma_load", "lse[", "dvec[", "__ldg", "ld_dsmem"):
            assert token not in pre, (f, name, token)
