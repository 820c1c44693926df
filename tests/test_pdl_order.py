"""Source check of the programmatic-dependent-launch ordering the kernels rely on (no GPU).

A kernel may start once every CTA of its predecessor has triggered (griddepcontrol.launch_dependents).
Data a kernel reads before its own wait is only guaranteed complete if it was written before the
nearest preceding kernel that waits before it triggers.  The library keeps that simple: every
kernel waits before it triggers except the fused GEMMs (their early reads are the packed weights,
never written inside a call) and the attention backward's item kernels (their early reads are the
forward's q/k/v and lse and the o-projection's dO, all written before the dvec kernel that always
precedes them and waits first).  A kernel added to the early set, or dvec losing its order, breaks
that argument, so this test pins the set."""
import glob
import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2510_03425_gb300", "csrc")

EARLY_TRIGGER = {"dequant_gemm_kernel", "dequant_gemm_narrow", "dkdv_kernel", "dq_kernel", "bwd_split_kernel"}


def _kernels():
    """(file, kernel name, body) of every __global__ function in the CUDA sources."""
    out = []
    for f in sorted(glob.glob(os.path.join(CSRC, "*.cu"))):
        src = open(f).read()
        for m in re.finditer(r"__global__\s+void\s+(?:__launch_bounds__\([^)]*\)\s*)?(\w+)\s*\(", src):
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
            out.append((os.path.basename(f), m.group(1), src[i:j]))
    return out


def test_kernels_are_found():
    names = {k for _, k, _ in _kernels()}
    assert {"dvec_kernel", "fwd_kernel", "rmsnorm_fwd_kernel", "skinny_slab_kernel"} <= names
    assert EARLY_TRIGGER <= names


def test_only_the_listed_kernels_trigger_before_they_wait():
    early = set()
    for f, name, body in _kernels():
        w, launch = body.find("griddep_wait()"), body.find("griddep_launch()")
        assert launch >= 0, f"{f}:{name} never triggers its dependents"
        if w < 0 or launch < w:
            early.add(name)
    assert early == EARLY_TRIGGER, early ^ EARLY_TRIGGER


def test_the_attention_backward_items_wait_before_reading_dvec():
    """Before the wait, dvec may only appear behind the fetch lambda's with_dvec guard, and every
    fetch issued before the wait passes with_dvec = false."""
    src = open(os.path.join(CSRC, "attention.cu")).read()
    for fn in ("dkdv_run", "dq_run"):
        body = src[src.index(f"void {fn}("):]
        body = body[:body.index("\n}\n")]
        pre = body[:body.index("griddep_wait()")]
        for line in pre.splitlines():
            if "a.dvec[" in line:
                assert "with_dvec" in line, (fn, line)
        for call in re.findall(r"fetch\(([^;]*)\);", pre):
            assert call.replace(" ", "").endswith("false"), (fn, call)
        assert "a.dvec[" in body[body.index("griddep_wait()"):], fn
