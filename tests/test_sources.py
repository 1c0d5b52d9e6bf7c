"""Static checks of the CUDA sources (no GPU, no compiler).

Every kernel is launched with programmatic dependent launch (the next kernel
may start while its predecessor drains), so each must begin by waiting for
the grids it depends on (pdl_prologue) before it touches memory.
"""
import os
import re

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2207_10731_gb300", "csrc")


def _kernels():
    for f in sorted(os.listdir(CSRC)):
        if not f.endswith((".cu", ".cuh")):
            continue
        src = open(os.path.join(CSRC, f)).read()
        for m in re.finditer(r"__global__", src):
            # the body opens at the first '{' after the parameter list closes
            j, depth, opened = m.end(), 0, False
            while True:
                c = src[j]
                if c == "(":
                    depth, opened = depth + 1, True
                elif c == ")":
                    depth -= 1
                elif c == "{" and depth == 0 and opened:
                    break
                j += 1
            names = re.findall(r"(\w+)\s*\(", src[m.end():j])
            yield f, names[-1] if names else "?", src[j + 1:j + 200].strip()


def test_every_kernel_waits_for_its_predecessor_first():
    kernels = list(_kernels())
    assert len(kernels) >= 15
    for f, name, body in kernels:
        assert body.startswith("pdl_prologue();"), f"{f}: {name} does not start with pdl_prologue()"

