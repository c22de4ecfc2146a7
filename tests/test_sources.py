"""Source-level checks of the CUDA path (no GPU): every kernel that can run
inside a captured hyperbatch graph waits for its predecessor before anything
else.  With programmatic edges a kernel's blocks start before the previous
kernel has finished; one that read first, or that returned without waiting,
could see unfinished results or let its successors overtake the chain."""
import os
import re

import pytest

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2601_01473_gb300", "csrc")
GRAPH_FILES = ["prepare.cu", "sample.cu", "dedup.cu", "scan.cu", "gather.cu", "gather_hbm.cu"]


def _kernel_bodies(text):
    """(name, first statement) of every __global__ function."""
    out = []
    for m in re.finditer(r"__global__", text):
        i = m.end()
        while True:  # skip __launch_bounds__(...) and find the parameter list
            p = text.index("(", i)
            if text[i:p].rstrip().endswith("__launch_bounds__"):
                i = text.index(")", p) + 1
                continue
            break
        name = re.findall(r"(\w+)\s*$", text[i:p])[0]
        depth, j = 0, p
        while True:
            depth += {"(": 1, ")": -1}.get(text[j], 0)
            if depth == 0:
                break
            j += 1
        brace = text.index("{", j)
        first = text[brace + 1:].lstrip().split(";", 1)[0]
        out.append((name, first.strip()))
    return out


@pytest.mark.parametrize("fname", GRAPH_FILES)
def test_every_kernel_waits_for_its_predecessor_first(fname):
    text = open(os.path.join(CSRC, fname)).read()
    kernels = _kernel_bodies(text)
    assert kernels, fname
    for name, first in kernels:
        assert first == "grid_dep_wait()", f"{fname}: {name} starts with {first!r}"


def test_the_check_sees_a_kernel_that_reads_first():
    text = ("__global__ void __launch_bounds__(256) k1(const int* s) {\n  grid_dep_wait();\n}\n"
            "template <int G>\n__global__ void k2(int* p, int n) {\n  if (p[0]) return;\n"
            "  grid_dep_wait();\n}\n")
    assert _kernel_bodies(text) == [("k1", "grid_dep_wait()"), ("k2", "if (p[0]) return")]
