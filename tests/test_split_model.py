"""The token-split rule of the dense scale gradient (host logic, no GPU).

sgrad_splits(tiles, clusters, M) in csrc/sq_internal.h picks how many token parts a
dense scale-gradient launch uses: with w(s) = ceil(tiles * s / clusters) / s, the launch's
length in units of one full-M tile per cluster, the largest part count s <= 8 (each part
>= 2048 tokens) whose w(s) is within 1 % of the smallest and no longer than w(1): more,
shorter parts keep the dY and X panels that a part's waves share in L2. Checked here by compiling
the header's inline function into a tiny host program and comparing it with the same
rule evaluated in Python, and on the shapes it is meant for.
"""
import math
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_04526_gb300", "csrc")
CUDA_INC = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")

PROGRAM = r"""
#include <cstdio>
#include "sq_internal.h"
int main() {
  long long t, c, m;
  while (std::scanf("%lld %lld %lld", &t, &c, &m) == 3)
    std::printf("%d\n", sqi::sgrad_splits(t, static_cast<int>(c), m));
  return 0;
}
"""


def _rule(tiles, clusters, M):
    top = max(1, min(8, M // 2048))
    w = {s: math.ceil(tiles * s / clusters) / s for s in range(1, top + 1)}
    limit = min(min(w.values()) * 1.01, w[1])
    return max(s for s in w if w[s] <= limit + 1e-9)


@pytest.fixture(scope="module")
def splits(tmp_path_factory):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None or not os.path.exists(os.path.join(CUDA_INC, "cuda.h")):
        pytest.skip("no host C++ compiler or CUDA headers")
    d = tmp_path_factory.mktemp("split_model")
    src, exe = d / "split_model.cpp", d / "split_model"
    src.write_text(PROGRAM)
    subprocess.run([cxx, "-std=c++17", "-O1", f"-I{CSRC}", f"-I{CUDA_INC}", str(src), "-o", str(exe)], check=True)

    def run(cases):
        out = subprocess.run([str(exe)], input="".join(f"{t} {c} {m}\n" for t, c, m in cases),
                             capture_output=True, text=True, check=True).stdout.split()
        return [int(x) for x in out]
    return run


def tiles_of(N, K):
    return math.ceil(N / 256) * math.ceil(K / 256)


def test_layer_shapes(splits):
    """The Llama-3-8B-shaped layer at 16 x 2048 tokens on 76 CTA pairs."""
    M, C = 32768, 76
    shapes = {"q/o": (4096, 4096), "k/v": (1024, 4096), "gate/up": (14336, 4096), "down": (4096, 14336)}
    got = splits([(tiles_of(N, K), C, M) for N, K in shapes.values()])
    assert got == [8, 7, 8, 8]


def test_few_tokens_never_split(splits):
    assert splits([(256, 76, 4095), (1, 76, 2048), (8, 76, 0)]) == [1, 1, 1]
    assert splits([(256, 76, 4096)]) == [2]                    # 4096 x 4096 MXFP4 at M = 4096


def test_matches_the_rule_everywhere(splits):
    cases = [(t, c, m) for t in (1, 7, 64, 75, 76, 77, 150, 256, 896, 3584, 10000)
             for c in (1, 16, 74, 76) for m in (0, 2047, 4096, 9000, 16384, 32768, 1 << 20)]
    assert splits(cases) == [_rule(*x) for x in cases]


def test_never_longer_than_unsplit(splits):
    cases = [(t, 76, 1 << 16) for t in range(1, 400)]
    for (t, c, m), s in zip(cases, splits(cases)):
        assert 1 <= s <= 8
        assert math.ceil(t * s / c) / s <= math.ceil(t / c) + 1e-12
