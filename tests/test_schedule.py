"""Host launch policy (csrc/mc_schedule.h): vocabulary splits per row block.

The header is plain C++; a tiny harness compiled here with the host compiler
calls `choose_splits` on a grid of launch shapes. Checked: the count lies in
[1, min(kMaxSplits, n_tiles)], honours the L2 budget for the wave's hidden
rows whenever some count can, and is the fewest splits whose critical path in
tiles, waves(s) x ceil(n_tiles / s), is within kPathSlack of the best allowed
count; plus the counts the configured workloads get.
"""

import itertools
import math
import os
import shutil
import subprocess

import pytest

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2606_04847_gb300", "csrc")

HARNESS = r"""
#include <cstdio>
#include "mc_schedule.h"
int main() {
  using namespace mc::sched;
  std::printf("%.17g %.17g %d\n", kWaveRowBytes, kPathSlack, kMaxSplits);
  long long m; int n, conc, rb, d;
  while (std::scanf("%lld %d %d %d %d", &m, &n, &conc, &rb, &d) == 5)
    std::printf("%d\n", choose_splits(m, n, conc, rb, d));
  return 0;
}
"""


@pytest.fixture(scope="module")
def splits(tmp_path_factory):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    d = tmp_path_factory.mktemp("sched")
    src, exe = d / "h.cpp", d / "h"
    src.write_text(HARNESS)
    subprocess.run([cxx, "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True)

    def run(shapes):
        inp = "".join(f"{m} {n} {c} {rb} {dd}\n" for m, n, c, rb, dd in shapes)
        out = subprocess.run([str(exe)], input=inp, capture_output=True, text=True, check=True).stdout.split()
        budget, slack, max_splits = float(out[0]), float(out[1]), int(out[2])
        return (budget, slack, max_splits), [int(v) for v in out[3:]]

    return run


def _path(m, n, conc, s):
    return math.ceil(m * s / conc) * math.ceil(n / s)


def test_split_rule_over_a_grid_of_shapes(splits):
    shapes = list(itertools.product([1, 2, 7, 19, 60, 128, 327, 501, 561, 2326, 5000],
                                    [1, 2, 16, 17, 243, 594, 970, 4096],
                                    [152, 148, 76], [128, 256], [64, 512, 4096, 5120, 8192]))
    (budget, slack, max_splits), got = splits(shapes)
    assert len(got) == len(shapes)
    for (m, n, conc, rb, d), s in zip(shapes, got):
        hi = min(max_splits, n)
        assert 1 <= s <= hi, (m, n, conc, rb, d, s)
        lo = max(1, math.ceil(conc * rb * d * 2.0 / budget))
        if lo <= hi:
            assert s >= lo, "the wave's hidden rows exceed the L2 budget"
        else:
            assert s == hi
            continue
        best = min(_path(m, n, conc, t) for t in range(lo, hi + 1))
        assert _path(m, n, conc, s) <= best * slack
        assert all(_path(m, n, conc, t) > best * slack for t in range(lo, s)), "not the fewest splits"


def test_splits_of_the_configured_workloads(splits):
    # (row blocks of 256, vocabulary tiles of 256, CTAs, rows per block, d)
    cases = {
        "9B fwd+bwd forward (128,236 tokens)": ((501, 970, 152, 256, 4096), 6),
        "9B fwd+bwd dZ (83,586 kept tokens)": ((327, 970, 152, 256, 4096), 6),
        "9B forward (143,463 tokens)": ((561, 970, 152, 256, 4096), 7),
        "27B forward (595,356 tokens)": ((2326, 970, 152, 256, 5120), 5),
        "mid forward (32,768 tokens, V = 151,936)": ((128, 594, 152, 256, 4096), 7),
        "one of 4 vocabulary slices (62,080 rows)": ((501, 243, 152, 256, 4096), 6),
    }
    _, got = splits([shape for shape, _ in cases.values()])
    for (name, (shape, want)), s in zip(cases.items(), got):
        assert s == want, f"{name}: {s} splits, expected {want}"
