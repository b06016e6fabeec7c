"""Host logic of the balanced tile lists (csrc/gs_plan.cu), compiled on its own with g++.

The tensor-core prefill kernels take their tiles from these lists, so a tile
missing or handed out twice would show up in the GPU parity tests; here the
list itself is pinned on the CPU: every tile exactly once, owners' ranges
contiguous, each owner's tiles longest first, the longest-first bound on the
largest load, and the fallback to the fixed stride beyond the list's size.
"""
import shutil
import subprocess
from pathlib import Path

import numpy as np
import pytest

CSRC = Path(__file__).resolve().parent.parent / "paper_2609_33977_gb300" / "csrc"

DRIVER = r"""
#include "gs_plan.cuh"
#include <cstdio>
int main() {
  int owners = 0, n = 0;
  if (std::scanf("%d %d", &owners, &n) != 2) return 2;
  std::vector<int32_t> cost(n);
  for (int i = 0; i < n; ++i) std::scanf("%d", &cost[i]);
  static gs::TileList L;
  gs::plan_tiles(cost, owners, L);
  std::printf("%d\n", L.on);
  if (L.on) {
    for (int b = 0; b <= owners; ++b) std::printf("%d ", (int)L.off[b]);
    std::printf("\n");
    for (int i = 0; i < n; ++i) std::printf("%d ", (int)L.order[i]);
    std::printf("\n");
  }
  return 0;
}
"""


@pytest.fixture(scope="module")
def planner(tmp_path_factory):
    gxx = shutil.which("g++")
    if not gxx:
        pytest.skip("g++ not available")
    d = tmp_path_factory.mktemp("plan")
    (d / "main.cpp").write_text(DRIVER)
    exe = d / "plan"
    subprocess.run([gxx, "-std=c++17", "-O2", "-x", "c++", str(CSRC / "gs_plan.cu"), "-x", "none", str(d / "main.cpp"),
                    f"-I{CSRC}", "-o", str(exe)], check=True, capture_output=True)

    def run(cost, owners):
        inp = f"{owners} {len(cost)}\n" + " ".join(str(int(c)) for c in cost) + "\n"
        out = subprocess.run([str(exe)], input=inp, capture_output=True, text=True, check=True).stdout.split("\n")
        on = int(out[0])
        if not on:
            return None
        off = np.array(out[1].split(), dtype=np.int64)
        order = np.array(out[2].split(), dtype=np.int64)
        return off, order
    return run


def loads(cost, off, order):
    cost = np.asarray(cost)
    return np.array([cost[order[off[b]:off[b + 1]]].sum() for b in range(len(off) - 1)])


def check_list(cost, owners, res):
    off, order = res
    cost = np.asarray(cost)
    assert off[0] == 0 and off[-1] == len(cost) and np.all(np.diff(off) >= 0)
    assert np.array_equal(np.sort(order), np.arange(len(cost)))          # every tile exactly once
    for b in range(owners):
        c = cost[order[off[b]:off[b + 1]]]
        assert np.all(np.diff(c) <= 0)                                   # longest first within an owner
    ld = loads(cost, off, order)
    opt_lb = max(cost.max(), -(-cost.sum() // owners))                    # no assignment does better
    assert ld.max() <= (4.0 / 3.0 - 1.0 / (3 * owners)) * max(opt_lb, 1) + 1e-9   # Graham's bound for longest-first
    return ld


def test_llama2_13b_block_at_128_tokens(planner):
    # single-CTA gathering tiles of one 13B block at T = 128: 32 down-projection windows of 54
    # chunks, then 302 windows of 20 (q/k/v/o 4 x 32, gate/up 2 x 87), over 152 CTAs
    cost = [54] * 32 + [20] * 302
    ld = check_list(cost, 152, planner(cost, 152))
    assert ld.max() == 60                    # the fixed stride gives 94 (54 + 20 + 20)
    stride = [sum(cost[t] for t in range(b, len(cost), 152)) for b in range(152)]
    assert max(stride) == 94


@pytest.mark.parametrize("seed", range(6))
def test_random_costs(planner, seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 2049))
    owners = int(rng.integers(1, 161))
    cost = rng.integers(1, 100, size=n)
    check_list(cost, owners, planner(cost, owners))


def test_equal_costs_spread_evenly(planner):
    cost = [20] * 432
    off, order = planner(cost, 76)
    counts = np.diff(off)
    assert counts.max() - counts.min() <= 1 and counts.sum() == 432


def test_fewer_tiles_than_owners(planner):
    cost = [7, 3, 9]
    off, order = planner(cost, 5)
    check_list(cost, 5, (off, order))
    assert np.array_equal(np.diff(off), [1, 1, 1, 0, 0])


def test_beyond_the_list_falls_back(planner):
    assert planner([1] * 2049, 76) is None          # more tiles than the list holds
    assert planner([1] * 10, 161) is None           # more owners than the list holds
    assert planner([1] * 2048, 160) is not None
