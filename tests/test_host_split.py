"""Host logic of the decode product's launch (CPU only): gemv_split, which
cuts a launch's 16-row blocks into one contiguous range per CTA with equal
shares of rows x columns, compiled from the library's own header with the
host compiler and checked for cover, order and balance."""
import os
import shutil
import subprocess
import tempfile

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_04048_gb300", "csrc")
CUDA_INCLUDE = "/usr/local/cuda/include"

HARNESS = r"""
#include <cstdio>
#include "rrq_internal.h"
// stdin: count grid, then rows cols per matrix; stdout: cta_begin[0..grid]
int main() {
  static rrq::GemvBatch p;
  int count = 0, grid = 0;
  if (std::scanf("%d %d", &count, &grid) != 2) return 1;
  p.count = count;
  int64_t blocks = 0;
  for (int i = 0; i < count; ++i) {
    long long r = 0, c = 0;
    if (std::scanf("%lld %lld", &r, &c) != 2) return 1;
    p.item[i].rows = r;
    p.item[i].cols = c;
    p.item[i].blk_begin = blocks;
    blocks += (r + rrq::kGemvRows - 1) / rrq::kGemvRows;
  }
  p.total_blocks = blocks;
  rrq::gemv_split(p, grid);
  for (int c = 0; c <= grid; ++c) std::printf("%lld\n", static_cast<long long>(p.cta_begin[c]));
  return 0;
}
"""


@pytest.fixture(scope="module")
def harness():
    gxx = shutil.which("g++")
    if gxx is None or not os.path.isdir(CUDA_INCLUDE):
        pytest.skip("needs g++ and the CUDA headers")
    d = tempfile.mkdtemp()
    src, exe = os.path.join(d, "split.cpp"), os.path.join(d, "split")
    with open(src, "w") as f:
        f.write(HARNESS)
    subprocess.run([gxx, "-std=c++17", "-O1", "-I", CSRC, "-I", CUDA_INCLUDE, src, "-o", exe], check=True)
    yield exe
    shutil.rmtree(d, ignore_errors=True)


def split(exe, shapes, grid):
    text = f"{len(shapes)} {grid}\n" + "".join(f"{r} {c}\n" for r, c in shapes)
    out = subprocess.run([exe], input=text, capture_output=True, text=True, check=True).stdout
    return [int(x) for x in out.split()]


def blocks_of(shapes):
    """(weights of each 16-row block) in launch order."""
    w = []
    for r, c in shapes:
        for b in range(0, r, 16):
            w.append(min(16, r - b) * c)
    return np.array(w, dtype=np.int64)


CASES = [
    ("qwen3_8b_layer", [(1024, 4096), (1024, 4096), (4096, 4096), (4096, 4096), (4096, 12288),
                        (12288, 4096), (12288, 4096)], (152, 304, 512)),
    ("tiny_mixed", [(1, 32), (3, 96), (17, 128), (33, 1056), (5, 57344)], (1, 2, 7, 12)),
    ("many_small", [(1 + (i * 7) % 39, 128 * (1 + i % 19)) for i in range(64)], (3, 152, 304)),
]


@pytest.mark.parametrize("name,shapes,grids", CASES, ids=[c[0] for c in CASES])
def test_split_covers_in_order_and_balances(harness, name, shapes, grids):
    w = blocks_of(shapes)
    total = int(w.sum())
    for grid in grids:
        grid = min(grid, len(w))
        cb = split(harness, shapes, grid)
        assert len(cb) == grid + 1
        assert cb[0] == 0 and cb[-1] == len(w)
        assert all(a <= b for a, b in zip(cb, cb[1:])), "ranges out of order"
        # every CTA's share is within one block of the equal share
        share = total / grid
        for c in range(grid):
            got = int(w[cb[c]:cb[c + 1]].sum())
            assert got <= share + w.max(), (grid, c, got, share)
        # the prefix boundaries sit where the running sum first reaches c/grid
        csum = np.concatenate([[0], np.cumsum(w)])
        for c in range(1, grid):
            if cb[c] < len(w):
                assert csum[cb[c]] * grid >= c * total
                assert cb[c] == 0 or csum[cb[c] - 1] * grid < c * total or cb[c] == cb[c - 1]
