"""Layout invariants of the streaming coefficient kernel's shared-memory stage
(host code only, no GPU): the row table the kernel is launched with is built
by make_stream_geom in pair_coeffs_stream.cuh; this test compiles a small
host program around it with nvcc and checks, for every G it serves
(4, 8, ..., 64), what the maskless row sweep relies on:
  * every row's staged columns land at Qt[i] + j, inside the stage, and no
    two rows or a row and a gap overlap;
  * column G of every row and every diagonal cell that is not staged fall in
    a gap (gaps hold +inf, so those reads weigh 0);
  * staged row starts are 16-byte aligned (bulk copies), and each row base
    falls in a different bank group (mod 32 words) from the previous three;
  * the expected byte count of a group is the bytes of its row copies plus
    the rewards.
Skipped where nvcc is not installed."""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_11368_gb300", "csrc")
TRI_FLOATS = 2620  # kTriFloats: the stage's triangle region

PROGRAM = r"""
#include <cstdio>
#include "pair_coeffs_stream.cuh"
int main() {
  for (int G = 4; G <= 64; G += 4) {
    pairk::StreamGeom g = pairk::make_stream_geom(G);
    std::printf("%d %u", G, g.group_bytes);
    for (int v = 0; v < 64; ++v) std::printf(" %d", g.Qt[v]);
    std::printf("\n");
  }
  return 0;
}
"""


def col0(i):
    return (i + 1) & ~3


@pytest.fixture(scope="module")
def tables(tmp_path_factory):
    nvcc = shutil.which("nvcc")
    if nvcc is None:
        pytest.skip("nvcc not installed")
    d = tmp_path_factory.mktemp("stream_layout")
    src = d / "layout.cu"
    src.write_text(PROGRAM)
    exe = d / "layout"
    subprocess.run([nvcc, "-std=c++17", "-I", CSRC, "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True, capture_output=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    rows = {}
    for line in out.splitlines():
        xs = [int(v) for v in line.split()]
        rows[xs[0]] = (xs[1], xs[2:])
    return rows


@pytest.mark.parametrize("G", list(range(4, 65, 4)))
def test_stream_layout_invariants(tables, G):
    group_bytes, Qt = tables[G]
    kind = np.zeros(TRI_FLOATS, np.int8)   # 0 unused, 1 row data, 2 gap
    # Rows: columns col0(i) .. G-1 at Qt[i] + j.
    tri = 0
    for i in range(G - 1):
        start = Qt[i] + col0(i)
        L = G - col0(i)
        assert start % 4 == 0 and L % 4 == 0 and L > 0
        assert 0 <= start and start + L <= TRI_FLOATS
        assert (kind[start:start + L] == 0).all(), "rows overlap"
        kind[start:start + L] = 1
        tri += L
    # Gaps: before each row, and 4 floats after row G-1 (which has no entries).
    for i in range(G):
        start = 0 if i == 0 else Qt[i - 1] + G
        D = Qt[i] + col0(i) if i <= G - 2 else Qt[i] + G
        assert D - start >= 4, "gap shorter than 4 floats"
        assert (kind[start:D] == 0).all(), "gap over row data"
        kind[start:D] = 2
        if i == G - 1:
            assert D + 4 <= TRI_FLOATS
            kind[D:D + 4] = 2
    for i in range(G):
        assert kind[Qt[i] + G] == 2, ("column G of row %d" % i)
        if not (i <= G - 2 and col0(i) <= i):
            assert kind[Qt[i] + i] == 2, ("unstaged diagonal of row %d" % i)
        else:
            assert kind[Qt[i] + i] == 1   # staged diagonal: overwritten with +inf per group
    # Bank groups of the row bases.
    res = [Qt[i] % 32 for i in range(G - 1)]
    for i in range(G - 1):
        assert res[i] not in res[max(0, i - 3):i], ("row base bank of row %d" % i)
    # Unused rows of the table point at row 0 (reads stay inside the stage).
    assert all(q == 0 for q in Qt[G:])
    assert group_bytes == 4 * (tri + G)
