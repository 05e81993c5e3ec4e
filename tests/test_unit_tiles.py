"""The attention's work decomposition (unit_tiles / attn_units in the
kernels' header), compiled for the host and checked exhaustively: every
(head, query tile) of a frame belongs to exactly one unit, a unit's two tiles
are two consecutive tiles of one head or the last tiles of heads 2g and
2g + 1, and only the last head of an odd head count has a unit with one tile.
No GPU is needed (nvcc compiles the header's host side)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_23286_gb300", "csrc")

PROGRAM = r"""
#include <cstdio>
#include "kernels.h"
using namespace regmem_dev;
int main() {
  for (int H = 1; H <= 40; ++H)
    for (int nqt = 1; nqt <= 40; ++nqt) {
      const long long n = attn_units(nqt, H);
      for (long long u = 0; u < n; ++u) {
        const UnitTiles t = unit_tiles(u, nqt, H);
        std::printf("%d %d %lld %d %d %d %d %d\n", H, nqt, u, t.h0, t.qt0, t.h1, t.qt1, t.has1 ? 1 : 0);
      }
    }
  return 0;
}
"""


@pytest.fixture(scope="module")
def table(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    d = tmp_path_factory.mktemp("units")
    src, exe = d / "units.cu", d / "units"
    src.write_text(PROGRAM)
    subprocess.run([nvcc, "-std=c++17", "-I", CSRC, "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True, capture_output=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    rows = {}
    for line in out.splitlines():
        H, nqt, u, h0, q0, h1, q1, has1 = map(int, line.split())
        rows.setdefault((H, nqt), []).append((u, h0, q0, h1, q1, has1))
    return rows


def test_every_tile_in_exactly_one_unit(table):
    for (H, nqt), units in table.items():
        seen = []
        for u, h0, q0, h1, q1, has1 in units:
            seen.append((h0, q0))
            if has1:
                seen.append((h1, q1))
        assert sorted(seen) == [(h, q) for h in range(H) for q in range(nqt)], (H, nqt)
        assert len(units) == H * (nqt // 2) + ((H + 1) // 2 if nqt % 2 else 0)


def test_unit_shapes(table):
    for (H, nqt), units in table.items():
        lone = 0
        for u, h0, q0, h1, q1, has1 in units:
            if not has1:
                lone += 1
                assert H % 2 == 1 and nqt % 2 == 1 and h0 == H - 1 and q0 == nqt - 1
            elif h0 == h1:
                assert q0 % 2 == 0 and q1 == q0 + 1 < nqt
            else:
                assert h0 % 2 == 0 and h1 == h0 + 1 and q0 == q1 == nqt - 1
        assert lone == (1 if H % 2 and nqt % 2 else 0)


def test_units_of_a_head_pair_are_contiguous(table):
    """Units are ordered by pairs of heads, so units that read the same K/V
    run close in time."""
    for (H, nqt), units in table.items():
        groups = [min(h0, h1) // 2 for _, h0, _, h1, _, _ in units]
        assert groups == sorted(groups)


SPLIT_PROGRAM = r"""
#include <cstdio>
#include "kernels.h"
#include "split.cuh"
using namespace regmem_dev;
int main() {
  // (units, bank tiles, frame tiles, CTAs)
  const int cases[][4] = {{88, 121, 11, 152}, {88, 0, 11, 152}, {88, 11, 11, 152}, {88, 230, 11, 152},
                          {1, 313, 1, 152}, {1, 159, 1, 152}, {1, 1, 1, 2}, {3, 40, 11, 152},
                          {8, 2, 1, 24}, {88, 2148, 11, 256}, {5, 0, 3, 15}};
  for (const auto& c : cases) {
    SplitBounds sb;
    attn_split_bounds(sb, c[0], c[1], c[2], c[3]);
    std::printf("case %d %d %d %d\n", c[0], c[1], c[2], c[3]);
    for (int b = 0; b <= c[3]; ++b) std::printf("%lld ", sb.x[b]);
    std::printf("\n");
    const long long total = (long long)c[0] * (c[1] + c[2]);
    for (long long x = 0; x < total; x += 1 + total / 997) std::printf("%lld:%d ", x, split::cta_of(sb, c[3], x));
    std::printf("\n");
  }
  return 0;
}
"""


def test_weighted_split_covers_every_tile_once_and_balances_cost(tmp_path):
    """attn_split_bounds cuts the (unit, key tile) sequence into G ranges:
    strictly increasing, from 0 to units * (nb + nf), each CTA's estimated
    cost (bank tile 100, frame tile 108, a unit start 170) within one tile
    and one unit start of the mean; cta_of inverts the cuts."""
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    src, exe = tmp_path / "split.cu", tmp_path / "split"
    src.write_text(SPLIT_PROGRAM)
    subprocess.run([nvcc, "-std=c++17", "-I", CSRC, "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True, capture_output=True)
    lines = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines()
    for i in range(0, len(lines), 3):
        units, nb, nf, G = map(int, lines[i].split()[1:])
        x = list(map(int, lines[i + 1].split()))
        nkv, total = nb + nf, units * (nb + nf)
        assert len(x) == G + 1 and x[0] == 0 and x[-1] == total
        assert all(a < b for a, b in zip(x, x[1:]))
        cost = []
        for b in range(G):
            c = 0
            for t in range(x[b], x[b + 1]):
                j = t % nkv
                c += (170 if j == 0 else 0) + (100 if j < nb else 108)
            cost.append(c)
        mean = sum(cost) / G
        if total >= 4 * G:  # enough tiles per CTA for the cut to balance cost
            assert max(cost) - mean <= 108 + 170 and mean - min(cost) <= 108 + 170, (units, nb, nf, G)
        for pair in lines[i + 2].split():
            t, b = map(int, pair.split(":"))
            assert x[b] <= t < x[b + 1]
