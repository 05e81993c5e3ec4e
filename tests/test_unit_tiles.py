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
  // (heads, query tiles per head, bank rows M, frame tiles, CTAs, phases allowed)
  const long long cases[][6] = {{16, 11, 15486, 11, 152, 2}, {16, 11, 0, 11, 152, 2},
                                {16, 11, 1374, 11, 152, 2}, {16, 11, 29360, 11, 152, 2},
                                {16, 11, 29360, 11, 152, 1}, {1, 1, 40000, 1, 152, 2},
                                {1, 1, 20352, 1, 152, 2}, {2, 1, 1, 1, 2, 2}, {3, 11, 5000, 11, 152, 2},
                                {4, 1, 90000, 1, 152, 2}, {4, 11, 12000, 11, 152, 2},
                                {16, 11, 274800, 11, 256, 2}, {5, 9, 0, 9, 15, 2}, {7, 3, 70000, 3, 152, 2}};
  for (const auto& c : cases) {
    const int H = (int)c[0], nqt = (int)c[1], nf = (int)c[3], G = (int)c[4], mp = (int)c[5];
    const long long M = c[2];
    const int nb = (int)((M + 127) / 128);
    const long long units = attn_units(nqt, H);
    SplitBounds sb;
    attn_split_bounds(sb, units, nb, nf, G, H, nqt, M, mp);
    std::printf("case %d %d %lld %d %d %d %lld %d %d\n", H, nqt, M, nf, G, mp, units, sb.P, sb.slots);
    for (int p = 0; p <= sb.P; ++p) std::printf("%lld ", sb.pbeg[p]);
    std::printf("\n");
    for (int p = 0; p < sb.P; ++p) {
      for (int b = 0; b <= G; ++b) std::printf("%lld ", sb.x[p][b]);
      std::printf("\n");
    }
    const long long total = units * (nb + nf);
    for (long long x = 0; x < total; x += 1 + total / 997) {
      const int p = split::phase_of(sb, x);
      std::printf("%lld:%d:%d ", x, p, split::cta_of(sb, p, G, x));
    }
    std::printf("\n");
  }
  return 0;
}
"""


def test_weighted_split_covers_every_tile_once_and_balances_cost(tmp_path):
    """attn_split_bounds cuts the (unit, key tile) sequence into G ranges per
    phase: strictly increasing, each phase a run of whole head-pair groups of
    units, the phases together from 0 to units * (nb + nf), each CTA's
    estimated cost (bank tile 100, frame tile 108, a unit start 170) within
    one tile and one unit start of the phase's mean; two phases exactly when
    the K/V bytes H M 256 exceed 80 MB, there are two head-pair groups and two
    phases are allowed; phase_of / cta_of invert the cuts."""
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    src, exe = tmp_path / "split.cu", tmp_path / "split"
    src.write_text(SPLIT_PROGRAM)
    subprocess.run([nvcc, "-std=c++17", "-I", CSRC, "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True, capture_output=True)
    lines = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines()
    i = 0
    seen_two = 0
    while i < len(lines):
        H, nqt, M, nf, G, mp, units, P, slots = map(int, lines[i].split()[1:])
        nb = -(-M // 128)
        nkv, total = nb + nf, units * (nb + nf)
        gs = 2 * (nqt // 2) + (nqt % 2)
        pbeg = list(map(int, lines[i + 1].split()))
        cuts = [list(map(int, lines[i + 2 + p].split())) for p in range(P)]
        want_two = mp > 1 and (H + 1) // 2 >= 2 and H * M * 256 > 80 * 2 ** 20
        assert P == (2 if want_two else 1) and slots == (4 if mp > 1 else 2)
        seen_two += P == 2
        assert pbeg[0] == 0 and pbeg[-1] == total
        for p in range(P):
            x = cuts[p]
            assert len(x) == G + 1 and x[0] == pbeg[p] and x[-1] == pbeg[p + 1]
            assert pbeg[p] % (gs * nkv) == 0  # phases begin at head-pair groups
            assert all(a < b for a, b in zip(x, x[1:]))
            cost = []
            for b in range(G):
                c = 0
                for t in range(x[b], x[b + 1]):
                    j = t % nkv
                    c += (170 if j == 0 else 0) + (100 if j < nb else 108)
                cost.append(c)
            mean = sum(cost) / G
            if pbeg[p + 1] - pbeg[p] >= 4 * G:  # enough tiles per CTA to balance cost
                assert max(cost) - mean <= 108 + 170 and mean - min(cost) <= 108 + 170, lines[i]
        for trip in lines[i + 2 + P].split():
            t, p, b = map(int, trip.split(":"))
            assert pbeg[p] <= t < pbeg[p + 1] and cuts[p][b] <= t < cuts[p][b + 1]
        i += 3 + P
    assert seen_two >= 3
