"""The element-wise O error bound of tests/helpers.py, checked on CPU against
an emulation of the kernel's rounding steps: P rounded to bf16 before P V
(normaliser from the unrounded values), a unit split into two pieces whose
normalised partials are stored in bf16, and the final bf16 rounding.  The
emulated result must lie inside the bound on every element, and plausible
mistakes -- a 128-key tile dropped from the sum, P V accumulated from the
wrong V tile, a softmax scale 1 % off -- must fall outside it on some
elements."""
import numpy as np
import pytest

import oracle as orc
from helpers import O_ATOL, O_BOUND_ABS, O_BOUND_FLOOR, O_BOUND_REF, O_RTOL


def bf16(a):
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    r = ((u + np.uint32(0x7FFF) + ((u >> 16) & np.uint32(1))) & np.uint32(0xFFFF0000))
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def emulate(q, kc, vc, scale, split, drop_tile=None, shift_v=False):
    """O as the kernel forms it (fp64 stands in for fp32 accumulation)."""
    z = (q @ kc.T) * scale
    L = kc.shape[0]
    keep = np.ones(L, dtype=bool)
    if drop_tile is not None:
        keep[drop_tile * 128:(drop_tile + 1) * 128] = False
    v_used = np.roll(vc, 128, axis=0) if shift_v else vc
    parts = []
    for lo, hi in ((0, split), (split, L)):
        zz = z[:, lo:hi]
        m = zz.max(axis=1, keepdims=True)
        p = np.exp(zz - m) * keep[None, lo:hi]
        l = p.sum(axis=1, keepdims=True)
        o_p = bf16((bf16(p) @ v_used[lo:hi]) / l)  # normalised partial in bf16
        lse_p = m[:, 0] + np.log(l[:, 0])
        parts.append((o_p, lse_p))
    lse = np.logaddexp(parts[0][1], parts[1][1])
    o = sum(np.exp(lp - lse)[:, None] * op for op, lp in parts)
    return bf16(o)


def inputs(seed, n, L):
    rng = np.random.default_rng(seed)
    q = bf16(rng.standard_normal((n, 64)))
    kc = bf16(rng.standard_normal((L, 64)) * np.exp(0.5 * rng.standard_normal((L, 1))))
    vc = bf16(rng.standard_normal((L, 64)))
    return q, kc, vc


def bound_ratio(o, q, kc, vc):
    o_ref, _, _, _ = orc.attend_head(q, kc, vc, 0.125)
    o_abs, _, _, _ = orc.attend_head(q, kc, np.abs(vc), 0.125)
    d = np.abs(o - o_ref)
    contract_ok = bool((d <= O_ATOL + O_RTOL * np.abs(o_ref)).all())
    return (d / (O_BOUND_REF * np.abs(o_ref) + O_BOUND_ABS * o_abs + O_BOUND_FLOOR)).max(), contract_ok


@pytest.mark.parametrize("L", [300, 2760, 9000])
def test_rounded_arithmetic_lies_inside_the_bound(L):
    q, kc, vc = inputs(L, 256, L)
    ratio, contract_ok = bound_ratio(emulate(q, kc, vc, 0.125, split=L // 2 + 7), q, kc, vc)
    assert contract_ok
    assert ratio <= 1.0


def test_dropped_key_tile_violates_the_bound():
    L = 9000
    q, kc, vc = inputs(5, 256, L)
    ratio, _ = bound_ratio(emulate(q, kc, vc, 0.125, split=4500, drop_tile=20), q, kc, vc)
    assert ratio > 1.0


def test_wrong_value_tile_violates_the_bound():
    L = 2760
    q, kc, vc = inputs(6, 256, L)
    ratio, _ = bound_ratio(emulate(q, kc, vc, 0.125, split=1380, shift_v=True), q, kc, vc)
    assert ratio > 1.0


def test_scale_one_percent_off_violates_the_bound():
    L = 29360
    q, kc, vc = inputs(7, 128, L)
    ratio, _ = bound_ratio(emulate(q, kc, vc, 0.125 * 1.01, split=L // 2), q, kc, vc)
    assert ratio > 1.0
