"""Failure detection on the GPU without a GPU fault: an attention launch in
which the first CTA's TMA producer skips one K/V load (regmem_debug_set), so
nothing ever lands in that ring stage.  The consumers' bounded waits run out
after the handle's limit, the kernel drains what it issued and returns, and
the timeout bit of the status word is reported by the next calls.  The GPU
context stays usable: a fresh handle afterwards matches the oracle."""
import time

import numpy as np
import pytest
import torch

import oracle as orc
from helpers import Stream, check_lse, check_o, check_saliency, o_abs_frame, to64
from paper_2609_23286_gb300 import regmem

pytestmark = pytest.mark.gpu

H, NS, GH, GW, M = 16, 5, 37, 37, 3000  # CTA 0 runs ~20 K/V loads, so load 2 exists


def _bank():
    g = torch.Generator().manual_seed(41)
    bk = (torch.randn(H, M, 64, generator=g) * 1.3).to(torch.bfloat16)
    bv = torch.randn(H, M, 64, generator=g).to(torch.bfloat16)
    return bk, bv


def test_expired_wait_reports_timeout_and_the_context_stays_usable():
    bk, bv = _bank()
    st = Stream(1, H, NS, GH, GW, budget=14, max_frames=400, seed=31)
    try:
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 5)
        out = torch.empty_like(q)
        sal = torch.empty(H, st.N, dtype=torch.float32, device=q.device)
        with pytest.raises(regmem.RegmemError) as e:
            st.rm.debug_set(wait_limit_us=0)
        assert e.value.status == regmem.ERR_ARG
        st.rm.debug_set(wait_limit_us=20000, skip_kv_load=2)  # 20 ms limit, one skipped load
        st.rm.attend_frame(0, q, k, v, out, sal)               # enqueued without error
        t0 = time.perf_counter()
        with pytest.raises(regmem.RegmemError) as e:
            st.rm.synchronize()
        assert e.value.status == regmem.ERR_TIMEOUT
        assert "bounded wait expired" in str(e.value)
        assert time.perf_counter() - t0 < 5.0  # the kernel gave up and returned
        # every later call on the handle reports it before enqueueing anything
        with pytest.raises(regmem.RegmemError) as e:
            st.rm.admit(0, 14)
        assert e.value.status == regmem.ERR_TIMEOUT
        torch.cuda.synchronize()  # no CUDA error: the context is intact
    finally:
        st.close()

    # a fresh handle on the same GPU: one frame against the oracle
    st = Stream(1, H, NS, GH, GW, budget=14, max_frames=400, seed=31)
    try:
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 5)
        out, sal, lse = st.attend(0, q, k, v)
        st.admit(0, 14)
        st.rm.synchronize()
        bk64 = [bk[h].double().numpy() for h in range(H)]
        bv64 = [bv[h].double().numpy() for h in range(H)]
        qi = orc.sampled_query_tokens(NS, GH, GW, 2)
        ref = orc.attend_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8, qi)
        check_o(out, ref["O"], "after timeout", o_abs=o_abs_frame(to64(q), to64(k), to64(v),
                                                                   bk64, bv64, 1 / 8))
        check_lse(lse, ref["LSE"], "after timeout")
        check_saliency(sal, ref["S"], "after timeout")
    finally:
        st.close()


def test_armed_fault_is_one_shot_and_default_limit_restored():
    """The fault applies to the next attention launch only; a launch with the
    limit back at its default completes normally."""
    bk, bv = _bank()
    st = Stream(1, H, NS, GH, GW, budget=14, max_frames=400, seed=32)
    try:
        st.rm.import_bank(0, bk, bv, M)
        st.rm.debug_set(wait_limit_us=2000000, skip_kv_load=-1)
        q, k, v = st.inputs(0, 6)
        out, sal, lse = st.attend(0, q, k, v)
        st.admit(0, 14)
        st.rm.synchronize()
        assert np.isfinite(to64(lse)).all()
    finally:
        st.close()
