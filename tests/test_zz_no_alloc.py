"""The allocation-free attend entry point against the handle-based one.

Callers that cannot allocate device memory (code running inside another
framework's memory pool, plugins given pre-sized buffers, real-time loops)
use regmem_attend_frame_noalloc, whose scratch is a fixed array inside the
library.  Here it is called twice in a row through the C ABI, with different
banks and frames, and each result is compared with regmem_attend_frame on the
same inputs, within the parity tolerances of the other tests.  This file is
collected last so that a failure here cannot stop the rest of the suite.
"""
import pytest
import torch

from helpers import check_o, check_saliency, to64
from paper_2609_23286_gb300 import regmem, synth

pytestmark = pytest.mark.gpu


def test_noalloc_matches_handle_path_on_two_calls():
    H, ns, gh, gw, budget = 16, 5, 37, 37, 14
    N = ns + gh * gw
    dev = torch.device("cuda")
    stream = torch.cuda.current_stream()
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    for call, (M, seed) in enumerate([(2760, 21), (1374 + 40 * budget, 22)]):
        g = torch.Generator(device=dev).manual_seed(seed)
        bk = (torch.randn(H, M, 64, generator=g, device=dev) * 1.3).to(torch.bfloat16)
        bv = torch.randn(H, M, 64, generator=g, device=dev).to(torch.bfloat16)
        q, k, v = synth.frame_qkv(seed, 0, call + 2, N, H, 64, device=dev)

        rm = regmem.RegMem(1, H, 64, budget)
        try:
            rm.set_frame(ns, gh, gw, ds=2, max_frames=400)
            rm.set_stream(stream)
            rm.import_bank(0, bk.cpu(), bv.cpu(), M)
            out_ref = torch.empty_like(q)
            sal_ref = torch.empty(H, N, device=dev)
            rm.attend_frame(0, q, k, v, out_ref, sal_ref)
            rm.synchronize()
        finally:
            rm.close()

        out = torch.empty_like(q)
        sal = torch.empty(H, N, device=dev)
        regmem.regmem_attend_frame_noalloc(ns, gh, gw, H, q, k, v, bk, bv, M, M, out, sal,
                                           status=status, stream=stream)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        check_o(out, to64(out_ref), f"call {call}")
        check_saliency(sal, to64(sal_ref), f"call {call}")


def test_noalloc_rejects_sizes_beyond_its_scratch():
    z = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(regmem.RegmemError) as e:
        # 64 heads x 4101 tokens > 262144 LSE rows held by the scratch
        regmem.regmem_attend_frame_noalloc(5, 64, 64, 64, z, z, z, None, None, 0, 0, z, z,
                                           status=status)
    assert e.value.status == regmem.ERR_UNSUPPORTED


def test_noalloc_requires_a_status_word():
    """Without a handle no later call could report an expired device wait, so
    the caller's status word is mandatory."""
    z = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(regmem.RegmemError) as e:
        regmem.regmem_attend_frame_noalloc(5, 2, 2, 2, z, z, z, None, None, 0, 0, z, z)
    assert e.value.status == regmem.ERR_ARG
