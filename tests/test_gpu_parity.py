"""Parity of the CUDA path (through the C ABI) against the fp64 oracle.

Every test feeds both sides the same seeded bf16 inputs.  The oracle gets the
exact values the GPU saw (bf16 widened to float64)."""
import math

import numpy as np
import pytest
import torch

import oracle as orc
from helpers import (Stream, check_indices, check_lse, check_o, check_saliency, o_abs_frame,
                     to64)
from paper_2609_23286_gb300 import regmem

pytestmark = pytest.mark.gpu


def run_stream(L, H, ns, gh, gw, k, frames, seed, ds=2, check_every=1, fused=False, candidates=0):
    """Free-running stream on GPU and oracle; the oracle adopts the GPU's
    admitted indices after they pass check_indices, so later frames stay
    comparable.  fused: each step is one regmem_attend_admit call (admission
    inside the saliency kernel) instead of regmem_attend_frame + regmem_admit."""
    st = Stream(L, H, ns, gh, gw, budget=k, max_frames=frames, seed=seed, ds=ds, candidates=candidates)
    ref = orc.OracleStream(L, H, 64, ns, gh, gw, ds=ds, candidates="all" if candidates else "patch")
    try:
        for t in range(1, frames + 1):
            for layer in range(L):
                q, kk_, v = st.inputs(layer, t)
                if fused:
                    out, sal, lse, idx = st.attend_admit(layer, q, kk_, v, k)
                else:
                    out, sal, lse = st.attend(layer, q, kk_, v)
                    idx = st.admit(layer, k)
                torch.cuda.synchronize()
                oa = o_abs_frame(to64(q), to64(kk_), to64(v), ref.bank_k[layer],
                                 ref.bank_v[layer], ref.scale)
                r = ref.attend(layer, to64(q), to64(kk_), to64(v))
                if t % check_every == 0 or t <= 2:
                    check_o(out, r["O"], f"t={t} l={layer}", o_abs=oa)
                    check_lse(lse, r["LSE"], f"t={t} l={layer}")
                    check_saliency(sal, r["S"], f"t={t} l={layer}")
                if ref.memory_len(layer) == 0:
                    ref.admit(layer, k)
                else:
                    gi = idx.cpu().numpy().astype(np.int64)
                    check_indices(gi, to64(sal), r["S"], ns, k, len(ref.qidx),
                                  "all" if candidates else "patch")
                    ref.admit(layer, k, indices=gi)
                assert st.rm.memory_len(layer) == ref.memory_len(layer) == st.N + (t - 1) * k
            if t in (1, 2, frames):
                for layer in range(L):
                    bk, bv = st.export(layer)
                    for h in range(H):
                        assert np.array_equal(bk[h].double().numpy(), ref.bank_k[layer][h])
                        assert np.array_equal(bv[h].double().numpy(), ref.bank_v[layer][h])
        st.rm.synchronize()
    finally:
        st.close()


@pytest.mark.parametrize("fused", [False, True])
def test_tiny_stream_full_oracle(fused):
    """1 layer, 2 heads, 8x8 patches + 5 specials = 69 tokens, 8 frames, k = 1,
    seed 0: the whole stream against the free-running oracle."""
    run_stream(1, 2, 5, 8, 8, 1, 8, seed=0, fused=fused)


@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("H,ns,gh,gw", [(1, 0, 1, 1), (3, 1, 1, 2), (2, 0, 3, 1)])
def test_degenerate_frames(H, ns, gh, gw, fused):
    """The smallest frames: one token (no special tokens, a 1 x 1 patch grid:
    one sampled query, one admission candidate), three tokens (one special,
    1 x 2 patches) and a 3 x 1 grid.  Every query and key tile is a single
    ragged row or a few; the stream admits one row per frame, against the
    oracle frame by frame."""
    run_stream(1, H, ns, gh, gw, 1, 5, seed=H * 10 + gh, fused=fused)


@pytest.mark.parametrize("k,fused", [(14, True), (40, False)])
def test_largest_candidate_set(k, fused):
    """Frames at the library's limit of admission candidates: 2 special tokens
    and 90 x 91 patches (N = 8,192, 8,190 candidates, 2,116 sampled queries):
    the fused selection over 64 key tiles' lists (k = 14) and the radix
    selection of the two-call path (k = 40), against the full oracle."""
    run_stream(1, 2, 2, 90, 91, k, 2, seed=77 + k, fused=fused)


@pytest.mark.parametrize("ds", [1, 3, 4])
def test_query_downsampling_factors(ds):
    """Sec. 3.3 with other windows (T6's sweep): 13 x 11 patches + 5 specials,
    4 heads, k = 3, 4 frames; ds = 1 samples every patch query, 3 and 4 keep
    the partial edge windows of the odd grid."""
    run_stream(1, 4, 5, 13, 11, 3, 4, seed=12, ds=ds, fused=True)


@pytest.mark.parametrize("fused", [False, True])
def test_all_tokens_as_candidates(fused):
    """candidates = 1: the special tokens may be admitted too (13 x 11 + 5,
    4 heads, k = 4, 4 frames)."""
    run_stream(1, 4, 5, 13, 11, 4, 4, seed=13, fused=fused, candidates=1)


def test_vggt_layer_first_frames():
    """16 heads, 37x37 + 5 = 1374 tokens, k = 14, seed 1, first 4 frames: several
    query tiles with a ragged last tile, bank tiles with ragged ends."""
    run_stream(1, 16, 5, 37, 37, 14, 4, seed=1)


def test_two_layers_nonsquare():
    """37x28 + 5 = 1041 tokens, k = 11, two layers with independent seeds."""
    run_stream(2, 16, 5, 37, 28, 11, 3, seed=5)


@pytest.mark.parametrize("M", [1, 127, 128, 129, 383, 2760])
def test_teacher_forced_bank_lengths(M):
    """Single frame against an imported bank of M rows: bank tiles that are
    tiny, exactly one tile, one row past a tile, and the 100-frame length."""
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    st = Stream(1, H, ns, gh, gw, budget=14, max_frames=400, seed=3)
    try:
        g = torch.Generator().manual_seed(M)
        bk = (torch.randn(H, M, 64, generator=g) * 1.3).to(torch.bfloat16)
        bv = torch.randn(H, M, 64, generator=g).to(torch.bfloat16)
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 7)
        out, sal, lse = st.attend(0, q, k, v)
        idx = st.admit(0, 14)
        torch.cuda.synchronize()
        bk64 = [bk[h].double().numpy() for h in range(H)]
        bv64 = [bv[h].double().numpy() for h in range(H)]
        ref = orc.attend_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8,
                               orc.sampled_query_tokens(ns, gh, gw, 2))
        oa = o_abs_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8)
        check_o(out, ref["O"], f"M={M}", o_abs=oa)
        check_lse(lse, ref["LSE"], f"M={M}")
        check_saliency(sal, ref["S"], f"M={M}")
        check_indices(idx.cpu().numpy(), to64(sal), ref["S"], ns, 14, 361)
        bk2, bv2 = st.export(0)
        gi = idx.cpu().numpy()
        for h in range(H):
            assert torch.equal(bk2[h, :M], bk[h]) and torch.equal(bv2[h, :M], bv[h])
            assert torch.equal(bk2[h, M:], k[gi[h], h].cpu())
            assert torch.equal(bv2[h, M:], v[gi[h], h].cpu())
    finally:
        st.close()


@pytest.mark.parametrize("H,ns,gh,gw,M", [
    (1, 1, 8, 8, 20352),   # 160 key tiles on the grid: one or two tiles per CTA
    (1, 1, 8, 8, 40000),   # one unit split over every CTA of the grid
    (2, 4, 14, 14, 30000),  # two query tiles per unit, each unit over half the grid
    (3, 5, 37, 37, 5000),  # eleven query tiles: heads 0 and 1 share a unit of their last
                           # tiles, head 2's last tile is a unit by itself
    (2, 1, 8, 8, 30000),   # one query tile per head: a single two-head unit over the grid
    (4, 5, 37, 37, 12000),  # two two-head units, each split over many CTAs
    (4, 5, 8, 8, 90000),   # K/V of 92 MB: two phases (heads 0-1, then 2-3), each unit over every CTA
])
def test_split_units_across_many_ctas(H, ns, gh, gw, M):
    """Few heads and a long bank: units whose key tiles are spread over many
    CTAs (more than 64 on a full GB300 grid), merged by the combine kernel."""
    N = ns + gh * gw
    st = Stream(1, H, ns, gh, gw, budget=14, max_frames=M // 14 + 2, seed=6)
    try:
        g = torch.Generator().manual_seed(M + H)
        bk = (torch.randn(H, M, 64, generator=g) * 1.3).to(torch.bfloat16)
        bv = torch.randn(H, M, 64, generator=g).to(torch.bfloat16)
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 3)
        out, sal, lse = st.attend(0, q, k, v)
        torch.cuda.synchronize()
        bk64 = [bk[h].double().numpy() for h in range(H)]
        bv64 = [bv[h].double().numpy() for h in range(H)]
        ref = orc.attend_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8,
                               orc.sampled_query_tokens(ns, gh, gw, 2))
        oa = o_abs_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8)
        check_o(out, ref["O"], f"H={H} N={N} M={M}", o_abs=oa)
        check_lse(lse, ref["LSE"], f"H={H} N={N} M={M}")
        check_saliency(sal, ref["S"], f"H={H} N={N} M={M}")
    finally:
        st.close()


def test_running_max_renewed_by_large_later_logits():
    """A row's running max grows by far more than the softmax lets it lag
    (2^8 in exp2 units) after its piece's first key tiles: a bank whose first
    600 rows are tiny and whose rows 1500-1503 are 50 * ones gives logits up
    to ~10^3 above the first tiles' maximum in the rows where sum(q) is
    large, so those rows rescale O and l mid-piece (in pieces that start
    before the large rows; pieces starting after them take the large max on
    their first tile).  All rows must still match the oracle."""
    H, ns, gh, gw, M = 2, 5, 37, 37, 2000
    st = Stream(1, H, ns, gh, gw, budget=14, max_frames=M // 14 + 2, seed=9)
    try:
        g = torch.Generator().manual_seed(99)
        bk = torch.randn(H, M, 64, generator=g)
        bk[:, :600] *= 0.05
        bk[:, 1500:1502] = 50.0
        bk[:, 1502:1504, ::2] = 50.0  # a second large row in the other half of its tile
        bk = bk.to(torch.bfloat16)
        bv = torch.randn(H, M, 64, generator=g).to(torch.bfloat16)
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 3)
        out, sal, lse = st.attend(0, q, k, v)
        torch.cuda.synchronize()
        bk64 = [bk[h].double().numpy() for h in range(H)]
        bv64 = [bv[h].double().numpy() for h in range(H)]
        ref = orc.attend_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8,
                               orc.sampled_query_tokens(ns, gh, gw, 2))
        oa = o_abs_frame(to64(q), to64(k), to64(v), bk64, bv64, 1 / 8)
        # the case is only meaningful if many rows' logits outgrow the first tiles' by far
        z_big = to64(q)[:, 0, :].sum(axis=1) * 50.0 / 8.0
        assert (z_big * 1.4426950408889634 > 64 + 5).sum() > 50
        check_o(out, ref["O"], "renewed running max", o_abs=oa)
        check_lse(lse, ref["LSE"], "renewed running max")
        check_saliency(sal, ref["S"], "renewed running max")
    finally:
        st.close()


def test_long_bank_sampled_rows():
    """Config-4 end size: a bank of 29360 rows per head (2000 frames at k = 14).
    O is checked on sampled query rows (the oracle computes rows one by one),
    LSE and saliency on all sampled queries / keys."""
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    M = N + 1999 * 14
    st = Stream(1, H, ns, gh, gw, budget=14, max_frames=2001, seed=4)
    try:
        g = torch.Generator().manual_seed(11)
        bk = (torch.randn(H, M, 64, generator=g) * torch.exp(0.5 * torch.randn(1, M, 1, generator=g))).to(torch.bfloat16)
        bv = torch.randn(H, M, 64, generator=g).to(torch.bfloat16)
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 2000)
        out, sal, lse = st.attend(0, q, k, v)
        torch.cuda.synchronize()
        qi = orc.sampled_query_tokens(ns, gh, gw, 2)
        rows = sorted(set(list(range(0, N, 97)) + [N - 1, 127, 128, 1279, 1280]))
        q64, k64, v64 = to64(q), to64(k), to64(v)
        for h in range(H):
            kc = np.concatenate([bk[h].double().numpy(), k64[:, h]])
            vc = np.concatenate([bv[h].double().numpy(), v64[:, h]])
            o_r, l_r, _, _ = orc.attend_head(q64[rows, h], kc, vc, 1 / 8)
            o_a, _, _, _ = orc.attend_head(q64[rows, h], kc, np.abs(vc), 1 / 8)
            check_o(out[rows, h], o_r, f"h={h}", o_abs=o_a)
            check_lse(lse[h, rows], l_r, f"h={h}")
            _, l_s, z_s, _ = orc.attend_head(q64[qi, h], kc, vc, 1 / 8)
            s_r = orc.saliency_lse(z_s, l_s, M, list(range(len(qi))))
            check_saliency(sal[h], s_r, f"h={h}")
        st.rm.admit(0, 14)
        st.rm.synchronize()
    finally:
        st.close()


def test_frame_attention_matches_sdpa_oracle():
    """Non-causal intra-frame attention (M = 0, no saliency), 1041 tokens."""
    H, ns, gh, gw = 16, 5, 37, 28
    st = Stream(1, H, ns, gh, gw, budget=11, max_frames=2, seed=9)
    try:
        q, k, v = st.inputs(0, 1)
        out = torch.empty_like(q)
        st.rm.frame_attention(q, k, v, out)
        torch.cuda.synchronize()
        ref = orc.attend_frame(to64(q), to64(k), to64(v), [np.zeros((0, 64))] * H,
                               [np.zeros((0, 64))] * H, 1 / 8, [0])
        oa = o_abs_frame(to64(q), to64(k), to64(v), [np.zeros((0, 64))] * H,
                         [np.zeros((0, 64))] * H, 1 / 8)
        check_o(out, ref["O"], "frame attention", o_abs=oa)
        assert st.rm.memory_len(0) == 0
    finally:
        st.close()


def test_k_zero_and_budget_edges():
    """k = 0 leaves the bank as it is (Eq. 5 layers); k = budget appends."""
    st = Stream(1, 4, 5, 8, 8, budget=3, max_frames=5, seed=2)
    try:
        for t, kk in ((1, 0), (2, 0), (3, 3), (4, 1)):
            q, k, v = st.inputs(0, t)
            st.attend(0, q, k, v)
            st.admit(0, kk)
        assert st.rm.memory_len(0) == 69 + 0 + 0 + 3 + 1
        st.rm.synchronize()
    finally:
        st.close()


def test_host_buffer_entry_point_matches_device_path():
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    a = Stream(1, H, ns, gh, gw, budget=14, max_frames=4, seed=6)
    b = Stream(1, H, ns, gh, gw, budget=14, max_frames=4, seed=6)
    try:
        for t in range(1, 4):
            q, k, v = a.inputs(0, t)
            out_d, sal_d, _ = a.attend(0, q, k, v)
            a.admit(0, 14)
            hq, hk, hv = q.cpu().pin_memory(), k.cpu().pin_memory(), v.cpu().pin_memory()
            ho = torch.empty_like(hq).pin_memory()
            hs = torch.empty(H, N, dtype=torch.float32).pin_memory()
            b.rm.attend_frame_host(0, hq, hk, hv, ho, hs)
            b.rm.admit(0, 14)
            b.rm.synchronize()
            torch.cuda.synchronize()
            assert torch.equal(ho, out_d.cpu())
            assert torch.equal(hs, sal_d.cpu())
    finally:
        a.close()
        b.close()


def test_host_entry_points_allocate_nothing_after_set_frame():
    """regmem_set_frame makes every staging buffer, copy stream and event of
    the host-buffer calls: once the kernels are loaded (two warm-up frames),
    a run of host calls that cycles through all six staging sets of
    regmem_attend_admit_host, plus the two-call host form, leaves the
    device's free memory (cudaMemGetInfo) unchanged."""
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    st = Stream(2, H, ns, gh, gw, budget=14, max_frames=16, seed=16)
    try:
        frames = [tuple(x.cpu().pin_memory() for x in st.inputs(l, t)) for t in range(1, 5)
                  for l in range(2)]
        ho = torch.empty(N, H, 64, dtype=torch.bfloat16).pin_memory()
        hs = torch.empty(H, N, dtype=torch.float32).pin_memory()

        def host_frame(i):
            for l in range(2):
                q, k, v = frames[(2 * i + l) % len(frames)]
                st.rm.attend_admit_host(l, q, k, v, ho, hs, 14)

        for i in range(2):  # anchor and first admitted frame: every kernel loaded
            host_frame(i)
        q, k, v = frames[0]
        st.rm.attend_frame_host(0, q, k, v, ho, hs)
        st.rm.admit(0, 14)
        st.rm.synchronize()
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        for i in range(2, 9):  # 14 calls: every staging set used twice or more
            host_frame(i)
        st.rm.attend_frame_host(1, q, k, v, ho, hs)
        st.rm.admit(1, 14)
        st.rm.synchronize()
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0
    finally:
        st.close()


def test_deterministic_repeat():
    """Same inputs twice -> bit-identical outputs, saliency and indices."""
    res = []
    for _ in range(2):
        st = Stream(1, 16, 5, 37, 37, budget=14, max_frames=3, seed=8)
        try:
            outs = []
            for t in (1, 2):
                q, k, v = st.inputs(0, t)
                out, sal, lse = st.attend(0, q, k, v)
                idx = st.admit(0, 14)
                torch.cuda.synchronize()
                outs += [out.cpu(), sal.cpu(), idx.cpu()]
            res.append(outs)
        finally:
            st.close()
    for x, y in zip(*res):
        assert torch.equal(x, y)


def test_state_machine_and_argument_errors():
    rm = regmem.RegMem(2, 2, 64, 1)
    try:
        with pytest.raises(regmem.RegmemError) as e:
            rm.admit(0, 1)
        assert e.value.status == regmem.ERR_STATE            # before set_frame
        rm.set_frame(5, 8, 8, ds=2, max_frames=3)
        with pytest.raises(regmem.RegmemError) as e:
            rm.set_frame(5, 8, 8)
        assert e.value.status == regmem.ERR_STATE            # twice
        N = 69
        q = torch.zeros(N, 2, 64, dtype=torch.bfloat16, device="cuda")
        out = torch.empty_like(q)
        sal = torch.empty(2, N, device="cuda")
        with pytest.raises(regmem.RegmemError) as e:
            rm.admit(0, 1)
        assert e.value.status == regmem.ERR_STATE            # admit before attend
        with pytest.raises(regmem.RegmemError) as e:
            rm.attend_frame(2, q, q, q, out, sal)
        assert e.value.status == regmem.ERR_ARG              # layer out of range
        with pytest.raises(regmem.RegmemError) as e:
            rm.attend_frame(0, q, q, q, None, sal)
        assert e.value.status == regmem.ERR_ARG              # null pointer
        with pytest.raises(regmem.RegmemError) as e:
            rm.attend_frame(0, q.data_ptr() + 2, q, q, out, sal)
        assert e.value.status == regmem.ERR_ARG              # misaligned
        rm.attend_frame(0, q, q, q, out, sal)
        with pytest.raises(regmem.RegmemError) as e:
            rm.attend_frame(0, q, q, q, out, sal)
        assert e.value.status == regmem.ERR_STATE            # second attend
        rm.admit(0, 1)                                       # anchor: k ignored
        assert rm.memory_len(0) == N
        for kk in (1, 1):
            rm.attend_frame(0, q, q, q, out, sal)
            with pytest.raises(regmem.RegmemError) as e:
                rm.admit(0, 2)
            assert e.value.status == regmem.ERR_ARG          # k > budget
            rm.admit(0, kk)
        assert rm.memory_len(0) == N + 2 == rm.capacity()
        rm.attend_frame(0, q, q, q, out, sal)
        with pytest.raises(regmem.RegmemError) as e:
            rm.admit(0, 1)
        assert e.value.status == regmem.ERR_CAPACITY         # bank full
        assert rm.memory_len(0) == N + 2
        rm.admit(0, 0)
        rm.reset()
        assert rm.memory_len(0) == 0
        rm.synchronize()
    finally:
        rm.close()
    with pytest.raises(regmem.RegmemError) as e:
        regmem.regmem_create(1, 1, 128, 1)
    assert e.value.status == regmem.ERR_UNSUPPORTED


def test_uniform_keys_tie_to_lowest_indices():
    """K = 0 makes every logit 0: softmax is uniform over the L attended keys,
    every frame key has saliency |Q~| / L, and the admitted tokens must be the
    k lowest candidate indices (ties go to the lower index)."""
    H, ns, gh, gw, k = 4, 5, 8, 8, 20
    N = ns + gh * gw
    st = Stream(1, H, ns, gh, gw, budget=k, max_frames=3, seed=12)
    try:
        for t in (1, 2):
            q, kk, v = st.inputs(0, t)
            out, sal, lse = st.attend(0, q, torch.zeros_like(kk), v)
            idx = st.admit(0, k)
            torch.cuda.synchronize()
            L = N if t == 1 else 2 * N
            assert torch.allclose(lse.cpu().double(), torch.full((H, N), math.log(L), dtype=torch.float64),
                                  atol=1e-4)
            s_ref = np.full((H, N), 16.0 / L)
            check_saliency(sal, s_ref, f"t={t}")
            if t == 2:
                assert (idx.cpu().numpy() == np.arange(ns, ns + k)[None, :]).all()
    finally:
        st.close()


def test_admit_every_candidate():
    """k equal to the number of candidates admits every patch token in order."""
    H, ns, gh, gw = 2, 5, 8, 8
    nc = gh * gw
    st = Stream(1, H, ns, gh, gw, budget=nc, max_frames=3, seed=13)
    try:
        for t in (1, 2):
            q, kk, v = st.inputs(0, t)
            st.attend(0, q, kk, v)
            idx = st.admit(0, nc)
        torch.cuda.synchronize()
        assert (idx.cpu().numpy() == np.arange(ns, ns + nc)[None, :]).all()
        bk, bv = st.export(0)
        assert torch.equal(bk[:, ns + gh * gw + 0:], kk[ns:, :, :].permute(1, 0, 2).cpu())
    finally:
        st.close()


def test_fused_step_matches_two_calls():
    """regmem_attend_admit (admission inside the saliency kernel) gives
    bit-identical outputs, saliency, admitted indices and banks to
    regmem_attend_frame + regmem_admit on a 1374-token, 16-head stream."""
    H, ns, gh, gw, k = 16, 5, 37, 37, 14
    a = Stream(2, H, ns, gh, gw, budget=k, max_frames=6, seed=21)
    b = Stream(2, H, ns, gh, gw, budget=k, max_frames=6, seed=21)
    try:
        for t in range(1, 6):
            for layer in range(2):
                q, kk, v = a.inputs(layer, t)
                o1, s1, l1 = a.attend(layer, q, kk, v)
                i1 = a.admit(layer, k)
                o2, s2, l2, i2 = b.attend_admit(layer, q, kk, v, k)
                torch.cuda.synchronize()
                assert torch.equal(o1, o2) and torch.equal(s1, s2) and torch.equal(l1, l2)
                if t > 1:
                    assert torch.equal(i1, i2)
        for layer in range(2):
            assert a.rm.memory_len(layer) == b.rm.memory_len(layer) == ns + gh * gw + 4 * k
            ka, va = a.export(layer)
            kb, vb = b.export(layer)
            assert torch.equal(ka, kb) and torch.equal(va, vb)
    finally:
        a.close()
        b.close()


def _enqueue_stream(st, frames, ks, high_priority=False):
    """Enqueue every (frame, layer) step of st back to back, without host
    synchronisation, each into buffers of its own; returns them after a
    device synchronisation.  ks[layer] rows are admitted per frame."""
    stream = (torch.cuda.Stream(priority=-1) if high_priority else torch.cuda.current_stream())
    torch.cuda.synchronize()
    st.rm.set_stream(stream)
    res = []
    inputs = [[st.inputs(layer, t) for layer in range(st.L)] for t in range(1, frames + 1)]
    torch.cuda.synchronize()
    for t in range(frames):
        for layer in range(st.L):
            q, kk, v = inputs[t][layer]
            out = torch.empty_like(q)
            sal = torch.empty(st.H, st.N, dtype=torch.float32, device="cuda")
            lse = torch.empty(st.H, st.N, dtype=torch.float32, device="cuda")
            idx = torch.full((st.H, max(ks[layer], 1)), -1, dtype=torch.int32, device="cuda")
            st.rm.attend_admit(layer, q, kk, v, out, sal, ks[layer], idx)
            st.rm.copy_lse(lse)
            res.append((out, sal, lse, idx))
    st.rm.join()
    torch.cuda.synchronize()
    st.rm.synchronize()
    return res, inputs


@pytest.mark.parametrize("ks", [(14, 14, 14), (14, 40, 1)])
def test_overlap_matches_one_stream(ks):
    """regmem_set_overlap(1): saliency and admission on the side stream,
    every step enqueued back to back (so side work of layer l runs beside the
    attention of layer l + 1 and the next frame's attention must wait for
    it), on a high-priority stream.  Outputs, LSE, saliency, indices and
    banks equal the one-stream run bit for bit; k = 40 takes the separate
    selection kernel on the side stream, k = 1 the fused one."""
    H, ns, gh, gw = 16, 5, 37, 37
    frames = 5
    a = Stream(3, H, ns, gh, gw, budget=max(ks), max_frames=frames, seed=31)
    b = Stream(3, H, ns, gh, gw, budget=max(ks), max_frames=frames, seed=31)
    try:
        b.rm.set_overlap(1)
        ra, _ = _enqueue_stream(a, frames, ks)
        rb, _ = _enqueue_stream(b, frames, ks, high_priority=True)
        for i, (x, y) in enumerate(zip(ra, rb)):
            t, layer = divmod(i, 3)
            for name, u, w in zip(("out", "saliency", "lse", "idx"), x, y):
                if name == "idx" and t == 0:
                    continue  # the first frame is stored whole: no indices
                assert torch.equal(u, w), f"{name} differs at t={t + 1} layer={layer}"
        for layer in range(3):
            assert a.rm.memory_len(layer) == b.rm.memory_len(layer)
            ka, va = a.export(layer)
            kb, vb = b.export(layer)
            assert torch.equal(ka, kb) and torch.equal(va, vb)
    finally:
        a.close()
        b.close()


def test_overlap_against_oracle_and_mode_switches():
    """Overlap on a 2-layer 13 x 11 + 5 stream checked against the oracle
    frame by frame; then the two-call path, the host-buffer path, an import
    and a reset on the same handle, each ordered after pending side work."""
    H, ns, gh, gw, k = 4, 5, 13, 11, 3
    st = Stream(2, H, ns, gh, gw, budget=k, max_frames=8, seed=32)
    ref = orc.OracleStream(2, H, 64, ns, gh, gw)
    try:
        st.rm.set_overlap(1)
        for t in range(1, 5):
            for layer in range(2):
                q, kk, v = st.inputs(layer, t)
                if t == 3 and layer == 1:   # two-call path between overlapped steps
                    out, sal, lse = st.attend(layer, q, kk, v)
                    idx = st.admit(layer, k)
                else:
                    out, sal, lse, idx = st.attend_admit(layer, q, kk, v, k)
                torch.cuda.synchronize()
                r = ref.attend(layer, to64(q), to64(kk), to64(v))
                check_o(out, r["O"], f"t={t} l={layer}")
                check_lse(lse, r["LSE"], f"t={t} l={layer}")
                check_saliency(sal, r["S"], f"t={t} l={layer}")
                if t == 1:
                    ref.admit(layer, k)
                else:
                    gi = idx.cpu().numpy().astype(np.int64)
                    check_indices(gi, to64(sal), r["S"], ns, k, len(ref.qidx))
                    ref.admit(layer, k, indices=gi)
        # host-buffer path with overlap: same outputs as the device path
        q, kk, v = st.inputs(0, 5)
        hq, hk, hv = q.cpu().pin_memory(), kk.cpu().pin_memory(), v.cpu().pin_memory()
        ho = torch.empty_like(hq).pin_memory()
        hs = torch.empty(H, st.N, dtype=torch.float32).pin_memory()
        st.rm.attend_admit_host(0, hq, hk, hv, ho, hs, k)
        st.rm.synchronize()
        r = ref.attend(0, to64(q), to64(kk), to64(v))
        check_o(ho, r["O"], "host path")
        check_saliency(hs, r["S"], "host path")
        # import and export follow the pending side work
        bk, bv = st.export(1)
        st.rm.import_bank(1, bk, bv, bk.shape[1])
        bk2, bv2 = st.export(1)
        assert torch.equal(bk, bk2) and torch.equal(bv, bv2)
        st.rm.reset()
        st.rm.set_overlap(0)
        assert st.rm.memory_len(0) == 0
    finally:
        st.close()


def test_fused_uniform_keys_and_every_candidate():
    """The fused selection: uniform saliency ties to the lowest indices, and
    k = all candidates admits every patch token in order."""
    H, ns, gh, gw = 4, 5, 8, 8
    nc = gh * gw
    for k, zero_keys in ((20, True), (nc, False)):
        st = Stream(1, H, ns, gh, gw, budget=k, max_frames=3, seed=22)
        try:
            for t in (1, 2):
                q, kk, v = st.inputs(0, t)
                if zero_keys:
                    kk = torch.zeros_like(kk)
                out, sal, lse, idx = st.attend_admit(0, q, kk, v, k)
            torch.cuda.synchronize()
            assert (idx.cpu().numpy() == np.arange(ns, ns + k)[None, :]).all()
            bk, _ = st.export(0)
            assert torch.equal(bk[:, ns + gh * gw:], kk[ns:ns + k].permute(1, 0, 2).cpu())
        finally:
            st.close()


def test_fused_host_entry_point_and_errors():
    H, ns, gh, gw, k = 16, 5, 37, 37, 14
    N = ns + gh * gw
    a = Stream(1, H, ns, gh, gw, budget=k, max_frames=4, seed=23)
    b = Stream(1, H, ns, gh, gw, budget=k, max_frames=4, seed=23)
    try:
        for t in range(1, 4):
            q, kk, v = a.inputs(0, t)
            o_d, s_d, _, _ = a.attend_admit(0, q, kk, v, k)
            hq, hk, hv = q.cpu().pin_memory(), kk.cpu().pin_memory(), v.cpu().pin_memory()
            ho = torch.empty_like(hq).pin_memory()
            hs = torch.empty(H, N, dtype=torch.float32).pin_memory()
            b.rm.attend_admit_host(0, hq, hk, hv, ho, hs, k)
            b.rm.synchronize()
            torch.cuda.synchronize()
            assert torch.equal(ho, o_d.cpu()) and torch.equal(hs, s_d.cpu())
        assert a.rm.memory_len(0) == b.rm.memory_len(0) == N + 2 * k
        q, kk, v = a.inputs(0, 4)
        out = torch.empty_like(q)
        sal = torch.empty(H, N, device="cuda")
        with pytest.raises(regmem.RegmemError) as e:
            a.rm.attend_admit(0, q, kk, v, out, sal, k + 1)
        assert e.value.status == regmem.ERR_ARG               # k above the budget
        a.rm.attend_frame(0, q, kk, v, out, sal)
        with pytest.raises(regmem.RegmemError) as e:
            a.rm.attend_admit(0, q, kk, v, out, sal, k)
        assert e.value.status == regmem.ERR_STATE             # attend pending
        a.rm.admit(0, 0)
        assert a.rm.memory_len(0) == N + 2 * k                # nothing appended by the refusals
        a.rm.synchronize()
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("pattern", ["duplicates", "constant", "spread"])
@pytest.mark.parametrize("k", [14, 32, 33])
def test_selection_on_crafted_saliency(pattern, k):
    """The admission selection against the oracle's sort on crafted saliency
    written between attend and admit (the library reads the caller's saliency
    buffer at admit time): many exact ties, a constant row, and a wide value
    range across 1369 candidates; k = 14 and 32 take the distributed list
    selection, k = 33 the single-block radix selection."""
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    st = Stream(1, H, ns, gh, gw, budget=k, max_frames=3, seed=24)
    g = torch.Generator().manual_seed(25)
    try:
        q, kk, v = st.inputs(0, 1)
        st.attend(0, q, kk, v)
        st.admit(0, k)
        q, kk, v = st.inputs(0, 2)
        out = torch.empty_like(q)
        sal = torch.empty(H, N, device="cuda")
        st.rm.attend_frame(0, q, kk, v, out, sal)
        if pattern == "duplicates":
            crafted = torch.randint(0, 6, (H, N), generator=g).float() * 0.25
        elif pattern == "constant":
            crafted = torch.full((H, N), 3.5)
        else:
            crafted = torch.exp(torch.randn(H, N, generator=g) * 8.0)
        sal.copy_(crafted.to("cuda"))
        idx = torch.full((H, k), -1, dtype=torch.int32, device="cuda")
        st.rm.admit(0, k, idx)
        torch.cuda.synchronize()
        c = crafted.double().numpy()
        for h in range(H):
            assert list(idx[h].cpu().numpy()) == orc.topk_admission(c[h], ns, k), f"head {h}"
    finally:
        st.close()


def test_profile_counters_events_and_launch_clock():
    """regmem_profile_*: launch counters, event timing of every launch
    (time_attention = 1) and the attention's launch clock agree with each
    other; with profiling off nothing is timed."""
    H, ns, gh, gw, k = 16, 5, 37, 37, 14
    st = Stream(2, H, ns, gh, gw, budget=k, max_frames=6, seed=33)
    try:
        st.rm.set_overlap(1)
        for layer in range(2):
            st.attend_admit(layer, *st.inputs(layer, 1), k)
        st.rm.profile_enable(1)
        for t in (2, 3, 4):
            for layer in range(2):
                st.attend_admit(layer, *st.inputs(layer, t), k)
        p = st.rm.profile_read()
        assert p.launches_attention == 6 and p.launches_saliency == 6
        assert p.launches_combine == (6 if p.attention_ctas > 1 else 0)
        assert p.attention_timed == 6 and p.attention_clocked == 6
        assert p.attention_clock_flops == pytest.approx(p.attention_flops, rel=1e-12)
        L = [ns + gh * gw + (ns + gh * gw) + (t - 2) * k for t in (2, 3, 4)]
        assert p.attention_flops == pytest.approx(sum(4.0 * (ns + gh * gw) * l * 64 * H * 2 for l in L))
        # the clock brackets the kernel after its dependency wait; the events
        # also hold its launch: clock <= events, and of the same order
        assert 0 < p.attention_clock_ms <= 1.05 * p.attention_ms + 0.005
        assert p.attention_clock_ms >= 0.3 * p.attention_ms
        st.rm.profile_enable(0)
        for layer in range(2):
            st.attend_admit(layer, *st.inputs(layer, 5), k)
        p = st.rm.profile_read()
        assert p.launches_attention == 2 and p.attention_timed == 0 and p.attention_clocked == 0
        assert p.attention_clock_ms == 0.0
        st.rm.synchronize()
    finally:
        st.close()
