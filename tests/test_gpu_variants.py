"""Parity of the variants the paper studies around its default configuration,
through the C ABI against the fp64 oracle:

* selection without head-specific retention (Sec. 4.5, Table 4):
  regmem_admit_shared;
* the unregulated full-KV memory the paper compares against (every frame's
  N rows kept; candidates = all tokens, k = N);
* the layer-specific allocation of Sec. 4.1 (Eq. 5 layers keep only the
  anchor, Eq. 6 layers admit k per frame);
* bank export / import as checkpoint and resume of a stream.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from helpers import Stream, check_indices, check_lse, check_o, check_saliency, to64

pytestmark = pytest.mark.gpu


def shared_choice_fp32(sal_gpu: torch.Tensor, n_special: int, k: int) -> list[int]:
    """The integer decision in the kernel's precision: fp32 head sum of the
    GPU's own fp32 saliency, heads added in ascending order."""
    s = sal_gpu.detach().cpu().numpy().astype(np.float32)
    acc = np.zeros(s.shape[1], dtype=np.float32)
    for h in range(s.shape[0]):
        acc = (acc + s[h]).astype(np.float32)
    return orc.topk_admission(acc.astype(np.float64), n_special, k)


@pytest.mark.parametrize("kk", [1, 14, 40])
def test_shared_admission_matches_oracle(kk):
    """Head-averaged admission on frame 3 of a VGGT-shaped stream: the chosen
    set equals the fp32 head-sum ranking of the GPU's saliency, differs from
    the oracle's fp64 head-mean ranking only inside the tie band, and every
    head's bank receives the same rows."""
    H, ns, gh, gw = 16, 5, 37, 37
    st = Stream(1, H, ns, gh, gw, budget=kk, max_frames=4, seed=31)
    ref = orc.OracleStream(1, H, 64, ns, gh, gw)
    try:
        for t in (1, 2, 3):
            q, k, v = st.inputs(0, t)
            out, sal, lse = st.attend(0, q, k, v)
            idx = torch.full((kk,), -1, dtype=torch.int32, device="cuda")
            st.rm.admit_shared(0, kk, idx)
            torch.cuda.synchronize()
            r = ref.attend(0, to64(q), to64(k), to64(v))
            check_o(out, r["O"], f"t={t}")
            check_lse(lse, r["LSE"], f"t={t}")
            check_saliency(sal, r["S"], f"t={t}")
            if t == 1:
                ref.admit(0, kk)
                continue
            gi = idx.cpu().numpy().astype(np.int64)
            assert list(gi) == shared_choice_fp32(sal, ns, kk)
            want = orc.topk_admission_shared(r["S"], ns, kk)
            if list(gi) != want:
                mean = r["S"].mean(axis=0)
                kth = sorted(mean[want])[0]
                for j in set(gi) ^ set(want):
                    assert abs(mean[j] - kth) <= 1e-3 * kth + 1e-7 * len(ref.qidx)
            ref.admit(0, kk, indices=np.tile(gi, (H, 1)))
            M = st.N + (t - 2) * kk
            bk, bv = st.export(0)
            assert bk.shape[1] == M + kk
            for h in range(H):
                assert torch.equal(bk[h, M:], k[gi, h].cpu())
                assert torch.equal(bv[h, M:], v[gi, h].cpu())
    finally:
        st.close()


@pytest.mark.parametrize("overlap,kk", [(0, 14), (1, 14), (1, 1), (1, 32), (1, 33)])
def test_one_call_shared_admission_matches_two_calls(overlap, kk):
    """regmem_attend_admit_shared (saliency and head-averaged selection on the
    side stream when overlap is on; fused into the saliency kernel for k <= 32,
    the separate selection kernel above) against regmem_attend_frame +
    regmem_admit_shared on another handle: O, saliency, the chosen tokens and
    every layer's bank bit for bit, over the anchor and four admitted frames of
    two layers."""
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    a = Stream(2, H, ns, gh, gw, budget=kk, max_frames=6, seed=35)
    b = Stream(2, H, ns, gh, gw, budget=kk, max_frames=6, seed=35)
    try:
        a.rm.set_overlap(overlap)
        for t in range(1, 6):
            for l in range(2):
                q, k, v = a.inputs(l, t)
                oa, sa = torch.empty_like(q), torch.empty(H, N, dtype=torch.float32, device=q.device)
                ia = torch.full((kk,), -1, dtype=torch.int32, device="cuda")
                a.rm.attend_admit_shared(l, q, k, v, oa, sa, kk, ia)
                ob, sb, _ = b.attend(l, q, k, v)
                ib = torch.full((kk,), -1, dtype=torch.int32, device="cuda")
                b.rm.admit_shared(l, kk, ib)
                a.rm.synchronize()
                b.rm.synchronize()
                assert torch.equal(oa, ob) and torch.equal(sa, sb), (t, l)
                if t > 1:
                    assert torch.equal(ia, ib), (t, l)
                assert a.rm.memory_len(l) == b.rm.memory_len(l) == N + (t - 1) * kk
        for l in range(2):
            ka, va = a.export(l)
            kb, vb = b.export(l)
            assert torch.equal(ka, kb) and torch.equal(va, vb)
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("H,ns,gh,gw,frames", [(2, 5, 8, 8, 6), (16, 5, 37, 37, 3)])
def test_unregulated_full_kv_stream(H, ns, gh, gw, frames):
    """The full-KV memory: candidates = all tokens and k = N keep every frame
    whole (a plain copy, nothing ranked); |M_t| = t N and the banks equal the
    frames' rows in order; attention over the growing memory matches the
    oracle frame by frame."""
    N = ns + gh * gw
    st = Stream(1, H, ns, gh, gw, budget=N, max_frames=frames, seed=32, candidates=1)
    ref = orc.OracleStream(1, H, 64, ns, gh, gw, candidates="all")
    try:
        for t in range(1, frames + 1):
            q, k, v = st.inputs(0, t)
            out, sal, lse, idx = st.attend_admit(0, q, k, v, N)
            torch.cuda.synchronize()
            r = ref.attend(0, to64(q), to64(k), to64(v))
            ref.admit(0, N)
            check_o(out, r["O"], f"t={t}")
            check_lse(lse, r["LSE"], f"t={t}")
            check_saliency(sal, r["S"], f"t={t}")
            assert st.rm.memory_len(0) == ref.memory_len(0) == t * N
            if t > 1:
                assert np.array_equal(idx.cpu().numpy(), np.tile(np.arange(N), (H, 1)))
        bk, bv = st.export(0)
        for h in range(H):
            assert np.array_equal(bk[h].double().numpy(), ref.bank_k[0][h])
            assert np.array_equal(bv[h].double().numpy(), ref.bank_v[0][h])
    finally:
        st.close()


def test_unregulated_end_size_sampled_rows():
    """The largest memory of the configurations: frame 200 of the unregulated
    stream attends the 199 whole frames before it (273,426 bank rows per
    head, 1.1 GB of K/V over 16 heads).  That launch runs in two phases, with
    every unit spread over the whole grid.  O and LSE are checked on sampled
    query rows of every head, the saliency on two heads (the oracle
    materialises their 361 x 274,800 logits).  The admission of all N
    candidates then fills the capacity exactly."""
    H, ns, gh, gw = 16, 5, 37, 37
    N = ns + gh * gw
    M = 199 * N
    st = Stream(1, H, ns, gh, gw, budget=N, max_frames=200, seed=33, candidates=1)
    try:
        g = torch.Generator().manual_seed(12)
        bk = (torch.randn(H, M, 64, generator=g)
              * torch.exp(0.5 * torch.randn(1, M, 1, generator=g))).to(torch.bfloat16)
        bv = torch.randn(H, M, 64, generator=g).to(torch.bfloat16)
        st.rm.import_bank(0, bk, bv, M)
        q, k, v = st.inputs(0, 200)
        out, sal, lse = st.attend(0, q, k, v)
        torch.cuda.synchronize()
        qi = orc.sampled_query_tokens(ns, gh, gw, 2)
        rows = sorted(set(list(range(0, N, 211)) + [N - 1, 127, 128]))
        q64, k64, v64 = to64(q), to64(k), to64(v)
        for h in range(H):
            kc = np.concatenate([bk[h].double().numpy(), k64[:, h]])
            vc = np.concatenate([bv[h].double().numpy(), v64[:, h]])
            o_r, l_r, _, _ = orc.attend_head(q64[rows, h], kc, vc, 1 / 8)
            o_a, _, _, _ = orc.attend_head(q64[rows, h], kc, np.abs(vc), 1 / 8)
            check_o(out[rows, h], o_r, f"h={h}", o_abs=o_a)
            check_lse(lse[h, rows], l_r, f"h={h}")
            if h in (0, H - 1):
                _, l_s, z_s, _ = orc.attend_head(q64[qi, h], kc, vc, 1 / 8)
                s_r = orc.saliency_lse(z_s, l_s, M, list(range(len(qi))))
                check_saliency(sal[h], s_r, f"h={h}")
                del z_s
        idx = st.admit(0, N)
        st.rm.synchronize()
        assert st.rm.memory_len(0) == M + N == 200 * N
        assert np.array_equal(idx.cpu().numpy(), np.tile(np.arange(N), (H, 1)))
    finally:
        st.close()


def test_paper_layer_split_stream():
    """Sec. 4.1 / Eq. 5-6 on a 24-layer stream of small frames: layers 11-17
    admit k per frame, the others keep only the anchor frame; outputs match
    the oracle and the memory lengths follow |M_t| = N + (t - 1) k_l."""
    L, H, ns, gh, gw, kk, frames = 24, 2, 5, 8, 8, 3, 4
    ks = orc.paper_layer_k(L, kk)
    st = Stream(L, H, ns, gh, gw, budget=kk, max_frames=frames, seed=33)
    ref = orc.OracleStream(L, H, 64, ns, gh, gw)
    try:
        for t in range(1, frames + 1):
            for layer in range(L):
                q, k, v = st.inputs(layer, t)
                out, sal, lse, idx = st.attend_admit(layer, q, k, v, ks[layer])
                torch.cuda.synchronize()
                r = ref.attend(layer, to64(q), to64(k), to64(v))
                if t == 1 or ks[layer] == 0:
                    ref.admit(layer, ks[layer])
                else:
                    gi = idx.cpu().numpy().astype(np.int64)
                    check_indices(gi, to64(sal), r["S"], ns, ks[layer], len(ref.qidx))
                    ref.admit(layer, ks[layer], indices=gi)
                if layer in (0, 10, 16, 17, 23):
                    check_o(out, r["O"], f"t={t} l={layer}")
                    check_saliency(sal, r["S"], f"t={t} l={layer}")
        for layer in range(L):
            assert st.rm.memory_len(layer) == st.N + (frames - 1) * ks[layer]
            bk, _ = st.export(layer)
            for h in range(H):
                assert np.array_equal(bk[h].double().numpy(), ref.bank_k[layer][h])
    finally:
        st.close()


def test_checkpoint_resume_is_bit_exact():
    """Export every layer's bank after frame 3, resume in a fresh handle from
    the imported banks, and run frames 4-5: outputs, saliency, admitted
    indices and final banks equal those of the uninterrupted stream bit for
    bit (the kernels are deterministic)."""
    L, H, ns, gh, gw, kk = 2, 16, 5, 37, 37, 14

    def run(frames, st, store):
        for t in frames:
            for layer in range(L):
                q, k, v = st.inputs(layer, t)
                out, sal, lse, idx = st.attend_admit(layer, q, k, v, kk)
                store[(t, layer)] = (out.cpu(), sal.cpu(), idx.cpu())
        torch.cuda.synchronize()

    whole, resumed = {}, {}
    a = Stream(L, H, ns, gh, gw, budget=kk, max_frames=5, seed=34)
    try:
        run(range(1, 6), a, whole)
        final_a = [a.export(layer) for layer in range(L)]
    finally:
        a.close()
    b = Stream(L, H, ns, gh, gw, budget=kk, max_frames=5, seed=34)
    try:
        run(range(1, 4), b, resumed)
        ckpt = [b.export(layer) for layer in range(L)]
    finally:
        b.close()
    c = Stream(L, H, ns, gh, gw, budget=kk, max_frames=5, seed=34)
    try:
        for layer, (bk, bv) in enumerate(ckpt):
            c.rm.import_bank(layer, bk, bv, bk.shape[1])
        run(range(4, 6), c, resumed)
        final_c = [c.export(layer) for layer in range(L)]
    finally:
        c.close()
    for key, (o, s, i) in whole.items():
        o2, s2, i2 = resumed[key]
        assert torch.equal(o, o2) and torch.equal(s, s2) and torch.equal(i, i2), key
    for (ka, va), (kc, vc) in zip(final_a, final_c):
        assert torch.equal(ka, kc) and torch.equal(va, vc)
