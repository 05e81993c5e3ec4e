"""Pins for the fp64 oracle: checks against things other than the oracle
itself -- brute-force loops, a library attention routine, closed forms and
invariants the paper fixes.  Each ``check_*`` helper is also run against a
deliberately broken copy of the oracle (``test_mutations_are_caught``) to show
that a plausible mistake fails at least one pin.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand(shape, rng, scale=1.0):
    return rng.standard_normal(shape) * scale


# --------------------------------------------------------------------------
# independent references used by the pins
# --------------------------------------------------------------------------

def brute_attention(q, kc, vc, scale):
    """Pure-Python loops: softmax attention of Eq. 2 written out element by
    element, with the LSE defined as log of the plain sum of exponentials."""
    n, d = len(q), len(q[0])
    L = len(kc)
    O, LSE, P = [], [], []
    for i in range(n):
        z = [sum(q[i][e] * kc[j][e] for e in range(d)) * scale for j in range(L)]
        tot = sum(math.exp(x) for x in z)
        lse = math.log(tot)
        p = [math.exp(x) / tot for x in z]
        O.append([sum(p[j] * vc[j][e] for j in range(L)) for e in range(d)])
        LSE.append(lse)
        P.append(p)
    return np.array(O), np.array(LSE), np.array(P)


def rank_topk(s, lo, k):
    """Top-k by ranks: token j is chosen iff fewer than k candidates beat it,
    where i beats j if s_i > s_j, or s_i == s_j and i < j."""
    chosen = []
    for j in range(lo, len(s)):
        beaten = sum(1 for i in range(lo, len(s))
                     if (s[i] > s[j]) or (s[i] == s[j] and i < j))
        if beaten < k:
            chosen.append(j)
    return chosen


# --------------------------------------------------------------------------
# pins, written as reusable checks (module = the oracle under test)
# --------------------------------------------------------------------------

def check_bruteforce(mod):
    rng = np.random.default_rng(11)
    d, n, m = 4, 5, 3
    q = rand((n, d), rng)
    kc = rand((m + n, d), rng)
    vc = rand((m + n, d), rng)
    o, lse, z, p = mod.attend_head(q, kc, vc, 0.5)
    bo, blse, bp = brute_attention(q.tolist(), kc.tolist(), vc.tolist(), 0.5)
    return (np.allclose(o, bo, rtol=1e-12, atol=1e-12)
            and np.allclose(lse, blse, rtol=1e-12, atol=1e-12)
            and np.allclose(p, bp, rtol=1e-12, atol=1e-14))


def check_sdpa(mod):
    """torch's scaled_dot_product_attention in float64 on CPU (scale 1/sqrt(d)
    is the library default, matching Eq. 2's 1/sqrt(D/H))."""
    rng = np.random.default_rng(12)
    H, N, M, d = 3, 9, 6, 8
    q = rand((N, H, d), rng)
    k = rand((N, H, d), rng)
    v = rand((N, H, d), rng)
    bk = [rand((M, d), rng) for _ in range(H)]
    bv = [rand((M, d), rng) for _ in range(H)]
    res = mod.attend_frame(q, k, v, bk, bv, 1.0 / math.sqrt(d), [0, 2])
    kc = torch.stack([torch.from_numpy(np.concatenate([bk[h], k[:, h]])) for h in range(H)])
    vc = torch.stack([torch.from_numpy(np.concatenate([bv[h], v[:, h]])) for h in range(H)])
    qt = torch.from_numpy(q).permute(1, 0, 2).contiguous()
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kc, vc).permute(1, 0, 2).numpy()
    # LSE via torch.logsumexp of the explicitly formed logits
    logits = torch.einsum("hnd,hld->hnl", qt, kc) / math.sqrt(d)
    ref_lse = torch.logsumexp(logits, dim=-1).numpy()
    return (np.allclose(res["O"], ref, rtol=1e-12, atol=1e-12)
            and np.allclose(res["LSE"], ref_lse, rtol=1e-12, atol=1e-12))


def check_closed_form(mod):
    """Two keys whose logits differ by ln 3: LSE = ln(e^0 + e^{ln 3}) = ln 4,
    P = (1/4, 3/4), O = (v1 + 3 v2)/4; saliency of key 2 from one query = 3/4."""
    d = 4
    scale = 0.5
    q = np.array([[1.0, 0, 0, 0]])
    kc = np.array([[0.0, 0, 0, 0], [2 * math.log(3), 0, 0, 0]])
    vc = np.array([[1.0, 2, 3, 4], [5.0, 6, 7, 8]])
    o, lse, z, p = mod.attend_head(q, kc, vc, scale)
    s = mod.saliency_lse(z, lse, 1, [0])
    return (abs(lse[0] - math.log(4)) < 1e-14
            and np.allclose(p[0], [0.25, 0.75], atol=1e-15)
            and np.allclose(o[0], (vc[0] + 3 * vc[1]) / 4, atol=1e-14)
            and abs(s[0] - 0.75) < 1e-15)


def check_uniform(mod):
    """K = 0 everywhere: every logit is 0, so softmax is uniform over the L
    attended keys: O = mean of V, LSE = ln L, S_j = |Q~| / L."""
    rng = np.random.default_rng(13)
    H, N, M, d = 2, 21, 7, 4   # 1 special + 4x5 grid
    q = rand((N, H, d), rng)
    k = np.zeros((N, H, d))
    v = rand((N, H, d), rng)
    bk = [np.zeros((M, d)) for _ in range(H)]
    bv = [rand((M, d), rng) for _ in range(H)]
    qidx = mod.sampled_query_tokens(1, 4, 5, 2)
    res = mod.attend_frame(q, k, v, bk, bv, 0.5, qidx)
    L = M + N
    ok = True
    for h in range(H):
        mean_v = np.concatenate([bv[h], v[:, h]]).mean(axis=0)
        ok &= np.allclose(res["O"][:, h], mean_v[None, :], atol=1e-13)
        ok &= np.allclose(res["LSE"][h], math.log(L), atol=1e-13)
        ok &= np.allclose(res["S"][h], len(qidx) / L, atol=1e-14)
    return bool(ok)


def check_mass(mod):
    """Softmax rows sum to 1; the sampled rows' total mass over all L keys is
    |Q~|; at frame 1 (M = 0) the saliency alone sums to |Q~|, afterwards to
    less (the memory takes the rest), and direct == LSE route."""
    rng = np.random.default_rng(14)
    H, d = 2, 8
    gh, gw, ns = 5, 6, 2
    N = ns + gh * gw
    qidx = mod.sampled_query_tokens(ns, gh, gw, 2)
    q = rand((N, H, d), rng)
    k = rand((N, H, d), rng)
    v = rand((N, H, d), rng)
    ok = True
    for M in (0, 11):
        bk = [rand((M, d), rng) for _ in range(H)]
        bv = [rand((M, d), rng) for _ in range(H)]
        res = mod.attend_frame(q, k, v, bk, bv, 1 / math.sqrt(d), qidx)
        for h in range(H):
            kc = np.concatenate([bk[h], k[:, h]])
            vc = np.concatenate([bv[h], v[:, h]])
            _, _, _, p = mod.attend_head(q[:, h], kc, vc, 1 / math.sqrt(d))
            ok &= np.allclose(p.sum(axis=1), 1.0, atol=1e-13)
            ok &= abs(p[qidx].sum() - len(qidx)) < 1e-11
            tot = res["S"][h].sum()
            ok &= (abs(tot - len(qidx)) < 1e-11) if M == 0 else (tot < len(qidx) - 1e-6)
            ok &= np.allclose(res["S"][h], res["S_direct"][h], rtol=1e-12, atol=1e-15)
    return bool(ok)


def check_topk(mod):
    """Top-k against the rank definition, on ties and on random values."""
    ok = True
    s = np.array([9.0, 9.0, 1.0, 3.0, 3.0, 3.0, 0.5, 3.0, 2.0])
    ok &= mod.topk_admission(s, 2, 2) == [3, 4]           # tie cut: lower indices win
    ok &= mod.topk_admission(s, 2, 5) == [3, 4, 5, 7, 8]
    ok &= mod.topk_admission(s, 0, 3) == [0, 1, 3]
    ok &= mod.topk_admission(s, 2, 0) == []
    rng = np.random.default_rng(15)
    for _ in range(30):
        n = int(rng.integers(3, 25))
        vals = rng.integers(0, 6, size=n).astype(float)     # many ties
        lo = int(rng.integers(0, 3))
        kk = int(rng.integers(0, n - lo + 1))
        ok &= mod.topk_admission(vals, lo, kk) == rank_topk(vals, lo, kk)
    return bool(ok)


def check_sampled_queries(mod):
    """Sampled set of the Head-Specific Token Retention step, on grids drawn
    by hand: a 4x4 patch grid after 5 specials, 2x2 windows -> the top-left
    patch of each window: patches (0,0),(0,2),(2,0),(2,2) -> tokens
    5, 7, 13, 15.  A 3x5 grid keeps the partial edge windows: rows 0,2 and
    cols 0,2,4."""
    ok = mod.sampled_query_tokens(5, 4, 4, 2) == [5, 7, 13, 15]
    ok &= mod.sampled_query_tokens(1, 3, 5, 2) == [1, 3, 5, 11, 13, 15]
    ok &= mod.sampled_query_tokens(1, 3, 5, 2, ds_floor=True) == [1, 3]
    ok &= mod.sampled_query_tokens(0, 2, 3, 1) == [0, 1, 2, 3, 4, 5]
    ok &= len(mod.sampled_query_tokens(5, 37, 37, 2)) == 361
    ok &= len(mod.sampled_query_tokens(5, 37, 28, 2)) == 266
    ok &= len(mod.sampled_query_tokens(4, 8, 8, 2)) == 16
    ok &= len(mod.sampled_query_tokens(5, 37, 37, 3)) == 13 * 13
    ok &= len(mod.sampled_query_tokens(5, 37, 37, 4)) == 10 * 10
    return bool(ok)


def check_stream(mod):
    """Eq. 4 - Eq. 6 on a short stream: frame 1 is stored whole (anchor),
    memory grows by exactly k per later frame, appended rows are bit-identical
    copies of the chosen frame rows, and k = 0 leaves the memory unchanged."""
    rng = np.random.default_rng(16)
    L_, H, d, ns, gh, gw = 2, 2, 4, 1, 3, 4
    N = ns + gh * gw
    st = mod.OracleStream(L_, H, d, ns, gh, gw, ds=2)
    ok = True
    for t in range(1, 7):
        for layer in range(L_):
            kk = 0 if layer == 1 else 2
            q, k, v = rand((N, H, d), rng), rand((N, H, d), rng), rand((N, H, d), rng)
            before = [st.bank_k[layer][h].copy() for h in range(H)]
            res = st.step(layer, q, k, v, kk)
            for h in range(H):
                rows = res["idx"][h]
                ok &= np.array_equal(st.bank_k[layer][h][len(before[h]):], k[rows, h])
                ok &= np.array_equal(st.bank_v[layer][h][-len(rows):] if len(rows) else
                                     np.zeros((0, d)), v[rows, h])
                ok &= np.array_equal(st.bank_k[layer][h][:len(before[h])], before[h])
            expect = N + (t - 1) * kk
            ok &= st.memory_len(layer) == expect
    return bool(ok)


def check_planted_key(mod):
    """A frame key aligned with every query and with a large norm gets most
    of the attention mass of every sampled query, so it must be admitted in
    every head."""
    rng = np.random.default_rng(17)
    H, d, ns, gh, gw = 3, 8, 5, 6, 6
    N = ns + gh * gw
    st = mod.OracleStream(1, H, d, ns, gh, gw, ds=2)
    q0, k0, v0 = rand((N, H, d), rng), rand((N, H, d), rng), rand((N, H, d), rng)
    st.step(0, q0, k0, v0, 1)
    q = rand((N, H, d), rng) * 0.1
    q[:, :, 0] += 1.0
    k = rand((N, H, d), rng)
    k[23, :, :] = 0.0
    k[23, :, 0] = 40.0
    res = st.step(0, q, k, rand((N, H, d), rng), 1)
    return bool(np.all(res["idx"][:, 0] == 23))


def check_permutation(mod):
    """Attention is a set operation over keys: permuting the memory rows (the
    same permutation for K and V) leaves O and LSE unchanged."""
    rng = np.random.default_rng(18)
    N, M, d = 6, 9, 4
    q = rand((N, d), rng)
    kc = rand((M + N, d), rng)
    vc = rand((M + N, d), rng)
    perm = np.concatenate([rng.permutation(M), np.arange(M, M + N)])
    o1, l1, _, _ = mod.attend_head(q, kc, vc, 0.5)
    o2, l2, _, _ = mod.attend_head(q, kc[perm], vc[perm], 0.5)
    return np.allclose(o1, o2, atol=1e-13) and np.allclose(l1, l2, atol=1e-13)


def check_shared_topk(mod):
    """Selection without head-specific retention (Sec. 4.5, Table 4): the
    chosen set equals the rank-based top-k of the plain head average written
    out in Python (ties included); with one head it is the per-head choice;
    and on a crafted case where each head prefers a different token, the
    shared choice is the token both heads rank second."""
    rng = np.random.default_rng(21)
    ok = True
    for trial in range(6):
        H, N, ns, k = 3, 12, 2, 1 + trial % 4
        s = np.round(rng.random((H, N)) * 4) / 4  # coarse values: many ties
        mean = [sum(float(s[h][j]) for h in range(H)) / H for j in range(N)]
        ok &= mod.topk_admission_shared(s, ns, k) == rank_topk(mean, ns, k)
        ok &= mod.topk_admission_shared(s[:1], ns, k) == mod.topk_admission(s[0], ns, k)
    crafted = np.zeros((2, 8))
    crafted[0, 3], crafted[1, 5] = 10.0, 10.0  # head 0 wants 3, head 1 wants 5
    crafted[:, 6] = 9.0                        # both rank token 6 second
    ok &= mod.topk_admission_shared(crafted, 1, 1) == [6]
    ok &= [mod.topk_admission(crafted[h], 1, 1) for h in range(2)] == [[3], [5]]
    # a stream with shared admission: every head appends the same tokens
    H, d, ns_, gh, gw = 2, 4, 1, 3, 3
    st = mod.OracleStream(1, H, d, ns_, gh, gw)
    Nn = ns_ + gh * gw
    for t in range(1, 5):
        q, kx, v = rand((Nn, H, d), rng), rand((Nn, H, d), rng), rand((Nn, H, d), rng)
        st.attend(0, q, kx, v)
        idx = st.admit(0, 2, shared=True)
        ok &= bool(np.all(idx == idx[0]))
        ok &= st.memory_len(0) == Nn + (t - 1) * 2
    return bool(ok)


def check_retention(mod):
    """k = floor(gamma N) (Eq. 6): gamma = 0.01 at N = 1374 keeps 13 tokens,
    gamma = 0.1 keeps 137; the paper's layer split (Sec. 4.1) makes layers
    11-17 of 24 (1-based) admit and the other 17 keep only the anchor; and
    the unregulated memory (every token admitted every frame) holds t N rows
    after t frames, the frames' rows in order."""
    ok = mod.retention_k(0.01, 1374) == 13 and mod.retention_k(0.1, 1374) == 137
    ok &= mod.retention_k(0.001, 1374) == 1 and mod.retention_k(1.0, 69) == 69
    lk = mod.paper_layer_k(24, 14)
    ok &= [i + 1 for i, x in enumerate(lk) if x == 14] == list(range(11, 18))
    ok &= sum(1 for x in lk if x == 0) == 17
    rng = np.random.default_rng(22)
    H, d, ns_, gh, gw = 2, 4, 1, 2, 3
    Nn = ns_ + gh * gw
    st = mod.OracleStream(1, H, d, ns_, gh, gw, candidates="all")
    ks = []
    for t in range(1, 5):
        q, kx, v = rand((Nn, H, d), rng), rand((Nn, H, d), rng), rand((Nn, H, d), rng)
        st.attend(0, q, kx, v)
        st.admit(0, Nn)
        ks.append(kx)
        ok &= st.memory_len(0) == t * Nn
    for h in range(H):
        ok &= np.array_equal(st.bank_k[0][h], np.concatenate([x[:, h] for x in ks]))
    return bool(ok)


PINS = [check_bruteforce, check_sdpa, check_closed_form, check_uniform, check_mass,
        check_topk, check_sampled_queries, check_stream, check_planted_key,
        check_permutation, check_shared_topk, check_retention]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    assert pin(orc)


def test_bf16_widening_exact():
    vals = torch.tensor([1.0, -2.5, 3.140625, 1e-3, -65280.0, 0.0], dtype=torch.bfloat16)
    bits = vals.view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(orc.bf16_bits_to_f64(bits), vals.double().numpy())


def test_golden_closed_form_fixture():
    """Hand-derived closed-form example stored as text (tests/golden)."""
    with open(os.path.join(GOLDEN, "closed_form_two_keys.json")) as f:
        g = json.load(f)
    o, lse, z, p = orc.attend_head(np.array(g["q"]), np.array(g["k"]), np.array(g["v"]),
                                   g["scale"])
    s = orc.saliency_lse(z, lse, g["m_rows"], g["qidx"])
    assert np.allclose(lse, g["lse"], atol=1e-12)
    assert np.allclose(o, g["o"], atol=1e-12)
    assert np.allclose(s, g["saliency"], atol=1e-12)


# --------------------------------------------------------------------------
# planted mistakes: a broken oracle must fail at least one pin
# --------------------------------------------------------------------------

class _Mutant:
    """A copy of the oracle module's namespace with one function replaced."""

    def __init__(self, **over):
        for name in dir(orc):
            if not name.startswith("__"):
                setattr(self, name, getattr(orc, name))
        for k, v in over.items():
            setattr(self, k, v)


def _attend_head_wrong_scale(q, kc, vc, scale):
    return orc.attend_head(q, kc, vc, scale * 2)


def _attend_head_kv_swapped(q, kc, vc, scale):
    return orc.attend_head(q, vc, kc, scale)


def _attend_head_no_max_in_lse(q, kc, vc, scale):
    o, lse, z, p = orc.attend_head(q, kc, vc, scale)
    return o, lse - z.max(axis=1), z, p


def _saliency_renormalised(z, lse, m_rows, qidx):
    qi = np.asarray(qidx)
    a = np.exp(z[qi, m_rows:])
    return (a / a.sum(axis=1, keepdims=True)).sum(axis=0)


def _saliency_off_by_one(z, lse, m_rows, qidx):
    return orc.saliency_lse(z, lse, m_rows - 1 if m_rows else 1, qidx)[: z.shape[1] - m_rows]


def _attend_frame_drops_memory(q, k, v, bank_k, bank_v, scale, qidx):
    h = len(bank_k)
    d = q.shape[2]
    return orc.attend_frame(q, k, v, [np.zeros((0, d))] * h, [np.zeros((0, d))] * h,
                            scale, qidx)


def _topk_ties_high(s, n_special, k, candidates="patch"):
    lo = n_special if candidates == "patch" else 0
    order = sorted(range(lo, len(s)), key=lambda j: (-float(s[j]), -j))
    return sorted(order[:k])


def _topk_includes_specials(s, n_special, k, candidates="patch"):
    return orc.topk_admission(s, 0, k)


def _sampled_transposed(n_special, grid_h, grid_w, ds, ds_floor=False):
    return orc.sampled_query_tokens(n_special, grid_w, grid_h, ds, ds_floor)


def _shared_first_head(s, n_special, k, candidates="patch"):
    return orc.topk_admission(np.asarray(s)[0], n_special, k, candidates)


def _shared_max_over_heads(s, n_special, k, candidates="patch"):
    return orc.topk_admission(np.asarray(s).max(axis=0), n_special, k, candidates)


def _retention_rounds(gamma, n_tokens):
    return int(round(gamma * n_tokens))


def _layer_split_shifted(layers, k):
    return [k if 10 <= layer + 1 <= 16 else 0 for layer in range(layers)]


MUTANTS = {
    "shared_from_first_head": dict(topk_admission_shared=_shared_first_head),
    "shared_max_not_mean": dict(topk_admission_shared=_shared_max_over_heads),
    "retention_rounded": dict(retention_k=_retention_rounds),
    "layer_split_shifted": dict(paper_layer_k=_layer_split_shifted),
    "wrong_scale": dict(attend_head=_attend_head_wrong_scale),
    "k_v_swapped": dict(attend_head=_attend_head_kv_swapped),
    "lse_missing_max": dict(attend_head=_attend_head_no_max_in_lse),
    "saliency_renormalised_over_frame": dict(saliency_lse=_saliency_renormalised),
    "saliency_column_offset": dict(saliency_lse=_saliency_off_by_one),
    "memory_dropped": dict(attend_frame=_attend_frame_drops_memory),
    "ties_to_higher_index": dict(topk_admission=_topk_ties_high),
    "specials_as_candidates": dict(topk_admission=_topk_includes_specials),
    "grid_transposed": dict(sampled_query_tokens=_sampled_transposed),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutations_are_caught(name, monkeypatch):
    mut = _Mutant(**MUTANTS[name])
    # OracleStream / attend_frame call module-level functions, so also patch
    # the real module for the duration of the check.
    import oracle.regmem_oracle as real
    for k, v in MUTANTS[name].items():
        monkeypatch.setattr(real, k, v)
    failed = []
    for pin in PINS:
        try:
            ok = pin(mut)
        except Exception:
            ok = False
        if not ok:
            failed.append(pin.__name__)
    assert failed, f"mutant {name} passed every pin"
