"""Shared helpers for the parity tests: run the CUDA path through the C ABI
and the fp64 oracle on the same bf16 inputs, and compare with the tolerances
the parity contract fixes."""
from __future__ import annotations

import numpy as np
import torch

import oracle as orc
from paper_2609_23286_gb300 import regmem, synth

# Tolerances (element-wise):
#   O (bf16 result, fp32 accumulation): |d| <= 2e-2 + 1e-2 |ref|
#   LSE (fp32): |d| <= 1e-3
#   saliency (fp32): |d| <= 1e-3 |ref| + 1e-6   (1e-6 absolute floor: a sum of
#       at most a few hundred probabilities in fp32 cannot resolve less)
#   O, element-wise error bound of the arithmetic (checked as well where the
#   test has O_abs = softmax(Z) |V|, the oracle run on |V|):
#       |d| <= 2^-8 |ref| + (2^-7 + 2^-10) O_abs + 1e-6
#   -- 2^-8 |ref|: O rounded to bf16 (RNE, 8 significant bits);
#   -- 2^-8 O_abs: P rounded to bf16 before P V (each term p_j v_j off by at
#      most 2^-8 |p_j v_j|, summed and normalised: at most 2^-8 O_abs);
#   -- 2^-8 O_abs: a split unit's normalised piece partials O_p stored in bf16
#      (|O_p| <= the piece's softmax |V|, whose weighted sum is O_abs);
#   -- 2^-10 O_abs + 1e-6: fp32 accumulation over up to ~3e4 keys and exp2.
#   Unlike the contract's 2e-2 absolute term, this does not loosen where |O|
#   is small (long banks average thousands of values), so a dropped or
#   doubled key tile cannot hide behind it.
O_ATOL, O_RTOL = 2e-2, 1e-2
O_BOUND_REF, O_BOUND_ABS, O_BOUND_FLOOR = 2.0 ** -8, 2.0 ** -7 + 2.0 ** -10, 1e-6
LSE_ATOL = 1e-3
S_RTOL, S_ATOL = 1e-3, 1e-6


def to64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu").double().numpy()


def check_o(o_gpu: torch.Tensor, o_ref: np.ndarray, what="", o_abs: np.ndarray | None = None):
    """Contract tolerance on every element; with o_abs also the arithmetic's
    own bound.  Returns (max |d|, max |d| / bound or None)."""
    d = np.abs(to64(o_gpu) - o_ref)
    bad = d > O_ATOL + O_RTOL * np.abs(o_ref)
    assert not bad.any(), f"{what} O: {bad.sum()} elements off, max |d| {d.max():.3e}"
    ratio = None
    if o_abs is not None:
        bound = O_BOUND_REF * np.abs(o_ref) + O_BOUND_ABS * o_abs + O_BOUND_FLOOR
        r = d / bound
        ratio = float(r.max())
        assert ratio <= 1.0, (f"{what} O: {(r > 1).sum()} elements beyond the bf16 error bound, "
                              f"max |d| / bound {ratio:.3f}")
    return float(d.max()), ratio


def o_abs_frame(q64, k64, v64, bank_k, bank_v, scale, qidx=(0,)):
    """O_abs = softmax(Z) |V| for every (token, head): the oracle's attention
    of the same queries and keys over |V| (the quantity the O error bound
    scales with)."""
    return orc.attend_frame(q64, k64, np.abs(v64), bank_k, [np.abs(b) for b in bank_v], scale,
                            list(qidx))["O"]


def check_lse(lse_gpu: torch.Tensor, lse_ref: np.ndarray, what=""):
    d = np.abs(to64(lse_gpu) - lse_ref)
    assert (d <= LSE_ATOL).all(), f"{what} LSE: max |d| {d.max():.3e}"
    return float(d.max())


def check_saliency(s_gpu: torch.Tensor, s_ref: np.ndarray, what=""):
    g = to64(s_gpu)
    d = np.abs(g - s_ref)
    bad = d > S_RTOL * np.abs(s_ref) + S_ATOL
    assert not bad.any(), f"{what} saliency: {bad.sum()} off, max rel {(d / (np.abs(s_ref) + 1e-30)).max():.3e}"
    return float((d / (np.abs(s_ref) + 1e-12)).max())


def check_indices(idx_gpu: np.ndarray, s_gpu: np.ndarray, s_ref: np.ndarray, n_special: int,
                  k: int, n_sampled: int, candidates="patch"):
    """(1) bit-exact: the GPU's choice equals the oracle's top-k taken on the
    GPU's own fp32 saliency (same precision decides the integer); (2) against
    the oracle's fp64 saliency, any differing index lies within the tie band
    |S_j - S_(k)| <= 1e-3 S_(k) + 1e-7 |Q~| of the k-th value."""
    H = idx_gpu.shape[0]
    for h in range(H):
        same_prec = orc.topk_admission(s_gpu[h], n_special, k, candidates)
        assert list(idx_gpu[h]) == same_prec, f"head {h}: {list(idx_gpu[h])} vs {same_prec}"
        ref = orc.topk_admission(s_ref[h], n_special, k, candidates)
        if list(idx_gpu[h]) != ref:
            kth = sorted(s_ref[h][ref])[0]
            band = 1e-3 * kth + 1e-7 * n_sampled
            for j in set(idx_gpu[h]) ^ set(ref):
                assert abs(s_ref[h][j] - kth) <= band, f"head {h} index {j} outside tie band"


class Stream:
    """One regulated stream on the GPU (through the C ABI) with inputs drawn
    by the shared seeded generator."""

    def __init__(self, layers, heads, n_special, grid_h, grid_w, budget, max_frames, seed,
                 ds=2, device="cuda", candidates=0):
        self.L, self.H, self.ns, self.gh, self.gw = layers, heads, n_special, grid_h, grid_w
        self.N = n_special + grid_h * grid_w
        self.budget, self.seed, self.ds, self.device = budget, seed, ds, device
        self.rm = regmem.RegMem(layers, heads, 64, budget)
        self.rm.set_frame(n_special, grid_h, grid_w, ds=ds, max_frames=max_frames,
                          candidates=candidates)
        self.rm.set_stream(torch.cuda.current_stream())
        self.scales = [synth.key_scale(seed, l, self.N, device=device) for l in range(layers)]

    def inputs(self, layer, frame):
        return synth.frame_qkv(self.seed, layer, frame, self.N, self.H, 64, device=self.device,
                               scale_cache=self.scales[layer])

    def attend(self, layer, q, k, v):
        out = torch.empty_like(q)
        sal = torch.empty(self.H, self.N, dtype=torch.float32, device=q.device)
        self.rm.attend_frame(layer, q, k, v, out, sal)
        lse = torch.empty(self.H, self.N, dtype=torch.float32, device=q.device)
        self.rm.copy_lse(lse)
        return out, sal, lse

    def admit(self, layer, k):
        idx = torch.full((self.H, max(k, 1)), -1, dtype=torch.int32, device="cuda")
        self.rm.admit(layer, k, idx)
        return idx[:, :k]

    def attend_admit(self, layer, q, k, v, kk):
        """The one-call step (attention, saliency and admission of kk rows)."""
        out = torch.empty_like(q)
        sal = torch.empty(self.H, self.N, dtype=torch.float32, device=q.device)
        idx = torch.full((self.H, max(kk, 1)), -1, dtype=torch.int32, device="cuda")
        self.rm.attend_admit(layer, q, k, v, out, sal, kk, idx)
        lse = torch.empty(self.H, self.N, dtype=torch.float32, device=q.device)
        self.rm.copy_lse(lse)
        return out, sal, lse, idx[:, :kk]

    def export(self, layer):
        n = self.rm.memory_len(layer)
        bk = torch.empty(self.H, n, 64, dtype=torch.bfloat16)
        bv = torch.empty(self.H, n, 64, dtype=torch.bfloat16)
        if n:
            self.rm.export_bank(layer, bk, bv)
        return bk, bv

    def close(self):
        self.rm.close()
