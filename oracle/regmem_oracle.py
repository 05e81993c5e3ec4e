"""Plain fp64 CPU oracle for regulated streaming attention (RegVGGT).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports, calls or links
this module: only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` may use it.  It shares no code with the CUDA library.

What it computes, per frame t, layer l and head h (paper notation):

* Eq. 2 / Eq. 3  --  temporal causal attention of the frame's queries over the
  regulated memory followed by the frame's own keys:
  ``O_t = softmax(Q_t [K_M ; K_t]^T / sqrt(D/H)) [V_M ; V_t]``, no mask inside
  the frame (causality is frame-granular).
* LSE-Saliency (Sec. 3.3, "FlashAttention-Compatible Saliency Estimation"):
  ``LSE_i = log sum_j exp(Z_ij)`` over every key actually attended, and
  ``A_ij = exp(Z_ij - LSE_i)`` for the current frame's keys.
* Head-Specific Token Retention (Sec. 3.3): the sampled query set is the
  top-left query of every non-overlapping ds x ds window of the patch grid and
  ``S_j = sum_{i in Q~} A_ij`` for each current-frame key j, per head.
* Eq. 6: per head, the k most salient candidate keys are appended to the
  memory; Eq. 4: the first frame's full K/V is the global anchor.
* Memory growth (Sec. 3.3, Layer-Specific Memory Allocation):
  ``|M_t| = |M_1| + (t - 1) k``, with ``k = floor(gamma N)`` on the layers
  that admit (Eq. 6) and k = 0 on the anchor-only layers (Eq. 5); Sec. 4.1
  makes layers 11-17 (1-based) the admitting ones.
* The selection without head-specific retention (the ablation of Sec. 4.5,
  Table 4): one set of k tokens for all heads, ranked by the saliency
  averaged over heads.
* The unregulated stream (the full-KV memory the paper compares against):
  every frame's N rows are kept, i.e. k = N over all tokens.

Everything is float64 and unblocked: the score matrix is materialised in full,
softmax is taken row by row as written, saliency is a plain column sum, and the
top-k is a full sort.  Library primitives used as single steps: ``@`` (matrix
product), ``np.exp``/``np.log`` and Python's ``sorted``.

Readings of points the paper leaves open (each one is a parameter or a
documented default here):

* LSE context: the keys actually attended, ``M_{t-1}`` followed by ``K_t``.
* A is the full-context softmax entry, not renormalised over ``K_t``.
* Saliency is produced for all N current-frame keys.
* Admission candidates are the patch tokens (index >= n_special) by default;
  ``candidates="all"`` admits from every token.
* Sampled queries are patch queries only; odd grids keep partial edge windows
  (stride-ds sampling, ceil(gh/ds) * ceil(gw/ds) queries); ``ds_floor=True``
  keeps only complete windows.
* Token order in a frame: special tokens first, then patches row-major.
* Frame 1 attends to itself only (M = 0) and then all N rows are stored.
* Frame t attends to M_{t-1}, never to its own admitted rows.
* Ties in saliency go to the lower token index; admitted rows are appended in
  ascending token index.

Parity status: every function here is pinned by the CPU tests in
``tests/test_oracle_pins.py`` (brute force, a library SDPA, closed forms and
invariants).  The two readings above about *which* tokens are candidates and
*which* queries are sampled are pinned only to the stated reading: no value
printed in the paper decides them.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "bf16_bits_to_f64",
    "sampled_query_tokens",
    "attend_head",
    "attend_frame",
    "saliency_direct",
    "saliency_lse",
    "topk_admission",
    "topk_admission_shared",
    "retention_k",
    "paper_layer_k",
    "OracleStream",
]


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of raw bfloat16 bit patterns (uint16) to float64.

    A bfloat16 is the upper half of an IEEE float32, so shifting the pattern
    into the top 16 bits of a uint32 gives the float32 with the same value.
    """
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def sampled_query_tokens(n_special: int, grid_h: int, grid_w: int, ds: int,
                         ds_floor: bool = False) -> list[int]:
    """Token indices of the sampled query subset Q~ (Sec. 3.3, Head-Specific
    Token Retention): the patch grid is cut into non-overlapping ds x ds
    windows and the top-left query of each window is kept.

    Patches follow the special tokens in row-major order, so patch (r, c) is
    token ``n_special + r * grid_w + c``.  With ``ds_floor`` only complete
    windows count; otherwise a partial window at the bottom/right edge still
    contributes its top-left query.
    """
    if ds < 1:
        raise ValueError("ds must be >= 1")
    rows = grid_h // ds if ds_floor else -(-grid_h // ds)
    cols = grid_w // ds if ds_floor else -(-grid_w // ds)
    return [n_special + (r * ds) * grid_w + (c * ds)
            for r in range(rows) for c in range(cols)]


def attend_head(q: np.ndarray, kc: np.ndarray, vc: np.ndarray, scale: float):
    """Softmax attention of one head (Eq. 2), materialising everything.

    q: [N, d] queries; kc, vc: [L, d] keys/values (memory rows, then frame
    rows).  Returns (O [N, d], LSE [N], Z [N, L], P [N, L]) with
    ``Z = q kc^T * scale``, ``LSE_i = log sum_j exp(Z_ij)`` and
    ``P_ij = exp(Z_ij - LSE_i)``.
    """
    z = (q @ kc.T) * scale
    m = z.max(axis=1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(z - m).sum(axis=1))
    p = np.exp(z - lse[:, None])
    o = p @ vc
    return o, lse, z, p


def saliency_direct(p: np.ndarray, m_rows: int, qidx) -> np.ndarray:
    """S_j = sum_{i in Q~} A_ij read straight off the materialised softmax:
    the column sums of the sampled rows over the current-frame columns
    (columns m_rows .. L-1)."""
    return p[np.asarray(qidx, dtype=np.int64), m_rows:].sum(axis=0)


def saliency_lse(z: np.ndarray, lse: np.ndarray, m_rows: int, qidx) -> np.ndarray:
    """Same saliency through the LSE route: ``A_ij = exp(Z_ij - LSE_i)`` with
    the LSE of the whole attended context (LSE-Saliency, Sec. 3.3)."""
    qi = np.asarray(qidx, dtype=np.int64)
    return np.exp(z[qi, m_rows:] - lse[qi, None]).sum(axis=0)


def topk_admission(s: np.ndarray, n_special: int, k: int,
                   candidates: str = "patch") -> list[int]:
    """Top-k of Eq. 6 for one head: the k most salient candidate tokens.

    Order is (saliency descending, token index ascending), so ties go to the
    lower index.  The chosen indices are returned in ascending token order,
    which is the order in which their rows are appended.
    """
    n = len(s)
    lo = n_special if candidates == "patch" else 0
    order = sorted(range(lo, n), key=lambda j: (-float(s[j]), j))
    return sorted(order[:k])


def topk_admission_shared(s: np.ndarray, n_special: int, k: int,
                          candidates: str = "patch") -> list[int]:
    """Top-k without head-specific retention (Sec. 4.5, Table 4, first row):
    the saliency of all heads ``s`` [H, N] is averaged over heads and one set
    of k tokens is chosen for every head, ordered and tie-broken as in
    ``topk_admission``."""
    mean = np.asarray(s, dtype=np.float64).mean(axis=0)
    return topk_admission(mean, n_special, k, candidates)


def retention_k(gamma: float, n_tokens: int) -> int:
    """k = floor(gamma N), the tokens a frame adds per head (Eq. 6)."""
    return int(math.floor(gamma * n_tokens))


def paper_layer_k(layers: int, k: int) -> list[int]:
    """Per-layer admission count of the paper's configuration (Sec. 4.1,
    Eq. 5 / Eq. 6): layers 11-17 (1-based) admit k rows per frame, every other
    layer keeps only its anchor frame (k = 0)."""
    return [k if 11 <= layer + 1 <= 17 else 0 for layer in range(layers)]


def attend_frame(q, k, v, bank_k, bank_v, scale, qidx):
    """One regulated-attention call for all heads.

    q, k, v: [N, H, d] float64; bank_k, bank_v: per-head lists of [M, d]
    arrays (M may be 0).  Returns dict with O [N, H, d], LSE [H, N],
    saliency via LSE [H, N], saliency read directly off P [H, N].
    """
    n, heads, d = q.shape
    o = np.empty((n, heads, d))
    lse = np.empty((heads, n))
    sal = np.empty((heads, n))
    sal_d = np.empty((heads, n))
    for h in range(heads):
        mk = bank_k[h]
        mv = bank_v[h]
        m_rows = mk.shape[0]
        kc = np.concatenate([mk, k[:, h, :]], axis=0)
        vc = np.concatenate([mv, v[:, h, :]], axis=0)
        oh, lh, zh, ph = attend_head(q[:, h, :], kc, vc, scale)
        o[:, h, :] = oh
        lse[h] = lh
        sal[h] = saliency_lse(zh, lh, m_rows, qidx)
        sal_d[h] = saliency_direct(ph, m_rows, qidx)
    return {"O": o, "LSE": lse, "S": sal, "S_direct": sal_d}


@dataclass
class OracleStream:
    """Frame-by-frame reference of the regulated memory (Eq. 4 - Eq. 6).

    Each layer keeps, per head, an append-only list of K rows and V rows.
    ``attend`` runs Eq. 3 against the memory as it stands (M_{t-1});
    ``admit`` appends either the first frame whole (Eq. 4, when the layer's
    memory is empty) or the per-head top-k of the current frame (Eq. 6).
    """

    layers: int
    heads: int
    head_dim: int
    n_special: int
    grid_h: int
    grid_w: int
    ds: int = 2
    scale: float | None = None
    candidates: str = "patch"
    ds_floor: bool = False
    bank_k: list = field(init=False)
    bank_v: list = field(init=False)
    _pending: dict = field(init=False)

    def __post_init__(self):
        if self.scale is None:
            self.scale = 1.0 / math.sqrt(self.head_dim)
        d = self.head_dim
        self.bank_k = [[np.zeros((0, d)) for _ in range(self.heads)]
                       for _ in range(self.layers)]
        self.bank_v = [[np.zeros((0, d)) for _ in range(self.heads)]
                       for _ in range(self.layers)]
        self._pending = {}

    @property
    def n_tokens(self) -> int:
        return self.n_special + self.grid_h * self.grid_w

    @property
    def qidx(self) -> list[int]:
        return sampled_query_tokens(self.n_special, self.grid_h, self.grid_w,
                                    self.ds, self.ds_floor)

    def memory_len(self, layer: int) -> int:
        return self.bank_k[layer][0].shape[0]

    def attend(self, layer: int, q, k, v) -> dict:
        q = np.asarray(q, dtype=np.float64)
        k = np.asarray(k, dtype=np.float64)
        v = np.asarray(v, dtype=np.float64)
        assert q.shape == (self.n_tokens, self.heads, self.head_dim)
        res = attend_frame(q, k, v, self.bank_k[layer], self.bank_v[layer],
                           self.scale, self.qidx)
        self._pending[layer] = (k, v, res["S"])
        return res

    def choose(self, layer: int, kk: int, saliency=None) -> np.ndarray:
        """Indices Eq. 6 would admit, [H, kk], without touching the memory.
        ``saliency`` overrides the oracle's own saliency (e.g. to take the
        integer decision on another implementation's fp32 values)."""
        _, _, s = self._pending[layer]
        if saliency is not None:
            s = np.asarray(saliency)
        return np.array([topk_admission(s[h], self.n_special, kk, self.candidates)
                         for h in range(self.heads)], dtype=np.int64).reshape(self.heads, kk)

    def admit(self, layer: int, kk: int, indices=None, shared: bool = False) -> np.ndarray:
        """Apply Eq. 4 (empty memory: store the whole frame) or Eq. 6 (append
        the top-kk rows per head).  ``indices`` ([H, kk]) teacher-forces the
        choice; ``shared`` takes one head-averaged choice for all heads.
        Returns the appended token indices per head."""
        k, v, s = self._pending.pop(layer)
        n = k.shape[0]
        if self.memory_len(layer) == 0:
            idx = np.tile(np.arange(n), (self.heads, 1))
        elif indices is not None:
            idx = np.asarray(indices, dtype=np.int64).reshape(self.heads, kk)
        elif shared:
            one = topk_admission_shared(s, self.n_special, kk, self.candidates)
            idx = np.tile(np.asarray(one, dtype=np.int64).reshape(1, kk), (self.heads, 1))
        else:
            idx = np.array([topk_admission(s[h], self.n_special, kk, self.candidates)
                            for h in range(self.heads)],
                           dtype=np.int64).reshape(self.heads, kk)
        for h in range(self.heads):
            rows = idx[h]
            self.bank_k[layer][h] = np.concatenate([self.bank_k[layer][h], k[rows, h, :]])
            self.bank_v[layer][h] = np.concatenate([self.bank_v[layer][h], v[rows, h, :]])
        return idx

    def step(self, layer: int, q, k, v, kk: int, indices=None) -> dict:
        """attend + admit in one call; returns the attend result plus 'idx'."""
        res = self.attend(layer, q, k, v)
        res["idx"] = self.admit(layer, kk, indices)
        return res
