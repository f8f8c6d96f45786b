"""Plain fp64 CPU oracle of HeteroFold's prefill-free K/V transfer.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
execute this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code, table or constant generator with the CUDA path in
``paper_2609_32259_gb300/``; the two are compared element by element.

What it computes (arxiv 2609.32259, "HeteroFold"):

* Token Alignment (TA), Section 3.1 "Token and Layer Alignment" and
  Appendix B.1 "Token Alignment (TA) Implementation": sender and receiver
  tokens of the same text are paired through shared character-end offsets;
  an unmatched receiver token takes the sender token at the latest preceding
  shared boundary, and receiver tokens before the first shared boundary take
  the first sender token.  Sender states are never averaged.
* Overlap mean-pooling (a second alignment reading, used by the tiny
  workload): receiver token j averages every sender token whose character
  span overlaps its own.
* Same-index pairing, Appendix A (baselines) and B.1: a(j) = min(j, n_S)
  with one-based indices.
* Layer Alignment, Eq. 1: pi(l) = 1 + round((l-1)(L_S-1)/(L_R-1)) and the
  clipped neighbourhood N(l) = (pi-4, pi, pi+4); plus the two-layer linear
  interpolation reading.
* Feature concatenation, Eq. 2: x = [c^{t1} || c^{t2} || c^{t3}].
* Recolor fitting (Section 3.2 "Moment-Matched Recoloring", Eq. 3-5): the
  sender RMS r over weighted samples (Eq. 3), weighted means and
  covariances of Z = X / r and Y, whitening and Procrustes alignment through
  the thin SVD of Sigma_Z^{-1/2} Sigma_ZY Sigma_Y^{-1/2} = U Lambda Q^T,
  R* = U Q^T (Eq. 4), and A = Sigma_Z^{-1/2} R* Sigma_Y^{1/2},
  b = mu_Y - mu_Z A (Eq. 5).
* The output-aware low-rank correction, Eq. 7: y_hat = y0 + (y0 B) G with
  y0 = (x / r) A + b, and its folding, Eq. 9: A_final = A (I + B G),
  b_final = b (I + B G).
* The KV Ridge + TA apply (Appendix A, baseline details; Section 4 setup;
  Appendix F, mapper size): each receiver layer reads k = 8 selected sender
  layers, and each receiver KV head has its own ridge map from all KV heads
  of those layers (their concatenation) to that head's features; with TA the
  token correspondence is Token Alignment, otherwise same-index pairing.
* The folded inference map, Eq. 9: Phi(x) = (x / r) A_final + b_final,
  one map per receiver layer and role, reshaped to receiver KV heads; keys
  then get the receiver's key normalisation and RoPE at receiver positions
  (Section 3 opening paragraph, Section 3.3 "Folding for inference",
  Appendix B.1 last paragraph).

Conventions (readings of passages the paper leaves open):

* Indices are zero-based in code; the paper's are one-based.
* Role 0 is K, role 1 is V.
* A role-c feature of a token is the head-major flattening h * D + d of its
  [H][D] KV entry.
* ``A`` has the paper's orientation: shape [K, d_R], applied as x @ A, with
  the rows of segment s at [s * d_S, (s + 1) * d_S).
* RoPE is the rotate-half form (pairs i and i + D/2), inv_freq_i is the
  fp32 rounding of theta ** (-2 i / D) evaluated in double precision, and the
  angle p * inv_freq_i is formed exactly in fp64.
* Key normalisation, when enabled, is a per-head RMS norm with a weight g[D].
* Sender keys are normally captured before RoPE (Section 3 opening
  paragraph).  For a sender cache whose keys already carry RoPE at the sender
  positions, the keys are first rotated back (the inverse rotation, by the
  negative angle, at each sender token's own position) and only then pooled
  and blended; values are never rotated.

Every routine here is a direct restatement of the definitions above in
numpy float64; nothing is blocked, fused or reordered beyond them.
"""

from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Dict, Iterable, List, Optional, Sequence, Tuple

import numpy as np

ROLE_K = 0
ROLE_V = 1

ALIGN_TA = "ta"
ALIGN_OVERLAP_MEAN = "overlap_mean"
ALIGN_SAME_INDEX = "same_index"

LAYER_PAPER3 = "paper3"
LAYER_INTERP = "interp"


# ---------------------------------------------------------------------------
# Input validation shared by the alignment routines
# ---------------------------------------------------------------------------

def _check_ends(ends: Sequence[int], name: str) -> List[int]:
    out = [int(e) for e in ends]
    prev = 0
    for e in out:
        if e <= prev:
            # Appendix B.1: TA pairs *nonempty* tokens, so every token ends
            # strictly after the previous one.
            raise ValueError(f"{name}: character-end offsets must be strictly "
                             f"increasing and positive (empty token?)")
        prev = e
    return out


def _check_pair(s_end: Sequence[int], r_end: Sequence[int]) -> Tuple[List[int], List[int]]:
    s = _check_ends(s_end, "sender")
    r = _check_ends(r_end, "receiver")
    if len(r) > 0 and len(s) == 0:
        raise ValueError("receiver tokens without any sender token")
    if len(r) > 0 and s[-1] != r[-1]:
        raise ValueError("sender and receiver must tokenize the same text "
                         "(their last character-end offsets differ)")
    return s, r


# ---------------------------------------------------------------------------
# Token alignment (Section 3.1, Appendix B.1)
# ---------------------------------------------------------------------------

def token_alignment(s_end: Sequence[int], r_end: Sequence[int]) -> np.ndarray:
    """TA: zero-based sender index a[j] for every receiver token j.

    Section 3.1 ("Token Alignment (TA)") and Appendix B.1: a receiver token
    whose end offset is also a sender end offset (a shared boundary) takes
    that sender token; otherwise it takes the sender token of the latest
    shared boundary before it; before the first shared boundary it takes the
    first sender token.  "Shared" is read literally: a sender-only boundary
    between two shared ones does not count.
    """
    s, r = _check_pair(s_end, r_end)
    sender_ending_at = {e: i for i, e in enumerate(s)}
    a = np.zeros(len(r), dtype=np.int64)
    current = 0  # first sender token before the first shared boundary
    for j, e in enumerate(r):
        if e in sender_ending_at:  # e is a shared boundary
            current = sender_ending_at[e]
        a[j] = current
    return a


def same_index_alignment(n_s: int, n_r: int) -> np.ndarray:
    """Same-index pairing, Appendix A/B.1: a(j) = min(j, n_S), one-based."""
    if n_r > 0 and n_s <= 0:
        raise ValueError("receiver tokens without any sender token")
    return np.array([min(j, n_s - 1) for j in range(n_r)], dtype=np.int64)


def overlap_alignment(s_end: Sequence[int], r_end: Sequence[int]) -> List[List[int]]:
    """Overlap reading: for receiver token j, the sender tokens whose
    character spans overlap j's span.

    Spans are half-open on the left: token j covers characters
    (end_{j-1}, end_j], with end_{-1} = 0.  Sender token k overlaps receiver
    token j iff start_k < end_j and end_k > start_j.  A two-pointer sweep
    over the two sorted end arrays.
    """
    s, r = _check_pair(s_end, r_end)
    members: List[List[int]] = []
    k = 0  # first sender token that may still overlap
    for j, e in enumerate(r):
        start_j = r[j - 1] if j > 0 else 0
        # advance past sender tokens that end at or before start_j
        while k < len(s) and s[k] <= start_j:
            k += 1
        row = []
        kk = k
        while kk < len(s):
            start_k = s[kk - 1] if kk > 0 else 0
            if start_k >= e:
                break
            row.append(kk)
            kk += 1
        members.append(row)
    return members


@dataclass
class CSR:
    """Alignment as a compressed sparse row matrix over global token indices.

    Row j (a receiver token) lists the sender tokens it draws from (``col``)
    with their pooling weights (``w``); TA and same-index rows have exactly
    one entry of weight 1.  ``w32`` holds the weights rounded to fp32, the
    stored form on the device; ``w`` holds the exact values the oracle uses.
    """

    row_ptr: np.ndarray
    col: np.ndarray
    w: np.ndarray

    @property
    def w32(self) -> np.ndarray:
        return self.w.astype(np.float32)

    @property
    def n_rows(self) -> int:
        return len(self.row_ptr) - 1

    @property
    def nnz(self) -> int:
        return int(self.row_ptr[-1])


def alignment_csr(mode: str, s_tok_ptr: Sequence[int], r_tok_ptr: Sequence[int],
                  s_end: Sequence[int], r_end: Sequence[int]) -> CSR:
    """Alignment of a batch of requests, concatenated.

    Request q owns sender tokens [s_tok_ptr[q], s_tok_ptr[q+1]) and receiver
    tokens [r_tok_ptr[q], r_tok_ptr[q+1]); its character offsets restart at
    zero.  Column indices are global sender token indices.
    """
    n_req = len(r_tok_ptr) - 1
    if len(s_tok_ptr) != n_req + 1:
        raise ValueError("s_tok_ptr and r_tok_ptr must have the same length")
    row_ptr = [0]
    col: List[int] = []
    w: List[float] = []
    for q in range(n_req):
        s0, s1 = int(s_tok_ptr[q]), int(s_tok_ptr[q + 1])
        r0, r1 = int(r_tok_ptr[q]), int(r_tok_ptr[q + 1])
        s_q = [int(x) for x in s_end[s0:s1]]
        r_q = [int(x) for x in r_end[r0:r1]]
        if mode == ALIGN_TA:
            rows = [[int(a)] for a in token_alignment(s_q, r_q)]
        elif mode == ALIGN_SAME_INDEX:
            _check_ends(s_q, "sender")
            _check_ends(r_q, "receiver")
            rows = [[int(a)] for a in same_index_alignment(len(s_q), len(r_q))]
        elif mode == ALIGN_OVERLAP_MEAN:
            rows = overlap_alignment(s_q, r_q)
        else:
            raise ValueError(f"unknown alignment mode {mode!r}")
        for members in rows:
            n = len(members)
            for k in members:
                col.append(s0 + k)
                w.append(1.0 / n)  # mean pooling; exactly 1 for one member
            row_ptr.append(len(col))
    return CSR(np.asarray(row_ptr, dtype=np.int64),
               np.asarray(col, dtype=np.int64),
               np.asarray(w, dtype=np.float64))


# ---------------------------------------------------------------------------
# Layer alignment (Eq. 1) and the interpolation reading
# ---------------------------------------------------------------------------

def proportional_depth(l1: int, L_s: int, L_r: int) -> int:
    """Eq. 1: pi(l) = 1 + round((l - 1)(L_S - 1)/(L_R - 1)), one-based.

    round() is read as round-half-away-from-zero, evaluated exactly in
    integers; with a single receiver layer pi(1) = 1.
    """
    if L_r == 1:
        return 1
    num = (l1 - 1) * (L_s - 1)
    den = L_r - 1
    return 1 + (2 * num + den) // (2 * den)


def layer_alignment(L_s: int, L_r: int) -> List[Tuple[int, int, int]]:
    """Eq. 1: clipped neighbourhood N(l) = clip(pi-4, pi, pi+4) to [1, L_S].

    Returned zero-based, one triple (t1, t2, t3) per receiver layer.
    Duplicates produced by the clip are kept as separate segments.
    """
    out = []
    for l1 in range(1, L_r + 1):
        pi = proportional_depth(l1, L_s, L_r)
        out.append(tuple(min(max(pi + off, 1), L_s) - 1 for off in (-4, 0, 4)))
    return out


def layer_interpolation(L_s: int, L_r: int) -> List[List[Tuple[int, float]]]:
    """Interpolation reading: receiver layer l (zero-based) blends sender
    layers floor(p) and floor(p) + 1 at p = l (L_S - 1)/(L_R - 1), with
    weights (1 - f, f), f = p - floor(p); the weights sum to one."""
    out = []
    for l in range(L_r):
        p = (l * (L_s - 1)) / (L_r - 1) if L_r > 1 else 0.0
        i0 = int(math.floor(p))
        f = p - i0
        terms = [(i0, 1.0 - f)]
        if f > 0.0:
            terms.append((min(i0 + 1, L_s - 1), f))
        out.append(terms)
    return out


def explicit_segments(seg_layer, seg_w) -> List[List[List[Tuple[int, float]]]]:
    """A caller-given layer table: seg_layer[l][s][t] (zero-based sender
    layer) and seg_w[l][s][t] give term t of segment s of receiver layer l.
    Segment s is the weighted sum of its terms (the same structure as Eq. 2's
    concatenation, with any layers and weights)."""
    out = []
    for layers_l, w_l in zip(seg_layer, seg_w):
        out.append([[(int(t), float(w)) for t, w in zip(ts, ws)] for ts, ws in zip(layers_l, w_l)])
    return out


def layer_segments(mode: str, L_s: int, L_r: int) -> List[List[List[Tuple[int, float]]]]:
    """Per receiver layer: the K-segments of the map input, each a weighted
    sum of sender layers.  Paper mode: three one-layer segments (Eq. 2);
    interpolation mode: one two-layer segment."""
    if mode == LAYER_PAPER3:
        return [[[(t, 1.0)] for t in trip] for trip in layer_alignment(L_s, L_r)]
    if mode == LAYER_INTERP:
        return [[terms] for terms in layer_interpolation(L_s, L_r)]
    raise ValueError(f"unknown layer mode {mode!r}")


def mapper_parameter_count(L_r: int, d_s: int, d_r: int, n_seg: int = 3) -> int:
    """Stored parameters of the folded maps (Appendix F "Mapper Size"):
    one [n_seg * d_S, d_R] matrix and one d_R bias per receiver layer and
    role, counted from the segment structure."""
    total = 0
    for _layer in range(L_r):
        for _role in (ROLE_K, ROLE_V):
            total += n_seg * d_s * d_r + d_r
    return total


# ---------------------------------------------------------------------------
# Receiver-side key processing
# ---------------------------------------------------------------------------

def rope_inv_freq(theta: float, D: int) -> np.ndarray:
    """inv_freq_i = fp32(theta ** (-2 i / D)), i < D/2, returned as fp64."""
    return np.array([np.float32(float(theta) ** (-(2.0 * i) / D)) for i in range(D // 2)],
                    dtype=np.float64)


def rope(x: np.ndarray, pos: np.ndarray, inv_freq: np.ndarray) -> np.ndarray:
    """Rotate-half RoPE at integer positions ``pos`` (one per leading row).

    x: [n, H, D]; pair (i, i + D/2) is rotated by the angle pos * inv_freq_i.
    """
    D = x.shape[-1]
    half = D // 2
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]  # exact in fp64
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1 = x[..., :half]
    x2 = x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def rope_inverse(x: np.ndarray, pos: np.ndarray, inv_freq: np.ndarray) -> np.ndarray:
    """The inverse of rope() at the same positions: pair (i, i + D/2) is
    rotated by the negative angle -pos * inv_freq_i.  x: [n, H, D]."""
    D = x.shape[-1]
    half = D // 2
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1 = x[..., :half]
    x2 = x[..., half:]
    return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=-1)


def key_norm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """Per-head RMS normalisation of receiver keys with weight g[D]."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(g, dtype=np.float64)


# ---------------------------------------------------------------------------
# The transfer (Eq. 2 + Eq. 9)
# ---------------------------------------------------------------------------

def pooled_features(sender_lc, csr: CSR, rows: np.ndarray, unrotate=None,
                    row_of=None) -> np.ndarray:
    """Pool one sender layer/role over the alignment rows: for receiver row j,
    sum_k w_k * c_k over the row's entries (a single copy for TA).

    unrotate: None, or (s_pos, inv_freq_s, H_s) for sender keys stored with
    RoPE: each sender token k is first rotated back at its position s_pos[k]
    (rope_inverse), then weighted and summed.
    row_of: None (sender token k is cache row k), or the cache row of every
    sender token (a message span inside a longer sender cache)."""
    starts = csr.row_ptr[rows]
    ends = csr.row_ptr[rows + 1]
    if np.any(ends <= starts):
        raise ValueError("every alignment row needs at least one sender token")
    lengths = ends - starts
    entry = np.concatenate([np.arange(a, b) for a, b in zip(starts, ends)])
    cols = csr.col[entry]
    feats = np.asarray(sender_lc[cols if row_of is None else np.asarray(row_of)[cols]],
                       dtype=np.float64)
    if unrotate is not None:
        s_pos, inv_freq_s, H_s = unrotate
        n, d_s = feats.shape
        feats = rope_inverse(feats.reshape(n, H_s, d_s // H_s), np.asarray(s_pos)[cols],
                             inv_freq_s).reshape(n, d_s)
    feats = feats * csr.w[entry][:, None]
    seg_start = np.concatenate([[0], np.cumsum(lengths)[:-1]])
    return np.add.reduceat(feats, seg_start, axis=0)


def map_input(sender, csr: CSR, segments_l, role: int, rows: np.ndarray,
              sender_rope=None, sender_row_of=None) -> np.ndarray:
    """Eq. 2: the concatenated map input x for receiver layer l and role c.

    Segment s is the weighted sum of its sender layers' pooled features;
    the segments are concatenated along the feature axis.  sender_rope
    (keys only): see pooled_features' unrotate; sender_row_of: its row_of.
    """
    unrot = sender_rope if role == ROLE_K else None
    parts = []
    for seg in segments_l:
        acc = None
        for (t, omega) in seg:
            term = omega * pooled_features(sender[t][role], csr, rows, unrot, sender_row_of)
            acc = term if acc is None else acc + term
        parts.append(acc)
    return np.concatenate(parts, axis=1)


def transfer(sender, csr: CSR, segments, A, b, r, *, H_r: int, D_r: int,
             pos: np.ndarray, inv_freq_r: np.ndarray,
             knorm_g: Optional[np.ndarray] = None, knorm_eps: float = 1e-6,
             layers: Optional[Iterable[int]] = None,
             rows: Optional[np.ndarray] = None,
             roles: Iterable[int] = (ROLE_K, ROLE_V),
             sender_rope=None, sender_row_of=None) -> Dict[Tuple[int, int], np.ndarray]:
    """The receiver cache entries for the requested layers, roles and rows.

    sender:  indexable as sender[t][c] -> [T_s, d_S] array (any float dtype)
    csr:     the alignment (receiver rows x sender tokens)
    segments: layer_segments(...) result, one entry per receiver layer
    A:       indexable as A[l][c] -> [K, d_R] (paper orientation, x @ A)
    b:       [L_R][2][d_R];  r: [L_R][2] positive scalars (Eq. 3's r)
    pos:     receiver position of every receiver row (RoPE position)
    sender_rope: None (sender keys captured before RoPE, the paper's case) or
             (s_pos, inv_freq_s, H_s) when the sender keys carry RoPE at
             sender positions s_pos: they are rotated back before pooling.
    sender_row_of: None, or the sender-cache row of every sender token of
             the alignment (message spans: only a span of each request's
             sender cache is transferred, Appendix "HiddenBench Evaluation").

    Returns {(l, c): [n_rows, H_r, D_r] float64}.  Eq. 9:
    Phi(x) = (x / r) A + b, reshaped to receiver heads; keys then get the
    optional key norm and RoPE at their receiver positions.
    """
    n_rows_total = csr.n_rows
    rows = np.arange(n_rows_total) if rows is None else np.asarray(rows, dtype=np.int64)
    layers = range(len(segments)) if layers is None else layers
    out: Dict[Tuple[int, int], np.ndarray] = {}
    for l in layers:
        for c in roles:
            x = map_input(sender, csr, segments[l], c, rows, sender_rope, sender_row_of)
            A_lc = np.asarray(A[l][c], dtype=np.float64)
            if A_lc.shape != (x.shape[1], H_r * D_r):
                raise ValueError(f"map shape {A_lc.shape} does not match input "
                                 f"width {x.shape[1]} and d_R {H_r * D_r}")
            y = (x / float(r[l][c])) @ A_lc + np.asarray(b[l][c], dtype=np.float64)
            y = y.reshape(len(rows), H_r, D_r)
            if c == ROLE_K:
                if knorm_g is not None:
                    y = key_norm(y, knorm_g, knorm_eps)
                y = rope(y, np.asarray(pos)[rows], inv_freq_r)
            out[(l, c)] = y
    return out


# ---------------------------------------------------------------------------
# KV Ridge + TA apply (Appendix A baseline details, Appendix F mapper size)
# ---------------------------------------------------------------------------

KV_RIDGE_K = 8  # sender layers per receiver layer (the method's default k)


def kv_ridge_segments(selected) -> List[List[List[Tuple[int, float]]]]:
    """KV Ridge's layer routing: receiver layer l reads the sender layers
    selected[l] (k of them, chosen offline by calibration R^2), each as one
    segment of weight 1, concatenated in the given order."""
    return [[[(int(t), 1.0)] for t in sel] for sel in selected]


def kv_ridge_transfer(sender, csr: CSR, selected, W_heads, b_heads, *, H_r: int, D_r: int,
                      pos: np.ndarray, inv_freq_r: np.ndarray,
                      layers: Optional[Iterable[int]] = None,
                      rows: Optional[np.ndarray] = None,
                      roles: Iterable[int] = (ROLE_K, ROLE_V)) -> Dict[Tuple[int, int], np.ndarray]:
    """The receiver cache entries of the KV Ridge apply.

    For receiver layer l, role c and receiver KV head h:
        y_h = x W_heads[l][c][h] + b_heads[l][c][h],
    x the concatenation of every KV head of the selected sender layers
    (kv_ridge_segments(selected)[l], Eq. 2's layout) at the aligned sender
    token; W_heads[l][c][h] is [k * d_S, D_r] and b_heads[l][c][h] is [D_r].
    A ridge map is a plain least-squares affine map: there is no Eq. 3
    normaliser.  Keys then get RoPE at their receiver positions, as in
    transfer().  Returns {(l, c): [n_rows, H_r, D_r] float64}."""
    rows = np.arange(csr.n_rows) if rows is None else np.asarray(rows, dtype=np.int64)
    segments = kv_ridge_segments(selected)
    layers = range(len(segments)) if layers is None else layers
    out: Dict[Tuple[int, int], np.ndarray] = {}
    for l in layers:
        for c in roles:
            x = map_input(sender, csr, segments[l], c, rows)
            y = np.empty((len(rows), H_r, D_r))
            for h in range(H_r):
                Wh = np.asarray(W_heads[l][c][h], dtype=np.float64)
                if Wh.shape != (x.shape[1], D_r):
                    raise ValueError(f"head map shape {Wh.shape} does not match input width "
                                     f"{x.shape[1]} and D_r {D_r}")
                y[:, h, :] = x @ Wh + np.asarray(b_heads[l][c][h], dtype=np.float64)
            if c == ROLE_K:
                y = rope(y, np.asarray(pos)[rows], inv_freq_r)
            out[(l, c)] = y
    return out


def token_positions(tok_ptr: Sequence[int], pos0: Optional[Sequence[int]] = None) -> np.ndarray:
    """RoPE position of every concatenated token of one model: the request's
    origin (default 0) plus the token's index within its request."""
    n_req = len(tok_ptr) - 1
    pos = []
    for q in range(n_req):
        base = 0 if pos0 is None else int(pos0[q])
        for t in range(int(tok_ptr[q + 1]) - int(tok_ptr[q])):
            pos.append(base + t)
    return np.asarray(pos, dtype=np.int64)


def span_rows(s_tok_ptr: Sequence[int], s_row0: Sequence[int]) -> np.ndarray:
    """Sender-cache row of every concatenated sender token when request q's
    tokens are the span starting at cache row s_row0[q]."""
    out = []
    for q in range(len(s_tok_ptr) - 1):
        for t in range(int(s_tok_ptr[q + 1]) - int(s_tok_ptr[q])):
            out.append(int(s_row0[q]) + t)
    return np.asarray(out, dtype=np.int64)


def sender_rms(X: np.ndarray, w: np.ndarray) -> float:
    """Eq. 3: r = sqrt(sum_n w_n |x_n|^2 / (d~_S sum_n w_n)), one scalar over
    all weighted samples and feature dimensions."""
    X = np.asarray(X, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    return float(np.sqrt(np.sum(w * np.sum(X * X, axis=1)) / (X.shape[1] * np.sum(w))))


def weighted_moments(Z: np.ndarray, Y: np.ndarray, w: np.ndarray):
    """Weighted means, covariances and cross-covariance (normalised by
    sum w): mu_Z, mu_Y, Sigma_Z, Sigma_Y, Sigma_ZY."""
    Z = np.asarray(Z, dtype=np.float64)
    Y = np.asarray(Y, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    W = np.sum(w)
    mu_z = (w @ Z) / W
    mu_y = (w @ Y) / W
    Zc = Z - mu_z
    Yc = Y - mu_y
    return (mu_z, mu_y, (Zc * w[:, None]).T @ Zc / W, (Yc * w[:, None]).T @ Yc / W,
            (Zc * w[:, None]).T @ Yc / W)


def _sym_power(S: np.ndarray, p: float) -> np.ndarray:
    """S^p of a symmetric positive definite matrix through its eigenvectors."""
    lam, V = np.linalg.eigh(S)
    return (V * lam ** p) @ V.T


def recolor(X: np.ndarray, Y: np.ndarray, w: np.ndarray, reg: float = 0.0):
    """Recolor fit (Eq. 3-5) for one receiver layer and role.

    X: [N, d~_S] sender features (Eq. 2 concatenation), Y: [N, d_R] receiver
    targets, w: [N] sample weights.  reg: numerical stabilisation, read as a
    ridge of reg * (mean eigenvalue) added to each covariance (the paper
    stabilises without giving the form).  Returns (A [d~_S, d_R], b [d_R], r).
    """
    r = sender_rms(X, w)
    Z = np.asarray(X, dtype=np.float64) / r
    mu_z, mu_y, S_z, S_y, S_zy = weighted_moments(Z, Y, w)
    if reg > 0.0:
        S_z = S_z + reg * np.trace(S_z) / S_z.shape[0] * np.eye(S_z.shape[0])
        S_y = S_y + reg * np.trace(S_y) / S_y.shape[0] * np.eye(S_y.shape[0])
    Sz_ih = _sym_power(S_z, -0.5)
    Sy_ih = _sym_power(S_y, -0.5)
    Sy_h = _sym_power(S_y, 0.5)
    U, _lam, Qt = np.linalg.svd(Sz_ih @ S_zy @ Sy_ih, full_matrices=False)
    R = U @ Qt
    A = Sz_ih @ R @ Sy_h
    b = mu_y - mu_z @ A
    return A, b, r


def fold(A: np.ndarray, b: np.ndarray, B: np.ndarray, G: np.ndarray):
    """Eq. 9 (folding for inference): A_final = A (I + B G), b_final =
    b (I + B G), for one receiver layer and role.  A: [K, d_R], b: [d_R],
    B: [d_R, rho], G: [rho, d_R]."""
    A = np.asarray(A, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    M = np.eye(A.shape[1]) + np.asarray(B, dtype=np.float64) @ np.asarray(G, dtype=np.float64)
    return A @ M, b @ M


def transfer_unfused(sender, csr: CSR, segments, A, b, r, B, G, *, H_r: int, D_r: int,
                     pos: np.ndarray, inv_freq_r: np.ndarray,
                     knorm_g: Optional[np.ndarray] = None, knorm_eps: float = 1e-6,
                     layers: Optional[Iterable[int]] = None,
                     rows: Optional[np.ndarray] = None,
                     roles: Iterable[int] = (ROLE_K, ROLE_V)) -> Dict[Tuple[int, int], np.ndarray]:
    """The receiver cache entries with the correction applied unfolded,
    in the order the paper defines it: y0 = (x / r) A + b (Eq. 5, the
    Recolor map), y_hat = y0 + (y0 B) G (Eq. 7), then heads, key norm and RoPE as in
    transfer().  B[l][c]: [d_R, rho], G[l][c]: [rho, d_R]."""
    n_rows_total = csr.n_rows
    rows = np.arange(n_rows_total) if rows is None else np.asarray(rows, dtype=np.int64)
    layers = range(len(segments)) if layers is None else layers
    out: Dict[Tuple[int, int], np.ndarray] = {}
    for l in layers:
        for c in roles:
            x = map_input(sender, csr, segments[l], c, rows)
            A_lc = np.asarray(A[l][c], dtype=np.float64)
            y0 = (x / float(r[l][c])) @ A_lc + np.asarray(b[l][c], dtype=np.float64)
            y = y0 + (y0 @ np.asarray(B[l][c], dtype=np.float64)) @ np.asarray(G[l][c],
                                                                               dtype=np.float64)
            y = y.reshape(len(rows), H_r, D_r)
            if c == ROLE_K:
                if knorm_g is not None:
                    y = key_norm(y, knorm_g, knorm_eps)
                y = rope(y, np.asarray(pos)[rows], inv_freq_r)
            out[(l, c)] = y
    return out


def receiver_positions(r_tok_ptr: Sequence[int], r_pos0: Optional[Sequence[int]] = None) -> np.ndarray:
    """Receiver RoPE positions (token_positions of the receiver side)."""
    return token_positions(r_tok_ptr, r_pos0)


def sender_positions(s_tok_ptr: Sequence[int], s_pos0: Optional[Sequence[int]] = None) -> np.ndarray:
    """Sender RoPE positions (token_positions of the sender side)."""
    return token_positions(s_tok_ptr, s_pos0)
