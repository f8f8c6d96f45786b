"""Pins that tie the fp64 oracle to the paper and to mathematics.

Each ``check_*`` function raises AssertionError when the oracle disagrees
with something fixed independently of it: a worked example printed in the
paper, a closed form, an invariant, a brute-force restatement on tiny
inputs, or a special case with a known answer.  ``test_oracle_pins.py`` runs
them against the oracle; ``test_oracle_mutations.py`` plants plausible
mistakes in the oracle and checks that some pin fails for each.
"""

from __future__ import annotations

import math
import os
import random

import numpy as np

import oracle
from oracle import heterofold_oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))


def _read_golden(name):
    out = {}
    with open(os.path.join(HERE, "golden", name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            if ":" in line:
                k, v = line.split(":", 1)
                out[k.strip()] = v.strip()
            else:
                out.setdefault("_rows", []).append(line.split())
    return out


def _ends(lengths):
    return list(np.cumsum(lengths).astype(int))


def _random_segmentation(rng, n_chars, lo, hi):
    ends, e = [], 0
    while e < n_chars:
        e = min(n_chars, e + rng.randint(lo, hi))
        ends.append(e)
    return ends


# ---------------------------------------------------------------------------
# Token alignment
# ---------------------------------------------------------------------------

def check_ta_worked_example():
    """Section 3.1's table: Qwen3 vs Ministral-3 tokenisations of
    "The unbelievable result." give a = [1,1,1,2,3,4] and [1,4,5,6]."""
    g = _read_golden("ta_worked_example.txt")
    qwen = [int(x) for x in g["qwen3_ends"].split()]
    mini = [int(x) for x in g["ministral3_ends"].split()]
    q2m = [int(x) for x in g["qwen3_to_ministral3"].split()]
    m2q = [int(x) for x in g["ministral3_to_qwen3"].split()]
    assert list(O.token_alignment(qwen, mini) + 1) == q2m
    assert list(O.token_alignment(mini, qwen) + 1) == m2q


def check_ta_literal_shared_boundary():
    """Reading of "latest preceding shared boundary": sender ends
    {1,2,4,6}, receiver ends {1,3,6}; the shared boundaries are {1,6}, so
    the receiver token ending at 3 takes the sender token ending at 1
    (zero-based 0), not the sender-only boundary at 2."""
    assert list(O.token_alignment([1, 2, 4, 6], [1, 3, 6])) == [0, 0, 3]


def _ta_brute(s_end, r_end):
    # For every receiver token scan all shared boundaries not after it.
    shared = [e for e in r_end if e in s_end]
    out = []
    for e in r_end:
        before = [x for x in shared if x <= e]
        out.append(s_end.index(max(before)) if before else 0)
    return out


def check_ta_brute_force(trials=300, seed=7):
    rng = random.Random(seed)
    for _ in range(trials):
        n = rng.randint(1, 60)
        s = _random_segmentation(rng, n, 1, rng.randint(1, 7))
        r = _random_segmentation(rng, n, 1, rng.randint(1, 7))
        a = list(O.token_alignment(s, r))
        assert a == _ta_brute(s, r), (s, r, a)
        # invariants: non-decreasing, end of text maps to end of text
        assert all(x <= y for x, y in zip(a, a[1:]))
        assert a[-1] == len(s) - 1


def check_ta_identity():
    rng = random.Random(3)
    for _ in range(50):
        s = _random_segmentation(rng, rng.randint(1, 80), 1, 6)
        assert list(O.token_alignment(s, s)) == list(range(len(s)))


def check_same_index():
    """Appendix B.1: a(j) = min(j, n_S) with one-based indices."""
    for n_s in range(1, 7):
        for n_r in range(0, 9):
            a = O.same_index_alignment(n_s, n_r)
            assert [int(x) + 1 for x in a] == [min(j, n_s) for j in range(1, n_r + 1)]


def _overlap_brute(s_end, r_end):
    # Token spans as explicit character sets; overlap = non-empty intersection.
    def spans(ends):
        out, prev = [], 0
        for e in ends:
            out.append(set(range(prev + 1, e + 1)))
            prev = e
        return out
    S, R = spans(s_end), spans(r_end)
    return [[k for k, sk in enumerate(S) if sk & rj] for rj in R]


def check_overlap_brute_force(trials=300, seed=11):
    rng = random.Random(seed)
    for _ in range(trials):
        n = rng.randint(1, 60)
        s = _random_segmentation(rng, n, 1, rng.randint(1, 7))
        r = _random_segmentation(rng, n, 1, rng.randint(1, 7))
        rows = O.overlap_alignment(s, r)
        assert rows == _overlap_brute(s, r), (s, r)
        csr = O.alignment_csr(O.ALIGN_OVERLAP_MEAN, [0, len(s)], [0, len(r)], s, r)
        for j in range(len(r)):
            w = csr.w[csr.row_ptr[j]:csr.row_ptr[j + 1]]
            assert abs(w.sum() - 1.0) < 1e-12  # a mean
        # the common refinement has one piece per overlapping pair
        assert csr.nnz == len(set(s) | set(r))


def check_csr_batching():
    """Concatenating requests offsets sender columns by the request start."""
    s1, r1 = [3, 16, 23, 24], [3, 9, 12, 16, 23, 24]
    s2, r2 = [2, 5], [1, 5]
    csr = O.alignment_csr(O.ALIGN_TA, [0, 4, 6], [0, 6, 8], s1 + s2, r1 + r2)
    assert list(csr.row_ptr) == list(range(9))
    assert list(csr.col) == [0, 0, 0, 1, 2, 3, 4, 5]
    assert np.all(csr.w == 1.0)


# ---------------------------------------------------------------------------
# Layer alignment
# ---------------------------------------------------------------------------

def check_layer_alignment_closed_form():
    """Eq. 1 properties: pi(1) = 1, pi(L_R) = L_S, monotone, identity when
    the depths agree, and the clip at the ends."""
    for L_s in range(1, 45):
        for L_r in range(2, 45):
            pis = [O.proportional_depth(l, L_s, L_r) for l in range(1, L_r + 1)]
            assert pis[0] == 1 and pis[-1] == L_s
            assert all(a <= b for a, b in zip(pis, pis[1:]))
            # |pi - (1 + exact)| <= 1/2
            for l, p in zip(range(1, L_r + 1), pis):
                exact = 1 + (l - 1) * (L_s - 1) / (L_r - 1)
                assert abs(p - exact) <= 0.5 + 1e-12
            if L_s == L_r:
                assert pis == list(range(1, L_r + 1))
            for trip in O.layer_alignment(L_s, L_r):
                assert all(0 <= t < L_s for t in trip)
                assert trip[0] <= trip[1] <= trip[2]


def check_layer_alignment_hand_tables():
    """Tables worked by hand from Eq. 1 (one-based pi)."""
    # L_S = 4 -> L_R = 6: (l-1)*3/5 = 0, .6, 1.2, 1.8, 2.4, 3
    assert [O.proportional_depth(l, 4, 6) for l in range(1, 7)] == [1, 2, 2, 3, 3, 4]
    # Llama (32) -> Ministral (40): (l-1)*31/39
    assert [O.proportional_depth(l, 32, 40) for l in range(1, 9)] == [1, 2, 3, 3, 4, 5, 6, 7]
    # the neighbourhood of receiver layer 1 is clip(-3, 1, 5) = (1, 1, 5)
    assert O.layer_alignment(32, 40)[0] == (0, 0, 4)
    # last receiver layer: pi = 32 -> clip(28, 32, 36) = (28, 32, 32)
    assert O.layer_alignment(32, 40)[-1] == (27, 31, 31)
    # Ministral (40) -> Llama (32): (l-1)*39/31, l = 2 -> 1.258 -> 1 -> pi 2
    assert [O.proportional_depth(l, 40, 32) for l in range(1, 5)] == [1, 2, 4, 5]


def check_layer_interpolation():
    for L_s in range(1, 41):
        for L_r in range(2, 41):
            rows = O.layer_interpolation(L_s, L_r)
            assert len(rows) == L_r
            assert rows[0] == [(0, 1.0)]
            assert rows[-1] == [(L_s - 1, 1.0)]
            for l, terms in enumerate(rows):
                assert abs(sum(w for _, w in terms) - 1.0) < 1e-12
                assert all(0.0 <= w <= 1.0 for _, w in terms)
                p = sum(t * w for t, w in terms)  # the blend position
                assert abs(p - l * (L_s - 1) / (L_r - 1)) < 1e-9


def check_mapper_size_table_f():
    """Appendix F's Table: 2 L_R (3 d_S d_R + d_R) parameters, in millions."""
    g = _read_golden("mapper_size_table_f.txt")
    for row in g["_rows"]:
        _, _, _Ls, Lr, ds, dr, millions = row
        n = O.mapper_parameter_count(int(Lr), int(ds), int(dr), n_seg=3)
        assert round(n / 1e6) == int(millions), (row, n)
        # and the same count from the segment structure of Eq. 1-2
        segs = O.layer_segments(O.LAYER_PAPER3, int(_Ls), int(Lr))
        assert sum(2 * (len(s) * int(ds) * int(dr) + int(dr)) for s in segs) == n


def check_mapper_size_table_f_kv_ridge():
    """Appendix F's Table, KV Ridge column: per receiver layer, role and
    receiver head, one map from the concatenated KV heads of k = 8 sender
    layers (8 H_S D_S inputs) to D_R outputs, plus a D_R bias.  Maps that
    read only the matching sender head (block-diagonal) would store H_S times
    fewer parameters and miss every entry of the column."""
    g = _read_golden("mapper_size_table_f_kv_ridge.txt")
    for row in g["_rows"]:
        _, _, _Ls, Lr, Hs, Ds, Hr, Dr, millions = row
        Lr, Hs, Ds, Hr, Dr = int(Lr), int(Hs), int(Ds), int(Hr), int(Dr)
        k = O.KV_RIDGE_K
        per_head = k * Hs * Ds * Dr + Dr
        n = 2 * Lr * Hr * per_head
        assert round(n / 1e6) == int(millions), (row, n)
        # the same count as one stacked [k d_S, d_R] map per layer and role
        assert O.mapper_parameter_count(Lr, Hs * Ds, Hr * Dr, n_seg=k) == n
        block_diag = 2 * Lr * Hr * (k * Ds * Dr + Dr)
        assert round(block_diag / 1e6) != int(millions)


# ---------------------------------------------------------------------------
# RoPE and key norm
# ---------------------------------------------------------------------------

def check_rope_two_dim_rotation():
    """D = 2, inv_freq = [1]: a plane rotation by angle p."""
    inv = O.rope_inv_freq(10000.0, 2)
    assert inv.tolist() == [1.0]
    rng = np.random.default_rng(0)
    x = rng.normal(size=(5, 1, 2))
    pos = np.array([0, 1, 7, 1000, 131071])
    y = O.rope(x, pos, inv)
    for n, p in enumerate(pos):
        c, s = math.cos(p), math.sin(p)
        a, b = x[n, 0]
        assert abs(y[n, 0, 0] - (a * c - b * s)) < 1e-12
        assert abs(y[n, 0, 1] - (b * c + a * s)) < 1e-12


def check_rope_complex_form():
    """Rotate-half RoPE equals multiplying z_i = x_i + 1j x_{i+D/2} by
    exp(1j p f_i); it preserves pair norms and is the identity at p = 0."""
    rng = np.random.default_rng(1)
    D = 16
    inv = O.rope_inv_freq(500000.0, D)
    x = rng.normal(size=(6, 3, D))
    pos = np.array([0, 3, 17, 4095, 32767, 131071])
    y = O.rope(x, pos, inv)
    z = x[..., : D // 2] + 1j * x[..., D // 2:]
    zr = z * np.exp(1j * pos[:, None, None] * inv[None, None, :])
    assert np.allclose(y[..., : D // 2], zr.real, atol=1e-9)
    assert np.allclose(y[..., D // 2:], zr.imag, atol=1e-9)
    assert np.allclose(np.abs(zr), np.abs(z))
    assert np.array_equal(y[0], x[0])


def check_rope_relative_position():
    """<RoPE_m q, RoPE_n k> depends only on m - n."""
    rng = np.random.default_rng(2)
    D = 8
    inv = O.rope_inv_freq(10000.0, D)
    q = rng.normal(size=(1, 1, D))
    k = rng.normal(size=(1, 1, D))
    for m, n in [(5, 3), (100, 98), (40000, 39998)]:
        lhs = float(np.sum(O.rope(q, np.array([m]), inv) * O.rope(k, np.array([n]), inv)))
        rhs = float(np.sum(O.rope(q, np.array([m - n]), inv) * k))
        assert abs(lhs - rhs) < 1e-8


def check_rope_inverse():
    """rope_inverse is the rotation by the negative angle: the complex form
    z * exp(-1j p f); it undoes rope at the same position, both ways round."""
    rng = np.random.default_rng(3)
    D = 16
    inv = O.rope_inv_freq(1e6, D)
    x = rng.normal(size=(5, 2, D))
    pos = np.array([0, 1, 29, 8191, 131071])
    y = O.rope_inverse(x, pos, inv)
    z = x[..., : D // 2] + 1j * x[..., D // 2:]
    zr = z * np.exp(-1j * pos[:, None, None] * inv[None, None, :])
    assert np.allclose(y[..., : D // 2], zr.real, atol=1e-9)
    assert np.allclose(y[..., D // 2:], zr.imag, atol=1e-9)
    assert np.allclose(O.rope(y, pos, inv), x, atol=1e-9)
    assert np.allclose(O.rope_inverse(O.rope(x, pos, inv), pos, inv), x, atol=1e-9)


def check_inv_freq():
    inv = O.rope_inv_freq(10000.0, 128)
    assert inv[0] == 1.0
    assert inv[32] == float(np.float32(0.01))  # 10000 ** (-64/128)
    assert all(a > b for a, b in zip(inv, inv[1:]))
    assert np.all(inv.astype(np.float32).astype(np.float64) == inv)  # fp32 values


def check_key_norm():
    rng = np.random.default_rng(4)
    x = rng.normal(size=(4, 2, 32)) * 3.0
    g = np.ones(32)
    y = O.key_norm(x, g, 0.0)
    assert np.allclose(np.mean(y * y, axis=-1), 1.0)
    assert np.allclose(O.key_norm(5.0 * x, g, 0.0), y)  # scale invariant
    g2 = rng.uniform(0.5, 2.0, size=32)
    assert np.allclose(O.key_norm(x, g2, 0.0), y * g2)


# ---------------------------------------------------------------------------
# The transfer
# ---------------------------------------------------------------------------

def _tiny_problem(seed, align_mode, layer_mode, L_s=3, L_r=4, H_s=2, D_s=4, H_r=2, D_r=4,
                  n_chars=23):
    rng = random.Random(seed)
    nrng = np.random.default_rng(seed)
    s_end = _random_segmentation(rng, n_chars, 1, 5)
    r_end = _random_segmentation(rng, n_chars, 1, 4)
    d_s, d_r = H_s * D_s, H_r * D_r
    sender = nrng.normal(size=(L_s, 2, len(s_end), d_s))
    segs = O.layer_segments(layer_mode, L_s, L_r)
    K = len(segs[0]) * d_s
    A = nrng.normal(size=(L_r, 2, K, d_r)) / math.sqrt(K)
    b = nrng.normal(size=(L_r, 2, d_r)) * 0.1
    r = nrng.uniform(0.5, 2.0, size=(L_r, 2))
    csr = O.alignment_csr(align_mode, [0, len(s_end)], [0, len(r_end)], s_end, r_end)
    inv = O.rope_inv_freq(10000.0, D_r)
    pos = O.receiver_positions([0, len(r_end)], [5])
    return dict(sender=sender, segs=segs, A=A, b=b, r=r, csr=csr, inv=inv, pos=pos,
                H_r=H_r, D_r=D_r, d_s=d_s, s_end=s_end, r_end=r_end)


def _transfer_brute(P, knorm_g=None, eps=1e-6, srope=None, row_of=None):
    """Every output element from the definitions, with Python loops.
    srope = (s_pos, inv_freq_s, H_s): sender keys carry RoPE and each sender
    feature is rotated back at its token's position before it is used."""
    sender, segs, A, b, r, csr = P["sender"], P["segs"], P["A"], P["b"], P["r"], P["csr"]
    H_r, D_r, d_s, inv, pos = P["H_r"], P["D_r"], P["d_s"], P["inv"], P["pos"]

    def feature(t, c, k, d):
        if row_of is not None:  # sender token k lives at cache row row_of[k]
            kr = row_of[k]
            v = sender[t, c, kr, d]
            if srope is None or c != 0:
                return v
            s_pos, inv_s, H_s = srope
            D_s = d_s // H_s
            h, i = divmod(d, D_s)
            hs = D_s // 2
            ang = s_pos[k] * inv_s[i % hs]
            if i < hs:
                return v * math.cos(ang) + sender[t, c, kr, h * D_s + i + hs] * math.sin(ang)
            return v * math.cos(ang) - sender[t, c, kr, h * D_s + i - hs] * math.sin(ang)
        v = sender[t, c, k, d]
        if srope is None or c != 0:
            return v
        s_pos, inv_s, H_s = srope
        D_s = d_s // H_s
        h, i = divmod(d, D_s)
        hs = D_s // 2
        f = inv_s[i % hs]
        ang = s_pos[k] * f
        if i < hs:  # x' = x cos + y sin
            return v * math.cos(ang) + sender[t, c, k, h * D_s + i + hs] * math.sin(ang)
        return v * math.cos(ang) - sender[t, c, k, h * D_s + i - hs] * math.sin(ang)

    out = {}
    for l in range(len(segs)):
        for c in (0, 1):
            res = np.zeros((csr.n_rows, H_r, D_r))
            for j in range(csr.n_rows):
                y = []
                for n in range(H_r * D_r):
                    acc = 0.0
                    for s, seg in enumerate(segs[l]):
                        for (t, omega) in seg:
                            for e in range(csr.row_ptr[j], csr.row_ptr[j + 1]):
                                k, wk = csr.col[e], csr.w[e]
                                for d in range(d_s):
                                    acc += omega * wk * feature(t, c, k, d) * A[l, c, s * d_s + d, n]
                    y.append(acc / r[l, c] + b[l, c, n])
                for h in range(H_r):
                    v = y[h * D_r:(h + 1) * D_r]
                    if c == 0:
                        if knorm_g is not None:
                            rms = math.sqrt(sum(t * t for t in v) / D_r + eps)
                            v = [t / rms * knorm_g[i] for i, t in enumerate(v)]
                        half = D_r // 2
                        w_ = list(v)
                        for i in range(half):
                            ang = pos[j] * inv[i]
                            w_[i] = v[i] * math.cos(ang) - v[i + half] * math.sin(ang)
                            w_[i + half] = v[i + half] * math.cos(ang) + v[i] * math.sin(ang)
                        v = w_
                    res[j, h] = v
            out[(l, c)] = res
    return out


def _run_oracle(P, **kw):
    return O.transfer(P["sender"], P["csr"], P["segs"], P["A"], P["b"], P["r"],
                      H_r=P["H_r"], D_r=P["D_r"], pos=P["pos"], inv_freq_r=P["inv"], **kw)


def check_transfer_brute_force():
    for seed, am, lm in [(0, O.ALIGN_TA, O.LAYER_PAPER3),
                         (1, O.ALIGN_OVERLAP_MEAN, O.LAYER_INTERP),
                         (2, O.ALIGN_OVERLAP_MEAN, O.LAYER_PAPER3),
                         (3, O.ALIGN_TA, O.LAYER_INTERP),
                         (4, O.ALIGN_SAME_INDEX, O.LAYER_PAPER3)]:
        P = _tiny_problem(seed, am, lm)
        got = _run_oracle(P)
        ref = _transfer_brute(P)
        for key in ref:
            assert np.allclose(got[key], ref[key], rtol=1e-10, atol=1e-10), (seed, key)
    P = _tiny_problem(5, O.ALIGN_TA, O.LAYER_PAPER3)
    g = np.random.default_rng(9).uniform(0.5, 1.5, size=P["D_r"])
    got = _run_oracle(P, knorm_g=g, knorm_eps=1e-6)
    ref = _transfer_brute(P, knorm_g=g, eps=1e-6)
    for key in ref:
        assert np.allclose(got[key], ref[key], rtol=1e-10, atol=1e-10)


def check_transfer_brute_force_rotated_sender():
    """Sender keys stored with RoPE: the brute force rotates each sender
    feature back at its own sender position; pooled and blended modes."""
    for seed, am, lm in [(10, O.ALIGN_TA, O.LAYER_PAPER3),
                         (11, O.ALIGN_OVERLAP_MEAN, O.LAYER_INTERP)]:
        P = _tiny_problem(seed, am, lm)
        n_s = len(P["s_end"])
        s_pos = O.sender_positions([0, n_s], [3])
        assert s_pos.tolist() == list(range(3, 3 + n_s))
        inv_s = O.rope_inv_freq(500000.0, 4)
        got = _run_oracle(P, sender_rope=(s_pos, inv_s, 2))
        ref = _transfer_brute(P, srope=(s_pos, inv_s, 2))
        for key in ref:
            assert np.allclose(got[key], ref[key], rtol=1e-10, atol=1e-10), (seed, key)


def check_message_spans():
    """Message spans: request q's sender tokens are the cache rows
    s_row0[q] .. s_row0[q] + n_q - 1 of a longer sender cache.  Brute force
    with explicit row arithmetic, and the same transfer on a cache that holds
    only the spans (concatenated) gives the same result."""
    rng = np.random.default_rng(16)
    L_s, L_r, H, D = 3, 4, 2, 4
    d = H * D
    s_ends = [_ends([2, 1, 3, 2]), _ends([1, 2, 2])]          # two messages
    r_ends = [_ends([3, 1, 2, 2]), _ends([2, 3])]
    s_ptr = [0, 4, 7]
    r_ptr = [0, 4, 6]
    s_row0 = [10, 3]                                          # spans inside a 20-row cache
    rows = O.span_rows(s_ptr, s_row0)
    assert rows.tolist() == [10, 11, 12, 13, 3, 4, 5]
    cache = rng.normal(size=(L_s, 2, 20, d))
    csr = O.alignment_csr(O.ALIGN_OVERLAP_MEAN, s_ptr, r_ptr, sum(s_ends, []), sum(r_ends, []))
    segs = O.layer_segments(O.LAYER_PAPER3, L_s, L_r)
    A = rng.normal(size=(L_r, 2, 3 * d, d)) / math.sqrt(3 * d)
    b = rng.normal(size=(L_r, 2, d)) * 0.1
    r = rng.uniform(0.5, 2.0, size=(L_r, 2))
    inv = O.rope_inv_freq(10000.0, D)
    pos = O.receiver_positions(r_ptr, [100, 7])
    s_pos = O.sender_positions(s_ptr, [40, 9])
    P = dict(sender=cache, segs=segs, A=A, b=b, r=r, csr=csr, inv=inv, pos=pos, H_r=H, D_r=D, d_s=d)
    srope = (s_pos, O.rope_inv_freq(5e5, D), H)
    got = _run_oracle(P, sender_rope=srope, sender_row_of=rows)
    ref = _transfer_brute(P, srope=srope, row_of=rows)
    for key in ref:
        assert np.allclose(got[key], ref[key], rtol=1e-10, atol=1e-10), key
    packed = cache[:, :, rows, :]                              # the spans alone
    alone = _run_oracle(dict(P, sender=packed), sender_rope=srope)
    for key in ref:
        assert np.allclose(alone[key], got[key], rtol=1e-12, atol=1e-12), key


def check_explicit_segments():
    """A caller-given layer table: the Eq. 1 triples given explicitly give
    the paper-mode table, and a hand-made two-term table maps as written."""
    L_s, L_r = 32, 40
    trip = O.layer_alignment(L_s, L_r)
    ex = O.explicit_segments([[[t] for t in tr] for tr in trip], [[[1.0]] * 3 for _ in trip])
    assert ex == O.layer_segments(O.LAYER_PAPER3, L_s, L_r)
    ex2 = O.explicit_segments([[[0, 2], [1, 1]]], [[[0.25, 0.75], [1.0, -2.0]]])
    assert ex2 == [[[(0, 0.25), (2, 0.75)], [(1, 1.0), (1, -2.0)]]]
    P = _tiny_problem(12, O.ALIGN_OVERLAP_MEAN, O.LAYER_PAPER3, L_s=3, L_r=1)
    P["segs"] = ex2
    P["A"] = P["A"][:, :, : 2 * P["d_s"], :]
    got = _run_oracle(P)
    ref = _transfer_brute(P)
    for key in ref:
        assert np.allclose(got[key], ref[key], rtol=1e-10, atol=1e-10), key
    # segment 1 is (1 - 2) * layer 1 = -layer 1
    A1 = np.zeros_like(P["A"])
    A1[:, :, P["d_s"]:, :] = P["A"][:, :, P["d_s"]:, :]
    y = _run_oracle(dict(P, A=A1), roles=(1,))[(0, 1)]
    rows = np.arange(P["csr"].n_rows)
    x = O.pooled_features(P["sender"][1, 1], P["csr"], rows)
    ref1 = -x @ P["A"][0, 1, P["d_s"]:, :] / P["r"][0, 1] + P["b"][0, 1]
    assert np.allclose(y.reshape(len(rows), -1), ref1)


def _kv_ridge_problem(seed, align_mode, L_s=5, L_r=3, H_s=2, D_s=4, H_r=2, D_r=4, k=3):
    P = _tiny_problem(seed, align_mode, O.LAYER_PAPER3, L_s=L_s, L_r=L_r, H_s=H_s, D_s=D_s,
                      H_r=H_r, D_r=D_r)
    rng = np.random.default_rng(seed + 100)
    sel = [sorted(rng.choice(L_s, size=k, replace=False).tolist()) for _ in range(L_r)]
    Kin = k * H_s * D_s
    Wh = rng.normal(size=(L_r, 2, H_r, Kin, D_r)) / math.sqrt(Kin)
    bh = rng.normal(size=(L_r, 2, H_r, D_r)) * 0.1
    return P, sel, Wh, bh


def check_kv_ridge_brute_force():
    """The KV Ridge apply element by element with Python loops: receiver head
    h of layer l, role c at receiver row j is sum over the selected sender
    layers s, every sender feature f (all heads) of the aligned token, of
    x[s][f] * W_h[s * d_S + f][d], plus the head's bias; keys rotated."""
    for seed, am in [(30, O.ALIGN_TA), (31, O.ALIGN_SAME_INDEX), (32, O.ALIGN_OVERLAP_MEAN)]:
        P, sel, Wh, bh = _kv_ridge_problem(seed, am)
        sender, csr, d_s = P["sender"], P["csr"], P["d_s"]
        H_r, D_r, inv, pos = P["H_r"], P["D_r"], P["inv"], P["pos"]
        got = O.kv_ridge_transfer(sender, csr, sel, Wh, bh, H_r=H_r, D_r=D_r, pos=pos,
                                  inv_freq_r=inv)
        for l in range(len(sel)):
            for c in (0, 1):
                for j in range(csr.n_rows):
                    y = np.zeros((H_r, D_r))
                    for h in range(H_r):
                        for d in range(D_r):
                            acc = bh[l, c, h, d]
                            for si, t in enumerate(sel[l]):
                                for e in range(csr.row_ptr[j], csr.row_ptr[j + 1]):
                                    for f in range(d_s):
                                        acc += (csr.w[e] * sender[t, c, csr.col[e], f]
                                                * Wh[l, c, h, si * d_s + f, d])
                            y[h, d] = acc
                    if c == 0:
                        half = D_r // 2
                        z = y.copy()
                        for i in range(half):
                            a = pos[j] * inv[i]
                            z[:, i] = y[:, i] * math.cos(a) - y[:, i + half] * math.sin(a)
                            z[:, i + half] = y[:, i + half] * math.cos(a) + y[:, i] * math.sin(a)
                        y = z
                    assert np.allclose(got[(l, c)][j], y, rtol=1e-10, atol=1e-10), (seed, l, c, j)


def check_kv_ridge_equals_stacked_map():
    """The per-head maps stacked column-wise (head-major, h * D_R + d) are one
    dense [k d_S, d_R] map: the KV Ridge apply equals transfer() with the
    k one-layer segments, that map, the stacked biases and r = 1."""
    for seed, am in [(33, O.ALIGN_TA), (34, O.ALIGN_OVERLAP_MEAN)]:
        P, sel, Wh, bh = _kv_ridge_problem(seed, am, L_s=9, L_r=4, k=8)
        H_r, D_r = P["H_r"], P["D_r"]
        L_r = len(sel)
        A = np.concatenate([Wh[:, :, h] for h in range(H_r)], axis=-1)  # [L_r, 2, K, d_R]
        b = bh.reshape(L_r, 2, H_r * D_r)
        ridge = O.kv_ridge_transfer(P["sender"], P["csr"], sel, Wh, bh, H_r=H_r, D_r=D_r,
                                    pos=P["pos"], inv_freq_r=P["inv"])
        segs = O.kv_ridge_segments(sel)
        assert all(len(sg) == 8 and all(len(t) == 1 and t[0][1] == 1.0 for t in sg)
                   for sg in segs)
        dense = O.transfer(P["sender"], P["csr"], segs, A, b, np.ones((L_r, 2)), H_r=H_r,
                           D_r=D_r, pos=P["pos"], inv_freq_r=P["inv"])
        for key in ridge:
            assert np.allclose(ridge[key], dense[key], rtol=1e-12, atol=1e-12), (seed, key)


def check_identity_map_reproduces_input():
    """Same depth, same tokenisation, A = [0; I; 0] (the middle block reads
    sender layer pi(l) = l), b = 0, r = 1: V is the sender V, K is the sender K
    rotated to its receiver position (the identity at position 0)."""
    L, H, D = 5, 2, 8
    d = H * D
    rng = np.random.default_rng(5)
    ends = _ends([2, 1, 3, 4, 1, 2, 5])
    sender = rng.normal(size=(L, 2, len(ends), d))
    segs = O.layer_segments(O.LAYER_PAPER3, L, L)
    A = np.zeros((L, 2, 3 * d, d))
    A[:, :, d:2 * d, :] = np.eye(d)
    b = np.zeros((L, 2, d))
    r = np.ones((L, 2))
    csr = O.alignment_csr(O.ALIGN_TA, [0, len(ends)], [0, len(ends)], ends, ends)
    inv = O.rope_inv_freq(10000.0, D)
    pos = O.receiver_positions([0, len(ends)])
    out = O.transfer(sender, csr, segs, A, b, r, H_r=H, D_r=D, pos=pos, inv_freq_r=inv)
    for l in range(L):
        assert np.array_equal(out[(l, 1)].reshape(len(ends), d), sender[l, 1])
        assert np.array_equal(out[(l, 0)][0].reshape(d), sender[l, 0, 0])
        z = sender[l, 0].reshape(len(ends), H, D)
        zc = z[..., : D // 2] + 1j * z[..., D // 2:]
        zc = zc * np.exp(1j * pos[:, None, None] * inv[None, None, :])
        assert np.allclose(out[(l, 0)][..., : D // 2], zc.real)
        assert np.allclose(out[(l, 0)][..., D // 2:], zc.imag)


def _recolor_data(seed, N, d_s, d_r, noise):
    rng = np.random.default_rng(seed)
    X = rng.normal(size=(N, d_s)) @ rng.normal(size=(d_s, d_s)) * 0.7 + rng.normal(size=d_s)
    A_true = rng.normal(size=(d_s, d_r)) / np.sqrt(d_s)
    Y = X @ A_true + 0.3 + noise * rng.normal(size=(N, d_r))
    w = rng.uniform(0.5, 2.0, size=N)
    return X, Y, w


def check_sender_rms():
    """Eq. 3: samples all of squared norm d~ s^2 give r = s, whatever the
    weights; doubling every weight leaves r unchanged."""
    rng = np.random.default_rng(19)
    X = rng.normal(size=(50, 6))
    X = X / np.linalg.norm(X, axis=1, keepdims=True) * np.sqrt(6) * 1.7
    w = rng.uniform(0.1, 3.0, size=50)
    assert abs(O.sender_rms(X, w) - 1.7) < 1e-12
    X2 = rng.normal(size=(40, 5))
    assert abs(O.sender_rms(X2, w[:40]) - O.sender_rms(X2, 2 * w[:40])) < 1e-12
    # brute force
    num = sum(w[n] * sum(X2[n, j] ** 2 for j in range(5)) for n in range(40))
    assert abs(O.sender_rms(X2, w[:40]) - math.sqrt(num / (5 * sum(w[:40])))) < 1e-12


def check_weighted_moments_brute_force():
    rng = np.random.default_rng(20)
    Z = rng.normal(size=(30, 4))
    Y = rng.normal(size=(30, 3))
    w = rng.uniform(0.2, 2.0, size=30)
    mu_z, mu_y, S_z, S_y, S_zy = O.weighted_moments(Z, Y, w)
    W = sum(w)
    for i in range(4):
        m = sum(w[n] * Z[n, i] for n in range(30)) / W
        assert abs(mu_z[i] - m) < 1e-12
        for j in range(3):
            my = sum(w[n] * Y[n, j] for n in range(30)) / W
            c = sum(w[n] * (Z[n, i] - m) * (Y[n, j] - my) for n in range(30)) / W
            assert abs(S_zy[i, j] - c) < 1e-12
    assert np.allclose(S_z, S_z.T) and np.allclose(S_y, S_y.T)


def check_recolor_moment_identities():
    """Eq. 5 (unregularised, nonsingular, d~_S >= d_R): mu_Z A + b = mu_Y and
    A^T Sigma_Z A = Sigma_Y."""
    X, Y, w = _recolor_data(21, 400, 7, 5, 0.5)
    A, b, r = O.recolor(X, Y, w)
    mu_z, mu_y, S_z, S_y, _ = O.weighted_moments(X / r, Y, w)
    assert np.allclose(mu_z @ A + b, mu_y, atol=1e-10)
    assert np.allclose(A.T @ S_z @ A, S_y, atol=1e-9)


def check_recolor_recovers_an_exact_rotation():
    """If Y = Z Q + c with Q orthogonal (d~_S = d_R), then Sigma_ZY =
    Sigma_Z Q, the whitened cross-covariance is Q itself, R* = Q, and the
    fit returns A = Q, b = c exactly."""
    rng = np.random.default_rng(22)
    d = 6
    X = rng.normal(size=(300, d)) @ rng.normal(size=(d, d)) + 2.0
    w = rng.uniform(0.5, 1.5, size=300)
    Q, _ = np.linalg.qr(rng.normal(size=(d, d)))
    c = rng.normal(size=d)
    r = O.sender_rms(X, w)
    Y = (X / r) @ Q + c
    A, b, r2 = O.recolor(X, Y, w)
    assert abs(r2 - r) < 1e-12
    assert np.allclose(A, Q, atol=1e-9) and np.allclose(b, c, atol=1e-9)


def check_fold_closed_forms():
    """Eq. 9 folding: G = 0 leaves the map unchanged; a rank-1 correction
    B = u, G = v^T gives A + (A u) v^T element by element; B = e_i, G = -e_i^T
    removes output feature i (I + B G is a projector)."""
    rng = np.random.default_rng(17)
    K, d, rho = 7, 5, 3
    A = rng.normal(size=(K, d))
    b = rng.normal(size=d)
    Af, bf = O.fold(A, b, rng.normal(size=(d, rho)), np.zeros((rho, d)))
    assert np.array_equal(Af, A) and np.array_equal(bf, b)
    u = rng.normal(size=(d, 1))
    v = rng.normal(size=(1, d))
    Af, bf = O.fold(A, b, u, v)
    for k in range(K):
        au = sum(A[k, n] * u[n, 0] for n in range(d))
        for n in range(d):
            assert abs(Af[k, n] - (A[k, n] + au * v[0, n])) < 1e-12
    bu = sum(b[n] * u[n, 0] for n in range(d))
    assert np.allclose(bf, b + bu * v[0])
    i = 2
    e = np.zeros((d, 1))
    e[i, 0] = 1.0
    Af, bf = O.fold(A, b, e, -e.T)
    assert np.allclose(Af[:, i], 0.0) and abs(bf[i]) < 1e-12
    keep = [n for n in range(d) if n != i]
    assert np.allclose(Af[:, keep], A[:, keep]) and np.allclose(bf[keep], b[keep])


def check_fold_equals_unfused_correction():
    """Eq. 7 applied at transfer time (y0 + (y0 B) G, then key norm and RoPE)
    equals the transfer with the Eq. 9 folded maps, keys and values."""
    P = _tiny_problem(18, O.ALIGN_OVERLAP_MEAN, O.LAYER_PAPER3)
    rng = np.random.default_rng(18)
    L_r, d_r = P["A"].shape[0], P["A"].shape[3]
    Bm = rng.normal(size=(L_r, 2, d_r, 2)) * 0.3
    Gm = rng.normal(size=(L_r, 2, 2, d_r)) * 0.3
    Af = np.zeros_like(P["A"])
    bf = np.zeros_like(P["b"])
    for l in range(L_r):
        for c in range(2):
            Af[l, c], bf[l, c] = O.fold(P["A"][l, c], P["b"][l, c], Bm[l, c], Gm[l, c])
    g = rng.uniform(0.5, 1.5, size=P["D_r"])
    folded = _run_oracle(dict(P, A=Af, b=bf), knorm_g=g)
    unfused = O.transfer_unfused(P["sender"], P["csr"], P["segs"], P["A"], P["b"], P["r"], Bm, Gm,
                                 H_r=P["H_r"], D_r=P["D_r"], pos=P["pos"], inv_freq_r=P["inv"],
                                 knorm_g=g)
    for key in unfused:
        assert np.allclose(folded[key], unfused[key], rtol=1e-10, atol=1e-10), key


def _identity_setup(L, H, D, lengths, seed):
    d = H * D
    rng = np.random.default_rng(seed)
    ends = _ends(lengths)
    sender = rng.normal(size=(L, 2, len(ends), d))
    segs = O.layer_segments(O.LAYER_PAPER3, L, L)
    A = np.zeros((L, 2, 3 * d, d))
    A[:, :, d:2 * d, :] = np.eye(d)
    csr = O.alignment_csr(O.ALIGN_TA, [0, len(ends)], [0, len(ends)], ends, ends)
    return sender, segs, A, np.zeros((L, 2, d)), np.ones((L, 2)), csr, ends


def check_identity_rotated_sender_keys():
    """The identity special case with sender keys stored rotated: same
    depth, same tokenisation, A = [0; I; 0], b = 0, r = 1, the same RoPE base
    and the same positions on both sides: un-rotate then rotate reproduces
    the sender keys, and values pass through unrotated."""
    L, H, D = 4, 2, 8
    sender, segs, A, b, r, csr, ends = _identity_setup(L, H, D, [1, 3, 2, 2, 4, 1], 13)
    n = len(ends)
    inv = O.rope_inv_freq(10000.0, D)
    pos = O.receiver_positions([0, n], [7])
    s_pos = O.sender_positions([0, n], [7])
    out = O.transfer(sender, csr, segs, A, b, r, H_r=H, D_r=D, pos=pos, inv_freq_r=inv,
                     sender_rope=(s_pos, inv, H))
    for l in range(L):
        assert np.allclose(out[(l, 0)].reshape(n, H * D), sender[l, 0], atol=1e-12)
        assert np.array_equal(out[(l, 1)].reshape(n, H * D), sender[l, 1])


def check_rotated_sender_position_shift():
    """Sender keys rotated at sender positions p (base theta_s), receiver at
    p + delta (base theta_r), identity map: in complex form each pair is
    multiplied by exp(1j ((p + delta) f_r - p f_s))."""
    L, H, D = 3, 1, 8
    sender, segs, A, b, r, csr, ends = _identity_setup(L, H, D, [2, 2, 1, 3, 2], 14)
    n = len(ends)
    inv_r = O.rope_inv_freq(1e6, D)
    inv_s = O.rope_inv_freq(5e5, D)
    pos = O.receiver_positions([0, n], [11])
    s_pos = O.sender_positions([0, n])
    out = O.transfer(sender, csr, segs, A, b, r, H_r=H, D_r=D, pos=pos, inv_freq_r=inv_r,
                     sender_rope=(s_pos, inv_s, H), roles=(0,))
    for l in range(L):
        z = sender[l, 0].reshape(n, H, D)
        zc = z[..., : D // 2] + 1j * z[..., D // 2:]
        ang = pos[:, None, None] * inv_r[None, None, :] - s_pos[:, None, None] * inv_s[None, None, :]
        zc = zc * np.exp(1j * ang)
        assert np.allclose(out[(l, 0)][..., : D // 2], zc.real, atol=1e-12)
        assert np.allclose(out[(l, 0)][..., D // 2:], zc.imag, atol=1e-12)


def check_rotated_sender_unrotates_before_pooling():
    """Every sender key is one vector v rotated to its own position; overlap
    mean pooling of the un-rotated keys gives v exactly, whatever the rows'
    spans, so with the identity map the receiver key is v rotated to the
    receiver position.  Rotating back after pooling would not give v."""
    L, H, D = 3, 2, 8
    d = H * D
    rng = np.random.default_rng(15)
    s_end = _ends([2, 1, 3, 1, 1, 4, 2])
    r_end = _ends([3, 4, 1, 3, 3])
    assert s_end[-1] == r_end[-1]
    n_s, n_r = len(s_end), len(r_end)
    inv = O.rope_inv_freq(10000.0, D)
    s_pos = O.sender_positions([0, n_s], [5])
    v = rng.normal(size=(1, H, D))
    rotated = O.rope(np.repeat(v, n_s, axis=0), s_pos, inv).reshape(n_s, d)
    sender = np.zeros((L, 2, n_s, d))
    sender[:, 0] = rotated
    segs = O.layer_segments(O.LAYER_PAPER3, L, L)
    A = np.zeros((L, 2, 3 * d, d))
    A[:, :, d:2 * d, :] = np.eye(d)
    csr = O.alignment_csr(O.ALIGN_OVERLAP_MEAN, [0, n_s], [0, n_r], s_end, r_end)
    assert max(csr.row_ptr[j + 1] - csr.row_ptr[j] for j in range(n_r)) > 1
    pos = O.receiver_positions([0, n_r])
    out = O.transfer(sender, csr, segs, A, np.zeros((L, 2, d)), np.ones((L, 2)), H_r=H, D_r=D,
                     pos=pos, inv_freq_r=inv, sender_rope=(s_pos, inv, H), roles=(0,))
    want = O.rope(np.repeat(v, n_r, axis=0), pos, inv)
    for l in range(L):
        assert np.allclose(out[(l, 0)], want, atol=1e-12)


def check_affine_structure():
    """Eq. 9 is affine in the sender features with slope 1/r: zero input gives
    the bias; scaling the sender scales (y - b); doubling r halves it."""
    P = _tiny_problem(6, O.ALIGN_OVERLAP_MEAN, O.LAYER_PAPER3)
    base = _run_oracle(P, roles=(1,))
    P0 = dict(P, sender=np.zeros_like(P["sender"]))
    zero = _run_oracle(P0, roles=(1,))
    for (l, c), y in zero.items():
        assert np.allclose(y.reshape(y.shape[0], -1), P["b"][l, c][None, :])
    P2 = dict(P, sender=2.5 * P["sender"])
    scaled = _run_oracle(P2, roles=(1,))
    Pr = dict(P, r=2.0 * P["r"])
    halved = _run_oracle(Pr, roles=(1,))
    for (l, c), y in base.items():
        bb = P["b"][l, c].reshape(1, P["H_r"], P["D_r"])
        assert np.allclose(scaled[(l, c)] - bb, 2.5 * (y - bb))
        assert np.allclose(halved[(l, c)] - bb, 0.5 * (y - bb))


def check_segment_blocks():
    """Segment s multiplies rows [s d_S, (s+1) d_S) of A: zeroing all but one
    block equals mapping that sender layer alone with that block."""
    P = _tiny_problem(8, O.ALIGN_TA, O.LAYER_PAPER3)
    d_s = P["d_s"]
    for s in range(3):
        A1 = np.zeros_like(P["A"])
        A1[:, :, s * d_s:(s + 1) * d_s, :] = P["A"][:, :, s * d_s:(s + 1) * d_s, :]
        got = _run_oracle(dict(P, A=A1), roles=(1,))
        for (l, c), y in got.items():
            t = P["segs"][l][s][0][0]
            a = P["csr"].col[P["csr"].row_ptr[:-1]]
            x = P["sender"][t, c][a]
            ref = x @ P["A"][l, c, s * d_s:(s + 1) * d_s, :] / P["r"][l, c] + P["b"][l, c]
            assert np.allclose(y.reshape(len(a), -1), ref)


ALL_CHECKS = [
    check_ta_worked_example, check_ta_literal_shared_boundary, check_ta_brute_force,
    check_ta_identity, check_same_index, check_overlap_brute_force, check_csr_batching,
    check_layer_alignment_closed_form, check_layer_alignment_hand_tables,
    check_layer_interpolation, check_mapper_size_table_f, check_mapper_size_table_f_kv_ridge,
    check_kv_ridge_brute_force, check_kv_ridge_equals_stacked_map,
    check_rope_two_dim_rotation, check_rope_complex_form, check_rope_relative_position,
    check_rope_inverse, check_inv_freq, check_key_norm,
    check_transfer_brute_force, check_transfer_brute_force_rotated_sender,
    check_explicit_segments, check_message_spans, check_identity_map_reproduces_input,
    check_identity_rotated_sender_keys, check_rotated_sender_position_shift,
    check_rotated_sender_unrotates_before_pooling,
    check_fold_closed_forms, check_fold_equals_unfused_correction,
    check_sender_rms, check_weighted_moments_brute_force, check_recolor_moment_identities,
    check_recolor_recovers_an_exact_rotation,
    check_affine_structure, check_segment_blocks,
]


def run_all():
    failures = []
    for chk in ALL_CHECKS:
        try:
            chk()
        except AssertionError as e:  # pragma: no cover - reported by the caller
            failures.append((chk.__name__, repr(e)[:200]))
        except Exception as e:  # a mutated oracle may also raise
            failures.append((chk.__name__, repr(e)[:200]))
    return failures
