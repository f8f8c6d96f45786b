"""Plant plausible mistakes in the oracle (on the CPU) and check that the
pins catch every one of them: evidence that the pins constrain each part of
the oracle, not just its happy path."""
import math

import numpy as np
import pytest

import oracle_pins as pins
from oracle import heterofold_oracle as O


def _ta_any_sender_boundary(s_end, r_end):
    # wrong reading: latest *sender* boundary, shared or not
    s, r = list(s_end), list(r_end)
    out = []
    for e in r:
        before = [i for i, x in enumerate(s) if x <= e]
        out.append(before[-1] if before else 0)
    return np.asarray(out)


def _ta_next_boundary(s_end, r_end):
    # wrong: the sender token that contains the receiver token's end
    s = list(s_end)
    return np.asarray([next(i for i, x in enumerate(s) if x >= e) for e in r_end])


def _depth_floor(l1, L_s, L_r):
    if L_r == 1:
        return 1
    return 1 + ((l1 - 1) * (L_s - 1)) // (L_r - 1)


def _layer_alignment_offsets3(L_s, L_r):
    return [tuple(min(max(O.proportional_depth(l, L_s, L_r) + o, 1), L_s) - 1
                  for o in (-3, 0, 3)) for l in range(1, L_r + 1)]


def _rope_sign(x, pos, inv):
    D = x.shape[-1]
    h = D // 2
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    return np.concatenate([x[..., :h] * c + x[..., h:] * s, x[..., h:] * c - x[..., :h] * s], -1)


def _rope_interleaved(x, pos, inv):
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    y = x.copy()
    y[..., 0::2] = x[..., 0::2] * c - x[..., 1::2] * s
    y[..., 1::2] = x[..., 1::2] * c + x[..., 0::2] * s
    return y


def _inv_freq_wrong(theta, D):
    return np.array([np.float32(float(theta) ** (-(1.0 * i) / D)) for i in range(D // 2)],
                    dtype=np.float64)


def _key_norm_no_weight(x, g, eps):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def _interp_swapped(L_s, L_r):
    out = []
    for l in range(L_r):
        p = (l * (L_s - 1)) / (L_r - 1) if L_r > 1 else 0.0
        i0 = int(math.floor(p))
        f = p - i0
        terms = [(i0, f)] if f > 0 else [(i0, 1.0)]
        if f > 0:
            terms.append((min(i0 + 1, L_s - 1), 1.0 - f))
        out.append(terms)
    return out


def _overlap_closed(s_end, r_end):
    # wrong: spans that merely touch count as overlapping
    s, r = list(s_end), list(r_end)
    rows = []
    for j, e in enumerate(r):
        st = r[j - 1] if j else 0
        rows.append([k for k in range(len(s)) if (s[k - 1] if k else 0) <= e and s[k] >= st])
    return rows


def _pool_unweighted(sender_lc, csr, rows, unrotate=None, row_of=None):
    out = []
    for j in rows:
        idx = csr.col[csr.row_ptr[j]:csr.row_ptr[j + 1]]
        x = np.asarray(sender_lc[idx if row_of is None else np.asarray(row_of)[idx]],
                       dtype=np.float64)
        if unrotate is not None:
            s_pos, inv, H_s = unrotate
            x = O.rope_inverse(x.reshape(len(idx), H_s, -1), np.asarray(s_pos)[idx], inv).reshape(len(idx), -1)
        out.append(x.sum(axis=0))
    return np.asarray(out)


def _rope_inverse_forward(x, pos, inv):
    # wrong: rotates forward instead of back
    return O.rope(x, pos, inv)


_orig_pooled = O.pooled_features


def _pool_then_unrotate(sender_lc, csr, rows, unrotate=None, row_of=None):
    # wrong: pools the rotated rows, then rotates back once at the row's
    # first sender position
    y = _orig_pooled(sender_lc, csr, rows, None, row_of)
    if unrotate is None:
        return y
    s_pos, inv, H_s = unrotate
    first = csr.col[csr.row_ptr[rows]]
    n, d = y.shape
    return O.rope_inverse(y.reshape(n, H_s, d // H_s), np.asarray(s_pos)[first], inv).reshape(n, d)


def _span_rows_from_zero(s_tok_ptr, s_row0):
    # wrong: ignores the span origins
    return np.arange(int(s_tok_ptr[-1]), dtype=np.int64)


def _fold_without_identity(A, b, B, G):
    # wrong: A B G instead of A (I + B G)
    M = np.asarray(B, dtype=np.float64) @ np.asarray(G, dtype=np.float64)
    return np.asarray(A, dtype=np.float64) @ M, np.asarray(b, dtype=np.float64) @ M


def _fold_bias_unchanged(A, b, B, G):
    # wrong: the bias is not folded
    M = np.eye(np.asarray(A).shape[1]) + np.asarray(B) @ np.asarray(G)
    return np.asarray(A, dtype=np.float64) @ M, np.asarray(b, dtype=np.float64)


def _rms_unweighted(X, w):
    X = np.asarray(X, dtype=np.float64)
    return float(np.sqrt(np.mean(X * X)))


_orig_recolor = O.recolor


def _recolor_transposed_rotation(X, Y, w, reg=0.0):
    # wrong: the transposed rotation (R*^T) where it is square
    r = O.sender_rms(X, w)
    Z = np.asarray(X, dtype=np.float64) / r
    mu_z, mu_y, S_z, S_y, S_zy = O.weighted_moments(Z, Y, w)
    lz, Vz = np.linalg.eigh(S_z)
    ly, Vy = np.linalg.eigh(S_y)
    Sz_ih = (Vz * lz ** -0.5) @ Vz.T
    Sy_ih = (Vy * ly ** -0.5) @ Vy.T
    Sy_h = (Vy * ly ** 0.5) @ Vy.T
    U, _, Qt = np.linalg.svd(Sz_ih @ S_zy @ Sy_ih, full_matrices=False)
    R = U @ Qt
    A = Sz_ih @ (R.T if R.shape[0] == R.shape[1] else R) @ Sy_h
    return A, mu_y - mu_z @ A, r


def _recolor_no_whitening(X, Y, w, reg=0.0):
    # wrong: Procrustes on the raw cross-covariance
    r = O.sender_rms(X, w)
    Z = np.asarray(X, dtype=np.float64) / r
    mu_z, mu_y, S_z, S_y, S_zy = O.weighted_moments(Z, Y, w)
    U, _, Qt = np.linalg.svd(S_zy, full_matrices=False)
    A = U @ Qt
    return A, mu_y - mu_z @ A, r


def _explicit_weights_swapped(seg_layer, seg_w):
    return [[[(int(t), float(w)) for t, w in zip(ts, reversed(ws))] for ts, ws in zip(ls, wl)]
            for ls, wl in zip(seg_layer, seg_w)]


_orig_map_input = O.map_input
_orig_transfer = O.transfer


def _map_input_reversed(sender, csr, segments_l, role, rows, sender_rope=None,
                        sender_row_of=None):
    return _orig_map_input(sender, csr, list(reversed(segments_l)), role, rows, sender_rope,
                           sender_row_of)


def _map_input_unrotates_values(sender, csr, segments_l, role, rows, sender_rope=None,
                                sender_row_of=None):
    # wrong: values are rotated back as well
    parts = []
    for seg in segments_l:
        acc = None
        for (t, omega) in seg:
            term = omega * _orig_pooled(sender[t][role], csr, rows, sender_rope, sender_row_of)
            acc = term if acc is None else acc + term
        parts.append(acc)
    return np.concatenate(parts, axis=1)


def _transfer_no_bias(sender, csr, segments, A, b, r, **kw):
    return _orig_transfer(sender, csr, segments, A, np.zeros_like(np.asarray(b, dtype=np.float64)), r, **kw)


def _transfer_times_r(sender, csr, segments, A, b, r, **kw):
    r2 = 1.0 / np.asarray(r, dtype=np.float64)
    return _orig_transfer(sender, csr, segments, A, b, r2, **kw)


def _kv_ridge_segments_reversed(selected):
    # wrong: the selected layers concatenated in reverse order
    return [[[(int(t), 1.0)] for t in reversed(list(sel))] for sel in selected]


_kv_ridge_ok = O.kv_ridge_transfer


def _kv_ridge_rotates_values(sender, csr, selected, W_heads, b_heads, *, H_r, D_r, pos,
                             inv_freq_r, **kw):
    out = _kv_ridge_ok(sender, csr, selected, W_heads, b_heads, H_r=H_r, D_r=D_r, pos=pos,
                       inv_freq_r=inv_freq_r, **kw)
    rows = np.arange(csr.n_rows) if kw.get("rows") is None else np.asarray(kw["rows"])
    for (l, c), y in out.items():
        if c == O.ROLE_V:
            out[(l, c)] = O.rope(y, np.asarray(pos)[rows], inv_freq_r)
    return out


MUTATIONS = {
    "kv_ridge_segments_reversed": ("kv_ridge_segments", _kv_ridge_segments_reversed),
    "kv_ridge_rotates_values": ("kv_ridge_transfer", _kv_ridge_rotates_values),
    "ta_any_sender_boundary": ("token_alignment", _ta_any_sender_boundary),
    "ta_next_boundary": ("token_alignment", _ta_next_boundary),
    "depth_floor": ("proportional_depth", _depth_floor),
    "offsets_3": ("layer_alignment", _layer_alignment_offsets3),
    "rope_sign": ("rope", _rope_sign),
    "rope_interleaved": ("rope", _rope_interleaved),
    "inv_freq_exponent": ("rope_inv_freq", _inv_freq_wrong),
    "key_norm_weight_dropped": ("key_norm", _key_norm_no_weight),
    "interp_weights_swapped": ("layer_interpolation", _interp_swapped),
    "overlap_touching": ("overlap_alignment", _overlap_closed),
    "pool_unweighted": ("pooled_features", _pool_unweighted),
    "segments_reversed": ("map_input", _map_input_reversed),
    "bias_dropped": ("transfer", _transfer_no_bias),
    "r_multiplies": ("transfer", _transfer_times_r),
    "rope_inverse_forward": ("rope_inverse", _rope_inverse_forward),
    "unrotate_after_pooling": ("pooled_features", _pool_then_unrotate),
    "values_unrotated": ("map_input", _map_input_unrotates_values),
    "explicit_weights_swapped": ("explicit_segments", _explicit_weights_swapped),
    "span_rows_from_zero": ("span_rows", _span_rows_from_zero),
    "fold_without_identity": ("fold", _fold_without_identity),
    "fold_bias_unchanged": ("fold", _fold_bias_unchanged),
    "rms_unweighted": ("sender_rms", _rms_unweighted),
    "recolor_transposed_rotation": ("recolor", _recolor_transposed_rotation),
    "recolor_no_whitening": ("recolor", _recolor_no_whitening),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, monkeypatch):
    attr, fn = MUTATIONS[name]
    monkeypatch.setattr(O, attr, fn)
    failures = pins.run_all()
    assert failures, f"no pin caught the planted mistake {name!r}"
    # a mutation with the wrong call signature would "fail" every pin for the
    # wrong reason; at least one pin must fail on an assertion
    assert any(msg.startswith("AssertionError") for _, msg in failures), failures
