"""Shared machinery of the GPU parity tests: generate a workload's inputs on
the device, run the transfer through the C ABI, and compare with the fp64
oracle fed from the same seeded inputs."""

from __future__ import annotations

import numpy as np
import torch

from oracle import heterofold_oracle as O
from paper_2609_32259_gb300 import pipeline
from paper_2609_32259_gb300 import workloads as W

# Tolerances of the transfer against the fp64 oracle (bf16 inputs, fp32
# accumulation): per receiver layer and role.
REL_FRO_TOL = 5e-3
MAX_ABS_TOL = 2e-2


class RowFetcher:
    """sender[t][c][rows] -> fp32 numpy rows, fetched from the device on demand."""

    def __init__(self, sender: torch.Tensor):
        self.s = sender

    class _LC:
        def __init__(self, t):
            self.t = t

        def __getitem__(self, idx):
            ix = torch.as_tensor(np.asarray(idx, dtype=np.int64), device=self.t.device)
            return self.t.index_select(0, ix).float().cpu().numpy()

    class _L:
        def __init__(self, t):
            self.t = t

        def __getitem__(self, c):
            return RowFetcher._LC(self.t[c])

    def __getitem__(self, t):
        return RowFetcher._L(self.s[t])


class MapFetcher:
    """A[l][c] = W[l][c]^T as fp64 numpy (the paper's x @ A orientation)."""

    def __init__(self, Wm: torch.Tensor):
        self.W = Wm

    class _L:
        def __init__(self, Wl):
            self.Wl = Wl

        def __getitem__(self, c):
            return self.Wl[c].float().cpu().numpy().T

    def __getitem__(self, l):
        return MapFetcher._L(self.W[l])


class HeadMapFetcher:
    """W_h[l][c][h] = the per-head map of receiver head h: columns
    h D_r .. (h+1) D_r - 1 of A = W[l][c]^T, as fp64 numpy."""

    def __init__(self, Wm: torch.Tensor, H_r: int, D_r: int):
        self.W, self.H, self.D = Wm, H_r, D_r

    def __getitem__(self, l):
        W, D = self.W, self.D

        class _LC:
            def __getitem__(_, c):
                A = W[l][c].float().cpu().numpy().T
                return [A[:, h * D:(h + 1) * D] for h in range(A.shape[1] // D)]
        return _LC()


class HeadBiasFetcher:
    """b_h[l][c][h] = the bias of receiver head h, fp64 numpy."""

    def __init__(self, b: torch.Tensor, H_r: int, D_r: int):
        self.b = b.double().cpu().numpy().reshape(b.shape[0], 2, H_r, D_r)

    def __getitem__(self, l):
        return self.b[l]


class Case:
    def __init__(self, w: W.Workload, device="cuda", sentinel=None, **desc_options):
        self.w = w
        self.dev = torch.device(device)
        self.tok = W.tokens(w)
        self.sender = W.sender_kv(w, W.sender_cache_rows(w, self.tok), self.dev)
        self.Wm, self.b, self.r = W.maps(w, self.dev)
        self.paged = W.paged_layout(w, self.tok) if w.paged else None
        self.knorm_w = W.knorm_weight(w)
        self.r_pos0 = W.r_pos0(w)
        self.job = pipeline.job_from_workload(w, self.tok, self.sender, self.Wm, self.b, self.r,
                                              paged=self.paged, knorm_w=self.knorm_w,
                                              r_pos0=self.r_pos0, device=self.dev,
                                              **desc_options)
        if sentinel is not None:
            self.job.receiver.fill_(sentinel)
        self.csr = O.alignment_csr(w.align_mode, self.tok.s_tok_ptr, self.tok.r_tok_ptr,
                                   self.tok.s_end, self.tok.r_end)
        if w.layer_mode == "explicit":
            self.segs = O.explicit_segments(w.seg_layer, np.asarray(w.seg_w, np.float32))
        else:
            self.segs = O.layer_segments(w.layer_mode, w.L_s, w.L_r)
        self.pos = O.receiver_positions(self.tok.r_tok_ptr, self.r_pos0)
        table = W.inv_freq_r_table(w)
        self.inv_freq_r = (O.rope_inv_freq(w.theta_r, w.D_r) if table is None
                           else table.astype(np.float64))
        sp = W.span_layout(w, self.tok)
        self.sender_row_of = None if sp is None else O.span_rows(self.tok.s_tok_ptr, sp[0])
        self.sender_rope = None
        if w.sender_k_rotated:
            self.sender_rope = (O.sender_positions(self.tok.s_tok_ptr, W.s_pos0(w)),
                                O.rope_inv_freq(w.theta_s, w.D_s), w.H_s)

    def run(self):
        self.job.step()
        torch.cuda.synchronize()
        return self

    # --------------------------------------------------------------- checks
    def check_csr(self):
        rp, col, wt = self.job.csr()
        assert self.job.align_status() == 0, self.job.align_status()
        assert np.array_equal(rp, self.csr.row_ptr.astype(np.int32))
        assert np.array_equal(col, self.csr.col.astype(np.int32))
        assert np.array_equal(wt.view(np.uint32), self.csr.w32.view(np.uint32))

    def dst_rows(self, rows):
        rows = np.asarray(rows, dtype=np.int64)
        if self.paged is None:
            return rows
        rp = self.tok.r_tok_ptr
        q = np.searchsorted(rp, rows, side="right") - 1
        t = rows - rp[q]
        bs = self.w.block_size
        return self.paged.block_table[q, t // bs].astype(np.int64) * bs + t % bs

    def gpu_rows(self, l, c, rows):
        d = torch.as_tensor(self.dst_rows(rows), device=self.dev)
        y = self.job.receiver[l, c].index_select(0, d).double().cpu().numpy()
        return y.reshape(len(rows), self.w.H_r, self.w.D_r)

    def oracle(self, layers, rows, roles=(0, 1)):
        if self.w.kv_ridge:  # the per-head formulation, against the stacked map on the GPU
            selected = [[t[0] for t in seg] for seg in self.w.seg_layer]
            return O.kv_ridge_transfer(RowFetcher(self.sender), self.csr, selected,
                                       HeadMapFetcher(self.Wm, self.w.H_r, self.w.D_r),
                                       HeadBiasFetcher(self.b, self.w.H_r, self.w.D_r),
                                       H_r=self.w.H_r, D_r=self.w.D_r, pos=self.pos,
                                       inv_freq_r=self.inv_freq_r, layers=layers, rows=rows,
                                       roles=roles)
        return O.transfer(RowFetcher(self.sender), self.csr, self.segs, MapFetcher(self.Wm),
                          self.b.cpu().numpy(), self.r, H_r=self.w.H_r, D_r=self.w.D_r,
                          pos=self.pos, inv_freq_r=self.inv_freq_r,
                          knorm_g=self.knorm_w, knorm_eps=1e-6, layers=layers, rows=rows,
                          roles=roles, sender_rope=self.sender_rope,
                          sender_row_of=self.sender_row_of)

    def check_parity(self, layers=None, rows=None, rel_tol=REL_FRO_TOL, abs_tol=MAX_ABS_TOL):
        """Every (layer, role) of `layers` on `rows` against the oracle; the
        per-(layer, role) errors are kept in self.errors (largest max-abs
        first in report())."""
        layers = list(range(self.w.L_r)) if layers is None else list(layers)
        rows = np.arange(self.tok.T_r) if rows is None else np.asarray(rows, dtype=np.int64)
        worst = {"rel_fro": 0.0, "max_abs": 0.0}
        if not hasattr(self, "errors"):
            self.errors = {}
        assert self.job.device_status() == 0
        for l in layers:
            ref = self.oracle([l], rows)
            for (ll, c), y in ref.items():
                g = self.gpu_rows(ll, c, rows)
                diff = g - y
                rel = float(np.linalg.norm(diff) / max(np.linalg.norm(y), 1e-30))
                mx = float(np.abs(diff).max()) if diff.size else 0.0
                worst["rel_fro"] = max(worst["rel_fro"], rel)
                worst["max_abs"] = max(worst["max_abs"], mx)
                old = self.errors.get((ll, c), (0.0, 0.0, 0))
                self.errors[(ll, c)] = (max(old[0], rel), max(old[1], mx), old[2] + diff.size)
                assert rel <= rel_tol, (ll, c, rel)
                assert mx <= abs_tol, (ll, c, mx)
        return worst

    def report(self, top=4):
        """One line: the workload, outputs compared, and the (layer, role)
        pairs with the largest max-abs error."""
        items = sorted(self.errors.items(), key=lambda kv: -kv[1][1])
        n = sum(v[2] for v in self.errors.values())
        worst = ", ".join(f"l{l}{'KV'[c]} max_abs={v[1]:.4g} rel_fro={v[0]:.3g}"
                          for (l, c), v in items[:top])
        return f"{self.w.name} {self.w.align_mode}+{self.w.layer_mode}: {n} outputs; {worst}"


def sampled_rows(tok, n, seed=0):
    """Seeded rows plus the edges: each request's first and last rows."""
    rng = np.random.default_rng(seed)
    T = tok.T_r
    rows = set(rng.choice(T, size=min(n, T), replace=False).tolist())
    for q in range(len(tok.r_tok_ptr) - 1):
        a, b = int(tok.r_tok_ptr[q]), int(tok.r_tok_ptr[q + 1])
        if b > a:
            rows.update({a, b - 1, min(a + 1, b - 1)})
    return np.array(sorted(rows), dtype=np.int64)


def run_boundary_rows(csr, r_tok_ptr, max_runs=None, seed=0):
    """First and last receiver row of every run of identical alignment rows
    (the rows where the kernel's epilogue starts or ends a distinct row's
    expansion), plus each request's first and last rows; with max_runs, of
    that many seeded runs only."""
    rp = np.asarray(csr.row_ptr, np.int64)
    col = np.asarray(csr.col, np.int64)
    w = np.asarray(csr.w, np.float64)
    T = len(rp) - 1
    starts = np.zeros(T, bool)
    for q in range(len(r_tok_ptr) - 1):
        a = int(r_tok_ptr[q])
        if a < int(r_tok_ptr[q + 1]):
            starts[a] = True
    one = np.all(rp[1:] - rp[:-1] == 1)
    if one:  # one entry per row: a run starts where the column or weight changes
        first = col[rp[:-1]]
        wt = w[rp[:-1]]
        starts[1:] |= (first[1:] != first[:-1]) | (wt[1:] != wt[:-1])
    else:
        for j in range(1, T):
            a0, a1, b0, b1 = rp[j - 1], rp[j], rp[j], rp[j + 1]
            if (a1 - a0 != b1 - b0 or not np.array_equal(col[a0:a1], col[b0:b1])
                    or not np.array_equal(w[a0:a1], w[b0:b1])):
                starts[j] = True
    first_rows = np.nonzero(starts)[0]
    last_rows = np.concatenate([first_rows[1:] - 1, [T - 1]]) if T else first_rows
    if max_runs is not None and len(first_rows) > max_runs:
        pick = np.random.default_rng(seed).choice(len(first_rows), max_runs, replace=False)
        first_rows, last_rows = first_rows[pick], last_rows[pick]
    return np.unique(np.concatenate([first_rows, last_rows]))


def section8c_rows(tok, csr, n_random=4096, seed=0, max_runs=4096):
    """The sampled rows of a long transfer: the first and last rows of the
    runs of identical alignment rows (of max_runs seeded runs when there are
    more), each request's first and last rows (the rows before the first
    shared boundary open the first run), and n_random seeded rows."""
    rows = set(run_boundary_rows(csr, tok.r_tok_ptr, max_runs, seed).tolist())
    rows.update(sampled_rows(tok, n_random, seed).tolist())
    return np.array(sorted(rows), dtype=np.int64)


def whole_layers(L_r):
    """First, last and two middle receiver layers."""
    return sorted({0, L_r // 3, (2 * L_r) // 3, L_r - 1})