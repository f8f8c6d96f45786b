"""Host logic around the transfer, on the CPU: bench workload names and
operand-path labels, the KV Ridge layer-selection stand-in, the sampled-row
helper of the GPU parity tests, and the bench's algorithmic-work counts."""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import bench  # noqa: E402
from gpu_harness import run_boundary_rows, section8c_rows, whole_layers  # noqa: E402
from oracle import heterofold_oracle as O  # noqa: E402
from paper_2609_32259_gb300 import workloads as W  # noqa: E402


@pytest.mark.parametrize("name,align,layer,T", [
    ("llama_to_ministral_32k", "ta", "paper3", 32768),
    ("llama_to_ministral_32k_overlap", "overlap_mean", "paper3", 32768),
    ("llama_to_ministral_32k_interp", "ta", "interp", 32768),
    ("llama_to_ministral_32k_overlap_interp", "overlap_mean", "interp", 32768),
    ("llama_to_ministral_32k_interp_overlap", "overlap_mean", "interp", 32768),
    ("llama_to_qwen25_4k_overlap", "overlap_mean", "paper3", 4096),
    ("ministral_to_llama_256", "ta", "paper3", 256),
    ("qwen25_to_llama_kv_ridge_4k", "ta", "explicit", 4096),
    ("qwen25_to_llama_kv_ridge_1024", "ta", "explicit", 1024),
])
def test_bench_workload_names(name, align, layer, T):
    w = bench.workload(name)
    assert (w.align_mode, w.layer_mode, sum(w.r_tokens)) == (align, layer, T)
    if align == "overlap_mean":
        assert "overlap_mean" in w.name
    if layer == "interp":
        assert w.name.endswith("interp")


def test_bench_unknown_workload_is_an_error():
    with pytest.raises(KeyError):
        bench.workload("llama_to_nowhere")


def test_copied_operand_label():
    assert bench._copied_operands(bench.workload("llama_to_ministral_32k"))
    assert bench._copied_operands(bench.workload("qwen25_to_llama_kv_ridge_4k"))
    assert not bench._copied_operands(bench.workload("llama_to_ministral_32k_interp"))
    # overlap pooling after the map copies sender rows; before it, pooled rows are computed
    assert bench._copied_operands(bench.workload("llama_to_qwen25_4k_overlap"))
    assert not bench._copied_operands(bench.workload("llama_to_qwen25_4k_overlap"),
                                      pool_before_map=True)
    assert not bench._copied_operands(bench.workload("llama_to_qwen25_4k_overlap_interp"))
    w = W.llama_to_ministral(64).with_(sender_k_rotated=True)
    assert not bench._copied_operands(w)
    assert not bench._copied_operands(w.with_(align_mode="overlap_mean"))


def test_launches_per_step():
    """Align + plan + transfer kernels, by mode (the bench's gpu_launches)."""
    assert bench.launches_per_step(bench.workload("llama_to_ministral_32k")) == 3 + 5 + 1
    ov = bench.workload("llama_to_qwen25_4k_overlap")
    assert bench.launches_per_step(ov) == 4 + 7 + 1
    assert bench.launches_per_step(ov, pool_before_map=True) == 4 + 5 + 1
    assert bench.launches_per_step(ov.with_(knorm=True)) == 4 + 5 + 1
    assert bench.launches_per_step(W.llama_to_ministral(64).with_(
        align_mode="same_index", span_gap=10)) == 1 + 6 + 1


def test_kv_ridge_selection_stand_in():
    sel = W.kv_ridge_selection(28, 32, 8, seed=13)
    assert len(sel) == 32
    for l, s in enumerate(sel):
        assert len(s) == 8 and len(set(s)) == 8
        assert list(s) == sorted(s) and 0 <= s[0] and s[-1] < 28
        # the stand-in ranks by distance to the proportional depth (+ U(0, 3)):
        # every selected layer is within 3 + 8 of it
        p = l * 27 / 31
        assert all(abs(t - p) <= 11 for t in s)
    assert W.kv_ridge_selection(28, 32, 8, seed=13) == sel
    w = W.qwen25_to_llama_kv_ridge(512)
    assert w.K == 8 * w.d_s and w.kv_ridge and w.n_seg == 8
    _, _, r = W.maps(w.with_(L_r=2, seg_layer=w.seg_layer[:2], seg_w=w.seg_w[:2]))
    assert np.all(r == 1.0)


def _runs_brute(csr):
    rows = []
    for j in range(csr.n_rows):
        a = (tuple(csr.col[csr.row_ptr[j]:csr.row_ptr[j + 1]]),
             tuple(csr.w[csr.row_ptr[j]:csr.row_ptr[j + 1]]))
        rows.append(a)
    starts = [j for j in range(len(rows)) if j == 0 or rows[j] != rows[j - 1]]
    ends = [s - 1 for s in starts[1:]] + [len(rows) - 1]
    return sorted(set(starts) | set(ends))


@pytest.mark.parametrize("mode", ["ta", "overlap_mean"])
def test_run_boundary_rows_against_brute_force(mode):
    w = W.llama_to_ministral(700).with_(align_mode=mode)
    tok = W.tokens(w)
    csr = O.alignment_csr(mode, tok.s_tok_ptr, tok.r_tok_ptr, tok.s_end, tok.r_end)
    got = run_boundary_rows(csr, tok.r_tok_ptr)
    assert got.tolist() == _runs_brute(csr)
    capped = run_boundary_rows(csr, tok.r_tok_ptr, max_runs=10, seed=1)
    assert set(capped.tolist()) <= set(got.tolist()) and len(capped) <= 20
    rows = section8c_rows(tok, csr, 100, seed=3, max_runs=50)
    assert rows[0] == 0 and rows[-1] == tok.T_r - 1 and len(set(rows)) == len(rows)


def test_whole_layers():
    assert whole_layers(40) == [0, 13, 26, 39]
    assert whole_layers(2) == [0, 1]


def test_algorithmic_work_counts():
    """FLOP = 2 * 2 L_r U K d_r; bytes add the receiver cache, the referenced
    sender rows of every sender layer the table reads, maps, biases, CSR."""
    w = W.llama_to_ministral(1000)
    tok = W.tokens(w)
    flops, by = bench.algorithmic_work(w, tok, 250, 300)
    assert flops == 2.0 * 2 * 40 * 250 * 3072 * 1024
    rec = 2 * 40 * tok.T_r * 1024 * 2
    snd = 32 * 2 * 300 * 1024 * 2
    maps = 2 * 40 * 3072 * 1024 * 2
    assert by == rec + snd + maps + 2 * 40 * 1024 * 4 + tok.T_r * 24
    kv = W.qwen25_to_llama_kv_ridge(1000)
    n_layers = len({t for l in kv.seg_layer for seg in l for t in seg})
    _, by2 = bench.algorithmic_work(kv, W.tokens(kv), 250, 300)
    assert 8 <= n_layers <= kv.L_s
    assert by2 == (2 * 32 * W.tokens(kv).T_r * 1024 * 2 + n_layers * 2 * 300 * 512 * 2
                   + 2 * 32 * 4096 * 1024 * 2 + 2 * 32 * 1024 * 4 + W.tokens(kv).T_r * 24)
