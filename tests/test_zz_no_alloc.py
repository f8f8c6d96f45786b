"""hf_transfer_noalloc against the workspace entry points.

Some callers cannot allocate device memory per call: a host framework or
plugin that owns every device allocation and hands in only the caches, or a
service held to a fixed memory budget.  hf_transfer_noalloc keeps the
per-transfer metadata in a device array built into the library instead of a
caller workspace.  These tests call it through the C ABI several times in a
row, on transfers of different sizes (stale contents of the shared array
would show), and compare each result with hf_plan_create + hf_transfer on
the same inputs: both run the same kernels, so the results must agree bit
for bit.

This file is collected last so that a run stopping at the first failure
has already run every other test."""

import ctypes

import numpy as np
import pytest
import torch

from gpu_harness import MAX_ABS_TOL, REL_FRO_TOL
from paper_2609_32259_gb300 import binding as B
from paper_2609_32259_gb300 import pipeline
from paper_2609_32259_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SENTINEL = 777.0


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


def _job(w):
    dev = torch.device("cuda")
    tok = W.tokens(w)
    sender = W.sender_kv(w, tok.T_s, dev)
    Wm, b, r = W.maps(w, dev)
    paged = W.paged_layout(w, tok) if w.paged else None
    job = pipeline.job_from_workload(w, tok, sender, Wm, b, r, paged=paged,
                                     knorm_w=W.knorm_weight(w), r_pos0=W.r_pos0(w), device=dev)
    job.receiver.fill_(SENTINEL)
    job.step()  # alignment CSR + the workspace plan + hf_transfer
    torch.cuda.synchronize()
    assert job.device_status() == 0
    return job


def _assert_close(ref, out):
    assert ref.shape == out.shape
    for l in range(ref.shape[0]):
        for c in range(2):
            a = ref[l, c].double()
            g = out[l, c].double()
            diff = g - a
            rel = float(diff.norm() / max(float(a.norm()), 1e-30))
            mx = float(diff.abs().max())
            assert rel <= REL_FRO_TOL and mx <= MAX_ABS_TOL, (l, c, rel, mx)


def _noalloc(job):
    out = torch.full_like(job.receiver, SENTINEL)
    B.transfer_noalloc(job.desc, job.sender, out)
    torch.cuda.synchronize()
    return out


def _assert_same(ref, out):
    # the two entry points run the same plan kernels and the same transfer
    # kernel, whose outputs involve no atomics: the results must agree bit for
    # bit (stale metadata, a shifted RoPE position for instance, would show
    # here even where it stays inside the oracle tolerance)
    if not torch.equal(ref, out):
        _assert_close(ref, out)  # a tolerance report says how far off it is
        raise AssertionError("hf_transfer_noalloc differs from hf_transfer")


def test_noalloc_matches_workspace_path_on_consecutive_calls():
    a = _job(W.llama_to_ministral(900).with_(L_s=4, L_r=5, r_pos0=(4000,)))
    b = _job(W.qwen25_to_llama_batched(n_req=3, lo=100, hi=700, seed=11).with_(L_s=4, L_r=3))
    _assert_same(a.receiver, _noalloc(a))   # first call
    _assert_same(b.receiver, _noalloc(b))   # second call, other sizes, paged
    _assert_same(a.receiver, _noalloc(a))   # and back
    a.close()
    b.close()


def test_noalloc_rejects_transfers_beyond_its_scratch():
    desc = B.Desc(L_s=4, H_s=8, D_s=128, L_r=4, H_r=8, D_r=128, dtype="bf16",
                  layer_mode="paper3", align_mode="ta", s_tok_ptr=[0, 10], r_tok_ptr=[0, 4_000_000],
                  d_row_ptr=256, d_col=512, d_w=768, d_W=1024, d_b=1280,
                  r=np.ones((4, 2)), theta_r=1e4)
    st = B.lib().hf_transfer_noalloc(ctypes.byref(desc.c), 4096, 8192, None)
    assert st == B.HF_ERR_UNSUPPORTED
    assert b"scratch" in B.lib().hf_last_error()
