"""hf_transfer_host: caches in page-locked host memory, copies overlapped
with the computation.  Its host result must equal, bit for bit, the device
result of hf_transfer on the same inputs (the same tiles run the same code;
only the launch split over receiver layers differs), for several group
counts, a paged pool included."""

import numpy as np
import pytest
import torch

from gpu_harness import Case
from paper_2609_32259_gb300 import binding as B
from paper_2609_32259_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SENTINEL = -321.0


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


CASES = {
    "contiguous": (lambda: W.llama_to_ministral(1000).with_(L_s=6, L_r=7), (0, 1, 3, 7)),
    "paged_batched": (lambda: W.qwen25_to_llama_batched(n_req=3, lo=60, hi=500, seed=8)
                      .with_(L_s=4, L_r=5), (2, 5)),
    "interp_f32": (W.tiny, (4,)),
    "kv_ridge_paged": (lambda: W.qwen25_to_llama_kv_ridge(1).with_(paged=True,
                                                                r_tokens=(300, 77)), (3, 32)),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_transfer_host_matches_device_path(name):
    make, groups = CASES[name]
    c = Case(make(), sentinel=SENTINEL).run()
    ref = c.job.receiver.cpu()
    h_sender = torch.empty(c.sender.shape, dtype=c.sender.dtype, pin_memory=True)
    h_sender.copy_(c.sender)
    h_recv = torch.empty(ref.shape, dtype=ref.dtype, pin_memory=True)
    for G in groups:
        c.sender.zero_()                  # the copy in must bring the sender back
        c.job.receiver.fill_(SENTINEL)
        h_recv.fill_(0.0)
        c.job.transfer_host(h_sender, h_recv, G)
        torch.cuda.synchronize()
        assert c.job.device_status() == 0
        assert torch.equal(h_recv, ref), (name, G)


def test_transfer_host_can_leave_the_receiver_on_the_device():
    c = Case(W.llama_to_ministral(800).with_(L_s=5, L_r=6), sentinel=SENTINEL).run()
    ref = c.job.receiver.clone()
    h_sender = torch.empty(c.sender.shape, dtype=c.sender.dtype, pin_memory=True)
    h_sender.copy_(c.sender)
    c.sender.zero_()
    c.job.receiver.fill_(SENTINEL)
    c.job.transfer_host(h_sender, None, 3)
    torch.cuda.synchronize()
    assert torch.equal(c.job.receiver, ref)


def test_transfer_host_rejects_pageable_memory_and_bad_groups():
    c = Case(W.llama_to_ministral(300).with_(L_s=3, L_r=2)).run()
    pageable = torch.empty(c.sender.shape, dtype=c.sender.dtype)
    h_recv = torch.empty(c.job.receiver.shape, dtype=c.job.receiver.dtype, pin_memory=True)
    with pytest.raises(B.HFError) as e:
        c.job.transfer_host(pageable, h_recv)
    assert e.value.status == B.HF_ERR_INVALID_ARGUMENT
    h_sender = torch.empty(c.sender.shape, dtype=c.sender.dtype, pin_memory=True)
    with pytest.raises(B.HFError) as e:
        c.job.transfer_host(h_sender, h_recv, n_groups=c.w.L_r + 1)
    assert e.value.status == B.HF_ERR_INVALID_ARGUMENT
