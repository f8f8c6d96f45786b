"""hf_transfer_batch: the six directions of a three-agent message round
(message spans after a context, every family pair) in one launch.  Each
direction must equal, bit for bit, its own hf_transfer (the same tiles, the
same code), and match the fp64 oracle within the parity tolerance."""

import numpy as np
import pytest
import torch

from gpu_harness import Case
from paper_2609_32259_gb300 import binding as B
from paper_2609_32259_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SENTINEL = 99.0


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


def test_message_round_batch_matches_single_transfers_and_oracle():
    cases = [Case(w, sentinel=SENTINEL).run() for w in W.message_round(msg_tokens=160)]
    single = [c.job.receiver.clone() for c in cases]
    for c in cases:
        c.job.receiver.fill_(SENTINEL)
    B.transfer_batch([c.job.plan for c in cases], [c.sender for c in cases],
                     [c.job.receiver for c in cases])
    torch.cuda.synchronize()
    for c, ref in zip(cases, single):
        assert torch.equal(c.job.receiver, ref), c.w.name
        c.check_parity()


def test_batch_mixing_operand_paths():
    """Plans that differ in dtype or operand path (copied rows vs built rows)
    go to separate launches; results equal their single transfers."""
    ws = [W.message_round(msg_tokens=60)[0], W.tiny(),
          W.llama_to_ministral(300).with_(L_s=3, L_r=3, align_mode="overlap_mean")]
    cases = [Case(w, sentinel=SENTINEL).run() for w in ws]
    single = [c.job.receiver.clone() for c in cases]
    for c in cases:
        c.job.receiver.fill_(SENTINEL)
    B.transfer_batch([c.job.plan for c in cases], [c.sender for c in cases],
                     [c.job.receiver for c in cases])
    torch.cuda.synchronize()
    for c, ref in zip(cases, single):
        assert torch.equal(c.job.receiver, ref), c.w.name


def test_batch_of_built_operand_rows():
    """Directions whose operand rows the loader warps build (layers blended
    per sender token, overlap pooling after the map; a Qwen2.5-shaped
    receiver is one 512-column wide tile) in one launch: each equals its
    single transfer and the oracle."""
    ws = [W.llama_to_ministral(700).with_(L_s=5, L_r=4, layer_mode="interp",
                                          align_mode="overlap_mean"),
          W.llama_to_qwen25(500).with_(L_s=6, L_r=3, layer_mode="interp",
                                       align_mode="overlap_mean"),
          W.qwen25_to_llama_batched(n_req=2, lo=80, hi=300, seed=61).with_(
              L_s=4, L_r=3, layer_mode="interp", align_mode="overlap_mean")]
    cases = [Case(w, sentinel=SENTINEL).run() for w in ws]
    single = [c.job.receiver.clone() for c in cases]
    for c in cases:
        c.job.receiver.fill_(SENTINEL)
    B.transfer_batch([c.job.plan for c in cases], [c.sender for c in cases],
                     [c.job.receiver for c in cases])
    torch.cuda.synchronize()
    for c, ref in zip(cases, single):
        assert torch.equal(c.job.receiver, ref), c.w.name
        c.check_parity()


def test_batch_mixing_layer_tables():
    """A KV Ridge direction (an explicit eight-segment table), a paper3
    direction and an interpolated one in one batch: each equals its single
    transfer and stays within the parity tolerance of the oracle."""
    ws = [W.qwen25_to_llama_kv_ridge(600),
          W.qwen25_to_llama_batched(n_req=2, lo=100, hi=400, seed=44).with_(L_s=28, L_r=32),
          W.llama_to_ministral(500).with_(L_s=5, L_r=6, layer_mode="interp")]
    cases = [Case(w, sentinel=SENTINEL).run() for w in ws]
    single = [c.job.receiver.clone() for c in cases]
    for c in cases:
        c.job.receiver.fill_(SENTINEL)
    B.transfer_batch([c.job.plan for c in cases], [c.sender for c in cases],
                     [c.job.receiver for c in cases])
    torch.cuda.synchronize()
    for c, ref in zip(cases, single):
        assert torch.equal(c.job.receiver, ref), c.w.name
    cases[0].check_parity(layers=[0, 13, 31])
    cases[2].check_parity()


def test_batch_of_one_and_empty_batch():
    c = Case(W.message_round(msg_tokens=40)[1], sentinel=SENTINEL).run()
    ref = c.job.receiver.clone()
    c.job.receiver.fill_(SENTINEL)
    B.transfer_batch([c.job.plan], [c.sender], [c.job.receiver])
    B.transfer_batch([], [], [])
    torch.cuda.synchronize()
    assert torch.equal(c.job.receiver, ref)


def test_batch_rejects_a_repeated_plan():
    c = Case(W.message_round(msg_tokens=40)[0]).run()
    with pytest.raises(B.HFError) as e:
        B.transfer_batch([c.job.plan, c.job.plan], [c.sender, c.sender],
                         [c.job.receiver, c.job.receiver])
    assert e.value.status == B.HF_ERR_INVALID_ARGUMENT
