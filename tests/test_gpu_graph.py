"""One transfer step recorded as CUDA graphs (alignment + plan, transfer)
and replayed: every replay must equal, bit for bit, an eager step on the
same buffer contents (the same kernels with the same parameters), also
after the sender cache changes between replays."""

import pytest
import torch

from gpu_harness import Case
from paper_2609_32259_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SENTINEL = 77.0


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


CASES = {
    "tiny_f32_overlap_interp": W.tiny,
    "ta_paper3": lambda: W.llama_to_ministral(600).with_(L_s=4, L_r=5),
    "overlap_after_map_paged": lambda: W.qwen25_to_llama_batched(
        n_req=3, lo=40, hi=300, seed=71).with_(L_s=4, L_r=3, align_mode="overlap_mean"),
    "interp_wide": lambda: W.llama_to_ministral(500).with_(L_s=5, L_r=3, layer_mode="interp"),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_graph_replay_equals_eager_step(name):
    c = Case(CASES[name](), sentinel=SENTINEL).run()
    c.job.capture()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    for trial in range(3):
        if trial:
            c.sender.copy_(torch.randn(c.sender.shape, generator=gen, device="cuda")
                           .to(c.sender.dtype))
        c.job.step()
        torch.cuda.synchronize()
        ref = c.job.receiver.clone()
        c.job.receiver.fill_(SENTINEL)
        c.job.replay()
        torch.cuda.synchronize()
        assert c.job.device_status() == 0
        assert torch.equal(c.job.receiver, ref), (name, trial)
    # the replayed step also matches the oracle on the last sender contents
    c.check_parity()
