"""The transfer kernel's bounded waits: a launch whose first map atom never
arrives ends with HF_CHECK_TIMEOUT in the plan's status instead of hanging,
and the CUDA context stays usable (a fresh plan then transfers correctly)."""

import time

import pytest
import torch

from gpu_harness import Case
from paper_2609_32259_gb300 import binding as B
from paper_2609_32259_gb300 import workloads as W

pytestmark = pytest.mark.gpu

HF_CHECK_TIMEOUT = 0x20


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


def test_stalled_transfer_times_out_and_context_recovers():
    c = Case(W.llama_to_ministral(700).with_(L_s=4, L_r=3))
    job = c.job
    job.align()
    job.make_plan()
    torch.cuda.synchronize()
    assert job.device_status() == 0
    t0 = time.perf_counter()
    B.debug_transfer_stalled(job.plan, job.sender, job.receiver)
    torch.cuda.synchronize()            # returns: no wait in the kernel is unbounded
    elapsed = time.perf_counter() - t0
    status = job.device_status()
    assert status & HF_CHECK_TIMEOUT, hex(status)
    assert elapsed < 60.0, elapsed     # each wait gives up after 2 s
    # the context is usable: a new plan (clear status) transfers correctly
    c.run()
    assert job.device_status() == 0
    c.check_csr()
    c.check_parity()

