"""Failure detection on the GPU without a fault: a bounded device wait that
nothing completes (an mbarrier no one arrives at) gives up after about a
second, reports SPEC_ERR_TIMEOUT through the caller's status word, and the
context stays usable for the next calls."""
import time

import pytest
import torch

from parity import compare, run_oracle, run_verify
from test_gpu_verify import _random_case

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_the_context_stays_usable():
    import paper_2607_25852_gb300 as spec
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    spec.spec_check_bounded_wait(status)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert int(status.item()) == spec.ERR_TIMEOUT
    assert 0.5 < waited < 30.0, waited
    # the same context still verifies correctly
    wl = _random_case(4097, "bf16", 0.7, "dense", B=4, K=3, seed=31)
    gpu = run_verify(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.7, wl.seeds, wl.request_ids, wl.pos_base)
    ref = run_oracle(wl.logits, wl.drafts, wl.q, 0.7, wl.seeds, wl.request_ids, wl.pos_base)
    assert gpu["status"] == 0 and (ref["status"] == 0).all()
    compare(gpu, ref, wl.K, 0.7)
