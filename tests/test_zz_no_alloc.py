"""spec_verify_static: verification for callers that cannot allocate device
memory.

Some users of this library run inside an inference engine that owns every
byte of GPU memory through its own pool, or on a latency-critical path where
cudaMalloc (which can synchronise the device) is not allowed.  They cannot
hand spec_verify a workspace, so spec_verify_static uses a fixed scratch
array that belongs to the library.  These tests call it through the C ABI and
check that, on two calls in a row, it gives the same results as spec_verify
with a caller-provided workspace (within the tolerances the other parity tests
use).  The file sorts last so that a run stopping at its first failure has
already run every other test.
"""
import numpy as np
import pytest
import torch

import paper_2607_25852_gb300 as spec
from parity import P_RTOL

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


def _inputs(V, B, K, t, dense_q, seed):
    g = torch.Generator().manual_seed(seed)
    base = torch.randn((B * (K + 1), V), generator=g) * 2.5
    logits = base.to(torch.bfloat16)
    q = None
    if dense_q:
        noisy = base.view(B, K + 1, V)[:, :K] + torch.randn((B, K, V), generator=g) * 0.7
        q = torch.softmax(noisy / 0.8, -1).to(torch.bfloat16)
        drafts = torch.multinomial(q.float().view(B * K, V), 1, generator=g).view(B, K)
    else:
        drafts = logits.float().view(B, K + 1, V)[:, :K].argmax(-1)
        drafts[:, K // 2:] = torch.randint(0, V, (B, K - K // 2), generator=g)
    return dict(logits=logits.to(DEV), q=None if q is None else q.to(DEV),
                drafts=drafts.to(torch.int32).to(DEV),
                seeds=torch.arange(B, dtype=torch.int64, device=DEV) * 7 + 1,
                request_ids=torch.arange(B, dtype=torch.int64, device=DEV) + 100,
                pos_base=torch.randint(0, 10**6, (B,), generator=g).to(DEV), B=B, K=K, V=V, t=t)


def _outputs(B, K):
    return dict(acc=torch.full((B,), -9, dtype=torch.int32, device=DEV),
                tok=torch.full((B, K + 1), -9, dtype=torch.int32, device=DEV),
                pdr=torch.zeros((B, K), dtype=torch.float32, device=DEV),
                rst=torch.zeros((B * (K + 1), 2), dtype=torch.float32, device=DEV),
                status=torch.zeros(1, dtype=torch.int32, device=DEV))


def _run(x, static):
    o = _outputs(x["B"], x["K"])
    args = (x["logits"], x["drafts"], x["q"], x["B"], x["K"], x["V"], x["t"], x["seeds"],
            x["request_ids"], x["pos_base"], o["acc"], o["tok"])
    kw = dict(p_draft_out=o["pdr"], row_stats_out=o["rst"], status=o["status"])
    if static:
        spec.spec_verify_static(*args, **kw)
    else:
        ws = spec.verify_workspace(x["B"], x["K"], x["V"], DEV)
        spec.spec_verify(*args, ws, **kw)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in o.items()}


@pytest.mark.parametrize("V,B,K,t,dense_q", [(20000, 8, 5, 0.8, True), (4097, 5, 3, 0.0, False),
                                            (65536, 64, 16, 1.0, True), (333, 3, 0, 1.3, False)])
def test_static_scratch_matches_caller_workspace_twice(V, B, K, t, dense_q):
    x = _inputs(V, B, K, t, dense_q, seed=V + B)
    want = _run(x, static=False)
    for _ in range(2):                                   # two calls in a row share the scratch
        got = _run(x, static=True)
        assert int(got["status"][0]) == 0 and int(want["status"][0]) == 0
        assert np.array_equal(got["acc"], want["acc"])
        assert np.array_equal(got["tok"], want["tok"])
        np.testing.assert_allclose(got["pdr"], want["pdr"], rtol=P_RTOL, atol=1e-30)
        np.testing.assert_allclose(got["rst"], want["rst"], rtol=P_RTOL, atol=P_RTOL)


def test_static_scratch_rejects_shapes_beyond_its_size():
    limit = 4 << 20
    B, K, V = 65536, 16, 201088                         # needs about 18 MB of partials
    assert spec.spec_verify_workspace(B, K, V) > limit
    o = _outputs(1, 1)
    dummy = torch.zeros(1, dtype=torch.int64, device=DEV)
    logits = torch.zeros(1, dtype=torch.bfloat16, device=DEV)   # never read: nothing launches
    with pytest.raises(spec.SpecError) as e:
        spec.spec_verify_static(logits, o["tok"], None, B, K, V, 1.0, dummy, dummy, dummy,
                                o["acc"], o["tok"])
    assert e.value.code == spec.ERR_TOO_LARGE


def test_static_scratch_over_a_sequence_of_shapes():
    """Shapes that change from call to call: the counters and records move
    inside the shared array, and a smaller call's counters start where a
    larger call left its partials.  Every call must still match spec_verify
    with a fresh caller workspace."""
    seq = [(65536, 64, 16, 1.0, True), (4097, 5, 3, 0.8, False), (65536, 64, 16, 1.0, True),
           (20000, 8, 5, 0.0, False), (4097, 5, 3, 0.8, False), (333, 3, 0, 1.3, False)]
    for n, (V, B, K, t, dense_q) in enumerate(seq):
        x = _inputs(V, B, K, t, dense_q, seed=V + B + n)
        want = _run(x, static=False)
        got = _run(x, static=True)
        assert int(got["status"][0]) == 0 and int(want["status"][0]) == 0, (V, B, K)
        assert np.array_equal(got["acc"], want["acc"]), (V, B, K)
        assert np.array_equal(got["tok"], want["tok"]), (V, B, K)
        np.testing.assert_allclose(got["pdr"], want["pdr"], rtol=P_RTOL, atol=1e-30)
        np.testing.assert_allclose(got["rst"], want["rst"], rtol=P_RTOL, atol=P_RTOL)


def test_static_scratch_argument_error_leaves_the_next_call_intact():
    """A call rejected on the host (negative temperature) queues nothing; the
    call after it is still correct."""
    x = _inputs(4097, 5, 3, 0.8, False, seed=77)
    o = _outputs(5, 3)
    with pytest.raises(spec.SpecError) as e:
        spec.spec_verify_static(x["logits"], x["drafts"], None, 5, 3, 4097, -1.0, x["seeds"], x["request_ids"],
                                x["pos_base"], o["acc"], o["tok"])
    assert e.value.code == spec.ERR_INVALID_ARG
    want = _run(x, static=False)
    got = _run(x, static=True)
    assert np.array_equal(got["acc"], want["acc"]) and np.array_equal(got["tok"], want["tok"])
