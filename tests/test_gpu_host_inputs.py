"""The large inputs read in place from pinned host memory: spec_verify's
logits and q and spec_commit's hidden rows may live in host memory that the
device reaches at the same address (read over the CPU-GPU link, no staging
copy).  The results must be bit-identical to those from device copies."""
import pytest
import torch

import workloads
import paper_2607_25852_gb300 as spec

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


def _pinned(t):
    h = t.cpu().pin_memory()
    if not spec.spec_pointer_device_readable(h):
        pytest.skip("pinned host memory is not mapped at the same address on this system")
    return h


def test_readability_of_device_pinned_and_pageable_memory():
    assert spec.spec_pointer_device_readable(torch.zeros(16, device=DEV))
    assert spec.spec_pointer_device_readable(torch.zeros(16).pin_memory())
    assert not spec.spec_pointer_device_readable(torch.zeros(16))      # pageable: not promised


def _round(wl, logits, q, hidden):
    B, K, V = wl.B, wl.K, wl.V
    z = lambda *s: torch.zeros(s, dtype=torch.int32, device=DEV)
    acc, tok, ctok, coff = z(B), z(B, K + 1), z(B * (K + 1)), z(B + 1)
    pd = torch.zeros((B, K), device=DEV)
    rs = torch.zeros((B * (K + 1), 2), device=DEV)
    hout = torch.zeros((B * (K + 1), wl.H), dtype=wl.hidden.dtype, device=DEV)
    status = z(1)
    ws = spec.verify_workspace(B, K, V, DEV)
    spec.spec_verify(logits, wl.drafts, q, B, K, V, wl.temperature, wl.seeds, wl.request_ids, wl.pos_base,
                     acc, tok, ws, p_draft_out=pd, row_stats_out=rs, status=status)
    spec.spec_commit(acc, tok, hidden, B, K, ctok, coff, hout, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return [t.cpu() for t in (acc, tok, pd, rs, ctok, coff, hout)]


@pytest.mark.parametrize("name,t", [("sampled", None), ("greedy", None), ("sampled", 1.3)])
def test_host_inputs_match_device_inputs(name, t):
    wl = workloads.make(name, V=20000, H=256, temperature=t, device=DEV)
    want = _round(wl, wl.logits, wl.q, wl.hidden)
    got = _round(wl, _pinned(wl.logits), None if wl.q is None else _pinned(wl.q), _pinned(wl.hidden))
    for a, b in zip(want, got):
        assert torch.equal(a, b)
