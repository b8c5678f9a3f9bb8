"""Pins for the oracle's commit gather (committed tokens and target hidden rows
feed the drafter's next round: Sections 1, 3.1 and 6) and for the seeded
workloads the parity tests draw from."""
import numpy as np
import torch

import oracle
import workloads
from conftest import bits16


def test_commit_equals_library_gather():
    rng = np.random.default_rng(1)
    B, K, H = 7, 5, 24
    depth = rng.integers(0, K + 1, B).astype(np.int32)
    off = np.concatenate([[0], np.cumsum(depth + 1)]).astype(np.int32)
    R = int(off[-1])
    accepted = np.array([rng.integers(0, d + 1) for d in depth], np.int32)
    tokens = np.full((B, K + 1), -1, np.int32)
    for i in range(B):
        tokens[i, :accepted[i] + 1] = rng.integers(0, 1000, accepted[i] + 1)
    hidden = torch.randn(R, H).to(torch.bfloat16)
    res = oracle.commit(accepted, tokens, off, bits16(hidden))
    idx = torch.cat([torch.arange(off[i], off[i] + accepted[i] + 1) for i in range(B)])
    want_hidden = bits16(hidden.index_select(0, idx))
    want_tokens = torch.cat([torch.as_tensor(tokens[i, :accepted[i] + 1]) for i in range(B)])
    assert res["total"] == int((accepted + 1).sum())
    assert np.array_equal(res["hidden"], want_hidden)
    assert res["packed_tokens"][:res["total"]].tolist() == want_tokens.tolist()
    assert res["commit_offsets"].tolist() == [0] + np.cumsum(accepted + 1).tolist()


def test_workloads_are_seeded_and_shaped():
    a = workloads.make("sampled", V=512, B=4)
    b = workloads.make("sampled", V=512, B=4)
    assert torch.equal(a.logits.view(torch.int16), b.logits.view(torch.int16))
    assert torch.equal(a.drafts, b.drafts) and torch.equal(a.q.view(torch.int16), b.q.view(torch.int16))
    assert a.logits.shape == (4 * 9, 512) and a.q.shape == (4, 8, 512) and a.logits.dtype == torch.bfloat16
    c = workloads.make("sampled", V=512, B=4, seed=99)
    assert not torch.equal(a.logits.view(torch.int16), c.logits.view(torch.int16))


def test_planted_peak_gives_geometric_acceptance_at_t0():
    """At temperature 0 with per-position match probability p, P(a >= k) = p^k,
    so E[a] = sum_{k=1}^{K} p^k (3.887 for p = 0.8, K = 16)."""
    wl = workloads.make("greedy", V=512, B=3000, with_hidden=False)
    res = oracle.verify_batch(bits16(wl.logits), wl.drafts.numpy(), None, 0.0,
                              wl.seeds.numpy().view(np.uint64), wl.request_ids.numpy().view(np.uint64),
                              wl.pos_base.numpy())
    a = res["accepted"].astype(np.float64)
    p, K = 0.8, wl.K
    expect = sum(p**k for k in range(1, K + 1))
    assert abs(a.mean() - expect) < 5 * a.std() / np.sqrt(len(a))
    for k in (1, 2, 4):
        frac = (a >= k).mean()
        assert abs(frac - p**k) < 5 * np.sqrt(p**k * (1 - p**k) / len(a))
