"""Pins for the oracle's Markov-head sequential draw (Section 3.2,
Eq. dspark-markov: b = W1[x_prev] W2, q = softmax(U + b); the block
distribution factorises over positions, Eq. ar-factorization).

Each test checks the oracle against something other than itself: the
already-pinned draft step (the bias vanishes with W1 = 0), library matmul /
logsumexp / softmax along the oracle's own draft chain, and the joint
distribution of two consecutive drafts.
"""
import numpy as np
import pytest
import torch
from scipy import stats

import oracle
from conftest import bf16_bits_from_float


def _bf16(x):
    return torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16).float().numpy().astype(np.float64)


def _case(B, K, V, r, seed, std=2.0, wstd=0.3):
    rng = np.random.default_rng(seed)
    U = rng.normal(0, std, (B, K, V)).astype(np.float32)
    W1 = rng.normal(0, wstd, (V, r)).astype(np.float32)
    W2 = rng.normal(0, wstd, (r, V)).astype(np.float32)
    x0 = rng.integers(0, V, B).astype(np.int32)
    seeds = rng.integers(0, 2**63, B, dtype=np.uint64)
    rids = rng.integers(0, 2**63, B, dtype=np.uint64)
    pos = rng.integers(0, 2**31, B).astype(np.int64)
    return U, bf16_bits_from_float(W1), bf16_bits_from_float(W2), _bf16(W1), _bf16(W2), x0, seeds, rids, pos


@pytest.mark.parametrize("tau", [0.0, 0.8, 1.0])
def test_zero_transition_is_the_draft_step(tau):
    """W1 = 0: every bias vanishes, so each position's q is the draft step's,
    and both draws race the same 256-entry blocks with the same variates
    (purposes DRAFT and DRAFT_IN_BLOCK at the drafted position): drafts,
    confidences, scores and row statistics all agree exactly, at tau = 0 and
    tau > 0.  V = 1100 puts the winner in any of five blocks, the last one
    partial."""
    U, _, _, _, _, x0, seeds, rids, pos = _case(16, 5, 1100, 8, 1)
    zero1 = np.zeros((1100, 8), np.uint16)
    zero2 = np.zeros((8, 1100), np.uint16)
    mk = oracle.markov_batch(U, zero1, zero2, x0, tau, seeds, rids, pos)
    dr = oracle.draft_batch(U, tau, seeds, rids, pos)
    for k in ("z", "c", "s", "m", "logS", "status"):
        assert np.array_equal(mk[k], dr[k]), k
    if tau > 0:
        assert len(set((mk["z"] // 256).ravel().tolist())) >= 3    # the draws span several blocks


def test_race_blocks_follow_q():
    """The Markov draw's level-1 blocks hold 256 entries: V = 1100 (five
    blocks, the last partial), 20000 requests with zero bias, the draft's
    histogram over the blocks against q's block masses (chi-square, 4 dof)."""
    V, N = 1100, 20000
    rng = np.random.default_rng(11)
    row = rng.normal(0, 1.0, V).astype(np.float32)
    U = np.broadcast_to(row, (N, 1, V)).copy()
    res = oracle.markov_batch(U, np.zeros((V, 2), np.uint16), np.zeros((2, V), np.uint16), np.zeros(N, np.int32),
                              1.0, np.full(N, 3, np.uint64), np.arange(N, dtype=np.uint64), np.full(N, 9, np.int64))
    q = np.exp(row.astype(np.float64) - row.max())
    q /= q.sum()
    mass = np.array([q[b * 256:(b + 1) * 256].sum() for b in range(5)])
    counts = np.bincount(res["z"][:, 0] // 256, minlength=5)
    chi2 = ((counts - N * mass) ** 2 / (N * mass)).sum()
    assert stats.chi2.sf(chi2, 4) > 1e-3


@pytest.mark.parametrize("tau", [0.0, 0.7, 1.3])
def test_biased_rows_match_library_matmul_and_softmax(tau):
    U, W1b, W2b, W1, W2, x0, seeds, rids, pos = _case(3, 4, 500, 16, 2)
    res = oracle.markov_batch(U, W1b, W2b, x0, tau, seeds, rids, pos)
    assert (res["status"] == 0).all()
    tc = tau if tau > 0 else 1.0
    for i in range(3):
        prev = int(x0[i])
        for k in range(4):
            l = torch.as_tensor(U[i, k].astype(np.float64) + W1[prev] @ W2) / tc
            z = int(res["z"][i, k])
            assert res["m"][i, k] == pytest.approx(float(l.max()), rel=1e-12, abs=1e-12)
            assert res["logS"][i, k] == pytest.approx(float(torch.logsumexp(l, 0) - l.max()), abs=1e-10)
            assert res["c"][i, k] == pytest.approx(float(torch.softmax(l, 0)[z]), rel=1e-10)
            if tau == 0:
                assert z == int(torch.argmax(l))
            prev = z


def test_scores_are_float32_prefix_products():
    U, W1b, W2b, _, _, x0, seeds, rids, pos = _case(4, 6, 300, 8, 3)
    res = oracle.markov_batch(U, W1b, W2b, x0, 1.0, seeds, rids, pos)
    c32 = res["c"].astype(np.float32)
    expect = np.concatenate([np.ones((4, 1), np.float32),
                             np.multiply.accumulate(c32, axis=1, dtype=np.float32)], axis=1)
    assert np.array_equal(res["s"], expect)


def test_two_drafts_follow_the_factorised_block_distribution():
    """V = 6, r = 2, 30000 requests with the same inputs: the histogram of
    (x_1, x_2) against q_1(x_1) q_2(x_2 | x_1) (chi-square, 35 dof)."""
    V, r, N, tau = 6, 2, 30000, 1.0
    rng = np.random.default_rng(4)
    U = rng.normal(0, 1.0, (1, 2, V)).astype(np.float32)
    W1 = rng.normal(0, 1.0, (V, r)).astype(np.float32)
    W2 = rng.normal(0, 1.0, (r, V)).astype(np.float32)
    W1v, W2v = _bf16(W1), _bf16(W2)
    x0 = 3
    res = oracle.markov_batch(np.broadcast_to(U, (N, 2, V)).copy(), bf16_bits_from_float(W1),
                              bf16_bits_from_float(W2), np.full(N, x0, np.int32), tau,
                              np.full(N, 17, np.uint64), np.arange(N, dtype=np.uint64), np.full(N, 5, np.int64))
    assert (res["status"] == 0).all()
    sm = lambda l: np.exp(l / tau - (l / tau).max()) / np.exp(l / tau - (l / tau).max()).sum()
    q1 = sm(U[0, 0].astype(np.float64) + W1v[x0] @ W2v)
    joint = np.array([[q1[a] * sm(U[0, 1].astype(np.float64) + W1v[a] @ W2v)[b] for b in range(V)]
                      for a in range(V)])
    counts = np.zeros((V, V))
    np.add.at(counts, (res["z"][:, 0], res["z"][:, 1]), 1)
    exp_ = N * joint
    chi2 = ((counts - exp_) ** 2 / exp_).sum()
    assert stats.chi2.sf(chi2, V * V - 1) > 1e-3
    # the bias matters: the second draft's distribution depends on the first
    assert not np.allclose(joint / joint.sum(1, keepdims=True), joint.sum(0), atol=1e-3)


def test_bad_inputs_flag_the_request():
    U, W1b, W2b, _, _, x0, seeds, rids, pos = _case(3, 3, 200, 4, 5)
    U[0, 1, 9] = np.nan
    x0 = x0.copy()
    x0[1] = 200                                   # last committed token out of range
    res = oracle.markov_batch(U, W1b, W2b, x0, 1.0, seeds, rids, pos)
    assert res["status"].tolist() == [oracle.ERR_BAD_INPUT, oracle.ERR_BAD_INPUT, 0]
    assert (res["z"][:2] == -1).all() and (res["s"][:2, 1:] == 0).all()
