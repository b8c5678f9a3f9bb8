"""Pins for the oracle's drafter producer step: the drafts and the token-level
confidences that D-cut reads (Section 4.2, Eq. dcut-score; the reading c =
q(z) is the design notes').

Each test checks the oracle against something other than itself: library
softmax / argmax / cumulative product, closed forms, and the distribution of
the drafts (they must follow q exactly).
"""
import numpy as np
import pytest
import torch
from scipy import stats

import oracle
from conftest import bf16_bits_from_float


def _softmax64(x, t):
    return torch.softmax(torch.as_tensor(np.asarray(x, np.float64)) / t, dim=-1).numpy()


def _case(B, K, V, seed, std=2.0, dtype="f32"):
    rng = np.random.default_rng(seed)
    x = rng.normal(0, std, (B, K, V)).astype(np.float32)
    logits = x if dtype == "f32" else bf16_bits_from_float(x)
    vals = x if dtype == "f32" else torch.as_tensor(x).to(torch.bfloat16).float().numpy()
    seeds = rng.integers(0, 2**63, B, dtype=np.uint64)
    rids = rng.integers(0, 2**63, B, dtype=np.uint64)
    pos = rng.integers(0, 2**31, B).astype(np.int64)
    return logits, vals, seeds, rids, pos


@pytest.mark.parametrize("tau", [0.0, 0.6, 1.0, 2.0])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_confidence_is_library_softmax_at_the_draft(tau, dtype):
    logits, vals, seeds, rids, pos = _case(3, 4, 777, 1, dtype=dtype)
    res = oracle.draft_batch(logits, tau, seeds, rids, pos)
    assert (res["status"] == 0).all()
    tc = tau if tau > 0 else 1.0
    for i in range(3):
        for k in range(4):
            q = _softmax64(vals[i, k], tc)
            z = res["z"][i, k]
            assert 0 <= z < 777
            assert res["c"][i, k] == pytest.approx(q[z], rel=1e-12)
            lt = torch.as_tensor(vals[i, k].astype(np.float64)) / tc
            assert res["m"][i, k] == float(lt.max())
            assert res["logS"][i, k] == pytest.approx(float(torch.logsumexp(lt, 0) - lt.max()), abs=1e-12)
            if tau == 0:
                assert z == int(np.argmax(vals[i, k]))     # numpy: first maximal index


def test_greedy_ties_go_to_the_lowest_index():
    x = np.zeros((1, 2, 16), np.float32)
    x[0, 0, [3, 9]] = 5.0
    x[0, 1, [0, 15]] = 1.0
    res = oracle.draft_batch(x, 0.0, np.array([1], np.uint64), np.array([2], np.uint64), np.array([0]))
    assert res["z"][0].tolist() == [3, 0]


def test_scores_are_float32_prefix_products_of_the_confidences():
    logits, _, seeds, rids, pos = _case(4, 9, 300, 2, std=1.0)
    res = oracle.draft_batch(logits, 0.8, seeds, rids, pos)
    c32 = res["c"].astype(np.float32)
    expect = np.concatenate([np.ones((4, 1), np.float32),
                             np.multiply.accumulate(c32, axis=1, dtype=np.float32)], axis=1)
    assert np.array_equal(res["s"], expect)
    assert (np.diff(res["s"], axis=1) <= 0).all()      # non-increasing (Eq. dcut-score)


def test_constant_rows_give_closed_form_scores():
    """Every row uniform over V: q(z) = 1/V at any draft, s_k = fl32 of (1/V)^k."""
    V, K = 64, 5
    x = np.zeros((1, K, V), np.float32)
    res = oracle.draft_batch(x, 1.0, np.array([7], np.uint64), np.array([3], np.uint64), np.array([10]))
    assert np.allclose(res["c"], 1.0 / V, rtol=1e-15)
    s = [np.float32(1.0)]
    for _ in range(K):
        s.append(np.float32(s[-1] * np.float32(1.0 / V)))
    assert res["s"][0].tolist() == [float(v) for v in s]


def test_one_hot_row_drafts_its_peak_with_confidence_one():
    x = np.full((1, 3, 500), -np.inf, np.float32)
    peaks = [0, 257, 499]
    for k, v in enumerate(peaks):
        x[0, k, v] = 2.0
    res = oracle.draft_batch(x, 1.0, np.array([5], np.uint64), np.array([6], np.uint64), np.array([0]))
    assert res["z"][0].tolist() == peaks
    assert res["c"][0].tolist() == [1.0, 1.0, 1.0]


@pytest.mark.parametrize("tau", [0.7, 1.5])
def test_drafts_follow_q(tau):
    """20000 requests with the same row and different request ids: the drafts'
    histogram against q (chi-square, 7 degrees of freedom)."""
    V, N = 8, 20000
    row = np.array([1.5, -0.3, 0.0, 2.2, -1.0, 0.7, 1.1, -2.0], np.float32)
    x = np.broadcast_to(row, (N, 1, V)).copy()
    res = oracle.draft_batch(x, tau, np.full(N, 11, np.uint64), np.arange(N, dtype=np.uint64),
                             np.full(N, 40, np.int64))
    q = _softmax64(row, tau)
    counts = np.bincount(res["z"][:, 0], minlength=V)
    chi2 = ((counts - N * q) ** 2 / (N * q)).sum()
    assert stats.chi2.sf(chi2, V - 1) > 1e-3


def test_drafts_follow_q_across_race_blocks():
    """V = 1000 (four race blocks): the block of the draft follows the blocks'
    mass (chi-square, 3 degrees of freedom), over 6000 positions."""
    V, N = 1000, 6000
    rng = np.random.default_rng(4)
    row = rng.normal(0, 1.0, V).astype(np.float32)
    row[600:700] += 1.5                  # more mass in block 2
    x = np.broadcast_to(row, (1, N, V)).copy()
    res = oracle.draft_batch(x, 1.0, np.array([3], np.uint64), np.array([8], np.uint64), np.array([0]))
    q = _softmax64(row, 1.0)
    mass = np.array([q[b * 256:(b + 1) * 256].sum() for b in range(4)])
    counts = np.bincount(res["z"][0] // 256, minlength=4)
    chi2 = ((counts - N * mass) ** 2 / (N * mass)).sum()
    assert stats.chi2.sf(chi2, 3) > 1e-3


def test_draw_streams_are_distinct_from_verification():
    """Same seed, request and position: the drafter's block variate is not the
    verification sampler's (distinct purposes of the counter)."""
    V = 512
    x = np.zeros((1, 1, V), np.float32)
    res = oracle.draft_batch(x, 1.0, np.array([9], np.uint64), np.array([4], np.uint64), np.array([99]))
    b = int(res["race"][0, 0, 1])
    e_draft = res["race"][0, 0, 0] * (256.0 / V)      # key * W_b with W_b = 256 / V
    e_verify = oracle.race_exponential(9, 4, 100, b, level=1)
    assert e_draft > 0 and abs(e_draft - e_verify) > 1e-9


def test_bad_rows_flag_only_their_request():
    logits, _, seeds, rids, pos = _case(3, 3, 200, 5)
    logits[0, 1, 17] = np.nan
    logits[1, 2, :] = -np.inf
    pos = pos.copy()
    pos[2] = 2**32 - 3                                # position past 2^32 - 1 at k = 3
    res = oracle.draft_batch(logits, 1.0, seeds, rids, pos)
    assert res["status"].tolist() == [oracle.ERR_BAD_INPUT] * 3
    assert (res["z"] == -1).all() and (res["s"][:, 1:] == 0).all() and (res["s"][:, 0] == 1).all()
    pos[2] = 2**32 - 4                                # the last draft at 2^32 - 1: fine
    logits2, _, _, _, _ = _case(1, 3, 200, 6)
    res = oracle.draft_batch(logits2, 1.0, seeds[2:], rids[2:], pos[2:])
    assert res["status"][0] == 0


def test_replay_is_bit_identical():
    logits, _, seeds, rids, pos = _case(2, 5, 3000, 7)
    a = oracle.draft_batch(logits, 0.9, seeds, rids, pos)
    b = oracle.draft_batch(logits, 0.9, seeds, rids, pos)
    for k in ("z", "c", "s", "m", "logS"):
        assert np.array_equal(a[k], b[k])
