"""Pins for the oracle's D-cut allocator (Section 4.2: Eqs. (dcut-score),
(dcut-expected-advance), (dcut-budget), (dcut-batch-utility), (dcut-select)).

The greedy top-T selection is checked against brute-force enumeration of all
depth vectors, the budget against worked values of Eq. (dcut-budget) and
exact rational arithmetic, and the packing against its definition.
"""
import itertools
import os
from fractions import Fraction
from math import ceil

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _scores(conf):
    """s_{i,k} as fp32 products in order (numpy's cumprod on float32)."""
    conf = np.asarray(conf, np.float32)
    B = conf.shape[0]
    return np.concatenate([np.ones((B, 1), np.float32), np.cumprod(conf, axis=1, dtype=np.float32)],
                          axis=1)


def _units(s):
    return np.floor(np.ldexp(s.astype(np.float64), 40)).astype(np.int64)


def _brute_force_best(conf, T):
    s = _units(_scores(conf))
    B, K1 = s.shape
    best = None
    for n in itertools.product(range(K1), repeat=B):
        if sum(n) + B != T:
            continue
        u = sum(int(s[i, :n[i] + 1].sum()) for i in range(B))
        if best is None or u > best[0]:
            best = (u, n)
    return best


def test_budget_matches_worked_values():
    ratios = [(1, 4), (1, 2), (3, 4), (1, 1)]
    rows = [l.split() for l in open(os.path.join(GOLDEN, "dcut_budget.txt")) if not l.startswith("#")]
    assert len(rows) >= 10
    for row in rows:
        B, D, *expected = map(int, row)
        got = [oracle.budget(B, D, n, d) for n, d in ratios]
        assert got == expected, (B, D)
        exact = [max(B, ceil(Fraction(n, d) * B * (D + 1))) for n, d in ratios]
        assert got == exact


@pytest.mark.parametrize("B,K", [(1, 3), (2, 2), (3, 2), (2, 4), (3, 3), (4, 2)])
def test_greedy_selection_is_the_brute_force_optimum(B, K):
    rng = np.random.default_rng(100 + 10 * B + K)
    for trial in range(12):
        if trial % 3 == 0:
            conf = rng.choice([0.0, 0.25, 0.5, 1.0], size=(B, K)).astype(np.float32)   # ties
        else:
            conf = rng.uniform(size=(B, K)).astype(np.float32)
        Ts = np.arange(B, B * (K + 1) + 1, dtype=np.int32)
        res = oracle.allocate(conf, Ts, np.ones(len(Ts)))
        assert res["status"] == 0
        s = _units(_scores(conf))
        for c, T in enumerate(Ts):
            u_best, _ = _brute_force_best(conf, int(T))
            n = res["all_depths"][c]
            assert (n >= 0).all() and (n <= K).all()
            assert int((n + 1).sum()) == T
            assert sum(int(s[i, :n[i] + 1].sum()) for i in range(B)) == u_best
            assert res["utility"][c] == np.ldexp(float(u_best), -40)


def test_ties_go_to_shallower_positions_then_lower_requests():
    B, K = 5, 3
    conf = np.ones((B, K), np.float32)                       # every score is 1
    Ts = np.array([B, B + 2, B + B, B + B + 1, B * (K + 1)], np.int32)
    res = oracle.allocate(conf, Ts, np.ones(len(Ts)))
    d = res["all_depths"]
    assert d[0].tolist() == [0] * B                             # bonus only
    assert d[1].tolist() == [1, 1, 0, 0, 0]                     # k = 1 of requests 0, 1
    assert d[2].tolist() == [1] * B                             # all k = 1 before any k = 2
    assert d[3].tolist() == [2, 1, 1, 1, 1]
    assert d[4].tolist() == [K] * B


def test_negative_zero_confidence_counts_as_zero():
    """-0 is the value 0 (Eq. dcut-score then gives s = 0): an allocation with
    -0 confidences equals the one with +0 everywhere, and the zero scores
    rank after every positive score with the tie rule (shallower k, then
    lower request)."""
    B, K = 4, 3
    pos = np.array([[0.9, -0.0, 0.5], [-0.0, 0.7, 0.7], [0.6, 0.6, 0.6], [-0.0, -0.0, -0.0]], np.float32)
    assert np.signbit(pos[1, 0]) and pos[1, 0] == 0.0
    plus = np.abs(pos)
    N = B * (K + 1)
    Ts = np.array([B, B + 3, B + 5, B + 7, N], np.int32)
    a = oracle.allocate(pos, Ts, np.ones(len(Ts)))
    b = oracle.allocate(plus, Ts, np.ones(len(Ts)))
    assert a["status"] == 0 and b["status"] == 0
    for k in ("depth", "row_offsets", "packed_tokens", "packed_pos", "utility", "all_depths"):
        assert np.array_equal(a[k], b[k]), k
    d = a["all_depths"]
    assert d[0].tolist() == [0, 0, 0, 0]                     # the bonus positions first
    assert d[1].tolist() == [1, 0, 2, 0]                     # s = 0.9, 0.6, 0.36
    assert d[2].tolist() == [1, 1, 3, 0]                     # 0.216, then the first zero: request 1, k = 1
    assert d[3].tolist() == [2, 1, 3, 1]                     # zeros: request 3 at k = 1, then request 0 at k = 2
    assert d[4].tolist() == [K] * B


def test_expected_advance_and_monotone_utility():
    rng = np.random.default_rng(5)
    B, K = 8, 6
    conf = rng.uniform(0.2, 1.0, size=(B, K)).astype(np.float32)
    Ts = np.arange(B, B * (K + 1) + 1, dtype=np.int32)
    res = oracle.allocate(conf, Ts, np.ones(len(Ts)))
    s = _scores(conf).astype(np.float64)
    for c, T in enumerate(Ts):
        n = res["all_depths"][c]
        # Eq. (dcut-expected-advance) summed per Eq. (dcut-batch-utility)
        a_hat = sum(s[i, :n[i] + 1].sum() for i in range(B))
        assert res["utility"][c] == pytest.approx(a_hat, abs=B * (K + 1) * 2.0**-40)
    assert (np.diff(res["utility"]) >= 0).all()
    assert res["all_depths"][-1].tolist() == [K] * B


def test_budget_choice_is_first_argmax_of_utility_over_cost():
    rng = np.random.default_rng(6)
    B, K = 16, 8
    conf = rng.beta(2, 2, size=(B, K)).astype(np.float32)
    Ts = np.array([oracle.budget(B, K, n, 4) for n in (1, 2, 3, 4)], np.int32)
    for costs in ([1.0, 1.0, 1.0, 1.0], [1.0, 1.9, 2.8, 3.7], [1.0, 1.2, 1.5, 10.0],
                  [float(T) for T in Ts]):
        res = oracle.allocate(conf, Ts, costs)
        obj = [Fraction(res["utility"][c]) / Fraction(costs[c]) for c in range(4)]
        # exact rationals agree with the fp64 ratio on these inputs; first maximiser wins
        want = max(range(4), key=lambda c: (obj[c], -c))
        assert res["chosen_T"] == Ts[want]
        assert res["depth"].tolist() == res["all_depths"][want].tolist()
    # all confidences zero: every candidate has utility B; the first (smallest T) wins
    res = oracle.allocate(np.zeros((B, K), np.float32), Ts, np.ones(4))
    assert res["chosen_T"] == Ts[0] and (res["utility"] == B).all()


def test_packing_layout():
    rng = np.random.default_rng(7)
    B, K = 6, 5
    conf = rng.uniform(size=(B, K)).astype(np.float32)
    last = rng.integers(0, 1000, B).astype(np.int32)
    drafts = rng.integers(0, 1000, (B, K)).astype(np.int32)
    pos = rng.integers(0, 10**6, B).astype(np.int64)
    res = oracle.allocate(conf, [17], [1.0], last, drafts, pos)
    n = res["depth"]
    off = np.concatenate([[0], np.cumsum(n + 1)])
    assert res["row_offsets"].tolist() == off.tolist() and off[-1] == 17
    for i in range(B):
        rows = slice(off[i], off[i + 1])
        assert res["packed_tokens"][rows].tolist() == [last[i]] + drafts[i, :n[i]].tolist()
        assert res["packed_pos"][rows].tolist() == list(range(pos[i], pos[i] + n[i] + 1))
    assert (res["packed_tokens"][17:] == -1).all() and (res["packed_pos"][17:] == -1).all()


def test_invalid_arguments_and_inputs():
    conf = np.full((2, 2), 0.5, np.float32)
    assert oracle.allocate(conf, [1], [1.0])["status"] == oracle.ERR_INVALID_ARG      # T < B
    assert oracle.allocate(conf, [7], [1.0])["status"] == oracle.ERR_INVALID_ARG      # T > B(K+1)
    assert oracle.allocate(conf, [4], [0.0])["status"] == oracle.ERR_INVALID_ARG      # cost <= 0
    bad = conf.copy()
    bad[1, 0] = np.nan
    res = oracle.allocate(bad, [4], [1.0])
    assert res["status"] == oracle.ERR_BAD_INPUT
    # the invalid confidence counts as 0: request 1 keeps only its bonus
    assert res["depth"].tolist() == [2, 0]
