"""Pins for the oracle's verification (rejection sampling, Section 1; the
overlap identity Eq. (mtp-acceptance-tv), Section 2; the deterministic-draft,
target-only protocol of Section 4.2).

Each test checks the oracle against something other than itself: a library
routine, a brute-force definition on tiny inputs, a closed form, or a
statistical property that the method guarantees (the committed tokens follow
the target distribution exactly).
"""
import numpy as np
import pytest
import torch
from scipy import stats

import oracle
from conftest import bf16_bits_from_float


def _softmax64(x, t):
    return torch.softmax(torch.as_tensor(np.asarray(x, np.float64)) / t, dim=-1).numpy()


# ---------------------------------------------------------------------------
# Softmax statistics and p(z) against torch (float64)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("t", [0.3, 0.8, 1.0, 2.5])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_row_statistics_match_library_softmax(t, dtype):
    rng = np.random.default_rng(1)
    n, V = 3, 1000
    x = rng.normal(0, 3, (n + 1, V)).astype(np.float32)
    logits = x if dtype == "f32" else bf16_bits_from_float(x)
    vals = x if dtype == "f32" else torch.as_tensor(x).to(torch.bfloat16).float().numpy()
    drafts = rng.integers(0, V, n)
    res = oracle.verify_request(logits, drafts, None, t, 9, 4, 100)
    assert res["status"] == 0
    lt = torch.as_tensor(vals.astype(np.float64)) / t
    np.testing.assert_allclose(res["row_m"], lt.max(dim=-1).values.numpy(), rtol=0, atol=0)
    np.testing.assert_allclose(res["row_logS"], (torch.logsumexp(lt, -1) - lt.max(-1).values).numpy(),
                               rtol=1e-12, atol=1e-12)
    for j in range(res["accepted"] + (1 if res["accepted"] < n else 0)):
        p = _softmax64(vals[j], t)
        assert res["p_draft"][j] == pytest.approx(p[drafts[j]], rel=1e-12)
        assert abs(p.sum() - 1.0) < 1e-12


# ---------------------------------------------------------------------------
# Temperature 0: longest argmax-matching prefix (brute force on tiny inputs)
# ---------------------------------------------------------------------------
def _greedy_brute(rows, drafts):
    n = len(drafts)
    g = []
    for row in rows:
        best = max(row)
        g.append(list(row).index(best))            # lowest index among ties
    a = 0
    while a < n and drafts[a] == g[a]:
        a += 1
    return a, list(drafts[:a]) + [g[a]]


def test_greedy_matches_brute_force_with_ties():
    rng = np.random.default_rng(2)
    for trial in range(300):
        n = int(rng.integers(0, 6))
        V = int(rng.integers(1, 9))
        rows = rng.integers(-2, 3, size=(n + 1, V)).astype(np.float32)   # many ties
        g = [list(r).index(max(r)) for r in rows]
        drafts = np.array([g[j] if rng.random() < 0.7 else int(rng.integers(0, V)) for j in range(n)],
                          dtype=np.int32)
        res = oracle.verify_request(rows, drafts, None, 0.0, 0, 0, 0)
        a, toks = _greedy_brute(rows.tolist(), drafts.tolist())
        assert res["accepted"] == a
        assert res["tokens"][:a + 1].tolist() == toks
        assert (res["tokens"][a + 1:] == -1).all()


def test_greedy_all_drafts_are_argmax_accepts_everything():
    rng = np.random.default_rng(3)
    rows = rng.normal(size=(9, 500)).astype(np.float32)
    drafts = rows[:8].argmax(-1).astype(np.int32)
    res = oracle.verify_request(rows, drafts, None, 0.0, 0, 0, 0)
    assert res["accepted"] == 8
    assert res["tokens"][:8].tolist() == drafts.tolist()
    assert res["tokens"][8] == int(rows[8].argmax())


# ---------------------------------------------------------------------------
# Acceptance: q <= p at the draft accepts surely; one-hot q accepts w.p. p(z);
# general q accepts w.p. sum_v min(p, q)  (Eq. mtp-acceptance-tv)
# ---------------------------------------------------------------------------
def test_q_equal_to_p_accepts_every_draft():
    rng = np.random.default_rng(4)
    n, V, t = 5, 64, 0.9
    rows = rng.normal(0, 2, (n + 1, V)).astype(np.float32)
    p = np.stack([_softmax64(r, t) for r in rows[:n]])
    p32 = p.astype(np.float32)
    q = np.where(p32.astype(np.float64) <= p, p32, np.nextafter(p32, np.float32(-np.inf)))  # q = p, rounded down
    for seed in range(2000):
        drafts = np.array([rng.choice(V, p=p[j]) for j in range(n)], np.int32)
        res = oracle.verify_request(rows, drafts, q, t, seed, seed, 10)
        assert res["accepted"] == n and res["mode"] == oracle.MODE_BONUS


def test_one_hot_acceptance_rate_is_target_probability():
    rng = np.random.default_rng(5)
    V, t = 32, 1.0
    rows = rng.normal(0, 1.5, (2, V)).astype(np.float32)
    z = 7
    pz = _softmax64(rows[0], t)[z]
    N = 40000
    acc = sum(oracle.verify_request(rows, [z], None, t, 123, i, 0)["accepted"] for i in range(N))
    assert abs(acc / N - pz) < 5 * np.sqrt(pz * (1 - pz) / N)


def test_acceptance_rate_is_distribution_overlap():
    rng = np.random.default_rng(6)
    V, t = 16, 0.7
    rows = rng.normal(0, 1.0, (2, V)).astype(np.float32)
    p = _softmax64(rows[0], t)
    qv = _softmax64(rows[0] + rng.normal(0, 1.0, V), 1.0).astype(np.float32)
    q = qv[None, :]
    alpha = np.minimum(p, qv.astype(np.float64)).sum()               # 1 - TV(p, q)
    N = 60000
    zs = rng.choice(V, size=N, p=qv.astype(np.float64) / qv.sum())
    acc = sum(oracle.verify_request(rows, [int(zs[i])], q, t, 77, i, 5)["accepted"] for i in range(N))
    assert abs(acc / N - alpha) < 5 * np.sqrt(alpha * (1 - alpha) / N)


# ---------------------------------------------------------------------------
# Distribution preservation: the committed stream follows the target exactly
# ---------------------------------------------------------------------------
class _MarkovToy:
    """Order-1 Markov target P and drafter Q over V tokens: every verification
    row's logits are log P[previous token]; drafts are drawn from Q."""

    def __init__(self, V, seed, t):
        rng = np.random.default_rng(seed)
        self.V, self.t = V, t
        self.logP = rng.normal(0, 1.2, (V, V)).astype(np.float32)
        self.Q = rng.dirichlet(np.ones(V) * 0.7, size=V).astype(np.float32)
        self.P = np.stack([_softmax64(r, t) for r in self.logP])   # target at temperature t

    def round_inputs(self, prev, K, rng, one_hot):
        """Inputs of one round for each context token in `prev` [N]."""
        N = len(prev)
        drafts = np.zeros((N, K), np.int32)
        cur = prev.copy()
        for j in range(K):
            if one_hot:
                nxt = self.Q[cur].argmax(-1)                         # deterministic drafter
            else:
                cdf = np.cumsum(self.Q[cur].astype(np.float64), axis=1)
                cdf /= cdf[:, -1:]
                nxt = (rng.random((N, 1)) > cdf).sum(1)
            drafts[:, j] = nxt
            cur = nxt
        ctx = np.concatenate([prev[:, None], drafts], axis=1)      # token before row j
        logits = self.logP[ctx].reshape(N * (K + 1), self.V)
        # q row j is the drafter's distribution of draft j+1 given the token before it
        q = None if one_hot else self.Q[ctx[:, :K]]
        return drafts, logits, q


def _first_two_tokens(toy, N, K, one_hot, seed):
    """Run rounds until every sequence has >= 2 committed tokens."""
    rng = np.random.default_rng(seed)
    start = np.zeros(N, np.int64)
    out = [[] for _ in range(N)]
    pos = np.zeros(N, np.int64)
    todo = np.arange(N)
    for _round in range(4):
        prev = np.array([out[i][-1] if out[i] else start[i] for i in todo], np.int64)
        drafts, logits, q = toy.round_inputs(prev, K, rng, one_hot)
        res = oracle.verify_batch(logits, drafts, q, toy.t, np.full(len(todo), 99, np.uint64),
                                  todo.astype(np.uint64), pos[todo])
        assert (res["status"] == 0).all()
        for r, i in enumerate(todo):
            a = res["accepted"][r]
            out[i].extend(res["tokens"][r, :a + 1].tolist())
            pos[i] += a + 1
        todo = np.array([i for i in todo if len(out[i]) < 2], np.int64)
        if len(todo) == 0:
            break
    assert len(todo) == 0
    return np.array([o[:2] for o in out])


@pytest.mark.parametrize("one_hot", [False, True])
def test_committed_tokens_follow_the_target_distribution(one_hot):
    V, K, t, N = 8, 2, 0.8, 1000000
    toy = _MarkovToy(V, seed=11, t=t)
    toks = _first_two_tokens(toy, N, K, one_hot, seed=12)
    # first token ~ P[start]
    c1 = np.bincount(toks[:, 0], minlength=V)
    assert stats.chisquare(c1, N * toy.P[0]).pvalue > 1e-3
    # first two tokens ~ P[start](x1) P[x1](x2)
    joint = (toy.P[0][:, None] * toy.P).reshape(-1)
    c2 = np.bincount(toks[:, 0] * V + toks[:, 1], minlength=V * V)
    assert stats.chisquare(c2, N * joint).pvalue > 1e-3


def test_bonus_draw_follows_the_bonus_row():
    rng = np.random.default_rng(13)
    V, t, N = 10, 1.3, 100000
    rows = rng.normal(0, 1.0, (2, V)).astype(np.float32)
    p0 = _softmax64(rows[0], t)
    q = np.full((1, V), 1e-30, np.float32)                            # q <= p: always accepted
    res = oracle.verify_batch(np.tile(rows, (N, 1)), np.full((N, 1), 3, np.int32),
                              np.tile(q[None], (N, 1, 1)), t, np.arange(N, dtype=np.uint64),
                              np.zeros(N, np.uint64), np.zeros(N, np.int64))
    assert (res["accepted"] == 1).all()
    counts = np.bincount(res["tokens"][:, 1], minlength=V)
    assert stats.chisquare(counts, N * _softmax64(rows[1], t)).pvalue > 1e-3
    assert p0.sum() == pytest.approx(1.0)


def test_one_hot_rejection_draws_target_without_the_draft():
    rng = np.random.default_rng(14)
    V, t, N = 6, 1.0, 120000
    rows = rng.normal(0, 0.5, (2, V)).astype(np.float32)
    z = 2
    res = oracle.verify_batch(np.tile(rows, (N, 1)), np.full((N, 1), z, np.int32), None, t,
                              np.full(N, 5, np.uint64), np.arange(N, dtype=np.uint64),
                              np.zeros(N, np.int64))
    rej = res["accepted"] == 0
    y = res["tokens"][rej, 0]
    assert (y != z).all()
    p = _softmax64(rows[0], t)
    w = p.copy()
    w[z] = 0
    counts = np.bincount(y, minlength=V)
    assert stats.chisquare(np.delete(counts, z), rej.sum() * np.delete(w / w.sum(), z)).pvalue > 1e-3


def _draws(rows, drafts, q, t, N, chunk=20000):
    """Outcomes of N requests that verify the same rows, seeds 0..N-1."""
    acc, tok = [], []
    for s0 in range(0, N, chunk):
        m = min(chunk, N - s0)
        res = oracle.verify_batch(np.tile(rows, (m, 1)), np.tile(drafts, (m, 1)),
                                  None if q is None else np.tile(q[None], (m, 1, 1)), t,
                                  np.arange(s0, s0 + m, dtype=np.uint64), np.zeros(m, np.uint64),
                                  np.zeros(m, np.int64))
        acc.append(res["accepted"])
        tok.append(res["tokens"])
    return np.concatenate(acc), np.concatenate(tok)


def test_draws_span_several_race_blocks():
    """V = 1100 spans five blocks of the two-level race (the last one partial):
    the bonus draw follows p and the residual draw follows norm(max(0, p - q))."""
    rng = np.random.default_rng(17)
    V, t, N = 1100, 1.0, 200000
    rows = rng.normal(0, 1.0, (2, V)).astype(np.float32)
    # bonus: q <= p at the draft, so it is always accepted and row 1 is drawn
    acc, tok = _draws(rows, np.array([[5]], np.int32), np.full((1, V), 1e-30, np.float32), t, N)
    assert (acc == 1).all()
    counts = np.bincount(tok[:, 1], minlength=V)
    assert stats.chisquare(counts, N * _softmax64(rows[1], t)).pvalue > 1e-3
    # residual: a draft distribution far from p, drafts drawn from it
    qv = _softmax64(rows[0] + rng.normal(0, 2.0, V), 1.0).astype(np.float32)
    p = _softmax64(rows[0], t)
    z = int(np.argmax(qv.astype(np.float64) - p))                      # q(z) > p(z): often rejected
    acc, tok = _draws(rows, np.array([[z]], np.int32), qv[None, :], t, N)
    rej = acc == 0
    resid = np.maximum(0.0, p - qv.astype(np.float64))
    assert rej.mean() == pytest.approx(1.0 - min(1.0, p[z] / float(qv[z])), abs=5e-3)
    counts = np.bincount(tok[rej, 0], minlength=V)
    keep = resid > 0
    assert counts[~keep].sum() == 0
    assert stats.chisquare(counts[keep], rej.sum() * resid[keep] / resid.sum()).pvalue > 1e-3


# ---------------------------------------------------------------------------
# Determinism (replay gives the same bits) and bad inputs
# ---------------------------------------------------------------------------
def test_replay_is_bit_identical():
    rng = np.random.default_rng(15)
    rows = rng.normal(0, 2, (5, 300)).astype(np.float32)
    d = rng.integers(0, 300, 4).astype(np.int32)
    a = oracle.verify_request(rows, d, None, 1.0, 42, 7, 1000)
    b = oracle.verify_request(rows, d, None, 1.0, 42, 7, 1000)
    assert a["tokens"].tolist() == b["tokens"].tolist() and a["race"].tolist() == b["race"].tolist()


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_bad_inputs_flag_the_request(t):
    rng = np.random.default_rng(16)
    rows = rng.normal(0, 2, (3, 50)).astype(np.float32)
    good = np.array([1, 2], np.int32)
    assert oracle.verify_request(rows, good, None, t, 0, 0, 0)["status"] == 0
    nan_rows = rows.copy()
    nan_rows[1, 7] = np.nan
    for bad in [dict(rows=nan_rows), dict(drafts=np.array([1, 50], np.int32)),
                dict(drafts=np.array([-1, 2], np.int32)), dict(pos=2**32 - 2)]:
        res = oracle.verify_request(bad.get("rows", rows), bad.get("drafts", good), None, t, 0, 0,
                                    bad.get("pos", 0))
        assert res["status"] == oracle.ERR_BAD_INPUT
        assert res["accepted"] == 0 and (res["tokens"] == -1).all()
    if t > 0:
        inf_rows = rows.copy()
        inf_rows[0] = -np.inf
        assert oracle.verify_request(inf_rows, good, None, t, 0, 0, 0)["status"] == oracle.ERR_BAD_INPUT
