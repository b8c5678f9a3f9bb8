"""Statistical checks of the CUDA path on its own (not through the oracle):
the committed tokens follow the target distribution exactly (Section 1), and
the acceptance rate equals the distribution overlap sum_v min(p, q)
(Eq. mtp-acceptance-tv).  The same 10^6-sequence run is also compared with the
oracle element by element."""
import numpy as np
import pytest
import torch
from scipy import stats

import oracle
import paper_2607_25852_gb300 as spec
from parity import ACCEPT_TIE, race_tie

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


def _softmax64(x, t):
    return torch.softmax(torch.as_tensor(np.asarray(x, np.float64)) / t, dim=-1).numpy()


class MarkovToy:
    """Order-1 Markov target P and drafter Q over V tokens."""

    def __init__(self, V, seed, t):
        rng = np.random.default_rng(seed)
        self.V, self.t = V, t
        self.logP = rng.normal(0, 1.2, (V, V)).astype(np.float32)
        self.Q = rng.dirichlet(np.ones(V) * 0.7, size=V).astype(np.float32)
        self.P = np.stack([_softmax64(r, t) for r in self.logP])

    def round_inputs(self, prev, K, rng, one_hot):
        N = len(prev)
        drafts = np.zeros((N, K), np.int32)
        cur = prev.copy()
        for j in range(K):
            if one_hot:
                nxt = self.Q[cur].argmax(-1)
            else:
                cdf = np.cumsum(self.Q[cur].astype(np.float64), axis=1)
                cdf /= cdf[:, -1:]
                nxt = (rng.random((N, 1)) > cdf).sum(1)
            drafts[:, j] = nxt
            cur = nxt
        ctx = np.concatenate([prev[:, None], drafts], axis=1)
        logits = self.logP[ctx].reshape(N * (K + 1), self.V)
        q = None if one_hot else self.Q[ctx[:, :K]]
        return drafts, logits, q


def _gpu_round(drafts, logits, q, t, seeds, reqs, pos):
    B, K = drafts.shape
    V = logits.shape[1]
    acc = torch.zeros(B, dtype=torch.int32, device=DEV)
    tok = torch.zeros((B, K + 1), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = spec.verify_workspace(B, K, V, DEV)
    spec.spec_verify(torch.as_tensor(logits, device=DEV), torch.as_tensor(drafts, device=DEV),
                     None if q is None else torch.as_tensor(np.ascontiguousarray(q), device=DEV),
                     B, K, V, t, torch.as_tensor(seeds.view(np.int64), device=DEV),
                     torch.as_tensor(reqs.view(np.int64), device=DEV), torch.as_tensor(pos, device=DEV),
                     acc, tok, ws, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return acc.cpu().numpy(), tok.cpu().numpy()


@pytest.mark.parametrize("one_hot", [False, True])
def test_gpu_committed_tokens_follow_the_target(one_hot):
    V, K, t, N = 8, 2, 0.8, 1000000
    toy = MarkovToy(V, seed=21, t=t)
    rng = np.random.default_rng(22)
    out = [[] for _ in range(N)]
    pos = np.zeros(N, np.int64)
    todo = np.arange(N)
    mismatches = positions = 0
    for _round in range(4):
        prev = np.array([out[i][-1] if out[i] else 0 for i in todo], np.int64)
        drafts, logits, q = toy.round_inputs(prev, K, rng, one_hot)
        seeds = np.full(len(todo), 77, np.uint64)
        reqs = todo.astype(np.uint64)
        acc, tok = _gpu_round(drafts, logits, q, t, seeds, reqs, pos[todo])
        if _round == 0:
            # element-wise parity with the oracle on the whole first round
            ref = oracle.verify_batch(logits, drafts, q, t, seeds, reqs, pos[todo])
            diff = np.nonzero((ref["accepted"] != acc) | (ref["tokens"] != tok).any(1))[0]
            for i in diff:
                a = min(acc[i], ref["accepted"][i])
                if acc[i] != ref["accepted"][i]:
                    assert abs(ref["u"][i, a] - ref["r"][i, a]) < ACCEPT_TIE
                else:
                    assert race_tie(ref["race"][i], int(tok[i, a]))
            mismatches = len(diff)
            positions = len(todo) * (K + 1)
        for r, i in enumerate(todo):
            a = acc[r]
            out[i].extend(tok[r, :a + 1].tolist())
            pos[i] += a + 1
        todo = np.array([i for i in todo if len(out[i]) < 2], np.int64)
        if len(todo) == 0:
            break
    assert mismatches <= 1e-4 * positions, (mismatches, positions)
    toks = np.array([o[:2] for o in out])
    c1 = np.bincount(toks[:, 0], minlength=V)
    assert stats.chisquare(c1, N * toy.P[0]).pvalue > 1e-3
    joint = (toy.P[0][:, None] * toy.P).reshape(-1)
    c2 = np.bincount(toks[:, 0] * V + toks[:, 1], minlength=V * V)
    assert stats.chisquare(c2, N * joint).pvalue > 1e-3


def test_gpu_acceptance_rate_is_overlap():
    rng = np.random.default_rng(23)
    V, t, N = 64, 0.9, 400000
    row = rng.normal(0, 1.5, V).astype(np.float32)
    p = _softmax64(row, t)
    qv = _softmax64(row + rng.normal(0, 1.0, V), 1.0).astype(np.float32)
    alpha = np.minimum(p, qv.astype(np.float64)).sum()
    pq = qv.astype(np.float64)
    drafts = rng.choice(V, size=(N, 1), p=pq / pq.sum()).astype(np.int32)
    logits = np.tile(row, (2 * N, 1))
    q = np.tile(qv, (N, 1, 1))
    acc, _ = _gpu_round(drafts, logits, q, t, np.arange(N, dtype=np.uint64), np.zeros(N, np.uint64),
                        np.zeros(N, np.int64))
    rate = acc.mean()
    assert abs(rate - alpha) < 5 * np.sqrt(alpha * (1 - alpha) / N)
