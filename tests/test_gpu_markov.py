"""GPU parity of spec_markov_draft (the Markov head's sequential draw,
Section 3.2 Eq. dspark-markov) against the CPU oracle.

The bias W1[x] W2 runs on the tensor cores: r exact bf16 x bf16 products
accumulated in fp32.  Each logit therefore carries an error of at most
r 2^-23 sum_j |W1[x, j] W2[j, v]| (the accumulation, with a unit roundoff of
2^-23 to cover truncating adders) plus 2^-24 |l| (the addition of U), the
bound `logit_error` computes.  Confidences and row statistics are compared to
5e-5 relative.  A draw may differ from the oracle's only where that bound
explains it: at tau = 0 the GPU's argmax must lie within the two entries'
bounds of the oracle's maximum; at tau > 0 the oracle's race must have had a
near tie (keys within 2 (max bound / tau) + 1e-5 relative) whose runner-up
the GPU took.  The request's chain then diverges and its later positions are
not compared.
"""
import numpy as np
import pytest
import torch

import oracle
from parity import RACE_TIE, bits, race_tie

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")
C_RTOL = 5e-5


def _case(B, K, V, r, seed, std=2.0, wstd=0.3):
    g = torch.Generator().manual_seed(seed)
    U = (torch.randn((B, K, V), generator=g) * std).to(torch.bfloat16)
    W1 = (torch.randn((V, r), generator=g) * wstd).to(torch.bfloat16)
    W2 = (torch.randn((r, V), generator=g) * wstd).to(torch.bfloat16)
    rng = np.random.default_rng(seed)
    x0 = torch.as_tensor(rng.integers(0, V, B), dtype=torch.int32)
    seeds = torch.as_tensor(rng.integers(0, 2**62, B))
    rids = torch.as_tensor(rng.integers(0, 2**62, B))
    pos = torch.as_tensor(rng.integers(0, 2**31, B))
    return U, W1, W2, x0, seeds, rids, pos


def run_markov(U, W1, W2, x0, tau, seeds, rids, pos):
    import paper_2607_25852_gb300 as spec
    B, K, V = U.shape
    r = W1.shape[1]
    d = lambda x: x.to(DEV).contiguous()
    ws = spec.markov_workspace(B, K, V, r, DEV)
    out = dict(z=torch.full((B, K), -7, dtype=torch.int32, device=DEV), c=torch.zeros((B, K), device=DEV),
               s=torch.zeros((B, K + 1), device=DEV), st=torch.zeros((B * K, 2), device=DEV),
               status=torch.zeros(1, dtype=torch.int32, device=DEV))
    spec.spec_markov_draft(d(U), d(W1), d(W2.t()), d(x0), tau, d(seeds), d(rids), d(pos), out["z"], out["c"], ws,
                           scores_out=out["s"], row_stats_out=out["st"], status=out["status"])
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["status"] = int(res["status"][0])
    return res


def run_oracle_markov(U, W1, W2, x0, tau, seeds, rids, pos, requests=None):
    return oracle.markov_batch(bits(U), bits(W1), bits(W2), x0.numpy(), tau, seeds.numpy().view(np.uint64),
                               rids.numpy().view(np.uint64), pos.numpy(), requests=requests, threads=8)


def _logits(U, W1, W2, i, k, prev):
    u = U[i, k].float().double().numpy()
    return u + W1[prev].float().double().numpy() @ W2.float().double().numpy()


def logit_error(W1, W2, prev, l):
    """Bound on |l_gpu - l_exact| for every entry of a row (module docstring)."""
    r = W1.shape[1]
    a = np.abs(W1[prev].float().double().numpy()) @ np.abs(W2.float().double().numpy())
    return r * 2.0 ** -23 * a + 2.0 ** -24 * np.abs(l) + 1e-30


def _race_tie_within(race, token, eps):
    b1k, _, b2k, _, _, yk, y2k, y2, yb2 = race
    close = lambda a, b: a > 0 and (b - a) / a < eps
    return (close(b1k, b2k) and int(yb2) == token) or (close(yk, y2k) and int(y2) == token)


def compare_markov(g, r, U, W1, W2, x0, tau, requests=None):
    """Assert parity; returns the number of draws explained as near ties."""
    B, K = r["z"].shape
    ties = 0
    for i in (range(B) if requests is None else requests):
        if r["status"][i] != 0:
            assert (g["z"][i] == -1).all() and (g["c"][i] == 0).all()
            continue
        prev = int(x0[i])
        for k in range(K):
            zg, zr = int(g["z"][i, k]), int(r["z"][i, k])
            np.testing.assert_allclose(g["st"][i * K + k, 0], r["m"][i, k], rtol=C_RTOL, atol=1e-6)
            np.testing.assert_allclose(g["st"][i * K + k, 1], r["logS"][i, k], rtol=0, atol=C_RTOL)
            if zg != zr:
                l = _logits(U, W1, W2, i, k, prev)
                bound = logit_error(W1, W2, prev, l)
                if tau > 0:
                    eps = 2 * (bound.max() / tau) + RACE_TIE
                    assert _race_tie_within(r["race"][i, k], zg, eps), (i, k, zg, zr, eps)
                else:
                    assert l[zg] >= l[zr] - (bound[zg] + bound[zr]), (i, k, zg, zr, l[zr] - l[zg])
                ties += 1
                break
            assert g["c"][i, k] == pytest.approx(r["c"][i, k], rel=C_RTOL, abs=1e-30), (i, k)
            prev = zr
    return ties


@pytest.mark.parametrize("V", [300, 4096, 12345])
@pytest.mark.parametrize("r", [64, 128, 256])
@pytest.mark.parametrize("tau", [0.0, 0.8])
def test_random_shapes(V, r, tau):
    U, W1, W2, x0, seeds, rids, pos = _case(5, 3, V, r, V + r)
    g = run_markov(U, W1, W2, x0, tau, seeds, rids, pos)
    o = run_oracle_markov(U, W1, W2, x0, tau, seeds, rids, pos)
    assert g["status"] == 0 and (o["status"] == 0).all()
    ties = compare_markov(g, o, U, W1, W2, x0, tau)
    assert ties <= 1


@pytest.mark.parametrize("B", [1, 33, 64, 128])
def test_batch_sizes(B):
    """B fills one to four TMEM lane quarters (and the M = 128 tile)."""
    U, W1, W2, x0, seeds, rids, pos = _case(B, 2, 2048, 64, 7 + B)
    g = run_markov(U, W1, W2, x0, 1.0, seeds, rids, pos)
    o = run_oracle_markov(U, W1, W2, x0, 1.0, seeds, rids, pos)
    assert g["status"] == 0
    assert compare_markov(g, o, U, W1, W2, x0, 1.0) <= max(1, B // 32)


@pytest.mark.parametrize("tau", [0.0, 0.9, 1.0])
def test_zero_transition_matches_the_draft_step(tau):
    """W1 = 0: every bias vanishes and both draws race the same 256-entry
    blocks with the same variates, so the Markov head's drafts are
    spec_draft's, and both are the oracle's (equal to each other there).  A
    draft may differ only at a near tie of the race; confidences agree to
    1e-5 relative."""
    import paper_2607_25852_gb300 as spec
    B, K, V = 16, 5, 3000
    U, W1, W2, x0, seeds, rids, pos = _case(B, K, V, 64, 8)
    g = run_markov(U, torch.zeros_like(W1), W2, x0, tau, seeds, rids, pos)
    assert g["status"] == 0
    ws = spec.draft_workspace(B, K, V, DEV)
    z = torch.zeros((B, K), dtype=torch.int32, device=DEV)
    c = torch.zeros((B, K), device=DEV)
    spec.spec_draft(U.to(DEV), tau, seeds.to(DEV), rids.to(DEV), pos.to(DEV), z, c, ws)
    torch.cuda.synchronize()
    zd, cd = z.cpu().numpy(), c.cpu().numpy()
    o = oracle.draft_batch(bits(U), tau, seeds.numpy().view(np.uint64), rids.numpy().view(np.uint64), pos.numpy())
    tied = 0
    for i in range(B):
        for k in range(K):
            if g["z"][i, k] != zd[i, k]:
                # one of the two left the oracle's draw at a near tie
                zo = int(o["z"][i, k])
                other = int(g["z"][i, k]) if zd[i, k] == zo else int(zd[i, k])
                assert race_tie(o["race"][i, k], other), (i, k)
                tied += 1
                break
            np.testing.assert_allclose(g["c"][i, k], cd[i, k], rtol=1e-5)
    assert tied <= 1
    if tau > 0:
        assert len(set((g["z"] // 256).ravel().tolist())) >= 3   # the draws span several blocks


@pytest.mark.parametrize("tau", [1.0, 0.0])
def test_block_of_seven_drafts_full_vocabulary(tau):
    """B = 64 requests, a block of 8 (K = 7 drafts), V = 201088, r = 256
    (the measured configuration): every request through the oracle."""
    import os
    U, W1, W2, x0, seeds, rids, pos = _case(64, 7, 201088, 256, 9, std=3.0, wstd=0.2)
    g = run_markov(U, W1, W2, x0, tau, seeds, rids, pos)
    assert g["status"] == 0
    o = oracle.markov_batch(bits(U), bits(W1), bits(W2), x0.numpy(), tau, seeds.numpy().view(np.uint64),
                            rids.numpy().view(np.uint64), pos.numpy(), threads=os.cpu_count() or 8)
    ties = compare_markov(g, o, U, W1, W2, x0, tau)
    print("markov full-size ties:", ties)
    assert ties <= 1


def test_bad_inputs_are_flagged_per_request():
    import paper_2607_25852_gb300 as spec
    U, W1, W2, x0, seeds, rids, pos = _case(4, 3, 1000, 64, 10)
    U[0, 1, 5] = float("nan")
    x0[1] = 1000
    pos[2] = 2**32 - 2
    g = run_markov(U, W1, W2, x0, 1.0, seeds, rids, pos)
    o = run_oracle_markov(U, W1, W2, x0, 1.0, seeds, rids, pos)
    assert g["status"] == spec.ERR_BAD_INPUT
    assert o["status"].tolist() == [oracle.ERR_BAD_INPUT] * 3 + [0]
    compare_markov(g, o, U, W1, W2, x0, 1.0)
    assert (g["s"][:3, 1:] == 0).all() and (g["s"][:3, 0] == 1).all()


@pytest.mark.parametrize("B,r", [(65, 64), (100, 192), (7, 192)])
def test_batches_past_the_repeated_rows_and_three_atom_rank(B, r):
    """B = 65 and 100: the operand is not repeated, every lane quarter takes
    its own rows over all columns (the last quarter part-filled); r = 192:
    three K-atoms per tile."""
    U, W1, W2, x0, seeds, rids, pos = _case(B, 3, 3000, r, 40 + B + r)
    g = run_markov(U, W1, W2, x0, 0.9, seeds, rids, pos)
    o = run_oracle_markov(U, W1, W2, x0, 0.9, seeds, rids, pos)
    assert g["status"] == 0 and (o["status"] == 0).all()
    assert compare_markov(g, o, U, W1, W2, x0, 0.9) <= max(1, B // 32)
