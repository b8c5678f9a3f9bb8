"""GPU parity of spec_draft (the drafter's producer step: drafts, token-level
confidences and D-cut scores, Section 4.2 Eq. dcut-score) against the CPU
oracle.  Comparison: drafts bit-exact (a draw may differ only where the
oracle's race had a near tie and the GPU took the runner-up, counted);
confidences and row statistics to 1e-5; scores bit-exact against the fp32
prefix products of the GPU's own confidences, and to 1e-5 against the
oracle's."""
import numpy as np
import pytest
import torch
from scipy import stats

import oracle
import workloads
from parity import P_RTOL, bits, race_tie

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


def run_draft(logits, tau, seeds, rids, pos, ws=None):
    import paper_2607_25852_gb300 as spec
    B, K, V = logits.shape
    d = lambda x: x.to(DEV).contiguous() if x.device != DEV or not x.is_contiguous() else x
    ws = spec.draft_workspace(B, K, V, DEV) if ws is None else ws
    out = dict(z=torch.full((B, K), -7, dtype=torch.int32, device=DEV),
               c=torch.full((B, K), -7.0, device=DEV), s=torch.full((B, K + 1), -7.0, device=DEV),
               st=torch.zeros((B * K, 2), device=DEV), status=torch.zeros(1, dtype=torch.int32, device=DEV))
    spec.spec_draft(d(logits), tau, d(seeds), d(rids), d(pos), out["z"], out["c"], ws, scores_out=out["s"],
                    row_stats_out=out["st"], status=out["status"])
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["status"] = int(res["status"][0])
    res["ws"] = ws
    return res


def run_oracle_draft(logits, tau, seeds, rids, pos):
    return oracle.draft_batch(bits(logits), tau, seeds.cpu().numpy().view(np.uint64),
                              rids.cpu().numpy().view(np.uint64), pos.cpu().numpy())


def compare_draft(g, r, tau):
    """Assert parity; returns the number of near-tie draws."""
    B, K = r["z"].shape
    ties = 0
    for i in range(B):
        if r["status"][i] != 0:
            assert (g["z"][i] == -1).all() and (g["c"][i] == 0).all()
            assert g["s"][i, 0] == 1 and (g["s"][i, 1:] == 0).all()
            continue
        tied = False
        for k in range(K):
            if g["z"][i, k] != r["z"][i, k]:
                assert tau > 0 and race_tie(r["race"][i, k], int(g["z"][i, k])), (
                    f"request {i} row {k}: draft {g['z'][i, k]} vs oracle {r['z'][i, k]}")
                ties += 1
                tied = True
                continue
            assert g["c"][i, k] == pytest.approx(r["c"][i, k], rel=P_RTOL, abs=1e-30), (i, k)
        np.testing.assert_allclose(g["st"][i * K:(i + 1) * K, 0], r["m"][i], rtol=P_RTOL, atol=0)
        np.testing.assert_allclose(g["st"][i * K:(i + 1) * K, 1], r["logS"][i], rtol=0, atol=P_RTOL)
        if not tied:
            np.testing.assert_allclose(g["s"][i], r["s"][i], rtol=P_RTOL, atol=1e-30)
    # the scores are the allocator's: fp32 prefix products of the GPU's own confidences
    ok = r["status"] == 0
    expect = np.concatenate([np.ones((B, 1), np.float32),
                             np.multiply.accumulate(g["c"].astype(np.float32), axis=1, dtype=np.float32)], 1)
    assert np.array_equal(g["s"][ok], expect[ok])
    assert ties <= max(1, 1e-4 * B * K), ties
    return ties


def _case(B, K, V, dtype, seed, std=2.0):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn((B, K, V), generator=g) * std
    x = x.to(torch.bfloat16 if dtype == "bf16" else torch.float32)
    rng = np.random.default_rng(seed)
    return (x, torch.as_tensor(rng.integers(0, 2**62, B)), torch.as_tensor(rng.integers(0, 2**62, B)),
            torch.as_tensor(rng.integers(0, 2**31, B)))


@pytest.mark.parametrize("V", [1, 7, 256, 257, 4096, 12345])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("tau", [0.0, 0.7, 1.5])
def test_random_shapes(V, dtype, tau):
    x, seeds, rids, pos = _case(3, 4, V, dtype, V + 7)
    compare_draft(run_draft(x, tau, seeds, rids, pos), run_oracle_draft(x, tau, seeds, rids, pos), tau)


@pytest.mark.parametrize("tau", [0.0, 1.0])
def test_misaligned_rows_take_the_scalar_path(tau):
    """Rows 2 bytes off a 16-byte boundary: the per-entry loads."""
    x, seeds, rids, pos = _case(4, 3, 4096, "bf16", 3)
    buf = torch.empty(x.numel() + 1, dtype=x.dtype, device=DEV)
    view = buf[1:].view(x.shape)
    view.copy_(x.to(DEV))
    assert view.data_ptr() % 16 == 2
    compare_draft(run_draft(view, tau, seeds, rids, pos), run_oracle_draft(x, tau, seeds, rids, pos), tau)


@pytest.mark.parametrize("tau", [0.05, 4.0])
def test_temperature_extremes(tau):
    x, seeds, rids, pos = _case(6, 5, 5000, "bf16", 11, std=3.0)
    compare_draft(run_draft(x, tau, seeds, rids, pos), run_oracle_draft(x, tau, seeds, rids, pos), tau)


def test_most_drafts_per_request():
    x, seeds, rids, pos = _case(2, 255, 700, "bf16", 12)
    compare_draft(run_draft(x, 1.0, seeds, rids, pos), run_oracle_draft(x, 1.0, seeds, rids, pos), 1.0)


def test_full_size_draft_block():
    """B = 64 requests, K = 16 drafts, V = 201088 bf16 at tau = 1 (the draft
    recipe): every row through the oracle."""
    di = workloads.make_draft()
    g = run_draft(di.logits, di.tau, di.seeds, di.request_ids, di.pos_base)
    r = run_oracle_draft(di.logits, di.tau, di.seeds, di.request_ids, di.pos_base)
    assert g["status"] == 0 and (r["status"] == 0).all()
    ties = compare_draft(g, r, di.tau)
    print("draft ties:", ties)


def test_bad_rows_are_flagged_per_request():
    import paper_2607_25852_gb300 as spec
    x, seeds, rids, pos = _case(5, 3, 1000, "bf16", 13)
    x[0, 1, 17] = float("nan")
    x[1, 2] = float("-inf")
    x[2, 0, 5] = float("inf")
    pos[3] = 2**32 - 3
    g = run_draft(x, 1.0, seeds, rids, pos)
    r = run_oracle_draft(x, 1.0, seeds, rids, pos)
    assert g["status"] == spec.ERR_BAD_INPUT
    assert r["status"].tolist() == [oracle.ERR_BAD_INPUT] * 4 + [0]
    compare_draft(g, r, 1.0)


def test_replay_and_workspace_reuse_are_bit_identical():
    x, seeds, rids, pos = _case(8, 6, 20000, "bf16", 14)
    a = run_draft(x, 0.9, seeds, rids, pos)
    b = run_draft(x, 0.9, seeds, rids, pos, ws=a["ws"])
    c = run_draft(x, 0.9, seeds, rids, pos, ws=a["ws"])
    for k in ("z", "c", "s", "st"):
        assert np.array_equal(a[k], b[k]) and np.array_equal(b[k], c[k]), k


def test_drafts_follow_q_on_the_gpu():
    """4096 requests x 4 rows over the same 8-entry row: the drafts' histogram
    against q (chi-square), drawn by the kernel."""
    B, K, V, tau = 4096, 4, 8, 0.8
    row = torch.tensor([1.5, -0.3, 0.0, 2.2, -1.0, 0.7, 1.1, -2.0])
    x = row.expand(B, K, V).contiguous()
    g = run_draft(x, tau, torch.full((B,), 3, dtype=torch.int64), torch.arange(B, dtype=torch.int64),
                  torch.full((B,), 9, dtype=torch.int64))
    q = torch.softmax(row.double() / tau, 0).numpy()
    counts = np.bincount(g["z"].ravel(), minlength=V)
    n = B * K
    chi2 = ((counts - n * q) ** 2 / (n * q)).sum()
    assert stats.chi2.sf(chi2, V - 1) > 1e-3


def test_draft_to_allocation():
    """The drafter's confidences feed spec_allocate as they are: the GPU and
    oracle allocations of the same confidences agree bit for bit."""
    from test_gpu_allocate_commit import assert_alloc_equal, gpu_allocate
    di = workloads.make_draft(B=32, K=8, V=4096)
    g = run_draft(di.logits, di.tau, di.seeds, di.request_ids, di.pos_base)
    conf = torch.as_tensor(g["c"])
    Ts, costs = workloads.budget_candidates(32, 8, sweep=(32, 288, 32))
    ga = gpu_allocate(conf, Ts, costs)
    ra = oracle.allocate(g["c"], Ts, costs)
    assert_alloc_equal(ga, ra)
