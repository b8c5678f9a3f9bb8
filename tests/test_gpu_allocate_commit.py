"""GPU parity of spec_allocate (D-cut, Section 4.2) and spec_commit against
the CPU oracle, and the allocate -> verify -> commit round on the alloc
workload (half chat-like, half code-like requests)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_25852_gb300 as spec
import workloads
from parity import bits, compare, run_oracle, run_verify

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


def gpu_allocate(conf, cand_T, cand_cost, last=None, drafts=None, pos=None):
    B, K = conf.shape
    N = B * (K + 1)
    last = torch.zeros(B, dtype=torch.int32) if last is None else last
    drafts = torch.zeros((B, K), dtype=torch.int32) if drafts is None else drafts
    pos = torch.zeros(B, dtype=torch.int64) if pos is None else pos
    out = dict(depth=torch.full((B,), -9, dtype=torch.int32, device=DEV),
               row_offsets=torch.full((B + 1,), -9, dtype=torch.int32, device=DEV),
               packed_tokens=torch.full((N,), -9, dtype=torch.int32, device=DEV),
               packed_pos=torch.full((N,), -9, dtype=torch.int64, device=DEV),
               chosen_T=torch.zeros(1, dtype=torch.int32, device=DEV),
               utility=torch.zeros(len(cand_T), dtype=torch.float64, device=DEV),
               status=torch.zeros(1, dtype=torch.int32, device=DEV))
    spec.spec_allocate(conf.to(DEV).contiguous(), cand_T, cand_cost, last.to(DEV), drafts.to(DEV),
                       pos.to(DEV), out["depth"], out["row_offsets"], out["packed_tokens"],
                       out["packed_pos"], out["chosen_T"], out["utility"], out["status"])
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def assert_alloc_equal(g, r):
    assert g["depth"].tolist() == r["depth"].tolist()
    assert g["row_offsets"].tolist() == r["row_offsets"].tolist()
    assert g["packed_tokens"].tolist() == r["packed_tokens"].tolist()
    assert g["packed_pos"].tolist() == r["packed_pos"].tolist()
    assert int(g["chosen_T"][0]) == r["chosen_T"]
    assert np.array_equal(g["utility"], r["utility"])


def test_alloc_workload_sweep_and_ratios():
    wl = workloads.make("alloc", V=256, with_hidden=False)
    B, K = wl.B, wl.K
    args = (wl.last_tokens, wl.drafts, wl.pos_base)
    Ts, costs = workloads.budget_candidates(B, K)
    for c in range(len(Ts)):                          # each fixed budget
        g = gpu_allocate(wl.conf, [Ts[c]], [costs[c]], *args)
        r = oracle.allocate(wl.conf.numpy(), [Ts[c]], [costs[c]], *[a.numpy() for a in args])
        assert_alloc_equal(g, r)
    g = gpu_allocate(wl.conf, Ts, costs, *args)       # argmax over the 16 candidates
    r = oracle.allocate(wl.conf.numpy(), Ts, costs, *[a.numpy() for a in args])
    assert_alloc_equal(g, r)
    ratios = spec.spec_budget_from_ratios(B, K, [1, 1, 3, 1], [4, 2, 4, 1])
    assert ratios == [272, 544, 816, 1088]
    g = gpu_allocate(wl.conf, ratios, [1.0 + 0.004 * max(0, T - 256) for T in ratios], *args)
    r = oracle.allocate(wl.conf.numpy(), ratios, [1.0 + 0.004 * max(0, T - 256) for T in ratios],
                        *[a.numpy() for a in args])
    assert_alloc_equal(g, r)
    # code-like requests (Beta(8,1)) keep deeper prefixes than chat-like (Beta(2,2))
    assert g["depth"][B // 2:].mean() > g["depth"][:B // 2].mean()


# The one-CTA kernel's paths: padded runs merged (B * KP <= 1024, KP the next
# power of two >= K: (7, 7), (64, 16), (32, 17), (4, 255) and (3, 200) with
# two merge levels, (1024, 1) and (1000, 1) with ten, pad runs past B), the
# bitonic network when the padded runs do not fit ((33, 17), (100, 10)); and
# the large kernel ((512, 15), (8192, 0)).
@pytest.mark.parametrize("B,K", [(1, 0), (1, 5), (3, 4), (7, 7), (64, 16), (32, 17), (4, 255), (3, 200),
                                 (1024, 1), (1000, 1), (33, 17), (100, 10), (512, 15), (8192, 0)])
def test_random_allocations(B, K):
    rng = np.random.default_rng(B * 100 + K)
    for trial in range(3):
        if trial == 0:
            conf = rng.choice([0.0, 0.5, 1.0], size=(B, K)).astype(np.float32)
        else:
            conf = rng.uniform(size=(B, K)).astype(np.float32)
        N = B * (K + 1)
        Ts = sorted(set(int(x) for x in rng.integers(B, N + 1, size=min(12, N - B + 1))) | {B, N})
        costs = list(rng.uniform(0.5, 3.0, len(Ts)))
        last = torch.as_tensor(rng.integers(0, 10**6, B), dtype=torch.int32)
        drafts = torch.as_tensor(rng.integers(0, 10**6, (B, K)), dtype=torch.int32)
        pos = torch.as_tensor(rng.integers(0, 10**9, B), dtype=torch.int64)
        g = gpu_allocate(torch.as_tensor(conf), Ts, costs, last, drafts, pos)
        r = oracle.allocate(conf, Ts, costs, last.numpy(), drafts.numpy(), pos.numpy())
        assert_alloc_equal(g, r)


@pytest.mark.parametrize("B,K", [(4, 3), (64, 16), (300, 7)])
def test_negative_zero_confidences(B, K):
    """-0 confidences (the value 0, sign bit set) rank as zero scores: the
    allocation is bit-exact with the oracle at T = B, T = B(K+1) and random
    budgets, and no depth is ever negative."""
    rng = np.random.default_rng(B + K)
    conf = rng.uniform(size=(B, K)).astype(np.float32)
    mask = rng.random((B, K)) < 0.3
    conf[mask] = np.float32(-0.0)
    conf[0, :] = np.float32(-0.0)
    assert np.signbit(conf[0, 0])
    N = B * (K + 1)
    Ts = sorted(set(int(x) for x in rng.integers(B, N + 1, size=6)) | {B, N})
    costs = list(rng.uniform(0.5, 3.0, len(Ts)))
    for cand in [[B], [N], Ts]:
        cc = costs[:len(cand)] if cand is Ts else [1.0]
        g = gpu_allocate(torch.as_tensor(conf), cand, cc)
        r = oracle.allocate(conf, cand, cc)
        assert int(g["status"][0]) == 0 and r["status"] == 0
        assert_alloc_equal(g, r)
        assert (g["depth"] >= 0).all()


def test_sixty_four_candidates():
    """The most candidates a call takes (SPEC_MAX_CANDIDATES), with tied scores."""
    rng = np.random.default_rng(64)
    B, K = 256, 15
    N = B * (K + 1)
    conf = rng.choice([0.25, 0.5, 0.75, 1.0], size=(B, K)).astype(np.float32)
    Ts = sorted(int(x) for x in rng.choice(np.arange(B, N + 1), size=64, replace=False))
    costs = list(rng.uniform(0.5, 3.0, 64))
    g = gpu_allocate(torch.as_tensor(conf), Ts, costs)
    r = oracle.allocate(conf, Ts, costs)
    assert_alloc_equal(g, r)


def test_invalid_confidence_is_flagged():
    conf = torch.full((4, 3), 0.7)
    conf[2, 1] = float("nan")
    conf[3, 0] = 1.5
    g = gpu_allocate(conf, [4, 9, 16], [1.0, 1.0, 1.0])
    r = oracle.allocate(conf.numpy(), [4, 9, 16], [1.0, 1.0, 1.0])
    assert int(g["status"][0]) == spec.ERR_BAD_INPUT and r["status"] == oracle.ERR_BAD_INPUT
    assert_alloc_equal(g, r)


def test_allocate_argument_errors():
    conf = torch.full((2, 2), 0.5)
    for Ts, costs in (([1], [1.0]), ([7], [1.0]), ([4], [0.0]), ([4], [float("inf")])):
        with pytest.raises(spec.SpecError) as e:
            gpu_allocate(conf, Ts, costs)
        assert e.value.code == spec.ERR_INVALID_ARG
    with pytest.raises(spec.SpecError):
        gpu_allocate(torch.zeros((8193, 0)), [8193], [1.0])     # beyond one-CTA capacity


def run_commit(acc, tok, hidden, B, K, row_offsets=None):
    ptok = torch.full((B * (K + 1),), -9, dtype=torch.int32, device=DEV)
    coff = torch.full((B + 1,), -9, dtype=torch.int32, device=DEV)
    hout = None if hidden is None else torch.zeros((B * (K + 1), hidden.shape[1]), dtype=hidden.dtype,
                                                   device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    spec.spec_commit(acc.to(DEV), tok.to(DEV), None if hidden is None else hidden.to(DEV), B, K, ptok,
                     coff, hout, row_offsets=None if row_offsets is None else row_offsets.to(DEV),
                     status=status)
    torch.cuda.synchronize()
    return ptok.cpu(), coff.cpu(), None if hout is None else hout.cpu(), int(status.item())


@pytest.mark.parametrize("B,K,H,dtype,packed", [(5, 4, 64, torch.bfloat16, False),
                                                 (9, 6, 33, torch.bfloat16, True),
                                                 (3, 2, 7, torch.float32, True),
                                                 (300, 3, 40, torch.bfloat16, True),
                                                 (2000, 1, 8, torch.float32, False)])
def test_commit_matches_oracle(B, K, H, dtype, packed):
    rng = np.random.default_rng(B + K + H)
    depth = rng.integers(0, K + 1, B) if packed else np.full(B, K)
    offs = np.concatenate([[0], np.cumsum(depth + 1)]).astype(np.int32)
    R = int(offs[-1])
    acc = np.array([rng.integers(0, d + 1) for d in depth], np.int32)
    tok = np.full((B, K + 1), -1, np.int32)
    for i in range(B):
        tok[i, :acc[i] + 1] = rng.integers(0, 10**5, acc[i] + 1)
    hidden = torch.randn((R, H)).to(dtype)
    ptok, coff, hout, st = run_commit(torch.as_tensor(acc), torch.as_tensor(tok), hidden, B, K,
                                      torch.as_tensor(offs) if packed else None)
    r = oracle.commit(acc, tok, offs, bits(hidden))
    assert st == 0
    assert coff.tolist() == r["commit_offsets"].tolist()
    assert ptok[:r["total"]].tolist() == r["packed_tokens"][:r["total"]].tolist()
    assert np.array_equal(bits(hout[:r["total"]]), r["hidden"])


def test_commit_flags_out_of_range_lengths():
    B, K = 4, 3
    acc = torch.tensor([1, 7, 0, -2], dtype=torch.int32)
    tok = torch.arange(B * (K + 1), dtype=torch.int32).view(B, K + 1)
    ptok, coff, _, st = run_commit(acc, tok, None, B, K)
    assert st == spec.ERR_BAD_INPUT
    assert coff.tolist() == [0, 2, 3, 4, 5]


def test_alloc_verify_commit_round():
    """The full round on the alloc workload: D-cut picks T*, the target rows of
    the kept prefixes are packed, verified at t = 1 (one-hot q), committed."""
    wl = workloads.make("alloc", V=8192, H=128)
    B, K = wl.B, wl.K
    Ts, costs = workloads.budget_candidates(B, K)
    g = gpu_allocate(wl.conf, Ts, costs, wl.last_tokens, wl.drafts, wl.pos_base)
    depth = torch.as_tensor(g["depth"])
    offs = torch.as_tensor(g["row_offsets"])
    logits = workloads.pack_rows(wl.logits, B, K, depth)
    hidden = workloads.pack_rows(wl.hidden, B, K, depth)
    gpu = run_verify(logits, wl.drafts, None, B, K, wl.V, 1.0, wl.seeds, wl.request_ids, wl.pos_base,
                     row_offsets=offs, depth=depth)
    ref = run_oracle(logits, wl.drafts, None, 1.0, wl.seeds, wl.request_ids, wl.pos_base,
                     row_offsets=offs, depth=depth)
    compare(gpu, ref, K, 1.0, depth=depth.numpy(), row_offsets=offs.numpy())
    ptok, coff, hout, st = run_commit(torch.as_tensor(gpu["accepted"]), torch.as_tensor(gpu["tokens"]),
                                      hidden, B, K, offs)
    r = oracle.commit(gpu["accepted"], gpu["tokens"], offs.numpy(), bits(hidden))
    assert st == 0 and coff.tolist() == r["commit_offsets"].tolist()
    assert np.array_equal(bits(hout[:r["total"]]), r["hidden"])
