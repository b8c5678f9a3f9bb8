"""GPU parity of spec_verify against the CPU oracle (Section 1 rejection
sampling; Section 4.2 deterministic-draft protocol; temperature 0 prefix)."""
import numpy as np
import pytest
import torch

import workloads
from parity import compare, run_oracle, run_verify

pytestmark = pytest.mark.gpu


def _check(wl, t, q="default", depth=None, row_offsets=None, logits=None):
    q = wl.q if q == "default" else q
    logits = wl.logits if logits is None else logits
    gpu = run_verify(logits, wl.drafts, q, wl.B, wl.K, wl.V, t, wl.seeds, wl.request_ids,
                     wl.pos_base, row_offsets=row_offsets, depth=depth)
    ref = run_oracle(logits, wl.drafts, q, t, wl.seeds, wl.request_ids, wl.pos_base,
                     row_offsets=row_offsets, depth=depth)
    assert gpu["status"] == 0 and (ref["status"] == 0).all()
    ties = compare(gpu, ref, wl.K, t, depth=None if depth is None else depth.cpu().numpy(),
                   row_offsets=None if row_offsets is None else row_offsets.cpu().numpy())
    return gpu, ref, ties


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_tiny_workload(t):
    wl = workloads.make("tiny")
    _check(wl, t)


def _random_case(V, dtype, t, qmode, B=3, K=3, seed=0):
    g = torch.Generator().manual_seed(seed * 1000 + V)
    rng = np.random.default_rng(seed * 1000 + V)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    base = torch.randn((B * (K + 1), V), generator=g) * 2.0
    logits = base.to(dt)
    q = None
    if qmode == "dense":
        noisy = base.view(B, K + 1, V)[:, :K] + torch.randn((B, K, V), generator=g) * 0.8
        qf = torch.softmax(noisy, -1)
        q = qf.to(dt)
        drafts = torch.multinomial(q.float().view(B * K, V) + 1e-12, 1, generator=g).view(B, K)
    else:
        amax = logits.float().view(B, K + 1, V)[:, :K].argmax(-1)
        drafts = torch.where(torch.as_tensor(rng.random((B, K)) < 0.6), amax,
                             torch.as_tensor(rng.integers(0, V, (B, K))))
    wl = workloads.Workload(
        name="random", B=B, K=K, V=V, H=8, dtype=dtype, temperature=t, logits=logits,
        drafts=drafts.to(torch.int32), q=q, seeds=torch.as_tensor(rng.integers(0, 2**62, B)),
        request_ids=torch.as_tensor(rng.integers(0, 2**62, B)),
        pos_base=torch.as_tensor(rng.integers(0, 2**31, B)), last_tokens=torch.zeros(B, dtype=torch.int32),
        hidden=None)
    return wl


@pytest.mark.parametrize("V", [1, 2, 7, 33, 4097, 8191, 12345])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("t", [0.0, 0.7])
@pytest.mark.parametrize("qmode", ["onehot", "dense"])
def test_ragged_shapes(V, dtype, t, qmode):
    wl = _random_case(V, dtype, t, qmode)
    _check(wl, t)


@pytest.mark.parametrize("t", [0.05, 3.0, 25.0])
def test_temperature_extremes(t):
    wl = _random_case(5000, "bf16", t, "dense", B=6, K=4, seed=3)
    _check(wl, t)


def test_greedy_workload_full_size():
    wl = workloads.make("greedy", with_hidden=False)
    gpu, ref, _ = _check(wl, 0.0)
    # planted peaks make the acceptance pattern known: a_i equals the run of hits
    hit = wl.extra["planted_hit"]
    run = np.array([np.argmin(np.append(h, False)) for h in hit])
    assert gpu["accepted"].tolist() == run.tolist()


def test_sampled_workload_full_size():
    wl = workloads.make("sampled", with_hidden=False)
    _check(wl, wl.temperature)


def test_stress_workload_full_size():
    wl = workloads.make("stress", with_hidden=False)
    gpu, ref, ties = _check(wl, wl.temperature)
    print("stress ties (accept, race, positions):", ties)


@pytest.mark.parametrize("V", [32768, 65536, 131072])
def test_stress_vocab_sweep(V):
    wl = workloads.make("stress", V=V, B=16, with_hidden=False)
    _check(wl, wl.temperature)


@pytest.mark.parametrize("t", [0.0, 1.0])
@pytest.mark.parametrize("qmode", ["onehot", "dense"])
def test_packed_depths_and_offsets(t, qmode):
    wl = _random_case(3001, "bf16", t, qmode, B=9, K=6, seed=5)
    rng = np.random.default_rng(9)
    depth = torch.as_tensor(rng.integers(0, wl.K + 1, wl.B), dtype=torch.int32)
    depth[0] = 0
    depth[1] = wl.K
    offs = torch.as_tensor(np.concatenate([[0], np.cumsum(depth.numpy() + 1)]), dtype=torch.int32)
    packed = workloads.pack_rows(wl.logits, wl.B, wl.K, depth)
    _check(wl, t, depth=depth, row_offsets=offs, logits=packed)
    # depth without offsets: rows stay at i*(K+1)
    _check(wl, t, depth=depth)


def test_no_drafts_samples_bonus_only():
    wl = _random_case(777, "f32", 1.0, "onehot", B=5, K=0, seed=6)
    gpu, ref, _ = _check(wl, 1.0)
    assert (gpu["accepted"] == 0).all()


def test_bad_inputs_are_flagged_per_request():
    import paper_2607_25852_gb300 as spec
    wl = _random_case(1000, "bf16", 1.0, "onehot", B=6, K=3, seed=7)
    logits = wl.logits.clone()
    drafts = wl.drafts.clone()
    depth = torch.full((wl.B,), wl.K, dtype=torch.int32)
    pos = wl.pos_base.clone()
    logits[0 * 4 + 1, 17] = float("nan")          # request 0: NaN logit
    drafts[1, 2] = wl.V                           # request 1: draft id out of range
    depth[2] = wl.K + 1                           # request 2: depth out of range
    pos[3] = 2**32 - 2                            # request 3: position overflow
    logits[4 * 4 + 0] = float("-inf")             # request 4: row without a finite logit
    gpu = run_verify(logits, drafts, None, wl.B, wl.K, wl.V, 1.0, wl.seeds, wl.request_ids, pos,
                     depth=depth)
    ref = run_oracle(logits, drafts, None, 1.0, wl.seeds, wl.request_ids, pos, depth=depth)
    assert gpu["status"] == spec.ERR_BAD_INPUT
    assert ref["status"][:5].tolist() == [spec.ERR_BAD_INPUT] * 5 and ref["status"][5] == 0
    for i in range(5):
        assert gpu["accepted"][i] == 0 and (gpu["tokens"][i] == -1).all()
    assert gpu["tokens"][5].tolist() == ref["tokens"][5].tolist()


def test_inconsistent_offsets_are_flagged():
    import paper_2607_25852_gb300 as spec
    wl = _random_case(500, "f32", 0.0, "onehot", B=4, K=2, seed=8)
    depth = torch.tensor([2, 1, 0, 2], dtype=torch.int32)
    offs = torch.tensor([0, 3, 4, 5, 8], dtype=torch.int32)     # request 1 spans 1 row, depth says 2
    packed = workloads.pack_rows(wl.logits, wl.B, wl.K, [2, 0, 0, 2])
    gpu = run_verify(packed, wl.drafts, None, wl.B, wl.K, wl.V, 0.0, wl.seeds, wl.request_ids,
                     wl.pos_base, row_offsets=offs, depth=depth)
    assert gpu["status"] == spec.ERR_BAD_INPUT
    assert gpu["accepted"][1] == 0 and (gpu["tokens"][1] == -1).all()


def test_replay_and_workspace_reuse_are_bit_identical():
    wl = _random_case(20000, "bf16", 0.9, "dense", B=8, K=5, seed=10)
    a = run_verify(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.9, wl.seeds, wl.request_ids,
                   wl.pos_base)
    b = run_verify(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.9, wl.seeds, wl.request_ids,
                   wl.pos_base, ws=a["ws"])
    c = run_verify(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.9, wl.seeds, wl.request_ids,
                   wl.pos_base, ws=a["ws"])
    for k in ("accepted", "tokens", "p_draft", "row_stats"):
        assert np.array_equal(a[k], b[k]) and np.array_equal(b[k], c[k]), k


def test_argument_errors_raise():
    import paper_2607_25852_gb300 as spec
    wl = _random_case(100, "f32", 1.0, "onehot", B=2, K=2, seed=11)
    small = torch.zeros(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(spec.SpecError) as e:
        run_verify(wl.logits, wl.drafts, None, wl.B, wl.K, wl.V, 1.0, wl.seeds, wl.request_ids,
                   wl.pos_base, ws=small)
    assert e.value.code == spec.ERR_WORKSPACE
    for t in (-1.0, float("nan"), float("inf")):
        with pytest.raises(spec.SpecError) as e:
            run_verify(wl.logits, wl.drafts, None, wl.B, wl.K, wl.V, t, wl.seeds, wl.request_ids,
                       wl.pos_base)
        assert e.value.code == spec.ERR_INVALID_ARG


@pytest.mark.parametrize("t", [0.0, 1.0])
@pytest.mark.parametrize("qmode", ["onehot", "dense"])
def test_most_drafts_per_request(t, qmode):
    """K = SPEC_MAX_DRAFTS = 255: the decision's per-lane loops over 256 rows."""
    wl = _random_case(600, "bf16", t, qmode, B=2, K=255, seed=5)
    _check(wl, t)


def test_many_requests():
    """B = 512, K = 15: 8192 rows, the most the allocator takes; one chunk per row."""
    wl = _random_case(2048, "bf16", 1.0, "dense", B=512, K=15, seed=6)
    _check(wl, 1.0)


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_misaligned_logits_and_q(t):
    """Row bases 2 bytes off a 16-byte boundary: the streaming pass takes its
    scalar head and tail, the sampling pass its scalar loads."""
    wl = _random_case(4096, "bf16", t, "dense", B=4, K=5, seed=7)
    dev = torch.device("cuda")

    def shifted(x):
        buf = torch.empty(x.numel() + 1, dtype=x.dtype, device=dev)
        view = buf[1:].view(x.shape)
        view.copy_(x.to(dev))
        assert view.data_ptr() % 16 == 2
        return view

    logits, q = shifted(wl.logits), shifted(wl.q)
    gpu = run_verify(logits, wl.drafts, q, wl.B, wl.K, wl.V, t, wl.seeds, wl.request_ids, wl.pos_base)
    ref = run_oracle(wl.logits, wl.drafts, wl.q, t, wl.seeds, wl.request_ids, wl.pos_base)
    assert gpu["status"] == 0 and (ref["status"] == 0).all()
    compare(gpu, ref, wl.K, t)
