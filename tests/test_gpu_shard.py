"""GPU parity of the vocabulary-sharded verification (spec_shard_stats /
decide / sample / finish) against the CPU oracle, and against spec_verify bit
for bit at temperature 0.  Shards of one GPU stand for tensor-parallel ranks
(the paper serves its target with TP = 8, Section 4.4); their records are
written side by side in place of the all-gathers."""
import numpy as np
import pytest
import torch

import workloads
from parity import compare, run_oracle, run_sharded, run_verify, shard_bounds
from test_gpu_verify import _random_case

pytestmark = pytest.mark.gpu


def _check(wl, t, bounds, q="default", depth=None, row_offsets=None, logits=None):
    q = wl.q if q == "default" else q
    logits = wl.logits if logits is None else logits
    gpu = run_sharded(logits, wl.drafts, q, wl.B, wl.K, wl.V, t, wl.seeds, wl.request_ids,
                      wl.pos_base, bounds, row_offsets=row_offsets, depth=depth)
    ref = run_oracle(logits, wl.drafts, q, t, wl.seeds, wl.request_ids, wl.pos_base,
                     row_offsets=row_offsets, depth=depth)
    assert gpu["status"] == 0 and (ref["status"] == 0).all()
    ties = compare(gpu, ref, wl.K, t, depth=None if depth is None else depth.cpu().numpy(),
                   row_offsets=None if row_offsets is None else row_offsets.cpu().numpy())
    return gpu, ref, ties


def _same_as_unsharded(wl, gpu, q="default", depth=None, row_offsets=None, logits=None):
    q = wl.q if q == "default" else q
    logits = wl.logits if logits is None else logits
    one = run_verify(logits, wl.drafts, q, wl.B, wl.K, wl.V, 0.0, wl.seeds, wl.request_ids,
                     wl.pos_base, row_offsets=row_offsets, depth=depth)
    for k in ("accepted", "tokens", "p_draft", "row_stats"):
        assert np.array_equal(gpu[k], one[k]), k


# shard layouts of V = 12345: one shard; 1024-aligned cuts; cuts inside race
# blocks (256 entries) and off the 8-entry grid; eight ranks of V // 8
LAYOUTS = {
    "one": lambda V: [0, V],
    "aligned3": lambda V: shard_bounds(V, 3, 1024),
    "ragged3": lambda V: [0, 4000, 4001 + 300, V],
    "tp8": lambda V: shard_bounds(V, 8),
}


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("qmode", ["onehot", "dense"])
def test_greedy_matches_unsharded_bit_for_bit(layout, dtype, qmode):
    wl = _random_case(12345, dtype, 0.0, qmode, B=5, K=4, seed=21)
    gpu, _, _ = _check(wl, 0.0, LAYOUTS[layout](wl.V))
    _same_as_unsharded(wl, gpu)


@pytest.mark.parametrize("layout", sorted(LAYOUTS))
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("qmode", ["onehot", "dense"])
def test_sampled_matches_oracle(layout, dtype, qmode):
    wl = _random_case(12345, dtype, 0.7, qmode, B=6, K=4, seed=22)
    _check(wl, 0.7, LAYOUTS[layout](wl.V))


@pytest.mark.parametrize("t", [0.0, 0.7])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_more_rows_than_one_wave_of_wide_stats_ctas(t, dtype):
    """Past four stats CTAs per SM (one CTA per row here: K = 3, B = SMs + 8,
    V_s < 16384), spec_shard_stats streams with 128-thread CTAs instead of
    256-thread ones; the result does not depend on which."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    wl = _random_case(12345, dtype, t, "dense", B=sms + 8, K=3, seed=24)
    gpu, _, _ = _check(wl, t, LAYOUTS["ragged3"](wl.V))
    if t == 0.0:
        _same_as_unsharded(wl, gpu)


@pytest.mark.parametrize("t", [0.0, 0.7])
@pytest.mark.parametrize("narrow", [False, True])
def test_stats_rows_with_a_short_last_round(t, narrow):
    """Shard rows whose 16-byte vectors run past whole load rounds by at most
    one per thread (2048 + 100 vectors with 256-thread stats CTAs, 1024 + 50
    with 128-thread ones): the remainder is loaded with the first round.
    Logits rounded to integers tie the maximum in many places; at t = 0 the
    lowest index must still win."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    B, K = (sms + 8, 3) if narrow else (5, 4)
    Vs = 8 * (1024 + 50) if narrow else 8 * (2048 + 100)
    wl = _random_case(Vs + 3000, "bf16", t, "dense", B=B, K=K, seed=25)
    wl.logits = wl.logits.float().round().to(wl.logits.dtype)
    gpu, _, _ = _check(wl, t, [0, Vs, wl.V])
    if t == 0.0:
        _same_as_unsharded(wl, gpu)


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_shards_inside_one_race_block(t):
    """V = 1000 (four race blocks, the last one partial): a shard that lies
    inside block 1, shards cut blocks 1 and 2, and a one-column shard.  With
    32 requests the draw lands in the cut blocks many times."""
    bounds = [0, 300, 350, 351, 700, 1000]
    for qmode in ("onehot", "dense"):
        wl = _random_case(1000, "bf16", t, qmode, B=32, K=3, seed=23)
        # flatter rows so that every block carries mass
        wl.logits = (wl.logits.float() * 0.25).to(wl.logits.dtype)
        gpu, ref, _ = _check(wl, t, bounds)
        if t == 0.0:
            _same_as_unsharded(wl, gpu)
        else:
            picked = np.array([gpu["tokens"][i, gpu["accepted"][i]] for i in range(wl.B)])
            assert ((picked >= 256) & (picked < 768)).any()


def test_empty_residual_falls_back_to_p():
    """A rejected draft with p <= q everywhere: the residual is empty and the
    token is drawn from p, here the one column that p and q both put all
    their mass on (Section 1; the p fallback of the verification rule)."""
    B, K, V = 4, 2, 3000
    g = torch.Generator().manual_seed(24)
    logits = torch.randn((B * (K + 1), V), generator=g) * 2.0
    q = torch.softmax(torch.randn((B, K, V), generator=g), -1)
    drafts = torch.randint(0, V, (B, K), generator=g, dtype=torch.int32)
    peaks = [5, 1500, 2100, 2999]
    for i, v in enumerate(peaks):
        logits[i * (K + 1)] = -1e4               # row 0: p is one-hot at v ...
        logits[i * (K + 1), v] = 0.0
        q[i, 0] = 0.0                            # ... and so is q
        q[i, 0, v] = 1.0
        drafts[i, 0] = (v + 7) % V               # a draft with p = q = 0: rejected
    wl = workloads.Workload(
        name="fallback", B=B, K=K, V=V, H=8, dtype="f32", temperature=1.0, logits=logits,
        drafts=drafts, q=q, seeds=torch.arange(B, dtype=torch.int64) + 5,
        request_ids=torch.arange(B, dtype=torch.int64), pos_base=torch.full((B,), 100, dtype=torch.int64),
        last_tokens=torch.zeros(B, dtype=torch.int32), hidden=None)
    ref = run_oracle(wl.logits, wl.drafts, wl.q, 1.0, wl.seeds, wl.request_ids, wl.pos_base)
    assert ref["accepted"].tolist() == [0] * B and ref["tokens"][:, 0].tolist() == peaks
    one = run_verify(wl.logits, wl.drafts, wl.q, B, K, V, 1.0, wl.seeds, wl.request_ids, wl.pos_base)
    assert one["tokens"][:, 0].tolist() == peaks
    for bounds in ([0, V], [0, 1000, 1700, V], shard_bounds(V, 8)):
        gpu, _, _ = _check(wl, 1.0, bounds)
        assert gpu["tokens"][:, 0].tolist() == peaks


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_packed_depths(t):
    wl = _random_case(3001, "bf16", t, "dense", B=9, K=6, seed=25)
    rng = np.random.default_rng(25)
    depth = torch.as_tensor(rng.integers(0, wl.K + 1, wl.B), dtype=torch.int32)
    depth[0], depth[1] = 0, wl.K
    offs = torch.as_tensor(np.concatenate([[0], np.cumsum(depth.numpy() + 1)]), dtype=torch.int32)
    packed = workloads.pack_rows(wl.logits, wl.B, wl.K, depth)
    bounds = [0, 999, 2048, 3001]
    gpu, _, _ = _check(wl, t, bounds, depth=depth, row_offsets=offs, logits=packed)
    if t == 0.0:
        _same_as_unsharded(wl, gpu, depth=depth, row_offsets=offs, logits=packed)


def test_bad_inputs_are_flagged_per_request():
    import paper_2607_25852_gb300 as spec
    wl = _random_case(1000, "bf16", 1.0, "onehot", B=6, K=3, seed=26)
    logits = wl.logits.clone()
    drafts = wl.drafts.clone()
    depth = torch.full((wl.B,), wl.K, dtype=torch.int32)
    pos = wl.pos_base.clone()
    logits[0 * 4 + 1, 17] = float("nan")          # request 0: NaN logit
    drafts[1, 2] = wl.V                           # request 1: draft id out of range
    depth[2] = wl.K + 1                           # request 2: depth out of range
    pos[3] = 2**32 - 2                            # request 3: position overflow
    logits[4 * 4 + 0] = float("-inf")             # request 4: row without a finite logit
    gpu = run_sharded(logits, drafts, None, wl.B, wl.K, wl.V, 1.0, wl.seeds, wl.request_ids, pos,
                      [0, 333, 1000], depth=depth)
    ref = run_oracle(logits, drafts, None, 1.0, wl.seeds, wl.request_ids, pos, depth=depth)
    assert gpu["status"] == spec.ERR_BAD_INPUT
    for i in range(5):
        assert gpu["accepted"][i] == 0 and (gpu["tokens"][i] == -1).all()
    assert gpu["tokens"][5].tolist() == ref["tokens"][5].tolist()


def test_uncovered_draft_column_is_flagged():
    """Shards that leave a draft's column uncovered (called through the C ABI
    directly: ShardedRound refuses such bounds): the request is flagged."""
    import paper_2607_25852_gb300 as spec
    wl = _random_case(2048, "f32", 1.0, "onehot", B=3, K=2, seed=27)
    wl.drafts[1, 0] = 2047
    B, K, V = wl.B, wl.K, wl.V
    dev = torch.device("cuda")
    d = lambda x: x.to(dev).contiguous()
    bounds = [0, 1024, 2047]
    R = B * (K + 1)
    stats = torch.zeros(2 * R * spec.SHARD_STAT_BYTES, dtype=torch.uint8, device=dev)
    races = torch.zeros(2 * B * spec.SHARD_RACE_BYTES, dtype=torch.uint8, device=dev)
    dec = torch.zeros(B * spec.SHARD_DECISION_BYTES, dtype=torch.uint8, device=dev)
    acc = torch.zeros(B, dtype=torch.int32, device=dev)
    tok = torch.zeros((B, K + 1), dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    dr, sd, ri, pb = d(wl.drafts), d(wl.seeds), d(wl.request_ids), d(wl.pos_base)
    lgs = [d(wl.logits[:, bounds[s]:bounds[s + 1]]) for s in range(2)]
    ws = [spec.shard_workspace(B, K, bounds[s + 1] - bounds[s], dev) for s in range(2)]
    sb, rb = R * spec.SHARD_STAT_BYTES, B * spec.SHARD_RACE_BYTES
    for s in range(2):
        spec.spec_shard_stats(lgs[s], dr, None, B, K, V, bounds[s], 1.0, pb, stats[s * sb:(s + 1) * sb], ws[s],
                              status=status)
    spec.spec_shard_decide(stats, 2, dr, False, B, K, V, 1.0, sd, ri, pb, acc, tok, decisions_out=dec,
                           status=status)
    for s in range(2):
        spec.spec_shard_sample(lgs[s], None, dec, B, K, V, bounds[s], 1.0, sd, ri, races[s * rb:(s + 1) * rb],
                               ws[s], status=status)
    spec.spec_shard_finish(races, 2, dec, B, K, V, 1.0, sd, ri, acc, tok, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == spec.ERR_BAD_INPUT
    assert int(acc[1]) == 0 and (tok[1] == -1).all()


def test_full_size_tp8_stress():
    """B = 64, K = 16, V = 201088 bf16 at t = 1 over eight shards of 25136
    columns, the split of a TP = 8 output layer."""
    wl = workloads.make("stress", with_hidden=False)
    gpu, _, ties = _check(wl, wl.temperature, shard_bounds(wl.V, 8))
    print("tp8 stress ties (accept, race, positions):", ties)


def test_full_size_tp8_greedy():
    wl = workloads.make("greedy", with_hidden=False)
    gpu, _, _ = _check(wl, 0.0, shard_bounds(wl.V, 8))
    _same_as_unsharded(wl, gpu)


def test_replay_and_workspace_reuse_are_bit_identical():
    wl = _random_case(20000, "bf16", 0.9, "dense", B=8, K=5, seed=28)
    bounds = shard_bounds(wl.V, 3)
    a = run_sharded(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.9, wl.seeds, wl.request_ids,
                    wl.pos_base, bounds)
    b = run_sharded(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.9, wl.seeds, wl.request_ids,
                    wl.pos_base, bounds, ws=a["ws"])
    c = run_sharded(wl.logits, wl.drafts, wl.q, wl.B, wl.K, wl.V, 0.9, wl.seeds, wl.request_ids,
                    wl.pos_base, bounds, ws=a["ws"])
    for k in ("accepted", "tokens", "p_draft", "row_stats"):
        assert np.array_equal(a[k], b[k]) and np.array_equal(b[k], c[k]), k
