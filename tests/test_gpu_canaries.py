"""Out-of-bounds writes, caught without a sanitizer: every output buffer and
workspace an entry point writes sits between two guard regions of a known
byte pattern, and the guards must come back untouched.  Each case also checks
that the guarded call gives the same results as the same call on plain
buffers, so a guard that shifted an output would show.

(compute-sanitizer is not available on the GPU pool this library is tested
on; these guards stand in for its out-of-bounds check on the outputs.)
"""
import math

import numpy as np
import pytest
import torch

import paper_2607_25852_gb300 as spec

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")
GUARD = 256      # bytes before and after; keeps the interior 256-byte aligned
PATTERN = 0xA5


class Guarded:
    """A tensor of `shape` and `dtype` between two guard regions."""

    def __init__(self, shape, dtype, fill=0):
        self.shape, self.dtype = tuple(shape), dtype
        self.nbytes = math.prod(self.shape) * torch.empty((), dtype=dtype).element_size()
        self.buf = torch.full((GUARD + self.nbytes + GUARD,), PATTERN, dtype=torch.uint8, device=DEV)
        self.t = self.buf[GUARD:GUARD + self.nbytes].view(dtype).view(self.shape)
        if fill is not None:
            self.t.fill_(fill)

    def intact(self):
        torch.cuda.synchronize()
        head = self.buf[:GUARD].cpu().numpy()
        tail = self.buf[GUARD + self.nbytes:].cpu().numpy()
        return bool((head == PATTERN).all() and (tail == PATTERN).all())


def guarded_workspace(nbytes):
    g = Guarded((nbytes,), torch.uint8, fill=0)  # workspaces start zeroed
    return g


def assert_intact(**bufs):
    bad = [name for name, g in bufs.items() if not g.intact()]
    assert not bad, f"guard bytes overwritten next to {bad}"


def _verify_inputs(B, K, V, t, dense_q, seed):
    g = torch.Generator().manual_seed(seed)
    R = B * (K + 1)
    base = torch.randn((R, V), generator=g) * 2.0
    logits = base.to(torch.bfloat16)
    if dense_q:
        q = torch.softmax(base.view(B, K + 1, V)[:, :K] + torch.randn((B, K, V), generator=g), -1)
        q = q.to(torch.bfloat16)
        drafts = torch.multinomial(q.float().view(B * K, V), 1, generator=g).view(B, K)
    else:
        q = None
        drafts = base.view(B, K + 1, V)[:, :K].argmax(-1)
        drafts[:, K // 2:] = torch.randint(0, V, (B, K - K // 2), generator=g)
    return dict(logits=logits.to(DEV), q=None if q is None else q.to(DEV),
                drafts=drafts.to(torch.int32).to(DEV),
                seeds=torch.arange(B, dtype=torch.int64, device=DEV) * 3 + 1,
                rids=torch.arange(B, dtype=torch.int64, device=DEV) + 50,
                pos=torch.randint(0, 10**6, (B,), generator=g).to(DEV), B=B, K=K, V=V, t=t)


def _verify_outputs(B, K, guarded):
    R = B * (K + 1)
    mk = (lambda s, d: Guarded(s, d, fill=-7 if d == torch.int32 else 0)) if guarded else \
         (lambda s, d: torch.full(s, -7, dtype=d, device=DEV) if d == torch.int32 else torch.zeros(s, dtype=d, device=DEV))
    status = Guarded((1,), torch.int32, fill=0) if guarded else torch.zeros(1, dtype=torch.int32, device=DEV)
    return dict(acc=mk((B,), torch.int32), tok=mk((B, K + 1), torch.int32), pdr=mk((B, K), torch.float32),
                rst=mk((R, 2), torch.float32), status=status)


def _t(x):
    return x.t if isinstance(x, Guarded) else x


@pytest.mark.parametrize("B,K,V,t,dense_q", [(8, 5, 4097, 1.0, True), (6, 3, 8191, 0.0, False),
                                            (64, 16, 33000, 1.0, True), (3, 0, 333, 0.7, False)])
def test_verify_writes_stay_inside_outputs_and_workspace(B, K, V, t, dense_q):
    x = _verify_inputs(B, K, V, t, dense_q, seed=B * 1000 + V)
    res = []
    for guarded in (False, True):
        o = _verify_outputs(B, K, guarded)
        n = spec.spec_verify_workspace(B, K, V)
        ws = guarded_workspace(n) if guarded else torch.zeros(n, dtype=torch.uint8, device=DEV)
        spec.spec_verify(x["logits"], x["drafts"], x["q"], B, K, V, t, x["seeds"], x["rids"], x["pos"],
                         _t(o["acc"]), _t(o["tok"]), _t(ws), p_draft_out=_t(o["pdr"]), row_stats_out=_t(o["rst"]),
                         status=_t(o["status"]))
        torch.cuda.synchronize()
        if guarded:
            assert_intact(ws=ws, **o)
        res.append({k: _t(v).cpu().numpy() for k, v in o.items()})
    for k in res[0]:
        assert np.array_equal(res[0][k], res[1][k]), k
    assert int(res[1]["status"][0]) == 0


def test_verify_static_writes_stay_inside_outputs():
    B, K, V = 16, 7, 12345
    x = _verify_inputs(B, K, V, 1.0, True, seed=7)
    o = _verify_outputs(B, K, True)
    spec.spec_verify_static(x["logits"], x["drafts"], x["q"], B, K, V, 1.0, x["seeds"], x["rids"], x["pos"],
                            o["acc"].t, o["tok"].t, p_draft_out=o["pdr"].t, row_stats_out=o["rst"].t,
                            status=o["status"].t)
    assert_intact(**o)
    assert int(o["status"].t.item()) == 0


@pytest.mark.parametrize("B,K", [(64, 16), (5, 3), (300, 3), (900, 8)])
def test_allocate_writes_stay_inside_outputs(B, K):
    g = torch.Generator().manual_seed(B * 31 + K)
    conf = torch.rand((B, K), generator=g).to(DEV)
    last = torch.randint(0, 1000, (B,), generator=g, dtype=torch.int32).to(DEV)
    drafts = torch.randint(0, 1000, (B, K), generator=g, dtype=torch.int32).to(DEV)
    pos = torch.randint(0, 1000, (B,), generator=g).to(DEV)
    N = B * (K + 1)
    cand = sorted({B, (B + N) // 2, N})
    cost = [1.0 + 0.001 * t for t in cand]
    res = []
    for guarded in (False, True):
        mk = (lambda s, d: Guarded(s, d, fill=0)) if guarded else (lambda s, d: torch.zeros(s, dtype=d, device=DEV))
        o = dict(depth=mk((B,), torch.int32), off=mk((B + 1,), torch.int32), ptok=mk((N,), torch.int32),
                 ppos=mk((N,), torch.int64), chosen=mk((1,), torch.int32), util=mk((len(cand),), torch.float64),
                 status=mk((1,), torch.int32))
        spec.spec_allocate(conf, cand, cost, last, drafts, pos, _t(o["depth"]), _t(o["off"]), _t(o["ptok"]),
                           _t(o["ppos"]), _t(o["chosen"]), _t(o["util"]), _t(o["status"]))
        torch.cuda.synchronize()
        if guarded:
            assert_intact(**o)
        res.append({k: _t(v).cpu().numpy() for k, v in o.items()})
    for k in res[0]:
        assert np.array_equal(res[0][k], res[1][k]), k


def test_commit_writes_stay_inside_the_committed_rows():
    B, K, H = 40, 6, 1000
    g = torch.Generator().manual_seed(5)
    R = B * (K + 1)
    acc = torch.randint(0, K + 1, (B,), generator=g, dtype=torch.int32).to(DEV)
    tok = torch.randint(0, 50000, (B, K + 1), generator=g, dtype=torch.int32).to(DEV)
    hidden = torch.randn((R, H), generator=g).to(torch.bfloat16).to(DEV)
    total = int((acc + 1).sum().item())
    o = dict(ptok=Guarded((total,), torch.int32, fill=-3), coff=Guarded((B + 1,), torch.int32, fill=-3),
             hout=Guarded((total, H), torch.bfloat16, fill=0), status=Guarded((1,), torch.int32, fill=0))
    spec.spec_commit(acc, tok, hidden, B, K, o["ptok"].t, o["coff"].t, o["hout"].t, status=o["status"].t)
    assert_intact(**o)
    a = acc.cpu().numpy()
    off = np.concatenate([[0], np.cumsum(a + 1)])
    assert np.array_equal(o["coff"].t.cpu().numpy(), off)
    rows = np.concatenate([np.arange(i * (K + 1), i * (K + 1) + a[i] + 1) for i in range(B)])
    assert torch.equal(o["hout"].t.cpu(), hidden.cpu()[torch.from_numpy(rows)])


@pytest.mark.parametrize("tau", [1.0, 0.0])
def test_draft_writes_stay_inside_outputs_and_workspace(tau):
    B, K, V = 12, 5, 20001
    g = torch.Generator().manual_seed(11)
    logits = (torch.randn((B, K, V), generator=g) * 2).to(torch.bfloat16).to(DEV)
    seeds = torch.arange(B, dtype=torch.int64, device=DEV) + 9
    rids = seeds * 2
    pos = torch.arange(B, dtype=torch.int64, device=DEV) * 5
    o = dict(z=Guarded((B, K), torch.int32, fill=-1), c=Guarded((B, K), torch.float32),
             s=Guarded((B, K + 1), torch.float32), rst=Guarded((B * K, 2), torch.float32),
             status=Guarded((1,), torch.int32))
    ws = guarded_workspace(spec.spec_draft_workspace(B, K, V))
    spec.spec_draft(logits, tau, seeds, rids, pos, o["z"].t, o["c"].t, ws.t, scores_out=o["s"].t,
                    row_stats_out=o["rst"].t, status=o["status"].t)
    assert_intact(ws=ws, **o)
    assert int(o["status"].t.item()) == 0


def test_markov_draft_writes_stay_inside_outputs_and_workspace():
    B, K, V, r = 16, 3, 5000, 64
    g = torch.Generator(device=DEV)
    g.manual_seed(3)
    U = (torch.randn((B, K, V), generator=g, device=DEV) * 2).to(torch.bfloat16)
    W1 = (torch.randn((V, r), generator=g, device=DEV) * 0.2).to(torch.bfloat16)
    W2T = (torch.randn((V, r), generator=g, device=DEV) * 0.2).to(torch.bfloat16)
    x0 = torch.randint(0, V, (B,), generator=g, device=DEV, dtype=torch.int32)
    seeds = torch.arange(B, dtype=torch.int64, device=DEV)
    o = dict(z=Guarded((B, K), torch.int32, fill=-1), c=Guarded((B, K), torch.float32),
             s=Guarded((B, K + 1), torch.float32), rst=Guarded((B * K, 2), torch.float32),
             status=Guarded((1,), torch.int32))
    ws = guarded_workspace(spec.spec_markov_workspace(B, K, V, r))
    spec.spec_markov_draft(U, W1, W2T, x0, 1.0, seeds, seeds + 1, seeds * 2, o["z"].t, o["c"].t, ws.t,
                           scores_out=o["s"].t, row_stats_out=o["rst"].t, status=o["status"].t)
    assert_intact(ws=ws, **o)
    assert int(o["status"].t.item()) == 0


@pytest.mark.parametrize("t", [1.0, 0.0])
def test_sharded_writes_stay_inside_records_and_workspaces(t):
    from parity import shard_bounds
    B, K, V, S = 8, 4, 9000, 3
    x = _verify_inputs(B, K, V, t, t > 0, seed=21)
    bounds = shard_bounds(V, S)
    R = B * (K + 1)
    stats = Guarded((S * R * 32,), torch.uint8)
    races = Guarded((S * B * 96,), torch.uint8)
    dec = Guarded((B * 32,), torch.uint8)
    o = _verify_outputs(B, K, True)
    shards = []
    for s in range(S):
        lo, hi = bounds[s], bounds[s + 1]
        ws = guarded_workspace(spec.spec_shard_workspace(B, K, hi - lo))
        lg = x["logits"][:, lo:hi].contiguous()
        qs = None if x["q"] is None else x["q"][:, :, lo:hi].contiguous()
        shards.append((lo, lg, qs, ws))
        spec.spec_shard_stats(lg, x["drafts"], qs, B, K, V, lo, t, x["pos"],
                              stats.t[s * R * 32:(s + 1) * R * 32], ws.t, status=o["status"].t)
    spec.spec_shard_decide(stats.t, S, x["drafts"], x["q"] is not None, B, K, V, t, x["seeds"], x["rids"], x["pos"],
                           o["acc"].t, o["tok"].t, decisions_out=dec.t, p_draft_out=o["pdr"].t,
                           row_stats_out=o["rst"].t, status=o["status"].t)
    if t > 0:
        for s, (lo, lg, qs, ws) in enumerate(shards):
            spec.spec_shard_sample(lg, qs, dec.t, B, K, V, lo, t, x["seeds"], x["rids"],
                                   races.t[s * B * 96:(s + 1) * B * 96], ws.t, status=o["status"].t)
        spec.spec_shard_finish(races.t, S, dec.t, B, K, V, t, x["seeds"], x["rids"], o["acc"].t, o["tok"].t,
                               status=o["status"].t)
    assert_intact(stats=stats, races=races, decisions=dec, **o,
                  **{f"ws{s}": sh[3] for s, sh in enumerate(shards)})
    assert int(o["status"].t.item()) == 0
