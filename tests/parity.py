"""Helpers for the GPU-vs-oracle parity tests.

The CUDA path is called through the C ABI (paper_2607_25852_gb300 binding);
the oracle runs on the CPU over the very same input bytes.  Comparison rules:

  * accepted lengths, committed tokens, depths, packed maps, gathered rows:
    bit-exact;
  * p_j(z_{j+1}) and the row statistics: relative 1e-5 (ln S: absolute 1e-5);
  * an acceptance decision may differ only where |u - min(1, p/q)| < 1e-6
    (the oracle's u and r); a sampled token may differ only where one level
    of the oracle's two-level race had its two best keys within a relative
    1e-5 of each other and the GPU took the runner-up there.  Each such case
    is counted; the rest of that request is not compared bit-exactly.
"""
import numpy as np
import torch

import oracle

P_RTOL = 1e-5
ACCEPT_TIE = 1e-6
RACE_TIE = 1e-5


def race_tie(race, token):
    """True if `token` is the runner-up of a near tie in the oracle's race."""
    b1k, _, b2k, _, _, yk, y2k, y2, yb2 = race

    def close(a, b):
        return a > 0 and (b - a) / a < RACE_TIE

    return (close(b1k, b2k) and int(yb2) == token) or (close(yk, y2k) and int(y2) == token)


def bits(t):
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def u64(t):
    return t.detach().cpu().numpy().view(np.uint64)


def run_verify(logits, drafts, q, B, K, V, t, seeds, request_ids, pos_base, row_offsets=None,
               depth=None, ws=None, device="cuda"):
    import paper_2607_25852_gb300 as spec
    dev = torch.device(device)
    d = lambda x: None if x is None else x.to(dev).contiguous()
    ws = spec.verify_workspace(B, K, V, dev) if ws is None else ws
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((B, K + 1), -7, dtype=torch.int32, device=dev)
    pdr = torch.full((B, max(K, 1)), -7.0, dtype=torch.float32, device=dev)
    rst = torch.zeros((B * (K + 1), 2), dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    spec.spec_verify(d(logits), d(drafts), d(q), B, K, V, t, d(seeds), d(request_ids), d(pos_base),
                     acc, tok, ws, row_offsets=d(row_offsets), depth=d(depth),
                     p_draft_out=pdr if K > 0 else None, row_stats_out=rst, status=status)
    torch.cuda.synchronize()
    return dict(accepted=acc.cpu().numpy(), tokens=tok.cpu().numpy(), p_draft=pdr.cpu().numpy()[:, :K],
                row_stats=rst.cpu().numpy(), status=int(status.item()), ws=ws)


def run_oracle(logits, drafts, q, t, seeds, request_ids, pos_base, row_offsets=None, depth=None):
    return oracle.verify_batch(bits(logits), drafts.cpu().numpy(), None if q is None else bits(q), t,
                               u64(seeds), u64(request_ids), pos_base.cpu().numpy(),
                               None if row_offsets is None else row_offsets.cpu().numpy(),
                               None if depth is None else depth.cpu().numpy())


def compare(gpu, ref, K, t, depth=None, row_offsets=None, check_stats=True):
    """Assert parity; returns (n_accept_ties, n_race_ties, n_positions)."""
    B = len(ref["accepted"])
    n_acc_ties = n_race_ties = 0
    positions = 0
    for i in range(B):
        n = K if depth is None else int(depth[i])
        positions += n + 1
        ga, ra = int(gpu["accepted"][i]), int(ref["accepted"][i])
        gt, rt = gpu["tokens"][i], ref["tokens"][i]
        if ref["status"][i] != 0:
            assert ga == 0 and (gt == -1).all(), f"request {i}: bad input not flagged"
            continue
        if ga != ra:
            j = min(ga, ra)
            assert t > 0 and j < n, f"request {i}: accepted {ga} vs oracle {ra}"
            gap = abs(ref["u"][i, j] - ref["r"][i, j])
            assert gap < ACCEPT_TIE, f"request {i}: decision at {j} differs, |u-r|={gap:.3g}"
            assert gt[:j].tolist() == rt[:j].tolist()
            n_acc_ties += 1
            continue
        assert gt[:ra].tolist() == rt[:ra].tolist(), f"request {i}: accepted drafts differ"
        assert (gt[ra + 1:] == -1).all(), f"request {i}: padding"
        if gt[ra] != rt[ra]:
            assert t > 0 and race_tie(ref["race"][i], int(gt[ra])), (
                f"request {i}: token {gt[ra]} vs oracle {rt[ra]} (race {ref['race'][i].tolist()})")
            n_race_ties += 1
        if t > 0 and n > 0:
            np.testing.assert_allclose(gpu["p_draft"][i, :n], ref["p_draft"][i, :n], rtol=P_RTOL,
                                       atol=1e-30, err_msg=f"request {i}: p_draft")
    if check_stats:
        rows = []
        for i in range(B):
            if ref["status"][i] != 0:
                continue
            n = K if depth is None else int(depth[i])
            row0 = i * (K + 1) if row_offsets is None else int(row_offsets[i])
            rows.extend(range(row0, row0 + n + 1))
        rows = np.asarray(rows, np.int64)
        np.testing.assert_allclose(gpu["row_stats"][rows, 0], ref["row_m"][rows], rtol=P_RTOL, atol=0)
        np.testing.assert_allclose(gpu["row_stats"][rows, 1], ref["row_logS"][rows], rtol=0, atol=P_RTOL)
    assert n_acc_ties + n_race_ties <= max(1, 1e-4 * positions), (n_acc_ties, n_race_ties, positions)
    return n_acc_ties, n_race_ties, positions


def shard_bounds(V, S, unit=1):
    """S contiguous ranges covering [0, V): equal parts rounded to `unit`
    columns, the last one taking the rest."""
    per = max(unit, (V // S) // unit * unit)
    b = [min(V, s * per) for s in range(S)] + [V]
    return b


def run_sharded(logits, drafts, q, B, K, V, t, seeds, request_ids, pos_base, bounds,
                row_offsets=None, depth=None, ws=None, device="cuda"):
    """The four shard calls over shards [bounds[s], bounds[s+1]) of one GPU
    (paper_2607_25852_gb300.sharded.ShardedRound with local=True: the S
    shards' records are written side by side, in place of the exchanges).
    `ws`: the ShardedRound of an earlier call, to reuse its workspaces."""
    from paper_2607_25852_gb300.sharded import ShardedRound
    dev = torch.device(device)
    d = lambda x: None if x is None else x.to(dev).contiguous()
    S = len(bounds) - 1
    R = B * (K + 1)
    lg, qq = d(logits), d(q)
    rnd = ShardedRound(B, K, V, bounds, device=dev, local=True) if ws is None else ws
    lgs = [lg[:, bounds[s]:bounds[s + 1]].contiguous() for s in range(S)]
    qs = None if qq is None else [qq[:, :, bounds[s]:bounds[s + 1]].contiguous() for s in range(S)]
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((B, K + 1), -7, dtype=torch.int32, device=dev)
    pdr = torch.full((B, max(K, 1)), -7.0, dtype=torch.float32, device=dev)
    rst = torch.zeros((R, 2), dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rnd.run(lgs, d(drafts), qs, t, d(seeds), d(request_ids), d(pos_base), acc, tok,
            row_offsets=d(row_offsets), depth=d(depth), p_draft_out=pdr if K > 0 else None,
            row_stats_out=rst, status=status)
    torch.cuda.synchronize()
    return dict(accepted=acc.cpu().numpy(), tokens=tok.cpu().numpy(), p_draft=pdr.cpu().numpy()[:, :K],
                row_stats=rst.cpu().numpy(), status=int(status.item()), ws=rnd)
