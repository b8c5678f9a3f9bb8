"""Host logic of vocabulary-sharded verification on CPU (Section 4.4 serves
the target with TP = 8): the column split, and the order in which two gloo
ranks' records reach the merging calls.  The four libspec calls are replaced
by fakes that stamp each shard's records, so no GPU is needed; what is tested
is the buffers, slices and exchanges of paper_2607_25852_gb300.sharded."""
import json
import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
from paper_2607_25852_gb300 import sharded  # noqa: E402


def test_even_bounds():
    assert sharded.even_bounds(201088, 8) == [25136 * s for s in range(9)]
    assert sharded.even_bounds(10, 4) == [0, 3, 6, 8, 10]
    assert sharded.even_bounds(5, 5) == [0, 1, 2, 3, 4, 5]
    with pytest.raises(ValueError):
        sharded.even_bounds(3, 4)


def _install_fakes(log, setattr_=None):
    """Fakes of the four calls: stats and sample stamp their output with the
    shard's index; decide and finish record what they were given.
    `setattr_`: how to install them (monkeypatch.setattr in-process)."""
    setattr_ = setattr_ or setattr
    def stamp_of(v_begin, bounds):
        return bounds.index(v_begin)

    def stats(lg, drafts, q, B, K, V, v_begin, t, pos, out, ws, **kw):
        out.fill_(1 + stamp_of(v_begin, log["bounds"]))

    def decide(stats_buf, S, *a, **kw):
        per = stats_buf.numel() // S
        log["decide"] = [int(stats_buf[s * per:(s + 1) * per].float().mean()) for s in range(S)]

    def sample(lg, q, dec, B, K, V, v_begin, t, seeds, rids, out, ws, **kw):
        out.fill_(100 + stamp_of(v_begin, log["bounds"]))

    def finish(races, S, *a, **kw):
        per = races.numel() // S
        log["finish"] = [int(races[s * per:(s + 1) * per].float().mean()) for s in range(S)]

    setattr_(sharded, "spec_shard_stats", stats)
    setattr_(sharded, "spec_shard_decide", decide)
    setattr_(sharded, "spec_shard_sample", sample)
    setattr_(sharded, "spec_shard_finish", finish)
    setattr_(sharded, "shard_workspace", lambda B, K, Vs, device: torch.zeros(256, dtype=torch.uint8, device=device))


def _round_args(B, K):
    z = lambda *s: torch.zeros(s, dtype=torch.int32)
    return dict(drafts=z(B, K), seeds=z(B), request_ids=z(B), pos_base=z(B), accepted_len_out=z(B),
                out_tokens=z(B, K + 1))


def test_local_round_writes_shards_side_by_side(monkeypatch):
    B, K, V = 3, 2, 5000
    bounds = sharded.even_bounds(V, 3)
    log = {"bounds": bounds}
    _install_fakes(log, monkeypatch.setattr)
    rnd = sharded.ShardedRound(B, K, V, bounds, device="cpu", local=True)
    lg = [torch.zeros(B * (K + 1), bounds[s + 1] - bounds[s]) for s in range(3)]
    rnd.run(lg, q=None, temperature=1.0, **_round_args(B, K))
    assert log["decide"] == [1, 2, 3] and log["finish"] == [100, 101, 102]
    log.pop("finish")
    rnd.run(lg, q=None, temperature=0.0, **_round_args(B, K))
    assert "finish" not in log      # t = 0: the decision writes every token


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    B, K, V = 4, 3, 201088
    bounds = sharded.even_bounds(V, world)
    log = {"bounds": bounds}
    _install_fakes(log)
    rnd = sharded.ShardedRound(B, K, V, bounds, rank=rank, device="cpu")
    lg = torch.zeros(B * (K + 1), bounds[rank + 1] - bounds[rank])
    rnd.run(lg, q=None, temperature=0.7, **_round_args(B, K))
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"decide": log["decide"], "finish": log["finish"]}, f)
    dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_gather_records_in_rank_order(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    for r in range(world):
        res = json.load(open(tmp_path / f"rank{r}.json"))
        assert res["decide"] == [1, 2]          # every rank sees both shards' stats, in order
        assert res["finish"] == [100, 101]      # and both shards' race records
