"""Host logic of the N > 1 bench path on CPU: two gloo ranks, as torchrun
launches them (RANK / WORLD_SIZE / MASTER_* in the environment).

The data path partitions by request, so ranks share no data; what crosses
ranks is the barrier around the timed region and the max of the per-rank
times, which these tests exercise with the gloo backend."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    w, r, _ = bench.dist_info()
    dist = bench.dist_init(w, "gloo")
    bench.barrier(dist)
    slowest = bench.max_over_ranks(dist, 1.5 + r, torch.device("cpu"))
    bench.barrier(dist)
    with open(os.path.join(out_dir, f"rank{r}.json"), "w") as f:
        json.dump({"rank": r, "world": w, "max_ms": slowest}, f)
    dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_time(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    assert [x["rank"] for x in res] == [0, 1]
    assert all(x["world"] == world for x in res)
    assert all(x["max_ms"] == 2.5 for x in res)   # max over ranks, on every rank


def test_weak_scaling_throughput_counts_every_rank():
    # 2 ranks x 1088 rows x 10 steps in 1.5 ms of the slowest rank
    assert bench.job_throughput(2, 1088, 10, 1.5) == pytest.approx(2 * 1088 * 10 / 1.5e-3)
    assert bench.job_throughput(1, 1088, 10, 1.5) * 2 == pytest.approx(bench.job_throughput(2, 1088, 10, 1.5))


def test_ranks_draw_their_own_inputs():
    class A:
        workload, V, B = "tiny", None, None
    a0 = bench.make_inputs(A, 0, "cpu")
    a1 = bench.make_inputs(A, 1, "cpu")
    assert a0.logits.shape == a1.logits.shape and a0.rows == a1.rows
    assert not torch.equal(a0.logits, a1.logits)      # per-rank seeds: independent batches
    assert not torch.equal(a0.conf, a1.conf)


def test_reference_arm_under_torchrun_prints_once():
    """`bench.py --impl reference` launched as two ranks: rank 0 times the
    oracle and prints one JSON line, rank 1 exits 0 without work."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
           "--steps", "1", "--warmup", "0", "--workload", "tiny"]
    env = {**os.environ, "CUDA_VISIBLE_DEVICES": ""}
    proc = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert proc.returncode == 0, proc.stderr[-2000:]
    lines = [l for l in proc.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"


class _Wl:
    """The fields of a workload that the byte accounting reads."""
    def __init__(self, B, K, V, H, dtype="bf16", q=True, hidden=True):
        self.B, self.K, self.V, self.H, self.dtype = B, K, V, H, dtype
        self.q = object() if q else None
        self.hidden = object() if hidden else None


def test_algorithmic_bytes_count_what_the_method_reads():
    """Every logits row once, a q row per rejecting request, the q(z)/l(z)
    sectors, the committed hidden rows read and written, the small arrays."""
    import numpy as np
    B, K, V, H = 4, 3, 1000, 64
    acc = np.array([3, 0, 1, 3])                    # two requests reject (a < K)
    ab = bench.algorithmic_bytes(_Wl(B, K, V, H), acc)
    assert ab["logits"] == B * (K + 1) * V * 2
    assert ab["q_rows"] == 2 * V * 2
    assert ab["gathers"] == B * K * 2 * 32
    assert ab["commit"] == 2 * int((acc + 1).sum()) * H * 2
    assert ab["total"] == ab["logits"] + ab["q_rows"] + ab["gathers"] + ab["commit"] + ab["small"]
    none = bench.algorithmic_bytes(_Wl(B, K, V, H, dtype="f32", q=False, hidden=False), acc)
    assert none["logits"] == B * (K + 1) * V * 4 and none["q_rows"] == 0 and none["commit"] == 0
