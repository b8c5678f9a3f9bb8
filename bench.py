"""Benchmark of the batched speculative-verification hot path on GB300.

One step = one round of the method over one batch of the stress workload
(B=64 requests, K=16 drafts, V=201088 bf16 logits, bf16 q, temperature 1,
hidden rows H=7168 bf16):

    spec_allocate  D-cut over the paper's ratios {1/4, 1/2, 3/4, 1} with a flat
                   cost table (light load: the full block wins, T* = B(K+1))
    spec_verify    rejection-sampling verification of all 1088 rows
    spec_commit    packing of the committed tokens and hidden rows

value = verified positions per second (rows verified / step time), inputs
resident in HBM.  The logits alone (437.6 MB) exceed L2 (129 MB), so no L2
flush is needed between steps.  The JSON line also carries the roofline of the
vocabulary-streaming kernel, clocks sampled during the timed region, an
end-to-end number through the same public API with host (pinned) buffers, and
the CPU oracle timed on a bounded sample.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Under torchrun (N > 1) each rank runs its own batch (weak scaling, no
collective on the data path); timing is the max over ranks.
"""
import argparse
import concurrent.futures as cf
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified positions/s"
UNIT = "positions/s"
L2_BYTES = 129 * 1000 * 1000  # GB300 L2, 129 MB
KERNEL_SAMPLES = 30  # event-bracketed launches of the streaming kernel, at least
FALLBACK_HBM_GBS = 6800.0


class L2Flush:
    """Evicts L2 between timed iterations: a write of twice the L2 size, then a
    read of another buffer of that size, so that L2 is left holding clean lines
    only.  (After the write alone, L2 is full of dirty lines, which the next
    kernel would write back to HBM while it reads its own inputs.)"""

    def __init__(self, device):
        import torch
        self.w = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=device)
        self.r = torch.ones(2 * L2_BYTES // 4, dtype=torch.float32, device=device)
        self.s = torch.empty((), dtype=torch.float32, device=device)

    def __call__(self, k):
        import torch
        self.w.fill_(k & 0xFF)
        torch.sum(self.r, 0, out=self.s)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="stress")
    ap.add_argument("--V", type=int, default=None)
    ap.add_argument("--B", type=int, default=None)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="skip the CUDA-graph replay timing")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--draft", action="store_true",
                    help="time the drafter's step (spec_draft) on B=64, K=16, V=201088 bf16 drafter logits")
    ap.add_argument("--tau", type=float, default=1.0, help="draft temperature for --draft")
    ap.add_argument("--markov", action="store_true",
                    help="time the Markov head's sequential draw: B=64 requests, a block of K=7 drafts, "
                         "V=201088, rank r=256")
    ap.add_argument("--round-graph", action="store_true",
                    help="time a round with the budget chosen on the device (one graph per candidate budget) "
                         "against the host reading the budget between allocation and verification")
    ap.add_argument("--shards", type=int, default=1,
                    help="S > 1: time vocabulary-sharded verification with S shards emulated on one GPU")
    return ap.parse_args()


# ---------------------------------------------------------------------------
# distributed plumbing (rank layout only; no collective touches the data path)
# ---------------------------------------------------------------------------
def dist_info():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_init(world, backend):
    if world <= 1:
        return None
    import torch.distributed as dist
    dist.init_process_group(backend=backend)
    return dist


def job_throughput(world, rows_per_rank, steps, total_ms):
    """Whole-job verified positions/s: every rank verifies rows_per_rank rows
    per step (weak scaling), timed as the slowest rank's total_ms."""
    return world * rows_per_rank * steps / (total_ms * 1e-3)


def max_over_ranks(dist, value, device):
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist):
    if dist is not None:
        dist.barrier()


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu_index = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu_index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# the workload
# ---------------------------------------------------------------------------
def make_inputs(args, rank, device):
    import torch
    import workloads
    wl = workloads.make(args.workload, device=device, seed=1234 + rank, V=args.V, B=args.B)
    B, K = wl.B, wl.K
    # Confidences for the allocator: the code/chat mix of the alloc workload.
    rng = np.random.default_rng(4321 + rank)
    half = B // 2
    conf = np.concatenate([rng.beta(2.0, 2.0, (half, K)), rng.beta(8.0, 1.0, (B - half, K))])
    wl.conf = torch.as_tensor(conf.astype(np.float32), device=device)
    return wl


class Step:
    """Buffers and one call sequence allocate -> verify -> commit."""

    def __init__(self, wl, device):
        import torch
        import paper_2607_25852_gb300 as spec
        self.spec = spec
        self.wl = wl
        B, K, V = wl.B, wl.K, wl.V
        if wl.name == "alloc":
            # the alloc workload's budget sweep T = 64..1024 with the profiled
            # piecewise-linear cost: D-cut picks T* < B(K+1)
            import workloads
            Ts, costs = workloads.budget_candidates(B, K)
            self.ratios, self.costs = [int(t) for t in Ts], [float(c) for c in costs]
        else:
            # the paper's ratios 1/4..1 with a flat cost table: the full block wins
            self.ratios = spec.spec_budget_from_ratios(B, K, [1, 1, 3, 1], [4, 2, 4, 1])
            self.costs = [1.0, 1.0, 1.0, 1.0]
        i32, i64 = torch.int32, torch.int64
        z = lambda *s, dt=i32: torch.zeros(s, dtype=dt, device=device)
        self.depth, self.row_off = z(B), z(B + 1)
        self.ptok, self.ppos = z(B * (K + 1)), z(B * (K + 1), dt=i64)
        self.chosen = z(1)
        self.util = z(len(self.ratios), dt=torch.float64)
        self.acc, self.tok = z(B), z(B, K + 1)
        self.ctok, self.coff = z(B * (K + 1)), z(B + 1)
        self.hout = None if wl.hidden is None else torch.empty_like(wl.hidden)
        self.status = z(1)
        self.ws = spec.verify_workspace(B, K, V, device)
        # The target forward writes its rows in the packed order of the
        # allocation; it is not part of this library, so the packed logits
        # and hidden rows of the (fixed) allocation are prepared once here.
        self.logits, self.hidden = wl.logits, wl.hidden
        spec.spec_allocate(wl.conf, self.ratios, self.costs, wl.last_tokens, wl.drafts, wl.pos_base,
                           self.depth, self.row_off, self.ptok, self.ppos, self.chosen, self.util, self.status)
        torch.cuda.synchronize()
        self.rows = int(self.chosen.item())
        if self.rows < wl.rows:
            import workloads
            depth = self.depth.cpu()
            self.logits = workloads.pack_rows(wl.logits, B, K, depth)
            self.hidden = None if wl.hidden is None else workloads.pack_rows(wl.hidden, B, K, depth)

    def run(self, inputs=None):
        wl = self.wl
        x = inputs or dict(conf=wl.conf, logits=self.logits, drafts=wl.drafts, q=wl.q, seeds=wl.seeds,
                           request_ids=wl.request_ids, pos_base=wl.pos_base,
                           last_tokens=wl.last_tokens, hidden=self.hidden)
        s = self.spec
        s.spec_allocate(x["conf"], self.ratios, self.costs, x["last_tokens"], x["drafts"],
                        x["pos_base"], self.depth, self.row_off, self.ptok, self.ppos, self.chosen,
                        self.util, self.status)
        s.spec_verify(x["logits"], x["drafts"], x["q"], wl.B, wl.K, wl.V, wl.temperature,
                      x["seeds"], x["request_ids"], x["pos_base"], self.acc, self.tok, self.ws,
                      row_offsets=self.row_off, depth=self.depth, status=self.status)
        s.spec_commit(self.acc, self.tok, x.get("hidden"), wl.B, wl.K, self.ctok, self.coff, self.hout,
                      row_offsets=self.row_off, status=self.status)

    def launches_per_step(self):
        # allocate (1) + verify: the streaming pass, then the decisions (t = 0)
        # or the sampling pass with the decisions (t > 0) (2) + commit (1 for
        # B <= 256, else 2)
        return 1 + 2 + (1 if self.wl.B <= 256 else 2)


def algorithmic_bytes(wl, acc, rows=None):
    """Bytes the method must move once per step (Section 4.2 verifies every
    retained position in one pass): every kept logits row (`rows`, all
    B(K+1) by default), the q row at each rejection, the q(z)/l(z) gathers,
    the committed hidden rows read and written, and the small per-request
    arrays."""
    B, K, V, H = wl.B, wl.K, wl.V, wl.H
    esize = 2 if wl.dtype == "bf16" else 4
    logits = (B * (K + 1) if rows is None else rows) * V * esize
    rejected = int(np.sum(acc < K))
    q_rows = rejected * V * esize if wl.q is not None else 0
    gathers = B * K * 2 * 32
    committed = int(np.sum(acc + 1))
    commit = 2 * committed * H * 2 if wl.hidden is not None else 0
    small = B * (K * 4 + K * 4 + 8 * 3 + (K + 1) * 4 * 2 + 4 * 4)
    return dict(logits=logits, q_rows=q_rows, gathers=gathers, commit=commit, small=small,
                total=logits + q_rows + gathers + commit + small)


def gpu_head_start(n_steps, host_us_per_step=80.0, max_ms=20.0):
    """Keep the GPU busy while the host queues `n_steps` steps ahead of a
    start event: the timed region then measures device time, not host launch
    latency or stalls of the host thread (the end-to-end figure covers the
    host).  About 80 us of host time per queued step, at most 20 ms."""
    import torch
    us = min(max_ms * 1e3, max(100.0, host_us_per_step * n_steps))
    torch.cuda._sleep(int(2100 * us))  # ~2.1 GHz SM clock: cycles per microsecond


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash():
    h = hashlib.sha256()
    for name in ("verify.cu", "verify_common.cuh", "spec_internal.cuh"):
        with open(os.path.join(ROOT, "paper_2607_25852_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload):
    """DRAM bytes per launch of the streaming kernel from the committed ncu
    summary, if it was taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", "stream_rows_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    entry = rec.get(workload)
    if not entry or entry.get("source_hash") != kernel_source_hash():
        return None
    return entry.get("dram_bytes_per_launch")


# ---------------------------------------------------------------------------
# CPU oracle timings (test infrastructure, timed as a reported baseline)
# ---------------------------------------------------------------------------
def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else platform)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def oracle_sample(wl, seconds, step_repeats=None, max_threads=None):
    """Run the CPU oracle over full batches of the same workload on the host
    cores (one request per task; at most `max_threads` threads) until
    `seconds` of wall time have passed."""
    import oracle
    import torch
    lg = wl.logits.detach().cpu()
    logits = lg.view(torch.int16).numpy().view(np.uint16) if lg.dtype == torch.bfloat16 else lg.numpy()
    q = None
    if wl.q is not None:
        qc = wl.q.detach().cpu()
        q = qc.view(torch.int16).numpy().view(np.uint16) if qc.dtype == torch.bfloat16 else qc.numpy()
    drafts = wl.drafts.cpu().numpy()
    seeds = wl.seeds.cpu().numpy().view(np.uint64)
    reqs = wl.request_ids.cpu().numpy().view(np.uint64)
    pos = wl.pos_base.cpu().numpy()
    B, K = wl.B, wl.K
    oracle.load()
    threads = os.cpu_count() or 1

    def one(i):
        return oracle.verify_batch(logits, drafts, q, wl.temperature, seeds, reqs, pos, requests=[i])

    rows = 0
    batches = 0
    t0 = time.perf_counter()
    if max_threads is not None:
        threads = max(1, min(threads, max_threads))
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        while True:
            list(ex.map(one, range(B)))
            rows += B * (K + 1)
            batches += 1
            el = time.perf_counter() - t0
            if (step_repeats is None and el >= seconds) or (step_repeats is not None and batches >= step_repeats):
                break
    el = time.perf_counter() - t0
    return rows, el, threads, batches


# ---------------------------------------------------------------------------
# arms
# ---------------------------------------------------------------------------
def run_reference(args):
    """The reference arm: the CPU oracle, timed on the host cores."""
    world, rank, local = dist_info()
    if rank != 0:
        return 0
    import torch
    wl = make_inputs(args, 0, "cpu")
    R = wl.rows
    # bounded sample per step: one full batch (all B requests) through the oracle
    if args.warmup:
        oracle_sample(wl, 0, step_repeats=1)
    times = []
    threads = os.cpu_count() or 1
    for _ in range(args.steps):
        rows, el, threads, _ = oracle_sample(wl, 0, step_repeats=1)
        times.append(el)
    total = sum(times)
    value = R * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": f"{wl.name}: B={wl.B} K={wl.K} V={wl.V} {wl.dtype} logits, "
                               f"t={wl.temperature}, q {'bf16' if wl.q is not None else 'one-hot'}",
                   "sample": "one full batch per step (verification of every request)"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"full batch of {wl.B} requests x {wl.K + 1} rows per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    import torch
    world, rank, local = dist_info()
    if not torch.cuda.is_available():
        print(json.dumps({"error": "no CUDA device"}))
        return 1
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    dist = dist_init(world, "nccl")
    import paper_2607_25852_gb300 as spec

    wl = make_inputs(args, rank, device)
    step = Step(wl, device)
    R = step.rows  # verified positions per step: the chosen budget T*
    stream = torch.cuda.current_stream()

    for _ in range(max(args.warmup, 3)):
        step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0, "device reported an input error"
    assert int(step.chosen.item()) == R, "the allocation changed between steps"
    acc = step.acc.cpu().numpy()
    alg = algorithmic_bytes(wl, acc, R)

    # ---- device-timed region ----
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    for pair in ev:                # torch creates the CUDA events lazily, at first record
        for e in pair:
            e.record(stream)
    # A step whose inputs fit in L2 would find them cached from the step
    # before: then L2 is flushed between steps (L2Flush) and
    # only the steps themselves are timed.
    flush = None
    if alg["logits"] < 2 * L2_BYTES:
        flush = L2Flush(device)
    torch.cuda.synchronize()
    barrier(dist)
    torch.cuda.synchronize()
    with ClockSampler(local) as clocks:
        start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        gpu_head_start(args.steps)
        # Steps follow one another as in a serving loop: an event between
        # two steps would keep the next step's first kernel from launching
        # while the last one drains, so steps are bracketed one by one only
        # where an L2 flush has to be left out of the time.
        start.record(stream)
        for k in range(args.steps):
            if flush is not None:
                flush(k)
                ev[k][0].record(stream)
            step.run()
            if flush is not None:
                ev[k][1].record(stream)
        stop.record(stream)
        torch.cuda.synchronize()
    barrier(dist)
    total_ms = start.elapsed_time(stop)
    if flush is not None:
        total_ms = sum(a.elapsed_time(b) for a, b in ev)
    total_ms = max_over_ranks(dist, total_ms, device)
    ms_per_step = total_ms / args.steps
    value = job_throughput(world, R, args.steps, total_ms)

    # ---- the streaming kernel alone: its own loop of event-bracketed steps ----
    # Events between two kernels break their programmatic overlap, so they
    # stay out of the timed steps above; here every step brackets the
    # streaming kernel, and the clocks are sampled over this loop.
    n_k = max(KERNEL_SAMPLES, args.steps)
    kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_k)]
    for pair in kev:
        for e in pair:
            e.record(stream)
    torch.cuda.synchronize()
    with ClockSampler(local) as kclocks:
        gpu_head_start(n_k)
        for k in range(n_k):
            if flush is not None:
                flush(k)
            spec.spec_profile_stream_pass(kev[k][0], kev[k][1])
            step.run()
        torch.cuda.synchronize()
    kern_ms = [a.elapsed_time(b) for a, b in kev]

    # ---- the spread of single steps: a loop of steps bracketed one by one
    # (each bracket keeps the step from overlapping the one before) ----
    if flush is None:
        sev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_k)]
        for pair in sev:
            for e in pair:
                e.record(stream)
        torch.cuda.synchronize()
        gpu_head_start(n_k)
        for k in range(n_k):
            sev[k][0].record(stream)
            step.run()
            sev[k][1].record(stream)
        torch.cuda.synchronize()
        step_ms = [a.elapsed_time(b) for a, b in sev]
    else:
        step_ms = [a.elapsed_time(b) for a, b in ev]

    # ---- the same step captured once in a CUDA graph and replayed ----
    graph = None
    if not args.no_graph and flush is None:
        try:
            g = torch.cuda.CUDAGraph()
            side = torch.cuda.Stream()
            side.wait_stream(stream)
            with torch.cuda.stream(side):
                step.run()          # warm the side stream before capture
            stream.wait_stream(side)
            torch.cuda.synchronize()
            with torch.cuda.graph(g):
                step.run()
            for _ in range(3):
                g.replay()
            torch.cuda.synchronize()
            barrier(dist)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            gpu_head_start(args.steps, host_us_per_step=20.0)
            a.record(stream)
            for _ in range(args.steps):
                g.replay()
            b.record(stream)
            torch.cuda.synchronize()
            g_ms = max_over_ranks(dist, a.elapsed_time(b), device)
            assert int(step.status.item()) == 0, "device reported an input error under the graph"
            graph = {"value": job_throughput(world, R, args.steps, g_ms), "unit": UNIT,
                     "ms_per_step": g_ms / args.steps,
                     "how": "allocate + verify + commit captured once with torch.cuda.graph, replayed"}
        except Exception as exc:  # report, do not hide: the line says why there is no number
            graph = {"error": f"{type(exc).__name__}: {exc}"[:300]}

    # ---- end to end through the same API with pinned host buffers ----
    # The large inputs (logits, q, hidden rows) are read in place by the
    # kernels when the device reaches the pinned buffers at the same address
    # (NVLink-C2C on Grace-Blackwell); the small ones are copied.  The
    # copy-engine variant (every input copied to device memory first) is
    # measured too.
    e2e = None
    if not args.no_e2e:
        src = dict(conf=wl.conf, logits=step.logits, drafts=wl.drafts, q=wl.q, seeds=wl.seeds,
                   request_ids=wl.request_ids, pos_base=wl.pos_base, last_tokens=wl.last_tokens,
                   hidden=step.hidden)  # the packed rows of the step's allocation
        host = {k: v.cpu().pin_memory() for k, v in src.items() if v is not None}
        dev_in = {k: torch.empty_like(v, device=device) for k, v in host.items()}
        dev_in.setdefault("q", None)
        outs_host = [torch.empty_like(t, device="cpu").pin_memory() for t in (step.acc, step.tok, step.ctok, step.coff)]
        h2d = sum(v.numel() * v.element_size() for v in host.values())
        d2h = sum(t.numel() * t.element_size() for t in outs_host)
        big = [k for k in ("logits", "q", "hidden") if k in host]
        in_place_ok = all(step.spec.spec_pointer_device_readable(host[k]) for k in big)

        def e2e_step(in_place):
            x = dict(dev_in)
            for k, v in host.items():
                if in_place and k in big:
                    x[k] = v
                else:
                    dev_in[k].copy_(v, non_blocking=True)
            step.run(x)
            for o, d in zip(outs_host, (step.acc, step.tok, step.ctok, step.coff)):
                o.copy_(d, non_blocking=True)

        def measure(in_place):
            for _ in range(2):
                e2e_step(in_place)
            torch.cuda.synchronize()
            n = max(3, min(args.steps, 10))
            barrier(dist)
            t0 = time.perf_counter()
            for _ in range(n):
                e2e_step(in_place)
            torch.cuda.synchronize()
            el = max_over_ranks(dist, time.perf_counter() - t0, device)
            return world * R * n / el, 1e3 * el / n, n

        v_copy, ms_copy, n_copy = measure(False)
        if in_place_ok:
            v, ms, n = measure(True)
            # what crosses the link in place: every logits row, the q row at
            # each rejection and the q(z) sectors, the committed hidden rows,
            # and the small inputs that are copied
            ab = algorithmic_bytes(wl, step.acc.cpu().numpy(), R)
            small_bytes = sum(t.numel() * t.element_size() for k, t in host.items() if k not in big)
            h2d_moved = (ab["logits"] + ab["q_rows"] + (wl.B * wl.K * 32 if wl.q is not None else 0)
                         + ab["commit"] // 2 + small_bytes)
            how = ("pinned host logits, q and hidden rows read in place by the kernels (only the bytes the "
                   "method reads cross the link); small inputs copied")
        else:
            v, ms, n, h2d_moved = v_copy, ms_copy, n_copy, h2d
            how = "every input copied to device memory first"
        e2e = {"value": v, "unit": UNIT, "h2d_bytes_per_step": h2d_moved, "d2h_bytes_per_step": d2h, "steps": n,
               "ms_per_step": ms, "h2d": how, "host_input_bytes_per_step": h2d,
               "copy_engine": {"value": v_copy, "ms_per_step": ms_copy, "h2d_bytes_per_step": h2d}}

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0

    peak, peak_kind = measured_peak()
    k_med = statistics.median(kern_ms)
    achieved = alg["logits"] / (k_med * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": recorded_traffic(wl.name),
                "kernel": "stream_rows_kernel", "peak_kind": peak_kind,
                "algorithmic_bytes_per_launch": alg["logits"],
                "median_launch_us": round(1e3 * k_med, 2),
                "avg_launch_us": round(1e3 * statistics.mean(kern_ms), 2),
                "launch_us_p10_p90": [round(1e3 * float(np.percentile(kern_ms, q)), 2) for q in (10, 90)],
                "launches_timed": len(kern_ms), "clocks": kclocks.summary(),
                "frac_of_8000": round(achieved / 8000.0, 4)}
    step_gbs = alg["total"] / (ms_per_step * 1e-3) / 1e9

    cpu = None
    if not args.no_cpu_baseline and world == 1:
        rows, el, threads, batches = oracle_sample(wl, args.cpu_seconds)
        rows1, el1, _, batches1 = oracle_sample(wl, args.cpu_seconds, max_threads=1)
        cpu = {"value": rows / el, "unit": UNIT, "cores": threads, "kind": "oracle",
               "sample": f"{batches} full batch(es) of the same workload ({wl.B} requests x "
                         f"{wl.K + 1} rows), {el:.1f} s wall on {threads} host threads",
               "single_thread": {"value": rows1 / el1, "unit": UNIT, "cores": 1,
                                 "sample": f"{batches1} full batch(es), {el1:.1f} s wall on 1 thread"},
               "nproc": os.cpu_count(), "cpu_model": cpu_model()}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": f"{wl.name}: B={wl.B} K={wl.K} V={wl.V} {wl.dtype} logits, "
                               f"t={wl.temperature}, q {'bf16 [B,K,V]' if wl.q is not None else 'one-hot'}, "
                               f"H={wl.H}; " + (f"D-cut over T = 64..1024 with cost 1 + 0.004 max(0, T - 256) "
                                                 f"(T*={R})" if wl.name == "alloc" else
                                                 f"D-cut ratios 1/4..1 with a flat cost table (T*={R})"),
                   "rows_per_step": R,
                   "l2": (f"inputs larger than L2 ({alg['logits'] / 1e6:.1f} MB logits per step, no flush)"
                          if flush is None else
                          f"L2 flushed between steps ({alg['logits'] / 1e6:.1f} MB logits per step); "
                          "the sum of per-step event times is timed"),
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "roofline": roofline,
        "step_hbm_gbs": round(step_gbs, 1),
        "step_frac_of_measured": round(step_gbs / peak, 4),
        "step_frac_of_8000": round(step_gbs / 8000.0, 4),
        "algorithmic_bytes_per_step": alg,
        "step_ms_p10_p50_p90": [float(np.percentile(step_ms, p)) for p in (10, 50, 90)],
        "step_ms_how": "single steps, each bracketed by events (no overlap with the step before)",
        "mean_accepted": float(acc.mean()),
        "accepted_histogram": [int(x) for x in np.bincount(acc, minlength=wl.K + 1)],
        "clocks": clocks.summary(),
        "e2e": e2e,
        "graph": graph,
        "gpu_launches": step.launches_per_step() * args.steps,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def run_sharded(args):
    """Vocabulary-sharded verification (the target's TP layout) with the S
    shards on this one GPU: the whole round (S x stats, decide, S x sample,
    finish; the records written side by side in place of the all-gathers),
    and the per-rank critical path (stats, decide, sample, finish), each call
    timed in a loop of back-to-back calls over the S shards and once alone
    after an L2 flush."""
    import torch
    import paper_2607_25852_gb300 as spec
    from paper_2607_25852_gb300.sharded import ShardedRound, even_bounds
    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    wl = make_inputs(args, 0, device)
    B, K, V, t = wl.B, wl.K, wl.V, wl.temperature
    S = args.shards
    bounds = even_bounds(V, S)
    rnd = ShardedRound(B, K, V, bounds, device=device, local=True)
    lgs = [wl.logits[:, bounds[s]:bounds[s + 1]].contiguous() for s in range(S)]
    qs = None if wl.q is None else [wl.q[:, :, bounds[s]:bounds[s + 1]].contiguous() for s in range(S)]
    acc = torch.zeros(B, dtype=torch.int32, device=device)
    tok = torch.zeros((B, K + 1), dtype=torch.int32, device=device)
    status = torch.zeros(1, dtype=torch.int32, device=device)
    stream = torch.cuda.current_stream()

    def round_():
        rnd.run(lgs, wl.drafts, qs, t, wl.seeds, wl.request_ids, wl.pos_base, acc, tok, status=status)

    for _ in range(max(args.warmup, 3)):
        round_()
    torch.cuda.synchronize()
    assert int(status.item()) == 0, "device reported an input error"
    R = B * (K + 1)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clocks:
        gpu_head_start(args.steps, host_us_per_step=40.0 * S)
        a.record(stream)
        for _ in range(args.steps):
            round_()
        b.record(stream)
        torch.cuda.synchronize()
    round_ms = a.elapsed_time(b) / args.steps

    # Per-rank calls.  Each is timed (1) in a loop of back-to-back calls that
    # cycles through the S shards, its mean per call: the stats and sample
    # calls then read S x a shard's logits in turn, more than L2, so that no
    # call finds its inputs in L2 (decide and finish read the records, which a
    # rank receives from the all-gather just before); and (2) alone, after an
    # L2 flush, the median of `steps` calls, which adds the latency of an
    # isolated launch and the event clock's granularity (about 1 us).
    sb, rb = R * spec.SHARD_STAT_BYTES, B * spec.SHARD_RACE_BYTES
    sl = [slice(s * sb, (s + 1) * sb) for s in range(S)]
    rl = [slice(s * rb, (s + 1) * rb) for s in range(S)]
    qsh = (lambda s: None) if qs is None else (lambda s: qs[s])
    calls = {
        "stats": lambda s: spec.spec_shard_stats(lgs[s], wl.drafts, qsh(s), B, K, V, bounds[s], t, wl.pos_base,
                                                 rnd.stats[sl[s]], rnd.ws[s], status=status),
        "decide": lambda s: spec.spec_shard_decide(rnd.stats, S, wl.drafts, qs is not None, B, K, V, t, wl.seeds,
                                                   wl.request_ids, wl.pos_base, acc, tok,
                                                   decisions_out=rnd.decisions, status=status),
        "sample": lambda s: spec.spec_shard_sample(lgs[s], qsh(s), rnd.decisions, B, K, V, bounds[s], t, wl.seeds,
                                                   wl.request_ids, rnd.races[rl[s]], rnd.ws[s], status=status),
        "finish": lambda s: spec.spec_shard_finish(rnd.races, S, rnd.decisions, B, K, V, t, wl.seeds,
                                                   wl.request_ids, acc, tok, status=status),
    }
    flush = L2Flush(device)
    n_loop = 4 * S
    per, alone = {}, {}
    for name, fn in calls.items():
        if t == 0 and name in ("sample", "finish"):
            continue
        ts, ts1 = [], []
        for k in range(args.steps):
            round_()                    # leaves every record of this round in place
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            gpu_head_start(1, host_us_per_step=40.0 * n_loop)  # queue the launches ahead of the start event
            e0.record(stream)
            for c in range(n_loop):
                fn(c % S)
            e1.record(stream)
            flush(k)
            e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(200000)
            e2.record(stream)
            fn(0)
            e3.record(stream)
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1) / n_loop)
            ts1.append(e2.elapsed_time(e3))
        per[name] = 1e3 * statistics.median(ts)
        alone[name] = 1e3 * statistics.median(ts1)
    assert int(status.item()) == 0
    peak, peak_kind = measured_peak()
    esize = 2 if wl.dtype == "bf16" else 4
    stats_bytes = R * (bounds[1] - bounds[0]) * esize
    achieved = stats_bytes / (per["stats"] * 1e-6) / 1e9
    line = {
        "metric": METRIC, "value": R * args.steps / (round_ms * 1e-3 * args.steps), "unit": UNIT,
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
        "data": "synthetic",
        "config": {"workload": f"{wl.name}: B={B} K={K} V={V} {wl.dtype} logits, t={t}, "
                               f"q {'bf16 [B,K,V]' if wl.q is not None else 'one-hot'}",
                   "shards": S, "bounds": bounds,
                   "parallelism": f"vocabulary split into {S} shards, all on one GPU (records written "
                                  "side by side in place of the all-gathers)"},
        "per_rank_us": {k: round(v, 2) for k, v in per.items()},
        "per_rank_us_how": (f"mean per call over {n_loop} back-to-back calls cycling through the {S} shards, "
                            f"median of {args.steps} loops"),
        "per_rank_alone_us": {k: round(v, 2) for k, v in alone.items()},
        "per_rank_alone_us_how": "one call alone after an L2 flush (L2Flush), event-bracketed, median",
        "per_rank_critical_path_us": round(sum(per.values()), 2),
        "exchange_bytes_per_rank": {"stats": sb, "races": rb if t > 0 else 0},
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None, "kernel": "shard_stats_kernel",
                     "peak_kind": peak_kind, "algorithmic_bytes_per_launch": stats_bytes,
                     "avg_launch_us": round(per["stats"], 2),
                     "alone": {"us": round(alone["stats"], 2),
                               "frac": round(stats_bytes / (alone["stats"] * 1e-6) / 1e9 / peak, 4)}},
        "clocks": clocks.summary(),
        "gpu_launches": (2 * S + 2 if t > 0 else S + 1) * args.steps,
    }
    print(json.dumps(line), flush=True)
    return 0


def run_draft(args):
    """The drafter's producer step (spec_draft) on the draft recipe: drafts,
    confidences and D-cut scores from B x K rows of drafter logits.  One
    launch per step; the logits (412 MB) exceed L2, so no flush."""
    import torch
    import paper_2607_25852_gb300 as spec
    import workloads
    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    di = workloads.make_draft(device=device, tau=args.tau, B=args.B or 64, V=args.V or 201088)
    B, K, V = di.B, di.K, di.V
    ws = spec.draft_workspace(B, K, V, device)
    z = torch.zeros((B, K), dtype=torch.int32, device=device)
    c = torch.zeros((B, K), device=device)
    sc = torch.zeros((B, K + 1), device=device)
    st = torch.zeros((B * K, 2), device=device)
    status = torch.zeros(1, dtype=torch.int32, device=device)
    stream = torch.cuda.current_stream()

    def step():
        spec.spec_draft(di.logits, di.tau, di.seeds, di.request_ids, di.pos_base, z, c, ws, scores_out=sc,
                        row_stats_out=st, status=status)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    assert int(status.item()) == 0, "device reported an input error"
    nbytes = di.logits.numel() * di.logits.element_size()
    flush = None
    if nbytes < 2 * L2_BYTES:
        flush = L2Flush(device)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(0) as clocks:
        gpu_head_start(args.steps)
        if flush is None:
            # steps back to back, as a drafter runs them (an event between two
            # launches would keep the next from launching while the last drains)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for k in range(args.steps):
                step()
            b.record(stream)
            torch.cuda.synchronize()
            ms_per_step = a.elapsed_time(b) / args.steps
        # single steps, each bracketed by events: their spread (and the time
        # itself where an L2 flush has to stay out of it)
        gpu_head_start(args.steps)
        for k in range(args.steps):
            if flush is not None:
                flush(k)
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        torch.cuda.synchronize()
    ms = [a.elapsed_time(b) for a, b in ev]
    if flush is not None:
        ms_per_step = statistics.mean(ms)
    peak, peak_kind = measured_peak()
    achieved = nbytes / (ms_per_step * 1e-3) / 1e9
    line = {
        "metric": "drafted positions/s", "value": B * K / (ms_per_step * 1e-3), "unit": "positions/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": di.dtype, "data": "synthetic",
        "config": {"workload": f"draft: B={B} K={K} V={V} {di.dtype} drafter logits, tau={di.tau}",
                   "l2": "inputs larger than L2, no flush" if flush is None else "L2 flushed between steps"},
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None, "kernel": "draft_rows_kernel",
                     "peak_kind": peak_kind, "algorithmic_bytes_per_launch": nbytes,
                     "avg_launch_us": round(1e3 * ms_per_step, 2)},
        "step_ms_p10_p50_p90": [float(np.percentile(ms, q)) for q in (10, 50, 90)],
        "step_ms_how": "single steps, each bracketed by events (no overlap with the step before)",
        "ms_per_step_how": ("steps back to back between two events" if flush is None
                            else "mean of single steps bracketed by events, L2 flushed between them"),
        "mean_confidence": float(c.mean().item()),
        "clocks": clocks.summary(),
        "gpu_launches": args.steps,
    }
    print(json.dumps(line), flush=True)
    return 0


def run_markov(args):
    """The Markov head's sequential draw (spec_markov_draft): per position, a
    [B, r] x [r, V] bias contraction on the tensor cores fused with the draw.
    Synthetic base logits N(0, 3^2) and factors N(0, 0.2^2), bf16."""
    import torch
    import paper_2607_25852_gb300 as spec
    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    B, K, V, r = args.B or 64, 7, args.V or 201088, 256
    g = torch.Generator(device=device)
    g.manual_seed(1234)
    U = (torch.randn((B, K, V), generator=g, device=device) * 3.0).to(torch.bfloat16)
    W1 = (torch.randn((V, r), generator=g, device=device) * 0.2).to(torch.bfloat16)
    W2T = (torch.randn((V, r), generator=g, device=device) * 0.2).to(torch.bfloat16)
    x0 = torch.randint(0, V, (B,), generator=g, device=device, dtype=torch.int32)
    seeds = torch.arange(B, dtype=torch.int64, device=device) + 11
    rids = torch.arange(B, dtype=torch.int64, device=device) + 7000
    pos = torch.randint(0, 4096, (B,), generator=g, device=device, dtype=torch.int64)
    ws = spec.markov_workspace(B, K, V, r, device)
    z = torch.zeros((B, K), dtype=torch.int32, device=device)
    c = torch.zeros((B, K), device=device)
    sc = torch.zeros((B, K + 1), device=device)
    status = torch.zeros(1, dtype=torch.int32, device=device)
    stream = torch.cuda.current_stream()
    tau = args.tau

    def step():
        spec.spec_markov_draft(U, W1, W2T, x0, tau, seeds, rids, pos, z, c, ws, scores_out=sc, status=status)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    assert int(status.item()) == 0, "device reported an error"
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(0) as clocks:
        # steps back to back (each step's 2K + 1 launches chained as always)
        gpu_head_start(args.steps, host_us_per_step=200.0)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for k in range(args.steps):
            step()
        b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / args.steps
        # single steps, each bracketed by events: their spread
        gpu_head_start(args.steps, host_us_per_step=200.0)
        for k in range(args.steps):
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        torch.cuda.synchronize()
    ms1 = [a.elapsed_time(b) for a, b in ev]
    peak, peak_kind = measured_peak()
    # per position: the whole W2 (V x r) and the position's base logits (B x V)
    per_pos = V * r * 2 + B * V * 2
    achieved = per_pos * K / (ms * 1e-3) / 1e9
    flops = 2.0 * B * r * V * K
    line = {
        "metric": "drafted positions/s (Markov head)", "value": B * K / (ms * 1e-3), "unit": "positions/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"markov: B={B} requests, K={K} drafts (block of 8), V={V}, r={r}, tau={tau}",
                   "l2": "W2 (%.0f MB) is read once per position; it fits in L2 between positions" % (V * r * 2 / 1e6)},
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None, "kernel": "markov_bias_kernel + markov_pick_kernel",
                     "peak_kind": peak_kind, "algorithmic_bytes_per_position": per_pos,
                     "avg_step_us": round(ms * 1e3, 2)},
        "tensor_tflops": round(flops / (ms * 1e-3) / 1e12, 2),
        "per_position_us": round(ms * 1e3 / K, 2),
        "ms_per_step_how": "steps back to back between two events",
        "step_ms_p10_p50_p90": [float(np.percentile(ms1, q)) for q in (10, 50, 90)],
        "step_ms_how": "single steps, each bracketed by events (no overlap with the step before)",
        "clocks": clocks.summary(),
        "gpu_launches": (1 + 2 * K) * args.steps,
    }
    print(json.dumps(line), flush=True)
    return 0


def run_round_graph(args):
    """A round of allocate -> verify -> commit on the stress workload with the
    D-cut ratios 1/4..1 and the piecewise-linear cost 1 + 0.004 max(0, T - 256).
    (a) host-driven: the host reads T* after spec_allocate, then launches the
    graph of verify + commit captured for that shape; (b) device-selected: one
    host-launched graph allocates and tail-launches the graph of T*.  The
    packed logits of every candidate shape are prepared once beforehand (the
    target forward, which would write them, is not part of this library)."""
    import torch
    import paper_2607_25852_gb300 as spec
    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    wl = make_inputs(args, 0, device)
    B, K, V = wl.B, wl.K, wl.V
    Ts = spec.spec_budget_from_ratios(B, K, [1, 1, 3, 1], [4, 2, 4, 1])
    costs = [1.0 + 0.004 * max(0, T - 256) for T in Ts]
    st = Step(wl, device)
    st.ratios, st.costs = Ts, costs
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        st.spec.spec_allocate(wl.conf, Ts, costs, wl.last_tokens, wl.drafts, wl.pos_base, st.depth, st.row_off,
                              st.ptok, st.ppos, st.chosen, st.util, st.status)
    s.synchronize()
    T_star = int(st.chosen.item())
    m_star = Ts.index(T_star)
    lg = []
    for T in Ts:
        buf = torch.zeros((T, V), dtype=wl.logits.dtype, device=device)
        with torch.cuda.stream(s):
            spec.spec_pack_rows(wl.logits, B, K, st.row_off, buf, status=st.status)  # this allocation's packing
        lg.append(buf)
    hid = torch.zeros((T_star, wl.H), dtype=torch.bfloat16, device=device)
    with torch.cuda.stream(s):
        spec.spec_pack_rows(wl.hidden, B, K, st.row_off, hid, status=st.status)
    s.synchronize()

    def after(m):
        spec.spec_verify(lg[m], wl.drafts, wl.q, B, K, V, wl.temperature, wl.seeds, wl.request_ids, wl.pos_base,
                         st.acc, st.tok, st.ws, row_offsets=st.row_off, depth=st.depth, status=st.status)
        spec.spec_commit(st.acc, st.tok, hid if m == m_star else None, B, K, st.ctok, st.coff,
                         st.hout if m == m_star else None, row_offsets=st.row_off, status=st.status)

    def allocate():
        spec.spec_allocate(wl.conf, Ts, costs, wl.last_tokens, wl.drafts, wl.pos_base, st.depth, st.row_off,
                           st.ptok, st.ppos, st.chosen, st.util, st.status)

    children = []
    launched = torch.zeros(1, dtype=torch.int32, device=device)
    with torch.cuda.stream(s):
        for m in range(len(Ts)):
            spec.spec_graph_begin_capture(s)
            after(m)
            children.append(spec.spec_graph_end_capture(s, device_launch=True))
        spec.spec_graph_begin_capture(s)
        allocate()
        spec.spec_select_round(st.chosen, Ts, children, launched, st.status)
        parent = spec.spec_graph_end_capture(s, device_launch=False)

    def host_round():
        with torch.cuda.stream(s):
            allocate()
            s.synchronize()
            m = Ts.index(int(st.chosen.item()))
            spec.spec_graph_launch(children[m], s)
            s.synchronize()

    def device_round():
        spec.spec_graph_launch(parent, s)
        s.synchronize()

    def timed(fn, n):
        for _ in range(max(args.warmup, 3)):
            fn()
        t0 = time.perf_counter()
        for _ in range(n):
            fn()
        return (time.perf_counter() - t0) / n

    n = args.steps
    host_s = timed(host_round, n)
    dev_s = timed(device_round, n)
    # back to back (no host wait between rounds): device time per round
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clocks:
        with torch.cuda.stream(s):
            gpu_head_start(n, host_us_per_step=20.0)
        a.record(s)
        for _ in range(n):
            spec.spec_graph_launch(parent, s)
        b.record(s)
        s.synchronize()
    chain_ms = a.elapsed_time(b) / n
    assert int(st.status.item()) == 0 and int(launched.item()) == m_star
    for g in children + [parent]:
        spec.spec_graph_destroy(g)
    line = {
        "metric": "round latency (allocate + verify + commit)", "value": dev_s * 1e6, "unit": "us",
        "n_gpus": 1, "steps": n, "warmup": args.warmup, "ms_per_step": dev_s * 1e3, "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": f"{wl.name}: B={B} K={K} V={V} {wl.dtype} logits, t={wl.temperature}; D-cut ratios "
                               f"1/4..1, cost 1 + 0.004 max(0, T - 256): T* = {T_star} of {Ts}",
                   "candidate_graphs": len(Ts)},
        "host_driven_round_us": round(host_s * 1e6, 2),
        "device_selected_round_us": round(dev_s * 1e6, 2),
        "device_selected_back_to_back_us": round(chain_ms * 1e3, 2),
        "saved_per_round_us": round((host_s - dev_s) * 1e6, 2),
        "how": "wall clock per round with a host wait at its end; back to back: CUDA events over consecutive "
               "parent-graph launches",
        "clocks": clocks.summary(),
        "gpu_launches": 6 * n,
    }
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.round_graph:
        return run_round_graph(args)
    if args.markov:
        return run_markov(args)
    if args.draft:
        return run_draft(args)
    if args.shards > 1:
        return run_sharded(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
