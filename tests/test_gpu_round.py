"""A round per candidate budget as CUDA graphs, the budget chosen on the
device (Section 4.3: one graph per reachable verification shape; the budget
choice off the host's critical path).  Each candidate's graph packs the rows
(standing in for the target forward), verifies and commits; a host-launched
parent graph allocates and tail-launches the graph of the chosen budget.  The
results must equal those of the same calls made directly from the host, and
those of the oracle: the allocation and the commit bit for bit, the
verification under the parity rules of the other verification tests."""
import numpy as np
import pytest
import torch

import oracle
import workloads
import paper_2607_25852_gb300 as spec
from parity import bits, compare, run_oracle

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


class Round:
    """Buffers of one round on the alloc workload (by default V = 8192,
    H = 128, the paper's ratios 1/4, 1/2, 3/4, 1; `sweep`: the budgets
    T = 64, 128, ..., 1024)."""

    def __init__(self, t=1.0, V=8192, H=128, sweep=False):
        wl = workloads.make("alloc", V=V, H=H, device=DEV)
        self.wl, self.t = wl, t
        B, K, V, H = wl.B, wl.K, wl.V, wl.H
        if sweep:
            self.Ts = [int(x) for x in workloads.budget_candidates(B, K)[0]]
        else:
            self.Ts = spec.spec_budget_from_ratios(B, K, [1, 1, 3, 1], [4, 2, 4, 1])
        z = lambda *s, dt=torch.int32: torch.zeros(s, dtype=dt, device=DEV)
        self.depth, self.row_off = z(B), z(B + 1)
        self.ptok, self.ppos = z(B * (K + 1)), z(B * (K + 1), dt=torch.int64)
        self.chosen, self.launched = z(1), z(1)
        self.util = z(len(self.Ts), dt=torch.float64)
        self.acc, self.tok = z(B), z(B, K + 1)
        self.pdr = z(B, K, dt=torch.float32)
        self.rst = z(B * (K + 1), 2, dt=torch.float32)
        self.ctok, self.coff = z(B * (K + 1)), z(B + 1)
        self.hout = torch.zeros((B * (K + 1), H), dtype=torch.bfloat16, device=DEV)
        self.status = z(1)
        self.ws = spec.verify_workspace(B, K, V, DEV)
        # per candidate: the packed target outputs at that shape
        self.lg = [torch.zeros((T, V), dtype=wl.logits.dtype, device=DEV) for T in self.Ts]
        self.hid = [torch.zeros((T, H), dtype=torch.bfloat16, device=DEV) for T in self.Ts]

    def allocate(self, costs):
        wl = self.wl
        spec.spec_allocate(wl.conf, self.Ts, costs, wl.last_tokens, wl.drafts, wl.pos_base, self.depth,
                           self.row_off, self.ptok, self.ppos, self.chosen, self.util, self.status)

    def after_allocation(self, m):
        """What follows the allocation at shape T_m."""
        wl = self.wl
        B, K, V = wl.B, wl.K, wl.V
        spec.spec_pack_rows(wl.logits, B, K, self.row_off, self.lg[m], status=self.status)
        spec.spec_pack_rows(wl.hidden, B, K, self.row_off, self.hid[m], status=self.status)
        spec.spec_verify(self.lg[m], wl.drafts, None, B, K, V, self.t, wl.seeds, wl.request_ids, wl.pos_base,
                         self.acc, self.tok, self.ws, row_offsets=self.row_off, depth=self.depth,
                         p_draft_out=self.pdr, row_stats_out=self.rst, status=self.status)
        spec.spec_commit(self.acc, self.tok, self.hid[m], B, K, self.ctok, self.coff, self.hout,
                         row_offsets=self.row_off, status=self.status)

    def outputs(self):
        torch.cuda.synchronize()
        return {k: getattr(self, k).cpu().numpy().copy() for k in
                ("depth", "row_off", "chosen", "acc", "tok", "pdr", "rst", "ctok", "coff", "status")} | \
               {"hout": self.hout.view(torch.int16).cpu().numpy().copy()}

    def reset_outputs(self):
        for k in ("acc", "tok", "pdr", "rst", "ctok", "coff", "status", "launched"):
            getattr(self, k).fill_(-5 if k != "status" else 0)
        self.hout.zero_()
        torch.cuda.synchronize()


def _costs_choosing(m, Ts):
    """A cost table whose utility / cost maximiser is candidate m."""
    return [1.0 if c == m else 1e6 for c in range(len(Ts))]


def _capture_children(rnd, stream):
    graphs = []
    for m in range(len(rnd.Ts)):
        with torch.cuda.stream(stream):
            spec.spec_graph_begin_capture(stream)
            rnd.after_allocation(m)
            graphs.append(spec.spec_graph_end_capture(stream, device_launch=True))
    return graphs


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_device_selected_round_matches_host_driven_round(t):
    rnd = Round(t)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graphs = _capture_children(rnd, s)
    try:
        for m in range(len(rnd.Ts)):
            costs = _costs_choosing(m, rnd.Ts)
            # host-driven: allocate, read T* on the host, then the rest
            rnd.reset_outputs()
            with torch.cuda.stream(s):
                rnd.allocate(costs)
                s.synchronize()
                mh = rnd.Ts.index(int(rnd.chosen.item()))
                assert mh == m
                rnd.after_allocation(mh)
            want = rnd.outputs()
            assert want["status"][0] == 0
            # device-selected: one parent graph per cost table
            rnd.reset_outputs()
            with torch.cuda.stream(s):
                spec.spec_graph_begin_capture(s)
                rnd.allocate(costs)
                spec.spec_select_round(rnd.chosen, rnd.Ts, graphs, rnd.launched, rnd.status)
                parent = spec.spec_graph_end_capture(s, device_launch=False)
                try:
                    for _ in range(2):          # replays are identical
                        spec.spec_graph_launch(parent, s)
                        s.synchronize()
                        got = rnd.outputs()
                        assert int(rnd.launched.item()) == m
                        for k, v in want.items():
                            assert np.array_equal(got[k], v), (m, k)
                finally:
                    spec.spec_graph_destroy(parent)
    finally:
        for g in graphs:
            spec.spec_graph_destroy(g)


def _assert_matches_oracle(rnd, got, costs):
    """The device-selected round's outputs against the oracle's round:
    allocation, verification of the packed rows, commit."""
    wl, t = rnd.wl, rnd.t
    B, K = wl.B, wl.K
    cpu = lambda x: x.detach().cpu()
    a = oracle.allocate(cpu(wl.conf).numpy(), rnd.Ts, costs, cpu(wl.last_tokens).numpy(), cpu(wl.drafts).numpy(),
                        cpu(wl.pos_base).numpy())
    assert int(got["chosen"][0]) == a["chosen_T"]
    assert got["depth"].tolist() == a["depth"].tolist()
    assert got["row_off"].tolist() == a["row_offsets"].tolist()
    depth = torch.as_tensor(a["depth"])
    offs = torch.as_tensor(a["row_offsets"])
    logits = workloads.pack_rows(cpu(wl.logits), B, K, depth)
    hidden = workloads.pack_rows(cpu(wl.hidden), B, K, depth)
    ref = run_oracle(logits, cpu(wl.drafts), None, t, cpu(wl.seeds), cpu(wl.request_ids), cpu(wl.pos_base),
                     row_offsets=offs, depth=depth)
    R = int(offs[-1])
    gpu = dict(accepted=got["acc"], tokens=got["tok"], p_draft=got["pdr"], row_stats=got["rst"][:R],
               status=int(got["status"][0]))
    assert gpu["status"] == 0 and (ref["status"] == 0).all()
    compare(gpu, ref, K, t, depth=depth.numpy(), row_offsets=offs.numpy())
    # the commit of the GPU's decisions (equal to the oracle's but at counted near ties)
    c = oracle.commit(got["acc"], got["tok"], offs.numpy(), bits(hidden))
    assert got["coff"].tolist() == c["commit_offsets"].tolist()
    assert got["ctok"][:c["total"]].tolist() == c["packed_tokens"][:c["total"]].tolist()
    assert np.array_equal(got["hout"][:c["total"]].view(np.uint16), c["hidden"])


@pytest.mark.parametrize("t", [0.0, 1.0])
def test_device_selected_round_matches_oracle(t):
    """Every candidate budget of the paper's ratios, chosen and launched on the
    device, against the oracle's round."""
    rnd = Round(t)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graphs = _capture_children(rnd, s)
    try:
        for m in range(len(rnd.Ts)):
            costs = _costs_choosing(m, rnd.Ts)
            rnd.reset_outputs()
            with torch.cuda.stream(s):
                spec.spec_graph_begin_capture(s)
                rnd.allocate(costs)
                spec.spec_select_round(rnd.chosen, rnd.Ts, graphs, rnd.launched, rnd.status)
                parent = spec.spec_graph_end_capture(s, device_launch=False)
                try:
                    spec.spec_graph_launch(parent, s)
                    s.synchronize()
                finally:
                    spec.spec_graph_destroy(parent)
            assert int(rnd.launched.item()) == m
            _assert_matches_oracle(rnd, rnd.outputs(), costs)
    finally:
        for g in graphs:
            spec.spec_graph_destroy(g)


def test_alloc_workload_at_full_vocabulary():
    """The alloc workload at its stated size -- B = 64, K = 16, V = 128256,
    t = 1 with one-hot q (Section 4.2's deterministic-draft protocol), the
    sixteen budgets T = 64..1024 with the profiled cost 1 + 0.004 max(0,
    T - 256) -- as one device-selected round, against the oracle."""
    rnd = Round(1.0, V=128256, H=64, sweep=True)
    costs = [float(x) for x in workloads.budget_candidates(rnd.wl.B, rnd.wl.K)[1]]
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graphs = _capture_children(rnd, s)
    try:
        rnd.reset_outputs()
        with torch.cuda.stream(s):
            spec.spec_graph_begin_capture(s)
            rnd.allocate(costs)
            spec.spec_select_round(rnd.chosen, rnd.Ts, graphs, rnd.launched, rnd.status)
            parent = spec.spec_graph_end_capture(s, device_launch=False)
            try:
                spec.spec_graph_launch(parent, s)
                s.synchronize()
            finally:
                spec.spec_graph_destroy(parent)
        got = rnd.outputs()
        T = int(got["chosen"][0])
        assert rnd.Ts.index(T) == int(rnd.launched.item())
        assert 64 < T < 1024                      # the cost table puts the optimum inside the sweep
        _assert_matches_oracle(rnd, got, costs)
    finally:
        for g in graphs:
            spec.spec_graph_destroy(g)


def test_budget_outside_the_captured_shapes_is_refused():
    rnd = Round(1.0)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graphs = _capture_children(rnd, s)
    try:
        rnd.reset_outputs()
        with torch.cuda.stream(s):
            spec.spec_graph_begin_capture(s)
            rnd.allocate(_costs_choosing(3, rnd.Ts))             # T* = the full block ...
            spec.spec_select_round(rnd.chosen, rnd.Ts[:3], graphs[:3], rnd.launched, rnd.status)  # ... not captured
            parent = spec.spec_graph_end_capture(s, device_launch=False)
            spec.spec_graph_launch(parent, s)
            s.synchronize()
            spec.spec_graph_destroy(parent)
        assert int(rnd.launched.item()) == -1
        assert int(rnd.status.item()) == spec.ERR_BAD_INPUT
        assert (rnd.acc.cpu() == -5).all()                     # nothing after the allocation ran
    finally:
        for g in graphs:
            spec.spec_graph_destroy(g)


def test_pack_rows_matches_the_allocation():
    rnd = Round(1.0)
    wl = rnd.wl
    B, K = wl.B, wl.K
    rnd.allocate(_costs_choosing(1, rnd.Ts))
    torch.cuda.synchronize()
    T = int(rnd.chosen.item())
    dst = torch.full((T + 3, wl.H), 7.0, dtype=torch.bfloat16, device=DEV)
    spec.spec_pack_rows(wl.hidden, B, K, rnd.row_off, dst, status=rnd.status)
    want = workloads.pack_rows(wl.hidden, B, K, rnd.depth.cpu())
    torch.cuda.synchronize()
    assert torch.equal(dst[:T].cpu(), want.cpu())
    assert (dst[T:].float() == 7.0).all()
