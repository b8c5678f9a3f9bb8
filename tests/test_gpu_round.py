"""A round per candidate budget as CUDA graphs, the budget chosen on the
device (Section 4.3: one graph per reachable verification shape; the budget
choice off the host's critical path).  Each candidate's graph packs the rows
(standing in for the target forward), verifies and commits; a host-launched
parent graph allocates and tail-launches the graph of the chosen budget.  The
results must equal those of the same calls made directly from the host."""
import numpy as np
import pytest
import torch

import workloads
import paper_2607_25852_gb300 as spec

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


class Round:
    """Buffers of one round on the alloc workload (V = 8192, H = 128)."""

    def __init__(self, t=1.0):
        wl = workloads.make("alloc", V=8192, H=128, device=DEV)
        self.wl, self.t = wl, t
        B, K, V, H = wl.B, wl.K, wl.V, wl.H
        self.Ts = spec.spec_budget_from_ratios(B, K, [1, 1, 3, 1], [4, 2, 4, 1])
        z = lambda *s, dt=torch.int32: torch.zeros(s, dtype=dt, device=DEV)
        self.depth, self.row_off = z(B), z(B + 1)
        self.ptok, self.ppos = z(B * (K + 1)), z(B * (K + 1), dt=torch.int64)
        self.chosen, self.launched = z(1), z(1)
        self.util = z(len(self.Ts), dt=torch.float64)
        self.acc, self.tok = z(B), z(B, K + 1)
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
                         self.acc, self.tok, self.ws, row_offsets=self.row_off, depth=self.depth, status=self.status)
        spec.spec_commit(self.acc, self.tok, self.hid[m], B, K, self.ctok, self.coff, self.hout,
                         row_offsets=self.row_off, status=self.status)

    def outputs(self):
        torch.cuda.synchronize()
        return {k: getattr(self, k).cpu().numpy().copy() for k in
                ("depth", "row_off", "chosen", "acc", "tok", "ctok", "coff", "status")} | \
               {"hout": self.hout.view(torch.int16).cpu().numpy().copy()}

    def reset_outputs(self):
        for k in ("acc", "tok", "ctok", "coff", "status", "launched"):
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
