"""Host-side checks of the C ABI that need no GPU: the library builds and
loads, exports every function include/spec.h declares, and rejects bad
arguments synchronously (before any CUDA call)."""
import ctypes
import os
import re
from fractions import Fraction
from math import ceil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "spec.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_25852_gb300 import build
    build.build()
    from paper_2607_25852_gb300 import _native
    return _native.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(spec_[a-z_]+)\s*\(", text, re.M)
    return sorted(set(names))


def test_every_declared_function_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 9, names
    from paper_2607_25852_gb300 import _native
    assert sorted(_native.SIGNATURES) == names
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_error_strings(lib):
    import paper_2607_25852_gb300 as spec
    assert spec.spec_version() == 1
    assert "bad input" in spec.spec_error_string(spec.ERR_BAD_INPUT)
    assert spec.spec_error_string(99) == "unknown error code"


def test_budget_from_ratios_is_exact(lib):
    import paper_2607_25852_gb300 as spec
    for B, K in [(1, 0), (3, 0), (4, 8), (5, 8), (64, 16), (7, 255)]:
        num, den = [1, 1, 3, 1, 0, 2, 5], [4, 2, 4, 1, 3, 3, 7]
        got = spec.spec_budget_from_ratios(B, K, num, den)
        want = [max(B, ceil(Fraction(n, d) * B * (K + 1))) for n, d in zip(num, den)]
        assert got == want
    for bad in ([1], [0]), ([2], [1]), ([-1], [2]):
        with pytest.raises(spec.SpecError):
            spec.spec_budget_from_ratios(4, 3, *bad)


def test_workspace_sizes(lib):
    import paper_2607_25852_gb300 as spec
    assert spec.spec_verify_workspace(0, 4, 100) == 0
    assert spec.spec_verify_workspace(4, 256, 100) == 0
    assert spec.spec_verify_workspace(4, 4, 1 << 30) == 0
    n = spec.spec_verify_workspace(64, 16, 201088)
    assert n > 0 and n % 256 == 0 and n < (1 << 20)
    assert spec.spec_allocate_workspace(64, 16, 4) == 0


def test_argument_errors_return_before_any_launch(lib):
    dummy = ctypes.c_void_p(16)          # never dereferenced: every call below fails its checks
    ws = ctypes.c_void_p(256)
    stream = ctypes.c_void_p(0)
    v = lambda B, K, V, t, ws_bytes=1 << 20, dt=0: lib.spec_verify(
        dummy, dt, None, None, dummy, None, 0, B, K, V, t, dummy, dummy, dummy, dummy, dummy,
        None, None, None, ws, ws_bytes, stream)
    assert v(0, 4, 100, 1.0) == 1
    assert v(4, 4, 0, 1.0) == 1
    assert v(4, 256, 100, 1.0) == 1
    assert v(4, 4, 100, -1.0) == 1
    assert v(4, 4, 100, float("nan")) == 1
    assert v(4, 4, 100, float("inf")) == 1
    assert v(4, 4, 100, 1.0, dt=7) == 1
    assert v(4, 4, 100, 1.0, ws_bytes=8) == 2
    assert lib.spec_verify(dummy, 0, None, None, dummy, None, 0, 4, 4, 100, 1.0, dummy, dummy, dummy,
                           dummy, dummy, None, None, None, ctypes.c_void_p(264), 1 << 20, stream) == 2
    a = lambda T, C, B=2, K=2: lib.spec_allocate(
        dummy, B, K, (ctypes.c_int32 * 1)(T), (ctypes.c_double * 1)(C), 1, dummy, dummy, dummy,
        dummy, dummy, dummy, dummy, dummy, None, None, None, 0, stream)
    assert a(1, 1.0) == 1 and a(7, 1.0) == 1 and a(4, 0.0) == 1 and a(4, float("nan")) == 1
    assert a(8193, 1.0, B=8193, K=0) == 1
    c = lambda B, K, hidden, hout, H=8, dt=0: lib.spec_commit(
        dummy, dummy, None, hidden, dt, B, K, H, dummy, dummy, hout, None, stream)
    assert c(0, 2, None, None) == 1
    assert c(2, 2, dummy, None) == 1
    assert c(2, 2, dummy, dummy, H=0) == 1
    assert c(2, 2, dummy, dummy, dt=3) == 1
    assert lib.spec_profile_stream_pass(dummy, None) == 1
    assert lib.spec_check_bounded_wait(None, stream) == 1  # no status word


def test_shard_workspace_and_argument_errors(lib):
    import paper_2607_25852_gb300 as spec
    assert spec.spec_shard_workspace(0, 4, 1024) == 0
    assert spec.spec_shard_workspace(4, 256, 1024) == 0
    n = spec.spec_shard_workspace(64, 16, 201088 // 8)
    assert n > 0 and n % 256 == 0 and n < (1 << 20)
    dummy = ctypes.c_void_p(16)          # never dereferenced: every call below fails its checks
    ws = ctypes.c_void_p(256)
    stream = ctypes.c_void_p(0)
    st = lambda V, vb, Vs, t=1.0, ws_bytes=1 << 20, out=dummy: lib.spec_shard_stats(
        dummy, 0, None, None, dummy, None, 0, 4, 3, V, vb, Vs, t, dummy, out, None, ws, ws_bytes,
        stream)
    assert st(5000, 4096, 1024) == 1       # past V
    assert st(5000, -1, 1024) == 1
    assert st(5000, 0, 0) == 1
    assert st(5000, 0, 1024, t=-1.0) == 1
    assert st(5000, 0, 1024, ws_bytes=8) == 2
    assert st(5000, 0, 1024, out=ctypes.c_void_p(24)) == 1   # records not 16-byte aligned
    d = lambda S, t, dec=dummy: lib.spec_shard_decide(
        dummy, S, None, None, dummy, 0, 4, 3, 5000, t, dummy, dummy, dummy, dummy, dummy, None, None,
        dec, None, stream)
    assert d(0, 1.0) == 1 and d(2, -1.0) == 1 and d(2, 1.0, dec=None) == 1
    s = lambda vb, Vs, t: lib.spec_shard_sample(
        dummy, 0, None, 0, dummy, 4, 3, 5000, vb, Vs, t, dummy, dummy, dummy, None, ws, 1 << 20, stream)
    assert s(4500, 1024, 1.0) == 1
    assert s(0, 1024, 0.0) == 0            # nothing to sample at t = 0: no launch
    f = lambda S, t: lib.spec_shard_finish(dummy, S, dummy, 4, 3, 5000, t, dummy, dummy, dummy, dummy,
                                           None, stream)
    assert f(0, 1.0) == 1 and f(2, 0.0) == 0


def test_draft_workspace_and_argument_errors(lib):
    import paper_2607_25852_gb300 as spec
    assert spec.spec_draft_workspace(0, 4, 100) == 0
    assert spec.spec_draft_workspace(4, 0, 100) == 0
    assert spec.spec_draft_workspace(4, 256, 100) == 0
    n = spec.spec_draft_workspace(64, 16, 201088)
    assert n > 0 and n % 256 == 0 and n < (1 << 20)
    dummy = ctypes.c_void_p(16)          # never dereferenced: every call below fails its checks
    stream = ctypes.c_void_p(0)
    d = lambda B, K, V, tau, ws=ctypes.c_void_p(256), ws_bytes=1 << 20, dt=0, stats=None: lib.spec_draft(
        dummy, dt, B, K, V, tau, dummy, dummy, dummy, dummy, dummy, None, stats, None, ws, ws_bytes, stream)
    assert d(0, 4, 100, 1.0) == 1
    assert d(4, 0, 100, 1.0) == 1
    assert d(4, 4, 0, 1.0) == 1
    assert d(4, 4, 100, -1.0) == 1 and d(4, 4, 100, float("nan")) == 1 and d(4, 4, 100, float("inf")) == 1
    assert d(4, 4, 100, 1.0, dt=5) == 1
    assert d(4, 4, 100, 1.0, stats=ctypes.c_void_p(20)) == 1     # row stats not 8-byte aligned
    assert d(4, 4, 100, 1.0, ws_bytes=8) == 2
    assert d(4, 4, 100, 1.0, ws=ctypes.c_void_p(264)) == 2


def test_markov_workspace_and_argument_errors(lib):
    """spec_markov_draft's shape, dtype, temperature, pointer and workspace
    checks fail before any CUDA launch."""
    import paper_2607_25852_gb300 as spec
    ws_size = lib.spec_markov_workspace
    for B, K, V, r in [(0, 7, 1000, 64), (129, 7, 1000, 64), (4, 0, 1000, 64), (4, 7, 0, 64), (4, 7, 1000, 32),
                       (4, 7, 1000, 100), (4, 7, 1000, 320)]:
        assert ws_size(B, K, V, r) == 0, (B, K, V, r)
    n = ws_size(64, 7, 201088, 256)
    assert n > 0 and n % 256 == 0 and n < (64 << 20)
    assert ws_size(128, 7, 201088, 256) > n                        # partials scale with B
    dummy = ctypes.c_void_p(16)                                    # never dereferenced: every call fails a check
    stream = ctypes.c_void_p(0)

    def d(B=4, K=3, V=1000, r=64, tau=1.0, dt=0, w1=dummy, w2=dummy, stats=None, ws=ctypes.c_void_p(256),
          ws_bytes=1 << 24, U=dummy):
        return lib.spec_markov_draft(U, dt, w1, w2, r, dummy, B, K, V, tau, dummy, dummy, dummy, dummy, dummy, None,
                                     stats, None, ws, ws_bytes, stream)
    assert d(B=0) == 1 and d(B=129) == 1 and d(K=0) == 1 and d(V=0) == 1
    assert d(r=0) == 1 and d(r=96) == 1 and d(r=512) == 1
    assert d(tau=-0.5) == 1 and d(tau=float("nan")) == 1 and d(tau=float("inf")) == 1
    assert d(dt=1) == 1                                             # U must be bf16
    assert d(U=None) == 1 and d(w1=None) == 1 and d(w2=None) == 1
    assert d(w1=ctypes.c_void_p(24)) == 1 and d(w2=ctypes.c_void_p(40)) == 1   # 16-byte alignment
    assert d(stats=ctypes.c_void_p(20)) == 1                        # row stats not 8-byte aligned
    assert d(ws_bytes=8) == 2                                       # workspace too small
    assert d(ws=ctypes.c_void_p(264)) == 2                          # workspace not 256-aligned
    assert d(ws=None) == 2


def test_round_graph_and_pack_rows_argument_errors(lib):
    """The graph helpers, spec_select_round and spec_pack_rows reject bad
    arguments before any CUDA call."""
    from paper_2607_25852_gb300 import _native
    hdr = open(HEADER).read()
    max_cand = int(re.search(r"#define SPEC_MAX_CANDIDATES\s+(\d+)", hdr).group(1))
    max_drafts = int(re.search(r"#define SPEC_MAX_DRAFTS\s+(\d+)", hdr).group(1))
    dummy = ctypes.c_void_p(16)                 # never dereferenced: every call fails a check
    stream = ctypes.c_void_p(0)
    assert lib.spec_graph_begin_capture(None) == 1          # the legacy stream cannot be captured
    assert lib.spec_graph_end_capture(stream, 0, None) == 1
    assert lib.spec_graph_launch(None, stream) == 1
    assert lib.spec_graph_destroy(None) == 0                # destroying nothing is fine
    cand = (ctypes.c_int32 * 2)(8, 16)
    graphs_ok = (ctypes.c_void_p * 2)(16, 32)
    graphs_hole = (ctypes.c_void_p * 2)(16, None)
    sel = lambda chosen, M, c, g: lib.spec_select_round(chosen, M, c, g, None, None, stream)
    assert sel(None, 2, cand, graphs_ok) == 1
    assert sel(dummy, 0, cand, graphs_ok) == 1
    assert sel(dummy, max_cand + 1, cand, graphs_ok) == 1
    assert sel(dummy, 2, None, graphs_ok) == 1
    assert sel(dummy, 2, cand, None) == 1
    assert sel(dummy, 2, cand, graphs_hole) == 1            # every candidate needs a graph
    pk = lambda src=dummy, rb=64, B=4, K=3, offs=dummy, dst=dummy, R=8: lib.spec_pack_rows(
        src, rb, B, K, offs, dst, R, None, stream)
    assert pk(src=None) == 1 and pk(dst=None) == 1 and pk(offs=None) == 1
    assert pk(rb=0) == 1 and pk(B=0) == 1 and pk(K=-1) == 1 and pk(K=max_drafts + 1) == 1 and pk(R=0) == 1
    assert _native.SIGNATURES["spec_pack_rows"][1][1] is ctypes.c_size_t


def test_pointer_readability_without_a_device(lib):
    """No pointer is promised device-readable when the query fails (no GPU
    here) or the pointer is NULL."""
    assert lib.spec_pointer_device_readable(None) == 0
    buf = ctypes.create_string_buffer(64)
    assert lib.spec_pointer_device_readable(ctypes.cast(buf, ctypes.c_void_p)) in (0, 1)
