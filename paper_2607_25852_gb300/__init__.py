"""GB300 (sm_103a) batched speculative verification: Python binding of libspec.

The functions below carry the names of the C ABI in ``include/spec.h`` and do
argument marshalling only (torch tensors -> device pointers, the current torch
stream -> cudaStream_t, error codes -> exceptions).  Every step of the path runs
in the CUDA kernels of ``libspec.so``; there is no CPU fallback.

Round of arxiv 2607.25852 (AngelSpec): ``spec_allocate`` (D-cut, Section 4.2)
-> target forward over the packed rows (caller) -> ``spec_verify`` (rejection
sampling, Section 1) -> ``spec_commit`` (packing for the next drafting step).
"""
import ctypes

import torch

from . import _native

BF16 = 0
F32 = 1

OK = 0
ERR_INVALID_ARG = 1
ERR_WORKSPACE = 2
ERR_CUDA = 3
ERR_BAD_INPUT = 4
ERR_TIMEOUT = 5
ERR_TOO_LARGE = 6

MAX_DRAFTS = 255
MAX_ALLOC_POSITIONS = 8192
MAX_CANDIDATES = 64

SHARD_STAT_BYTES = 32
SHARD_DECISION_BYTES = 32
SHARD_RACE_BYTES = 96

__all__ = [
    "SpecError", "spec_version", "spec_error_string", "spec_budget_from_ratios",
    "spec_allocate_workspace", "spec_allocate", "spec_verify_workspace", "spec_verify",
    "spec_verify_static", "spec_commit", "spec_profile_stream_pass", "verify_workspace", "library",
    "spec_shard_workspace", "spec_shard_stats", "spec_shard_decide", "spec_shard_sample",
    "spec_shard_finish", "shard_workspace", "spec_draft_workspace", "spec_draft", "draft_workspace",
    "spec_graph_begin_capture", "spec_graph_end_capture", "spec_graph_launch", "spec_graph_destroy",
    "spec_select_round", "spec_pack_rows", "spec_markov_workspace", "spec_markov_draft", "markov_workspace",
    "spec_pointer_device_readable", "spec_check_bounded_wait",
]


class SpecError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {spec_error_string(code)} (code {code})")


def library():
    """The loaded ctypes handle of libspec.so."""
    return _native.load()


def _ptr(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch.Tensor or None")
    if not t.is_contiguous():
        raise ValueError("tensors passed to libspec must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _dtype(t):
    if t is None:
        return BF16
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported element type {t.dtype} (bf16 or fp32)")


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(code, where):
    if code != OK:
        raise SpecError(code, where)


def spec_version() -> int:
    return library().spec_version()


def spec_error_string(code: int) -> str:
    return library().spec_error_string(code).decode()


def spec_pointer_device_readable(t) -> bool:
    """True if the library's kernels may read tensor t in place: device
    memory, or pinned host memory mapped at the same address (read over the
    CPU-GPU link with no staging copy)."""
    return bool(library().spec_pointer_device_readable(_ptr(t)))


def spec_budget_from_ratios(B: int, K: int, num, den):
    """Eq. (dcut-budget) for ratios num/den; host integers in, list out."""
    M = len(num)
    n = (ctypes.c_int32 * M)(*num)
    d = (ctypes.c_int32 * M)(*den)
    out = (ctypes.c_int32 * M)()
    _check(library().spec_budget_from_ratios(B, K, n, d, M, out), "spec_budget_from_ratios")
    return list(out)


def spec_allocate_workspace(B: int, K: int, M: int) -> int:
    return library().spec_allocate_workspace(B, K, M)


def spec_allocate(conf, cand_T, cand_cost, last_tokens, draft_tokens, pos_base, depth_out,
                  row_offsets_out, packed_tokens_out, packed_pos_out, chosen_T_out,
                  utility_out=None, status=None, ws=None, stream=None):
    """conf [B, K] fp32 device; cand_T / cand_cost host sequences; see spec.h."""
    B, K = conf.shape
    M = len(cand_T)
    T = (ctypes.c_int32 * M)(*[int(x) for x in cand_T])
    C = (ctypes.c_double * M)(*[float(x) for x in cand_cost])
    code = library().spec_allocate(
        _ptr(conf), B, K, T, C, M, _ptr(last_tokens), _ptr(draft_tokens), _ptr(pos_base),
        _ptr(depth_out), _ptr(row_offsets_out), _ptr(packed_tokens_out), _ptr(packed_pos_out),
        _ptr(chosen_T_out), _ptr(utility_out), _ptr(status), _ptr(ws),
        0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))
    _check(code, "spec_allocate")


def spec_verify_workspace(B: int, K: int, V: int) -> int:
    return library().spec_verify_workspace(B, K, V)


def verify_workspace(B: int, K: int, V: int, device="cuda"):
    """A zero-filled workspace tensor of the size spec_verify needs."""
    n = spec_verify_workspace(B, K, V)
    if n == 0:
        raise SpecError(ERR_INVALID_ARG, "spec_verify_workspace")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def spec_verify(logits, draft_tokens, q, B, K, V, temperature, seeds, request_ids, pos_base,
                accepted_len_out, out_tokens, ws, row_offsets=None, depth=None, p_draft_out=None,
                row_stats_out=None, status=None, stream=None):
    """logits [R, V] bf16/fp32, q [B, K, V] or None; seeds/request_ids int64 (uint64 bits)."""
    code = library().spec_verify(
        _ptr(logits), _dtype(logits), _ptr(row_offsets), _ptr(depth), _ptr(draft_tokens),
        _ptr(q), _dtype(q), B, K, V, float(temperature), _ptr(seeds), _ptr(request_ids),
        _ptr(pos_base), _ptr(accepted_len_out), _ptr(out_tokens), _ptr(p_draft_out),
        _ptr(row_stats_out), _ptr(status), _ptr(ws), ws.numel() * ws.element_size(),
        _stream(stream))
    _check(code, "spec_verify")


def spec_verify_static(logits, draft_tokens, q, B, K, V, temperature, seeds, request_ids,
                       pos_base, accepted_len_out, out_tokens, row_offsets=None, depth=None,
                       p_draft_out=None, row_stats_out=None, status=None, stream=None):
    """spec_verify without a workspace argument, for callers that may not
    allocate device memory (the scratch is a static array of the library)."""
    code = library().spec_verify_static(
        _ptr(logits), _dtype(logits), _ptr(row_offsets), _ptr(depth), _ptr(draft_tokens),
        _ptr(q), _dtype(q), B, K, V, float(temperature), _ptr(seeds), _ptr(request_ids),
        _ptr(pos_base), _ptr(accepted_len_out), _ptr(out_tokens), _ptr(p_draft_out),
        _ptr(row_stats_out), _ptr(status), _stream(stream))
    _check(code, "spec_verify_static")


def spec_commit(accepted_len, out_tokens, hidden, B, K, packed_tokens_out, commit_offsets_out,
                hidden_out=None, row_offsets=None, status=None, stream=None):
    """hidden [R, H] bf16/fp32 or None; see spec.h."""
    H = 0 if hidden is None else hidden.shape[-1]
    code = library().spec_commit(
        _ptr(accepted_len), _ptr(out_tokens), _ptr(row_offsets), _ptr(hidden), _dtype(hidden),
        B, K, H, _ptr(packed_tokens_out), _ptr(commit_offsets_out), _ptr(hidden_out),
        _ptr(status), _stream(stream))
    _check(code, "spec_commit")


def spec_markov_workspace(B: int, K: int, V: int, r: int) -> int:
    return library().spec_markov_workspace(B, K, V, r)


def markov_workspace(B: int, K: int, V: int, r: int, device="cuda"):
    n = spec_markov_workspace(B, K, V, r)
    if n == 0:
        raise SpecError(ERR_INVALID_ARG, "spec_markov_workspace")
    return torch.empty(n, dtype=torch.uint8, device=device)


def spec_markov_draft(U, W1, W2T, x0, tau, seeds, request_ids, pos_base, drafts_out, conf_out, ws,
                      scores_out=None, row_stats_out=None, status=None, stream=None):
    """U [B, K, V] bf16; W1 and W2T [V, r] bf16 (W2T = W2 transposed); x0 [B] int32."""
    B, K, V = U.shape
    r = W1.shape[1]
    code = library().spec_markov_draft(
        _ptr(U), _dtype(U), _ptr(W1), _ptr(W2T), r, _ptr(x0), B, K, V, float(tau), _ptr(seeds),
        _ptr(request_ids), _ptr(pos_base), _ptr(drafts_out), _ptr(conf_out), _ptr(scores_out),
        _ptr(row_stats_out), _ptr(status), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(code, "spec_markov_draft")


def spec_graph_begin_capture(stream):
    """Begin capturing `stream` (a torch.cuda.Stream, not the default stream)."""
    _check(library().spec_graph_begin_capture(_stream(stream)), "spec_graph_begin_capture")


def spec_graph_end_capture(stream, device_launch: bool):
    """End the capture; returns the instantiated graph handle (an int)."""
    out = ctypes.c_void_p()
    _check(library().spec_graph_end_capture(_stream(stream), int(bool(device_launch)), ctypes.byref(out)),
           "spec_graph_end_capture")
    return out.value


def spec_graph_launch(graph, stream=None):
    _check(library().spec_graph_launch(ctypes.c_void_p(graph), _stream(stream)), "spec_graph_launch")


def spec_graph_destroy(graph):
    _check(library().spec_graph_destroy(ctypes.c_void_p(graph)), "spec_graph_destroy")


def spec_select_round(chosen_T, cand_T, graphs, launched_out=None, status=None, stream=None):
    """chosen_T: device int32 [1]; cand_T: host ints [M]; graphs: handles [M]."""
    M = len(cand_T)
    if len(graphs) != M:
        raise SpecError(ERR_INVALID_ARG, "spec_select_round: one graph per candidate")
    Ts = (ctypes.c_int32 * M)(*[int(t) for t in cand_T])
    gs = (ctypes.c_void_p * M)(*graphs)
    _check(library().spec_select_round(_ptr(chosen_T), M, Ts, gs, _ptr(launched_out), _ptr(status),
                                       _stream(stream)), "spec_select_round")


def spec_pack_rows(src, B, K, row_offsets, dst, status=None, stream=None):
    """src [B(K+1), ...], dst [R_dst, ...] with the same row size."""
    row_bytes = src[0].numel() * src.element_size()
    if dst[0].numel() * dst.element_size() != row_bytes:
        raise SpecError(ERR_INVALID_ARG, "spec_pack_rows: row sizes differ")
    _check(library().spec_pack_rows(_ptr(src), row_bytes, B, K, _ptr(row_offsets), _ptr(dst), dst.shape[0],
                                    _ptr(status), _stream(stream)), "spec_pack_rows")


def spec_draft_workspace(B: int, K: int, V: int) -> int:
    return library().spec_draft_workspace(B, K, V)


def draft_workspace(B: int, K: int, V: int, device="cuda"):
    """A zero-filled workspace for spec_draft."""
    n = spec_draft_workspace(B, K, V)
    if n == 0:
        raise SpecError(ERR_INVALID_ARG, "spec_draft_workspace")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def spec_draft(logits, tau, seeds, request_ids, pos_base, drafts_out, conf_out, ws, scores_out=None,
               row_stats_out=None, status=None, stream=None):
    """logits [B, K, V] bf16/fp32 (the drafter's); see spec.h."""
    B, K, V = logits.shape
    code = library().spec_draft(
        _ptr(logits), _dtype(logits), B, K, V, float(tau), _ptr(seeds), _ptr(request_ids), _ptr(pos_base),
        _ptr(drafts_out), _ptr(conf_out), _ptr(scores_out), _ptr(row_stats_out), _ptr(status), _ptr(ws),
        _nbytes(ws), _stream(stream))
    _check(code, "spec_draft")


def spec_shard_workspace(B: int, K: int, V_shard: int) -> int:
    return library().spec_shard_workspace(B, K, V_shard)


def shard_workspace(B: int, K: int, V_shard: int, device="cuda"):
    """A zero-filled workspace for spec_shard_stats / spec_shard_sample."""
    n = spec_shard_workspace(B, K, V_shard)
    if n == 0:
        raise SpecError(ERR_INVALID_ARG, "spec_shard_workspace")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def spec_shard_stats(logits_shard, draft_tokens, q_shard, B, K, V, v_begin, temperature, pos_base,
                     stats_out, ws, row_offsets=None, depth=None, status=None, stream=None):
    """logits_shard [R, V_shard]; q_shard [B, K, V_shard] or None; stats_out >= R * 32 bytes."""
    R = B * (K + 1)
    if _nbytes(stats_out) < R * SHARD_STAT_BYTES:
        raise SpecError(ERR_INVALID_ARG, "spec_shard_stats: stats_out too small")
    code = library().spec_shard_stats(
        _ptr(logits_shard), _dtype(logits_shard), _ptr(row_offsets), _ptr(depth), _ptr(draft_tokens),
        _ptr(q_shard), _dtype(q_shard), B, K, V, v_begin, logits_shard.shape[-1], float(temperature),
        _ptr(pos_base), _ptr(stats_out), _ptr(status), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(code, "spec_shard_stats")


def spec_shard_decide(stats, S, draft_tokens, q_dense, B, K, V, temperature, seeds, request_ids,
                      pos_base, accepted_len_out, out_tokens, decisions_out=None, row_offsets=None,
                      depth=None, p_draft_out=None, row_stats_out=None, status=None, stream=None):
    """stats: the S shards' records [S, B(K+1)] (>= S * B(K+1) * 32 bytes)."""
    if _nbytes(stats) < S * B * (K + 1) * SHARD_STAT_BYTES:
        raise SpecError(ERR_INVALID_ARG, "spec_shard_decide: stats too small")
    if decisions_out is not None and _nbytes(decisions_out) < B * SHARD_DECISION_BYTES:
        raise SpecError(ERR_INVALID_ARG, "spec_shard_decide: decisions_out too small")
    code = library().spec_shard_decide(
        _ptr(stats), S, _ptr(row_offsets), _ptr(depth), _ptr(draft_tokens), int(bool(q_dense)), B, K, V,
        float(temperature), _ptr(seeds), _ptr(request_ids), _ptr(pos_base), _ptr(accepted_len_out),
        _ptr(out_tokens), _ptr(p_draft_out), _ptr(row_stats_out), _ptr(decisions_out), _ptr(status),
        _stream(stream))
    _check(code, "spec_shard_decide")


def spec_shard_sample(logits_shard, q_shard, decisions, B, K, V, v_begin, temperature, seeds,
                      request_ids, race_out, ws, status=None, stream=None):
    """race_out >= B * 96 bytes."""
    if _nbytes(race_out) < B * SHARD_RACE_BYTES or _nbytes(decisions) < B * SHARD_DECISION_BYTES:
        raise SpecError(ERR_INVALID_ARG, "spec_shard_sample: record buffer too small")
    code = library().spec_shard_sample(
        _ptr(logits_shard), _dtype(logits_shard), _ptr(q_shard), _dtype(q_shard), _ptr(decisions), B, K,
        V, v_begin, logits_shard.shape[-1], float(temperature), _ptr(seeds), _ptr(request_ids),
        _ptr(race_out), _ptr(status), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(code, "spec_shard_sample")


def spec_shard_finish(races, S, decisions, B, K, V, temperature, seeds, request_ids,
                      accepted_len_out, out_tokens, status=None, stream=None):
    """races: the S shards' race records [S, B] (>= S * B * 96 bytes)."""
    if _nbytes(races) < S * B * SHARD_RACE_BYTES or _nbytes(decisions) < B * SHARD_DECISION_BYTES:
        raise SpecError(ERR_INVALID_ARG, "spec_shard_finish: record buffer too small")
    code = library().spec_shard_finish(
        _ptr(races), S, _ptr(decisions), B, K, V, float(temperature), _ptr(seeds), _ptr(request_ids),
        _ptr(accepted_len_out), _ptr(out_tokens), _ptr(status), _stream(stream))
    _check(code, "spec_shard_finish")


def spec_check_bounded_wait(status):
    """Launch a warp whose bounded mbarrier wait has nothing to wait for: after
    about a second it gives up and sets ERR_TIMEOUT in `status` (int32 [1])."""
    _check(library().spec_check_bounded_wait(_ptr(status), _stream(None)), "spec_check_bounded_wait")


def spec_profile_stream_pass(before=None, after=None):
    """Record torch.cuda.Event `before`/`after` around the next verify's streaming kernel."""
    b = None if before is None else ctypes.c_void_p(before.cuda_event)
    a = None if after is None else ctypes.c_void_p(after.cuda_event)
    _check(library().spec_profile_stream_pass(b, a), "spec_profile_stream_pass")
