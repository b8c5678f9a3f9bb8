"""CPU oracle for batched speculative verification (test infrastructure).

A plain, slow, double-precision restatement of the method, in C
(``spec_oracle.c``), with this thin numpy wrapper.  Only the tests, the smoke
check and the benchmark's CPU-baseline leg use it.  It shares no code with the
CUDA library and imports nothing from it.

Array conventions: bf16 tensors are passed as ``uint16`` arrays of raw bits,
fp32 as ``float32``; 64-bit seeds and request ids as ``uint64``.
"""
import ctypes
import os

import numpy as np

from . import build as _build

BF16 = 0
F32 = 1

MODE_GREEDY = 0
MODE_RESIDUAL = 1
MODE_BONUS = 2
MODE_RESIDUAL_EMPTY = 3

OK = 0
ERR_INVALID_ARG = 1
ERR_BAD_INPUT = 4

_lib = None
_P = ctypes.c_void_p


def load(path: str = None):
    """Load (building first if needed) the oracle shared library."""
    global _lib
    if path is not None:
        return _declare(ctypes.CDLL(path))
    if _lib is None:
        _lib = _declare(ctypes.CDLL(_build.build()))
    return _lib


def _declare(lib):
    lib.oracle_philox4x32_10.argtypes = [_P, _P, _P]
    lib.oracle_philox4x32_10.restype = None
    lib.oracle_accept_uniform.argtypes = [ctypes.c_uint64] * 3
    lib.oracle_accept_uniform.restype = ctypes.c_double
    lib.oracle_race_exponential.argtypes = [ctypes.c_uint64] * 3 + [ctypes.c_uint32, ctypes.c_int]
    lib.oracle_race_variate.argtypes = [ctypes.c_uint32]
    lib.oracle_race_variate.restype = ctypes.c_double
    lib.oracle_race_exponential.restype = ctypes.c_double
    lib.oracle_row_stats.argtypes = [_P, ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                     _P, _P, _P]
    lib.oracle_row_stats.restype = None
    lib.oracle_verify_request.argtypes = [
        _P, ctypes.c_int, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
        ctypes.c_double, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
        _P, _P, _P, _P, _P, _P, _P, _P, _P]
    lib.oracle_verify_request.restype = ctypes.c_int
    lib.oracle_verify_batch.argtypes = [
        _P, ctypes.c_int, _P, _P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
        ctypes.c_int, ctypes.c_double, _P, _P, _P,
        _P, _P, _P, _P, _P, _P, _P, _P, _P, _P]
    lib.oracle_verify_batch.restype = ctypes.c_int
    lib.oracle_draft_batch.argtypes = [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                       ctypes.c_double, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P]
    lib.oracle_draft_batch.restype = ctypes.c_int
    lib.oracle_markov_request.argtypes = [_P, ctypes.c_int, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                          ctypes.c_int32, ctypes.c_double, ctypes.c_uint64, ctypes.c_uint64,
                                          ctypes.c_int64, _P, _P, _P, _P, _P, _P]
    lib.oracle_markov_request.restype = ctypes.c_int
    lib.oracle_budget.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64, ctypes.c_int64]
    lib.oracle_budget.restype = ctypes.c_int
    lib.oracle_allocate.argtypes = [
        _P, ctypes.c_int, ctypes.c_int, _P, _P, ctypes.c_int, _P, _P, _P,
        _P, _P, _P, _P, _P, _P, _P]
    lib.oracle_allocate.restype = ctypes.c_int
    lib.oracle_commit.argtypes = [_P, _P, _P, _P, ctypes.c_int64, ctypes.c_int,
                                  ctypes.c_int, _P, _P, _P]
    lib.oracle_commit.restype = None
    return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(a):
    if a is None:
        return BF16
    if a.dtype == np.uint16:
        return BF16
    if a.dtype == np.float32:
        return F32
    raise TypeError(f"unsupported element type {a.dtype}: use uint16 (bf16 bits) or float32")


def _c(a, dtype=None):
    if a is None:
        return None
    return np.ascontiguousarray(a if dtype is None else np.asarray(a, dtype=dtype))


# --------------------------------------------------------------------------
# Philox4x32-10 and the two variates derived from it.
# --------------------------------------------------------------------------
def philox4x32_10(ctr, key):
    """One Philox4x32-10 block: four 32-bit counter words, two key words."""
    c = np.asarray(ctr, dtype=np.uint32).copy()
    k = np.asarray(key, dtype=np.uint32).copy()
    out = np.zeros(4, dtype=np.uint32)
    load().oracle_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def accept_uniform(seed: int, request: int, position: int) -> float:
    return load().oracle_accept_uniform(seed, request, position)


def race_variate(word: int) -> float:
    """Unit exponential variate of one Philox output word."""
    return load().oracle_race_variate(word)


def race_exponential(seed: int, request: int, position: int, index: int, level: int = 2) -> float:
    """Race variate of block `index` (level 1) or entry `index` (level 2)."""
    return load().oracle_race_exponential(seed, request, position, index, level)


# Layout of the race record (9 values per request).
RACE_FIELDS = ("block_key", "block", "block2_key", "block2", "y", "y_key", "y2_key", "y2", "y_in_block2")


def row_stats(row, t: float):
    """(m, S, ok) of one logits row at temperature t > 0."""
    row = _c(row)
    m, S, ok = ctypes.c_double(), ctypes.c_double(), ctypes.c_int32()
    load().oracle_row_stats(_ptr(row), _dtype_code(row), row.shape[-1], t,
                            ctypes.byref(m), ctypes.byref(S), ctypes.byref(ok))
    return m.value, S.value, bool(ok.value)


# --------------------------------------------------------------------------
# Verification
# --------------------------------------------------------------------------
def verify_request(logits, drafts, q, t, seed, request, pos_base):
    """Verify one request: logits [n+1, V], drafts [n], q [n, V] or None."""
    logits = _c(logits)
    drafts = _c(drafts, np.int32)
    q = _c(q)
    n = drafts.shape[0]
    V = logits.shape[-1]
    assert logits.shape == (n + 1, V)
    out = dict(
        accepted=np.zeros(1, np.int32), tokens=np.zeros(n + 1, np.int32),
        p_draft=np.zeros(max(n, 1), np.float64), row_m=np.zeros(n + 1, np.float64),
        row_logS=np.zeros(n + 1, np.float64), u=np.zeros(max(n, 1), np.float64),
        r=np.zeros(max(n, 1), np.float64), race=np.zeros(9, np.float64),
        mode=np.zeros(1, np.int32))
    st = load().oracle_verify_request(
        _ptr(logits), _dtype_code(logits), _ptr(drafts), _ptr(q), _dtype_code(q),
        n, V, float(t), int(seed), int(request), int(pos_base),
        _ptr(out["accepted"]), _ptr(out["tokens"]), _ptr(out["p_draft"]),
        _ptr(out["row_m"]), _ptr(out["row_logS"]), _ptr(out["u"]), _ptr(out["r"]),
        _ptr(out["race"]), _ptr(out["mode"]))
    out["status"] = st
    out["accepted"] = int(out["accepted"][0])
    out["mode"] = int(out["mode"][0])
    out["p_draft"] = out["p_draft"][:n]
    out["u"] = out["u"][:n]
    out["r"] = out["r"][:n]
    return out


def verify_batch(logits, drafts, q, t, seeds, request_ids, pos_base,
                 row_offsets=None, depth=None, requests=None):
    """Verify a batch laid out like the device entry point.

    logits [R, V] (rows of request i start at row_offsets[i], or i*(K+1));
    drafts [B, K]; q [B, K, V] or None; depth [B] or None (= K).
    ``requests`` optionally restricts the work to a subset of request indices
    (the outputs of the others are left at their fill values).
    """
    logits = _c(logits)
    drafts = _c(drafts, np.int32)
    q = _c(q)
    B, K = drafts.shape
    V = logits.shape[-1]
    seeds = _c(seeds, np.uint64)
    request_ids = _c(request_ids, np.uint64)
    pos_base = _c(pos_base, np.int64)
    row_offsets = _c(row_offsets, np.int32)
    depth = _c(depth, np.int32)
    R = logits.shape[0]
    out = dict(
        accepted=np.zeros(B, np.int32), tokens=np.full((B, K + 1), -1, np.int32),
        p_draft=np.zeros((B, K), np.float64), row_m=np.zeros(R, np.float64),
        row_logS=np.zeros(R, np.float64), u=np.zeros((B, K), np.float64),
        r=np.zeros((B, K), np.float64), race=np.zeros((B, 9), np.float64),
        mode=np.zeros(B, np.int32), status=np.zeros(B, np.int32))
    lib = load()
    if requests is None:
        lib.oracle_verify_batch(
            _ptr(logits), _dtype_code(logits), _ptr(row_offsets), _ptr(depth),
            _ptr(drafts), _ptr(q), _dtype_code(q), B, K, V, float(t),
            _ptr(seeds), _ptr(request_ids), _ptr(pos_base),
            _ptr(out["accepted"]), _ptr(out["tokens"]), _ptr(out["p_draft"]),
            _ptr(out["row_m"]), _ptr(out["row_logS"]), _ptr(out["u"]), _ptr(out["r"]),
            _ptr(out["race"]), _ptr(out["mode"]), _ptr(out["status"]))
        return out
    for i in requests:
        n = int(depth[i]) if depth is not None else K
        row0 = int(row_offsets[i]) if row_offsets is not None else i * (K + 1)
        res = verify_request(logits[row0:row0 + n + 1], drafts[i, :n],
                             None if q is None else q[i, :n], t,
                             int(seeds[i]), int(request_ids[i]), int(pos_base[i]))
        out["accepted"][i] = res["accepted"]
        out["tokens"][i, :n + 1] = res["tokens"]
        out["p_draft"][i, :n] = res["p_draft"]
        out["u"][i, :n] = res["u"]
        out["r"][i, :n] = res["r"]
        out["row_m"][row0:row0 + n + 1] = res["row_m"]
        out["row_logS"][row0:row0 + n + 1] = res["row_logS"]
        out["race"][i] = res["race"]
        out["mode"][i] = res["mode"]
        out["status"][i] = res["status"]
    return out


# --------------------------------------------------------------------------
# The drafter's producer step
# --------------------------------------------------------------------------
def draft_batch(logits, tau, seeds, request_ids, pos_base):
    """Drafts, confidences and D-cut scores from the drafter's logits
    [B, K, V] (see oracle_draft_request in spec_oracle.c)."""
    logits = _c(logits)
    B, K, V = logits.shape
    seeds = _c(seeds, np.uint64)
    request_ids = _c(request_ids, np.uint64)
    pos_base = _c(pos_base, np.int64)
    out = dict(z=np.full((B, K), -1, np.int32), c=np.zeros((B, K), np.float64),
               s=np.zeros((B, K + 1), np.float32), m=np.zeros((B, K), np.float64),
               logS=np.zeros((B, K), np.float64), race=np.zeros((B, K, 9), np.float64),
               status=np.zeros(B, np.int32))
    load().oracle_draft_batch(
        _ptr(logits), _dtype_code(logits), B, K, V, float(tau), _ptr(seeds), _ptr(request_ids),
        _ptr(pos_base), _ptr(out["z"]), _ptr(out["c"]), _ptr(out["s"]), _ptr(out["m"]),
        _ptr(out["logS"]), _ptr(out["race"]), _ptr(out["status"]))
    return out


def markov_batch(U, W1, W2, x0, tau, seeds, request_ids, pos_base, requests=None, threads=1):
    """The Markov head's sequential draw (oracle_markov_request) for each
    request: U [B, K, V] base logits; W1 [V, r] and W2 [r, V] as bf16 bits
    (uint16); x0 [B] the last committed tokens.  ``requests`` restricts the
    work to some requests (the others keep their fill values); ``threads``
    runs requests side by side (each call is independent)."""
    U = _c(U)
    B, K, V = U.shape
    W1 = _c(W1, np.uint16)
    W2 = _c(W2, np.uint16)
    r = W1.shape[1]
    assert W1.shape == (V, r) and W2.shape == (r, V)
    x0 = _c(x0, np.int32)
    seeds = _c(seeds, np.uint64)
    request_ids = _c(request_ids, np.uint64)
    pos_base = _c(pos_base, np.int64)
    out = dict(z=np.full((B, K), -1, np.int32), c=np.zeros((B, K), np.float64),
               s=np.zeros((B, K + 1), np.float32), m=np.zeros((B, K), np.float64),
               logS=np.zeros((B, K), np.float64), race=np.zeros((B, K, 9), np.float64),
               status=np.zeros(B, np.int32))
    lib = load()

    def one(i):
        row = U[i]
        out["status"][i] = lib.oracle_markov_request(
            _ptr(row), _dtype_code(U), _ptr(W1), _ptr(W2), K, V, r, int(x0[i]), float(tau), int(seeds[i]),
            int(request_ids[i]), int(pos_base[i]), out["z"][i].ctypes.data, out["c"][i].ctypes.data,
            out["s"][i].ctypes.data, out["m"][i].ctypes.data, out["logS"][i].ctypes.data,
            out["race"][i].ctypes.data)

    idx = list(range(B)) if requests is None else list(requests)
    if threads > 1:
        import concurrent.futures as cf
        with cf.ThreadPoolExecutor(threads) as ex:
            list(ex.map(one, idx))
    else:
        for i in idx:
            one(i)
    return out


# --------------------------------------------------------------------------
# Allocation and commit
# --------------------------------------------------------------------------
def budget(B: int, K: int, num: int, den: int) -> int:
    """Eq. (dcut-budget) for ratio num/den, exact integers."""
    return load().oracle_budget(B, K, num, den)


def allocate(conf, cand_T, cand_cost, last_tokens=None, drafts=None, pos_base=None):
    conf = _c(conf, np.float32)
    B, K = conf.shape
    cand_T = _c(cand_T, np.int32)
    cand_cost = _c(cand_cost, np.float64)
    M = cand_T.shape[0]
    last_tokens = _c(np.zeros(B, np.int32) if last_tokens is None else last_tokens, np.int32)
    drafts = _c(np.zeros((B, K), np.int32) if drafts is None else drafts, np.int32)
    pos_base = _c(np.zeros(B, np.int64) if pos_base is None else pos_base, np.int64)
    N = B * (K + 1)
    out = dict(depth=np.zeros(B, np.int32), row_offsets=np.zeros(B + 1, np.int32),
               packed_tokens=np.zeros(N, np.int32), packed_pos=np.zeros(N, np.int64),
               chosen_T=np.zeros(1, np.int32), utility=np.zeros(M, np.float64),
               all_depths=np.zeros((M, B), np.int32))
    st = load().oracle_allocate(
        _ptr(conf), B, K, _ptr(cand_T), _ptr(cand_cost), M, _ptr(last_tokens),
        _ptr(drafts), _ptr(pos_base), _ptr(out["depth"]), _ptr(out["row_offsets"]),
        _ptr(out["packed_tokens"]), _ptr(out["packed_pos"]), _ptr(out["chosen_T"]),
        _ptr(out["utility"]), _ptr(out["all_depths"]))
    out["status"] = st
    out["chosen_T"] = int(out["chosen_T"][0])
    return out


def commit(accepted, tokens, row_offsets, hidden):
    """Pack committed tokens and gather hidden rows 0..a_i of each request.

    hidden: [R, H] array of any element type (copied as raw bytes) or None.
    """
    accepted = _c(accepted, np.int32)
    tokens = _c(tokens, np.int32)
    B, K1 = tokens.shape
    row_offsets = _c(row_offsets, np.int32)
    total = int(np.sum(accepted.astype(np.int64) + 1))
    packed = np.full(B * K1, -1, np.int32)
    offsets = np.zeros(B + 1, np.int32)
    hidden_out = None
    row_bytes = 0
    if hidden is not None:
        hidden = _c(hidden)
        row_bytes = hidden.shape[1] * hidden.itemsize
        hidden_out = np.zeros((B * K1, hidden.shape[1]), hidden.dtype)
    load().oracle_commit(_ptr(accepted), _ptr(tokens), _ptr(row_offsets), _ptr(hidden),
                         row_bytes, B, K1 - 1, _ptr(packed), _ptr(offsets), _ptr(hidden_out))
    return dict(packed_tokens=packed, commit_offsets=offsets,
                hidden=None if hidden_out is None else hidden_out[:total], total=total)
