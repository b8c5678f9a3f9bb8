"""Seeded generators for the five verification workloads.

The paper measures on public benchmarks and live serving traffic (Section 4.4,
Section 5) that are not available here.  These recipes stand in for them with
the same shapes: concurrency 4-64 (the c4-c64 sweeps of Section 4.4), a draft
block of 16, vocabularies of 128K-201K entries, and acceptance behaviour that
mimics the code/maths versus chat gap in accepted length the paper reports.

Every tensor is drawn from a ``torch.Generator`` (large arrays) or a
``numpy.random.Generator`` (small arrays) seeded from ``seed``; the same call
gives the same bytes on any machine for a given device type.

Recipes (std = standard deviation):
  tiny     B=4,  K=4,  V=4096,   fp32 logits ~ N(0, 2^2); draft j+1 equals the
           argmax of row j with probability 0.7, else uniform over V;
           one-hot q; Philox seed 0 for every request; request ids 0..3.
  greedy   B=16, K=16, V=128256, bf16 logits ~ N(0, 3^2); a planted peak
           (row max + 8) sits at draft j+1 with probability 0.8, else at a
           uniform other token; the bonus row gets a peak at a uniform token;
           hidden rows H=4096 bf16.
  sampled  B=32, K=8,  V=151936, bf16 logits ~ N(0, 2.5^2); draft logits =
           target + N(0, 0.7^2); q = softmax(draft / 0.8) stored bf16
           [B, K, V]; draft j+1 ~ q_j; temperature 0.8; seed_i = i.
  alloc    B=64, K=16, V=128256, bf16 logits as in `greedy`; requests 0..31
           chat-like (confidence ~ Beta(2,2), match probability 0.5),
           32..63 code-like (Beta(8,1), match 0.9); temperature 1, one-hot q;
           budget sweep T = 64..1024 with cost 1.0 + 0.004 * max(0, T - 256).
  stress   B=64, K=16, V=201088, bf16 logits ~ N(0, 3^2); q = softmax(target
           + N(0, 1)) stored bf16 [B, K, V]; draft j+1 ~ q_j; temperature 1;
           seed_i = i; hidden rows H=7168 bf16.
  draft    (make_draft) the drafter's logits [B, K, V] = N(0, 3^2) + N(0, 1),
           B=64, K=16, V=201088 bf16, tau = 1: the input of the drafter's
           producer step.
"""
from dataclasses import dataclass, field
from typing import Optional

import numpy as np
import torch

CONFIGS = {
    "tiny": dict(B=4, K=4, V=4096, dtype="f32", std=2.0, H=64, temperature=1.0),
    "greedy": dict(B=16, K=16, V=128256, dtype="bf16", std=3.0, H=4096, temperature=0.0),
    "sampled": dict(B=32, K=8, V=151936, dtype="bf16", std=2.5, H=64, temperature=0.8),
    "alloc": dict(B=64, K=16, V=128256, dtype="bf16", std=3.0, H=64, temperature=1.0),
    "stress": dict(B=64, K=16, V=201088, dtype="bf16", std=3.0, H=7168, temperature=1.0),
}


@dataclass
class Workload:
    name: str
    B: int
    K: int
    V: int
    H: int
    dtype: str                      # "bf16" or "f32": element type of logits and q
    temperature: float
    logits: torch.Tensor            # [B*(K+1), V], rows of request i at i*(K+1)
    drafts: torch.Tensor            # [B, K] int32
    q: Optional[torch.Tensor]       # [B, K, V] or None (one-hot at the draft)
    seeds: torch.Tensor             # [B] int64 (bit pattern of a uint64)
    request_ids: torch.Tensor       # [B] int64
    pos_base: torch.Tensor          # [B] int64
    last_tokens: torch.Tensor       # [B] int32
    hidden: Optional[torch.Tensor]  # [B*(K+1), H] bf16 or None
    conf: Optional[torch.Tensor] = None   # [B, K] fp32 (allocator input)
    extra: dict = field(default_factory=dict)

    @property
    def rows(self) -> int:
        return self.B * (self.K + 1)


def _torch_dtype(name):
    return torch.bfloat16 if name == "bf16" else torch.float32


def _normal(shape, std, gen, device):
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32) * std


def _plant_peaks(logits, drafts, match_prob, rng, device):
    """Plant a peak (row max + 8) per row at the draft token or elsewhere."""
    B, K = drafts.shape
    V = logits.shape[-1]
    rows = logits.view(B, K + 1, V)
    rowmax = rows.amax(dim=-1)                                   # [B, K+1]
    match_prob = np.broadcast_to(np.asarray(match_prob, dtype=np.float64), (B,))
    hit = rng.random((B, K)) < match_prob[:, None]
    other = rng.integers(0, V - 1, size=(B, K))
    d = drafts.cpu().numpy()
    other = np.where(other >= d, other + 1, other)               # uniform over V minus the draft
    peak_at = np.where(hit, d, other)
    bonus_at = rng.integers(0, V, size=(B, 1))
    peak_at = np.concatenate([peak_at, bonus_at], axis=1)        # [B, K+1]
    idx = torch.as_tensor(peak_at, dtype=torch.int64, device=device)
    rows.scatter_(2, idx.unsqueeze(-1), (rowmax + 8.0).unsqueeze(-1))
    return hit


def make(name: str, *, device="cpu", seed: int = 1234, V: Optional[int] = None,
         B: Optional[int] = None, K: Optional[int] = None,
         temperature: Optional[float] = None, with_q: Optional[bool] = None,
         with_hidden: bool = True, H: Optional[int] = None) -> Workload:
    """Draw workload `name` (see module docstring), optionally resized."""
    cfg = dict(CONFIGS[name])
    B = B or cfg["B"]
    K = cfg["K"] if K is None else K
    V = V or cfg["V"]
    H = H or cfg["H"]
    t = cfg["temperature"] if temperature is None else temperature
    dt = _torch_dtype(cfg["dtype"])
    std = cfg["std"]
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    rng = np.random.default_rng(seed)
    R = B * (K + 1)
    extra = {}

    logits = _normal((R, V), std, gen, device)
    q = None
    conf = None
    if name == "tiny":
        amax = logits.view(B, K + 1, V)[:, :K].argmax(dim=-1).cpu().numpy()
        uni = rng.integers(0, V, size=(B, K))
        drafts_np = np.where(rng.random((B, K)) < 0.7, amax, uni)
        drafts = torch.as_tensor(drafts_np, dtype=torch.int32)
    elif name in ("greedy", "alloc"):
        drafts = torch.as_tensor(rng.integers(0, V, size=(B, K)), dtype=torch.int32)
        if name == "alloc":
            half = B // 2
            match = np.concatenate([np.full(half, 0.5), np.full(B - half, 0.9)])
            conf_np = np.concatenate([rng.beta(2.0, 2.0, size=(half, K)),
                                      rng.beta(8.0, 1.0, size=(B - half, K))]).astype(np.float32)
            conf = torch.as_tensor(conf_np)
            extra["match_prob"] = match
        else:
            match = 0.8
        extra["planted_hit"] = _plant_peaks(logits, drafts, match, rng, device)
    elif name in ("sampled", "stress"):
        noise_std, q_temp = (0.7, 0.8) if name == "sampled" else (1.0, 1.0)
        rows = logits.view(B, K + 1, V)
        draft_logits = rows[:, :K] + _normal((B, K, V), noise_std, gen, device)
        qf = torch.softmax(draft_logits / q_temp, dim=-1)
        del draft_logits
        qs = qf.to(dt)
        del qf
        # Drafts are drawn from the stored q (as the caller's drafter would).
        flat = qs.view(B * K, V).float()
        drafts = torch.multinomial(flat, 1, generator=gen).view(B, K).to(torch.int32)
        del flat
        q = qs
    else:
        raise KeyError(name)

    logits = logits.to(dt)
    use_q = (q is not None) if with_q is None else with_q
    if not use_q:
        q = None
    seeds = torch.arange(B, dtype=torch.int64) if name != "tiny" else torch.zeros(B, dtype=torch.int64)
    request_ids = torch.arange(B, dtype=torch.int64) + (1000 if name == "stress" else 0)
    pos_base = torch.as_tensor(rng.integers(0, 4096, size=B), dtype=torch.int64)
    if name == "tiny":
        pos_base = torch.zeros(B, dtype=torch.int64)
    last_tokens = torch.as_tensor(rng.integers(0, V, size=B), dtype=torch.int32)
    hidden = None
    if with_hidden:
        hidden = torch.randn((R, H), generator=gen, device=device).to(torch.bfloat16)
    wl = Workload(name=name, B=B, K=K, V=V, H=H, dtype=cfg["dtype"], temperature=t,
                  logits=logits, drafts=drafts.to(device), q=q, seeds=seeds.to(device),
                  request_ids=request_ids.to(device), pos_base=pos_base.to(device),
                  last_tokens=last_tokens.to(device), hidden=hidden,
                  conf=None if conf is None else conf.to(device), extra=extra)
    return wl


@dataclass
class DraftInputs:
    """Inputs of the drafter's producer step (spec_draft)."""
    B: int
    K: int
    V: int
    dtype: str
    tau: float
    logits: torch.Tensor        # [B, K, V], the drafter's logits for drafts 1..K
    seeds: torch.Tensor         # int64 [B] (uint64 bits)
    request_ids: torch.Tensor   # int64 [B]
    pos_base: torch.Tensor      # int64 [B]


def make_draft(B: int = 64, K: int = 16, V: int = 201088, *, tau: float = 1.0, dtype: str = "bf16",
               std: float = 3.0, device="cpu", seed: int = 4321) -> DraftInputs:
    """The drafter's logits for one block of K drafts per request: rows of
    N(0, std^2) (the stress recipe's target rows) plus N(0, 1) noise, the same
    construction the stress recipe uses for q before its softmax.  B=64, K=16,
    V=201088 bf16 at tau = 1 by default."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    rng = np.random.default_rng(seed)
    logits = _normal((B, K, V), std, gen, device)
    logits += _normal((B, K, V), 1.0, gen, device)
    return DraftInputs(B=B, K=K, V=V, dtype=dtype, tau=tau, logits=logits.to(_torch_dtype(dtype)),
                       seeds=torch.arange(B, dtype=torch.int64, device=device) + 77,
                       request_ids=torch.arange(B, dtype=torch.int64, device=device) + 5000,
                       pos_base=torch.as_tensor(rng.integers(0, 4096, size=B), dtype=torch.int64).to(device))


def pack_rows(full: torch.Tensor, B: int, K: int, depth, row_offsets=None):
    """Gather rows 0..n_i of each request from a full-depth [B*(K+1), ...]
    tensor into the dense packed layout of an allocation (input preparation for
    a target forward over the packed batch)."""
    depth = [int(x) for x in depth]
    idx = []
    for i, n in enumerate(depth):
        idx.extend(range(i * (K + 1), i * (K + 1) + n + 1))
    idx = torch.as_tensor(idx, dtype=torch.int64, device=full.device)
    return full.index_select(0, idx)


def budget_candidates(B: int, K: int, sweep=(64, 1024, 64)):
    """The fixed budget sweep T = 64, 128, ..., 1024 (clipped to [B, B(K+1)])
    with the piecewise-linear profiled cost 1.0 + 0.004 * max(0, T - 256)."""
    lo, hi, step = sweep
    Ts = [min(max(T, B), B * (K + 1)) for T in range(lo, hi + 1, step)]
    costs = [1.0 + 0.004 * max(0, T - 256) for T in Ts]
    return np.asarray(Ts, np.int32), np.asarray(costs, np.float64)
