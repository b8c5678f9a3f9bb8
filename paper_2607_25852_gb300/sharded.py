"""One rank's round of vocabulary-sharded verification (arxiv 2607.25852
serves its target with TP = 8, Section 4.4): the four ``spec_shard_*`` calls
of libspec and the two all-gathers of their records between them.

Every arithmetic step runs in libspec's kernels.  This module only owns the
record buffers and makes the exchanges, through ``torch.distributed``
(``all_gather_into_tensor`` over the tensor-parallel group, in rank order) or,
when every shard lives on one device, by letting each shard write its records
straight into its slice of the gathered buffer.
"""
import torch

from . import (SHARD_DECISION_BYTES, SHARD_RACE_BYTES, SHARD_STAT_BYTES, shard_workspace,
               spec_shard_decide, spec_shard_finish, spec_shard_sample, spec_shard_stats)


def even_bounds(V: int, S: int):
    """Column ranges of an S-way split of V columns: contiguous, in rank
    order, the first V mod S ranks one column wider (V = 201088, S = 8 gives
    25136 columns each)."""
    if not (1 <= S <= V):
        raise ValueError("need 1 <= S <= V")
    base, extra = divmod(V, S)
    bounds = [0]
    for s in range(S):
        bounds.append(bounds[-1] + base + (1 if s < extra else 0))
    return bounds


def all_gather_records(local, out, group=None):
    """The exchange: `out` receives the ranks' `local` byte tensors one after
    another in rank order (torch.distributed.all_gather_into_tensor)."""
    import torch.distributed as dist
    dist.all_gather_into_tensor(out, local, group=group)


class ShardedRound:
    """Buffers and calls of one rank (shard `rank` of `bounds`) for batches of
    B requests with K drafts over a V-column vocabulary.

    gather(local, out): the exchange; None means torch.distributed over
    `group`.  Pass `local=True` to run all S shards on this device (rank is
    then ignored and `run` takes the S shards' tensors)."""

    def __init__(self, B, K, V, bounds, rank=0, device="cuda", group=None, gather=None, local=False):
        self.B, self.K, self.V = B, K, V
        self.bounds = list(bounds)
        self.S = len(self.bounds) - 1
        if self.bounds[0] != 0 or self.bounds[-1] != V or any(
                self.bounds[s + 1] <= self.bounds[s] for s in range(self.S)):
            raise ValueError("bounds must split [0, V) into non-empty ranges in order")
        self.rank = rank
        self.local = local
        self.group = group
        self.gather = gather
        self.device = torch.device(device)
        R = B * (K + 1)
        u8 = dict(dtype=torch.uint8, device=self.device)
        self.stats = torch.zeros(self.S * R * SHARD_STAT_BYTES, **u8)
        self.races = torch.zeros(self.S * B * SHARD_RACE_BYTES, **u8)
        self.decisions = torch.zeros(B * SHARD_DECISION_BYTES, **u8)
        mine = range(self.S) if local else [rank]
        self.ws = {s: shard_workspace(B, K, self.bounds[s + 1] - self.bounds[s], self.device) for s in mine}
        if not local:
            self.stats_local = torch.zeros(R * SHARD_STAT_BYTES, **u8)
            self.races_local = torch.zeros(B * SHARD_RACE_BYTES, **u8)

    def _exchange(self, local, out):
        if self.gather is not None:
            self.gather(local, out)
        else:
            all_gather_records(local, out, self.group)

    def _slice(self, buf, per, s):
        return buf[s * per:(s + 1) * per]

    def run(self, logits, drafts, q, temperature, seeds, request_ids, pos_base, accepted_len_out,
            out_tokens, row_offsets=None, depth=None, p_draft_out=None, row_stats_out=None, status=None,
            stream=None):
        """logits / q: this rank's [R, V_s] / [B, K, V_s] tensors, or with
        local=True lists of the S shards' tensors (q: None or a list)."""
        B, K, V, t = self.B, self.K, self.V, temperature
        R = B * (K + 1)
        sb, rb = R * SHARD_STAT_BYTES, B * SHARD_RACE_BYTES
        shards = list(range(self.S)) if self.local else [self.rank]
        lg = logits if self.local else {self.rank: logits}
        qq = (q if q is not None else [None] * self.S) if self.local else {self.rank: q}
        for s in shards:
            out = self._slice(self.stats, sb, s) if self.local else self.stats_local
            spec_shard_stats(lg[s], drafts, qq[s], B, K, V, self.bounds[s], t, pos_base, out, self.ws[s],
                             row_offsets=row_offsets, depth=depth, status=status, stream=stream)
        if not self.local:
            self._exchange(self.stats_local, self.stats)
        dense = (q is not None) if not self.local else (q is not None and q[0] is not None)
        spec_shard_decide(self.stats, self.S, drafts, dense, B, K, V, t, seeds, request_ids, pos_base,
                          accepted_len_out, out_tokens, decisions_out=self.decisions, row_offsets=row_offsets,
                          depth=depth, p_draft_out=p_draft_out, row_stats_out=row_stats_out, status=status,
                          stream=stream)
        if t == 0:
            return
        for s in shards:
            out = self._slice(self.races, rb, s) if self.local else self.races_local
            spec_shard_sample(lg[s], qq[s], self.decisions, B, K, V, self.bounds[s], t, seeds, request_ids,
                              out, self.ws[s], status=status, stream=stream)
        if not self.local:
            self._exchange(self.races_local, self.races)
        spec_shard_finish(self.races, self.S, self.decisions, B, K, V, t, seeds, request_ids,
                          accepted_len_out, out_tokens, status=status, stream=stream)
