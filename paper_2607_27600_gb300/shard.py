"""One counter-causal refresh split over the ranks of a torch.distributed
process group by query rows.

Given the cache, a row's score depends only on its own input and on the
cached K/V of the later slots, which the pass reuses (Sec. 3.1), so the rows
of one refresh can be scored by different GPUs that each hold the cache:

1. plan: cc_partition_rows splits every sequence into one contiguous block
   of rows per rank, of equal estimated cost (early rows attend more later
   slots, so they get shorter blocks);
2. score: each rank runs cc_score_rows over its block; every other entry of
   its score buffer is -inf;
3. exchange: one MAX all-reduce of the [batch][cap] fp32 scores, which is
   exact (max(-inf, x) = x for every score, signed zeros and infinities
   included), so every rank holds the scores a single cc_score_* call gives;
4. select and compact: every rank runs the same cc_select_keep on the same
   scores (identical keep-sets) and compacts its own replica of the cache.

Each rank keeps a full replica because a row attends every later slot; the
compaction is then local and needs no second exchange.  Every step runs in
the library's kernels; this module only plans, marshals and calls the
collective.
"""
import torch
import torch.distributed as dist

from . import cc


class RowShard:
    """Rank `rank`'s share of a refresh over sequences of (host-known)
    lengths `seq_lens`: rows [lo[rank][b], hi[rank][b]) of sequence b."""

    def __init__(self, cfg, full: bool, seq_lens, rank: int, world: int, align: int = 128,
                 device=None):
        if not 0 <= rank < world:
            raise ValueError("rank outside [0, world)")
        self.lo, self.hi = cc.cc_partition_rows(cfg, full, seq_lens, world, align)
        self.full, self.rank, self.world = bool(full), rank, world
        self.device = device
        self.row_lo = self.row_hi = None
        if device is not None:
            self.row_lo = torch.from_numpy(self.lo[rank].copy()).to(device)
            self.row_hi = torch.from_numpy(self.hi[rank].copy()).to(device)

    def rows(self, rank: int = None) -> int:
        r = self.rank if rank is None else rank
        return int((self.hi[r] - self.lo[r]).sum())

    def score(self, cfg, weights, cache, mode, scores, ws, stream=None):
        """This rank's rows into `scores` (-inf everywhere else)."""
        cc.cc_score_rows(cfg, weights, cache, mode, self.full, self.row_lo, self.row_hi, scores,
                         ws, stream)


def merge_scores(scores: torch.Tensor, group=None) -> torch.Tensor:
    """Element-wise maximum of every rank's score buffer, in place (one
    all-reduce); a no-op without an initialised group of more than one rank."""
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(scores, op=dist.ReduceOp.MAX, group=group)
    return scores


def sharded_refresh(shard: RowShard, cfg, weights, cache, mode, scores, ws, budget, n_sink,
                    keep_idx, keep_count, compact_ws, group=None):
    """One refresh: this rank's rows, the exchange, then select and compaction
    of this rank's replica (identical on every rank)."""
    b, cap = scores.shape
    shard.score(cfg, weights, cache, mode, scores, ws)
    merge_scores(scores, group)
    cc.cc_select_keep(scores, cache.d["seq_len"], b, cap, budget, n_sink, keep_idx, keep_count)
    cc.cc_compact_kv(cfg, cache, keep_idx, keep_count, compact_ws)
