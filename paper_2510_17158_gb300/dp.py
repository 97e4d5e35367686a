"""Host-side data-parallel sharding of a GRPO batch over ranks (whole groups per rank).

Advantages are normalised within a group (Alg. 1), so a rank must own whole groups; the loss
normaliser of Eq. 1's expectation must be the global one (S' sequences for seq_mean, N' scored
tokens for token_mean), passed to grpo_loss_bwd as `norm`. With that, the per-rank losses and
dW sum to the single-process values and each rank's dH rows equal the matching rows of the
single-process dH.
"""
from __future__ import annotations

import numpy as np


def shard_groups(group_offsets, world_size: int, rank: int):
    """Contiguous block of whole groups for `rank`, balanced by number of groups.

    Returns (seq_lo, seq_hi, local_offsets) where local_offsets start at 0."""
    go = np.asarray(group_offsets, dtype=np.int64)
    ng = len(go) - 1
    g_lo = (ng * rank) // world_size
    g_hi = (ng * (rank + 1)) // world_size
    lo, hi = int(go[g_lo]), int(go[g_hi])
    return lo, hi, (go[g_lo:g_hi + 1] - lo).astype(np.int32)


def global_norm(agg: str, local_seqs: int, local_tokens: int, all_reduce_sum) -> float:
    """Global normaliser for `norm`: total sequences (seq_mean) or total scored tokens
    (token_mean) over all ranks; `all_reduce_sum(x: float) -> float` performs the exchange."""
    if agg == "seq_mean":
        return float(all_reduce_sum(float(local_seqs)))
    if agg == "token_mean":
        return float(all_reduce_sum(float(local_tokens)))
    raise ValueError(agg)
