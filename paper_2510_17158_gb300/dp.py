"""Host-side sharding of a GRPO batch over ranks: data-parallel (whole groups per rank) and
vocabulary-parallel (rows of the LM head per rank).

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


def vocab_shard_bounds(V: int, world_size: int, rank: int, align: int = 256):
    """Rows [v0, v1) of the LM head held by `rank` when the vocabulary is split over
    `world_size` ranks in blocks aligned to `align` rows (the last shard takes the remainder)."""
    blocks = (V + align - 1) // align
    b0 = (blocks * rank) // world_size
    b1 = (blocks * (rank + 1)) // world_size
    return min(V, b0 * align), min(V, b1 * align)
