"""CPU float64 oracle of the GRPO scoring + loss + backward path.

Test infrastructure: only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s
``cpu_baseline`` leg use it. It shares no code with the CUDA path.
"""
from .grpo_oracle import (SEQ_MEAN, TOKEN_MEAN, aggregate, group_advantages, grpo_step,  # noqa: F401
                          logit_grads, merge_shard_stats, param_grads, perf_reward, reward,
                          score_tokens, shard_stats,
                          sft_objective, sft_step, token_objective, tool_reward, valid_counts)
