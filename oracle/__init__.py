"""CPU float64 oracle of the GRPO scoring + loss + backward path.

Test infrastructure: only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s
``cpu_baseline`` leg use it. It shares no code with the CUDA path.
"""
from .grpo_oracle import (SEQ_MEAN, TOKEN_MEAN, aggregate, exact_kl, exact_kl_logit_grads,  # noqa: F401
                          group_advantages, grpo_step, grpo_step_exact_kl,
                          logit_grads, merge_shard_stats, param_grads, perf_reward, reward,
                          score_tokens, shard_stats,
                          sft_objective, sft_step, token_objective, tool_reward, valid_counts)
