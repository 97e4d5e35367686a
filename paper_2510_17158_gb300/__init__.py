"""Fused GRPO token-scoring + loss + backward on GB300 (sm_103a)."""
