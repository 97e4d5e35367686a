"""Seeded synthetic GRPO rollout batches (the inputs of one GRPO update).

A batch stands in for the rollouts of Alg. 1: P prompts, each with a group of G sampled
completions of ragged length (Sec. 2.1 describes the group of completions per prompt; Sec. 6.1
sets K = 12 and Sec. 5 explains that tool-result text is appended inside a completion).
The paper's datasets and model weights are not available, so every tensor is drawn from the
distributions listed with each workload below.

This module is the only code shared by the oracle side and the CUDA side of the tests and of
the benchmark, so it holds none of the path's arithmetic: no log-softmax, no normaliser, no
advantage, no surrogate, no gradient. It draws random numbers and shapes them:

* hidden states ``H`` ~ N(0, 1), RMS-normalised per token, optionally divided by a per-token
  temperature; rounded to bf16 for bf16 workloads;
* LM-head weight ``W`` ~ N(0, 0.02^2);
* completion lengths, prefix masks, optional interior masked spans (tool-result tokens);
* rewards (Bernoulli or speedup law) and degenerate groups;
* noise vectors for the behaviour and reference log-probs (``old = logp + noise_old``,
  ``ref = logp + noise_ref``), which callers add to a log-prob they obtain elsewhere;
* sampled tokens: the rollout sampler of Alg. 1 draws ``y_t ~ softmax(W h_t)`` with the
  Gumbel-max trick, ``y_t = argmax_v (z_tv + G_tv)`` with ``z = W h_t`` from a library matmul.
  Sampling is the rollout's step, not the scoring path: it forms no normaliser or log-prob.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass
from typing import Optional, Tuple

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    prompts: int
    group_sizes: Tuple[int, ...]      # G of each prompt, cycled over the prompts
    T: int                            # padded completion length
    len_lo: int                       # completion lengths ~ U{len_lo .. len_hi}
    len_hi: int
    d: int
    V: int
    dtype: str                        # "f32" or "bf16": storage type of H and W
    reward_law: str                   # "bernoulli" or "speedup"
    temperature: Optional[Tuple[float, float]] = None   # per-token temperature ~ U[lo, hi]
    degenerate_frac: float = 0.0      # fraction of groups whose rewards are all equal
    eps: float = 0.2
    beta: float = 0.04
    old_sigma: float = 0.05
    ref_sigma: float = 0.1
    holes: bool = False               # interior masked spans standing in for tool output
    seed: int = 0

    @property
    def S(self) -> int:
        return sum(self.group_sizes[p % len(self.group_sizes)] for p in range(self.prompts))

    def scaled(self, **kw) -> "Workload":
        """Same laws, fewer or shorter sequences (oracle-sized parity cases)."""
        return dataclasses.replace(self, **kw)


# The five synthetic workloads. Tokens are sampled from softmax(W h); old/ref log-probs are the
# current log-prob plus Gaussian noise; rewards follow the stated laws.
WORKLOADS = {
    # 1 prompt x G=4, T=64, lengths U{16..64}, d=64, V=512, FP32, Bernoulli(0.5)+N(0,0.1^2).
    "tiny_f32": Workload("tiny_f32", 1, (4,), 64, 16, 64, 64, 512, "f32", "bernoulli", seed=0),
    # 8 prompts x G=8, T=1024, lengths U{256..1024}, d=2048, V=32000, BF16, speedup rewards.
    "g8_t1k_d2048_v32k": Workload("g8_t1k_d2048_v32k", 8, (8,), 1024, 256, 1024, 2048, 32000,
                                  "bf16", "speedup", seed=1),
    # 4 prompts x G=8, T=4096, lengths U{1024..4096}, d=4096, V=151936, BF16.
    "g8_t4k_d4096_v152k": Workload("g8_t4k_d4096_v152k", 4, (8,), 4096, 1024, 4096, 4096,
                                   151936, "bf16", "speedup", seed=2),
    # 2 prompts x G=16, T=16384, lengths U{4096..16384}, d=5120, V=151936, BF16, per-token
    # temperature U[0.5, 2] (heavy-tailed logit scale).
    "g16_t16k_d5120_v152k": Workload("g16_t16k_d5120_v152k", 2, (16,), 16384, 4096, 16384, 5120,
                                     151936, "bf16", "speedup", temperature=(0.5, 2.0), seed=3),
    # 64 prompts x G in {4, 8, 16}, lengths U{32..512}, T=512, d=3584, V=152064, BF16,
    # 10% degenerate groups.
    "g4_t512_d3584_v152k": Workload("g4_t512_d3584_v152k", 64, (4,), 512, 32, 512, 3584, 152064,
                                    "bf16", "speedup", degenerate_frac=0.1, seed=4),
    "g8_t512_d3584_v152k": Workload("g8_t512_d3584_v152k", 64, (8,), 512, 32, 512, 3584, 152064,
                                    "bf16", "speedup", degenerate_frac=0.1, seed=4),
    "g16_t512_d3584_v152k": Workload("g16_t512_d3584_v152k", 64, (16,), 512, 32, 512, 3584,
                                     152064, "bf16", "speedup", degenerate_frac=0.1, seed=4),
    # Parity-only mixed batch: G cycling {4, 8, 12, 16} (K = 12 is the paper's group size).
    "mixed_t512_d3584_v152k": Workload("mixed_t512_d3584_v152k", 64, (4, 8, 12, 16), 512, 32, 512,
                                       3584, 152064, "bf16", "speedup", degenerate_frac=0.1,
                                       seed=5),
}


@dataclass
class Batch:
    """One synthetic GRPO batch. Tensors live on ``device``; H and W have the workload dtype."""
    workload: Workload
    H: torch.Tensor            # [S, T, d]  bf16 or f32
    W: torch.Tensor            # [V, d]     bf16 or f32
    tokens: torch.Tensor       # [S, T]     int32
    mask: torch.Tensor         # [S, T]     uint8 (1 = scored completion token)
    lengths: torch.Tensor      # [S]        int32 (completion length before interior holes)
    rewards: torch.Tensor      # [S]        f32
    group_offsets: torch.Tensor  # [num_groups + 1] int32
    noise_old: torch.Tensor    # [S, T]     f32, N(0, old_sigma^2)
    noise_ref: torch.Tensor    # [S, T]     f32, N(0, ref_sigma^2)

    @property
    def S(self) -> int:
        return self.H.shape[0]

    @property
    def T(self) -> int:
        return self.H.shape[1]


def _group_sizes(w: Workload):
    return [w.group_sizes[p % len(w.group_sizes)] for p in range(w.prompts)]


class _NumpyDraws:
    """Independent numpy sub-streams, one per tensor, from one workload seed."""

    def __init__(self, seed: int):
        self.children = np.random.SeedSequence(seed).spawn(12)

    def rng(self, k: int) -> np.random.Generator:
        return np.random.Generator(np.random.PCG64(self.children[k]))


def _lengths_and_mask(w: Workload, rng_len, rng_hole):
    S, T = w.S, w.T
    lengths = rng_len.integers(w.len_lo, w.len_hi + 1, size=S).astype(np.int32)
    lengths = np.minimum(lengths, T)
    mask = np.zeros((S, T), dtype=np.uint8)
    for i in range(S):
        mask[i, : lengths[i]] = 1
        if w.holes and lengths[i] > 8:
            # two interior spans of tool-result text, each 1..max(1, n/8) tokens long
            for _ in range(2):
                span = int(rng_hole.integers(1, max(2, lengths[i] // 8)))
                start = int(rng_hole.integers(1, max(2, lengths[i] - span)))
                mask[i, start : start + span] = 0
    return lengths, mask


def _rewards(w: Workload, rng):
    S = w.S
    if w.reward_law == "bernoulli":
        r = rng.binomial(1, 0.5, size=S).astype(np.float64) + rng.normal(0.0, 0.1, size=S)
    elif w.reward_law == "speedup":
        # 0 with p = 0.4, else log2(s) with s log-uniform on [0.5, 8]  =>  log2 s ~ U[-1, 3]
        zero = rng.random(S) < 0.4
        r = np.where(zero, 0.0, rng.uniform(-1.0, 3.0, size=S))
    else:
        raise ValueError(w.reward_law)
    sizes = _group_sizes(w)
    offsets = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    if w.degenerate_frac > 0:
        ng = len(sizes)
        n_deg = max(1, int(round(w.degenerate_frac * ng)))
        deg = rng.choice(ng, size=n_deg, replace=False)
        for g in deg:
            r[offsets[g] : offsets[g + 1]] = r[offsets[g]]
    return r.astype(np.float32), offsets


def _sample_tokens_numpy(Hq64, Wq64, mask, rng_gumbel, rng_unif, V):
    """Rollout sampler: y = argmax(z + Gumbel) over z = W h (library matmul), per valid token."""
    S, T, d = Hq64.shape
    tokens = rng_unif.integers(0, V, size=(S, T)).astype(np.int32)   # unscored positions
    idx = np.argwhere(mask != 0)
    chunk = max(1, (1 << 24) // V)
    for c0 in range(0, len(idx), chunk):
        sel = idx[c0 : c0 + chunk]
        z = Hq64[sel[:, 0], sel[:, 1]] @ Wq64.T
        u = rng_gumbel.random(z.shape)
        g = -np.log(-np.log(np.clip(u, 1e-300, 1.0 - 1e-16)))
        tokens[sel[:, 0], sel[:, 1]] = np.argmax(z + g, axis=1).astype(np.int32)
    return tokens


def make_batch_numpy(w: Workload) -> Batch:
    """CPU batch from numpy PCG64 sub-streams: bit-reproducible on any host."""
    S, T, d, V = w.S, w.T, w.d, w.V
    dr = _NumpyDraws(w.seed)
    lengths, mask = _lengths_and_mask(w, dr.rng(0), dr.rng(1))
    H = dr.rng(2).standard_normal((S, T, d), dtype=np.float32)
    rms = np.sqrt(np.mean(H.astype(np.float64) ** 2, axis=-1, keepdims=True))
    H = (H / rms).astype(np.float32)
    if w.temperature is not None:
        tau = dr.rng(3).uniform(w.temperature[0], w.temperature[1], size=(S, T, 1))
        H = (H / tau).astype(np.float32)
    Wm = (dr.rng(4).standard_normal((V, d), dtype=np.float32) * np.float32(0.02)).astype(np.float32)
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    Ht = torch.from_numpy(H).to(tdt)
    Wt = torch.from_numpy(Wm).to(tdt)
    tokens = _sample_tokens_numpy(Ht.double().numpy(), Wt.double().numpy(), mask,
                                  dr.rng(5), dr.rng(6), V)
    rewards, offsets = _rewards(w, dr.rng(7))
    noise_old = dr.rng(8).normal(0.0, w.old_sigma, size=(S, T)).astype(np.float32)
    noise_ref = dr.rng(9).normal(0.0, w.ref_sigma, size=(S, T)).astype(np.float32)
    return Batch(w, Ht, Wt, torch.from_numpy(tokens), torch.from_numpy(mask),
                 torch.from_numpy(lengths), torch.from_numpy(rewards), torch.from_numpy(offsets),
                 torch.from_numpy(noise_old), torch.from_numpy(noise_ref))


def make_batch_torch(w: Workload, device: str = "cuda", sample_chunk_tokens: int = 2048) -> Batch:
    """Device batch from a seeded torch generator: used where the batch is too large for numpy
    (reproducible on one device type and torch build; the draws differ from ``make_batch_numpy``)."""
    S, T, d, V = w.S, w.T, w.d, w.V
    dr = _NumpyDraws(w.seed)                 # host-side small draws stay on numpy streams
    lengths, mask = _lengths_and_mask(w, dr.rng(0), dr.rng(1))
    rewards, offsets = _rewards(w, dr.rng(7))
    gen = torch.Generator(device=device)
    gen.manual_seed(int(dr.children[2].generate_state(1)[0]))
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    H = torch.empty((S, T, d), dtype=tdt, device=device)
    for i in range(S):                       # one sequence at a time bounds the f32 scratch
        h = torch.randn((T, d), generator=gen, device=device, dtype=torch.float32)
        h = h * torch.rsqrt(torch.mean(h * h, dim=-1, keepdim=True))
        if w.temperature is not None:
            tau = torch.empty((T, 1), device=device).uniform_(w.temperature[0], w.temperature[1],
                                                               generator=gen)
            h = h / tau
        H[i].copy_(h)
        del h
    Wt = torch.empty((V, d), dtype=tdt, device=device)
    for v0 in range(0, V, 16384):
        v1 = min(V, v0 + 16384)
        Wt[v0:v1].copy_(torch.randn((v1 - v0, d), generator=gen, device=device) * 0.02)
    mask_t = torch.from_numpy(mask).to(device)
    tokens = torch.randint(0, V, (S, T), generator=gen, device=device, dtype=torch.int64)
    valid = mask_t.reshape(-1).nonzero().squeeze(1)
    Hf = H.reshape(S * T, d)
    tok_flat = tokens.reshape(-1)
    for c0 in range(0, valid.numel(), sample_chunk_tokens):
        sel = valid[c0 : c0 + sample_chunk_tokens]
        z = torch.matmul(Hf[sel], Wt.t()).float()
        u = torch.rand(z.shape, generator=gen, device=device).clamp_(1e-30, 1.0 - 1e-7)
        z.sub_(torch.log(-torch.log(u)))
        tok_flat[sel] = torch.argmax(z, dim=1)
        del z, u
    noise_old = torch.randn((S, T), generator=gen, device=device) * w.old_sigma
    noise_ref = torch.randn((S, T), generator=gen, device=device) * w.ref_sigma
    return Batch(w, H, Wt, tokens.to(torch.int32), mask_t,
                 torch.from_numpy(lengths).to(device), torch.from_numpy(rewards).to(device),
                 torch.from_numpy(offsets).to(device), noise_old.float(), noise_ref.float())


def reference_model_inputs(batch: Batch, seed: int = 7, h_sigma: float = 0.3,
                           w_sigma: float = 0.004):
    """Hidden states and LM head of the frozen reference model (Alg. 1) for a batch: the policy's
    tensors plus Gaussian perturbations (h: sigma h_sigma, then rescaled to the policy token's
    RMS; W: sigma w_sigma), in the batch's dtype and on its device (seeded torch generator on
    that device). Draws only."""
    dev = batch.H.device
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    Hr = torch.empty_like(batch.H)
    for i in range(batch.H.shape[0]):           # one sequence at a time bounds the f32 scratch
        h = batch.H[i].float()
        x = h + h_sigma * torch.randn(h.shape, generator=gen, device=dev)
        x = x * torch.sqrt(torch.mean(h * h, dim=-1, keepdim=True) /
                           torch.mean(x * x, dim=-1, keepdim=True))
        Hr[i].copy_(x)
    Wr = torch.empty_like(batch.W)
    for v0 in range(0, batch.W.shape[0], 16384):
        wv = batch.W[v0:v0 + 16384].float()
        Wr[v0:v0 + 16384].copy_(wv + w_sigma * torch.randn(wv.shape, generator=gen, device=dev))
    return Hr, Wr


def token_count_mean(w: Workload) -> float:
    """Expected number of scored tokens of a workload (mean of its length law, no holes)."""
    return w.S * min(w.T, (w.len_lo + w.len_hi) / 2.0)


def lm_head_flops(n_tokens: int, d: int, V: int) -> float:
    """Algorithmic flops of one forward+backward over n scored tokens: 6 n d V."""
    return 6.0 * n_tokens * d * V


__all__ = ["Workload", "WORKLOADS", "Batch", "make_batch_numpy", "make_batch_torch",
           "reference_model_inputs", "token_count_mean", "lm_head_flops"]
