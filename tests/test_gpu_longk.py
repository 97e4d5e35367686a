"""Long-K parity: the dW GEMM sums over K = every scored token of the batch, and the workloads of
the benchmark reach K ~ 3e5. Oracle-sized cases stop at a few hundred tokens, so this test keeps
the long-rollout workload's hidden size, temperature law, lengths and token count
(2 prompts x G=12, T=16384, lengths U{8192..16384}: ~2.9e5 scored tokens, d = 5120) and only
shrinks the vocabulary to V = 4096, which the float64 oracle can afford for every token:
dW [V, d] and dH of every scored token are compared element-wise (relative Frobenius), as are
every token's logp / lse / entropy / argmax and the loss. The oracle runs over token chunks (dW is
the sum over tokens of dz_t h_t^T, so the chunk sums add up to the definition).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import Workload, make_batch_torch
from tests.parity_util import GRAD_RTOL, LOGP_ATOL, check_loss

pytestmark = pytest.mark.gpu

LONG_K = Workload("longk_g12_t16k_d5120_v4096", 2, (12,), 16384, 8192, 16384, 5120, 4096, "bf16",
                  "speedup", temperature=(0.5, 2.0), seed=31)
CHUNK = 8192   # tokens per oracle chunk


MODES = {"default": (0, 0, 2, 2), "single_cta": (0, 0, 0, 0)}


def test_long_k_gradients_and_loss_match_oracle():
    """Both the default tile modes (dH and dW on 256 x 512 CTA-pair tiles) and single-CTA tiles
    everywhere, against one oracle pass."""
    w = LONG_K
    dev = "cuda"
    b = make_batch_torch(w, dev)
    S, T, d, V = w.S, w.T, w.d, w.V
    mask = b.mask.cpu().numpy()
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    N = len(si)
    assert N > 250_000
    si_t, ti_t = torch.from_numpy(si).to(dev), torch.from_numpy(ti).to(dev)
    W64 = b.W.double().cpu().numpy()
    y = b.tokens.cpu().numpy()[si, ti].astype(np.int64)

    def h_chunk(sl):
        return b.H[si_t[sl], ti_t[sl]].double().cpu().numpy()

    # oracle forward, chunk by chunk (every token)
    sc = {k: np.empty(N) for k in ("logp", "lse", "entropy")}
    am = np.empty(N, np.int64)
    for c0 in range(0, N, CHUNK):
        sl = slice(c0, min(N, c0 + CHUNK))
        o = oracle.score_tokens(h_chunk(sl), W64, y[sl])
        for k in sc:
            sc[k][sl] = o[k]
        am[sl] = o["argmax"]
    old = np.zeros((S, T), np.float32)
    ref = np.zeros((S, T), np.float32)
    old[si, ti] = (sc["logp"] + b.noise_old.cpu().numpy()[si, ti]).astype(np.float32)
    ref[si, ti] = (sc["logp"] + b.noise_ref.cpu().numpy()[si, ti]).astype(np.float32)
    counts = oracle.valid_counts(mask)
    adv_o = oracle.group_advantages(b.rewards.cpu().numpy(), b.group_offsets.cpu().numpy())
    t = oracle.token_objective(sc["logp"], old[si, ti], ref[si, ti], adv_o[si], w.eps, w.eps,
                               w.beta)
    L, g, mass = oracle.aggregate(t["ell"], t["dell"], si, counts, S)

    # CUDA path through the C ABI, once per tile-mode set
    outs, reps = {}, {}
    try:
        for name, modes in MODES.items():
            for role, m in enumerate(modes):
                G.grpo_set_role_tile_mode(role, m)
            ws = G.Workspace.for_problem(S, T, d, V, b.H.dtype)
            adv = G.group_advantages(b.rewards, b.group_offsets, ws)
            f = G.grpo_score_fwd(b.H, b.W, b.tokens, b.mask, ws)
            r = G.grpo_loss_bwd(b.H, b.W, b.tokens, b.mask, f["logp"], f["lse"],
                                torch.from_numpy(old).to(dev), torch.from_numpy(ref).to(dev),
                                adv, f["valid_count"], ws, eps_low=w.eps, eps_high=w.eps,
                                beta=w.beta)
            torch.cuda.synchronize()
            assert G.grpo_last_device_error(ws)[0] == 0
            del ws
            outs[name] = (adv, f, r)
    finally:
        G.grpo_set_tile_mode(G.TILE_DEFAULT)

    for name, (adv, f, r) in outs.items():
        rep = reps.setdefault(name, {})
        assert np.array_equal(f["valid_count"].cpu().numpy(), counts)
        np.testing.assert_allclose(adv.cpu().numpy(), adv_o, rtol=1e-5, atol=2e-6)
        for k in sc:
            e = float(np.abs(f[k].cpu().numpy()[si, ti] - sc[k]).max())
            rep[k] = e
            assert e <= LOGP_ATOL, (name, k, e)
        am_g = f["argmax"].cpu().numpy()[si, ti]
        miss = np.flatnonzero(am_g != am)
        for j in miss:                     # near-ties within the f32 accumulation bound only
            h = b.H[si[j], ti[j]].double().cpu().numpy()
            a, c = am[j], am_g[j]
            bound = 2.0 * d * 2.0 ** -24 * (np.abs(h) @ (np.abs(W64[a]) + np.abs(W64[c])))
            assert abs(h @ W64[a] - h @ W64[c]) <= bound, (name, j, a, c)
        rep["argmax_near_ties"] = len(miss)
        check_loss(float(r["loss"].item()), L, mass, rep)
        assert bool(torch.all(r["dH"][~b.mask.bool()] == 0))

    # oracle gradients, chunk by chunk: dH rows compared as they come, dW summed over chunks
    dW_o = np.zeros((V, d))
    num = {name: 0.0 for name in outs}
    den = 0.0
    for c0 in range(0, N, CHUNK):
        sl = slice(c0, min(N, c0 + CHUNK))
        dH_c, dW_c = oracle.param_grads(h_chunk(sl), W64, y[sl], sc["lse"][sl], g[sl])
        dW_o += dW_c
        den += float((dH_c ** 2).sum())
        for name, (_, _, r) in outs.items():
            dH_g = r["dH"][si_t[sl], ti_t[sl]].double().cpu().numpy()
            num[name] += float(((dH_g - dH_c) ** 2).sum())
    nW = np.linalg.norm(dW_o)
    for name, (_, _, r) in outs.items():
        rep = reps[name]
        rep["dH"] = (num[name] / den) ** 0.5
        rep["dW"] = float(np.linalg.norm(r["dW"].double().cpu().numpy() - dW_o) / nW)
        print(name, MODES[name], "N", N, rep)
        assert rep["dH"] <= GRAD_RTOL, (name, rep)
        assert rep["dW"] <= GRAD_RTOL, (name, rep)
