"""Full-size workloads in the launch configuration bench.py times (whole-vocabulary dz scratch),
checked on outputs the oracle can compute one token at a time, and by identities that hold at
any size.

Sampled tokens (a seeded subset of scored positions -- 4096 on the two largest workloads, 40 on
the others -- plus the first and last scored token of a few completions): logp, lse, entropy,
argmax and the dH row are recomputed by the oracle from H, W, the sampled token and the
per-sequence advantage and count; the dH rows of the subset are compared by relative Frobenius
norm. dW needs every token's log-normaliser (a float64 forward over all 3e5 tokens and the whole
vocabulary, ~5e14 flop), so it is compared element-wise by the long-K test instead
(test_gpu_longk.py: the same token count and hidden size at V = 4096). The behaviour/reference log-probs of
the sampled tokens are the oracle's log-prob plus the batch noise; for the other tokens (never
seen by the oracle) they are the GPU's own log-prob plus noise, as a trainer's would be.

Identities at any size: counts and advantages for every completion; dH = 0 at unscored
positions; every row sum of dz is 0, so the rows of dW sum to ~0; and
<dH, H> = sum_t,v dz_tv z_tv = <dW, W>.
"""
import gc

import numpy as np
import pytest
import torch

import oracle
from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_torch
from tests.parity_util import GRAD_RTOL, LOGP_ATOL, rel_fro

pytestmark = pytest.mark.gpu

FULL = ["g8_t1k_d2048_v32k", "g8_t4k_d4096_v152k", "g16_t16k_d5120_v152k",
        "g16_t512_d3584_v152k", "g4_t512_d3584_v152k"]
# Random scored tokens checked one by one against the oracle: a seeded 4096-token subset on the
# two largest workloads (the long-rollout one the benchmark times, and the many-short one at
# G = 16), 40 on the others. The oracle scores them over the whole vocabulary in chunks.
SAMPLED = {"g16_t16k_d5120_v152k": 4096, "g16_t512_d3584_v152k": 4096}
CHUNK = 512


def _sample_positions(mask, n_random, rng):
    valid = np.argwhere(mask != 0)
    pick = [valid[i] for i in rng.choice(len(valid), size=min(n_random, len(valid)),
                                         replace=False)]
    for s in rng.choice(mask.shape[0], size=min(4, mask.shape[0]), replace=False):
        ts = np.flatnonzero(mask[s])
        if len(ts):
            pick += [np.array([s, ts[0]]), np.array([s, ts[-1]])]
    pick = np.unique(np.array(pick), axis=0)
    return pick[:, 0], pick[:, 1]


@pytest.mark.parametrize("name", FULL)
def test_fullsize_sampled_outputs_and_identities(name):
    w = WORKLOADS[name]
    dev = "cuda"
    b = make_batch_torch(w, dev)
    S, T, d, V = w.S, w.T, w.d, w.V
    ws = G.Workspace.for_problem(S, T, d, V, b.H.dtype)
    f0 = G.grpo_score_fwd(b.H, b.W, b.tokens, b.mask, ws)
    mask = b.mask.cpu().numpy()
    rng = np.random.default_rng(2026)
    si, ti = _sample_positions(mask, SAMPLED.get(name, 40), rng)
    Hs = b.H[torch.from_numpy(si).to(dev), torch.from_numpy(ti).to(dev)].double().cpu().numpy()
    W64 = b.W.double().cpu().numpy()
    y = b.tokens.cpu().numpy()[si, ti]
    sc = {k: np.empty(len(si)) for k in ("logp", "lse", "entropy")}
    sc["argmax"] = np.empty(len(si), np.int64)
    for c0 in range(0, len(si), CHUNK):
        o = oracle.score_tokens(Hs[c0:c0 + CHUNK], W64, y[c0:c0 + CHUNK])
        for k in sc:
            sc[k][c0:c0 + CHUNK] = o[k]

    no, nr = b.noise_old.cpu().numpy(), b.noise_ref.cpu().numpy()
    old = (f0["logp"] + b.noise_old).contiguous()
    ref = (f0["logp"] + b.noise_ref).contiguous()
    old_s = (sc["logp"] + no[si, ti]).astype(np.float32)
    ref_s = (sc["logp"] + nr[si, ti]).astype(np.float32)
    idx = (torch.from_numpy(si).to(dev), torch.from_numpy(ti).to(dev))
    old[idx] = torch.from_numpy(old_s).to(dev)
    ref[idx] = torch.from_numpy(ref_s).to(dev)

    adv = G.group_advantages(b.rewards, b.group_offsets, ws)
    f = G.grpo_score_fwd(b.H, b.W, b.tokens, b.mask, ws)
    r = G.grpo_loss_bwd(b.H, b.W, b.tokens, b.mask, f["logp"], f["lse"], old, ref, adv,
                        f["valid_count"], ws, eps_low=w.eps, eps_high=w.eps, beta=w.beta)
    torch.cuda.synchronize()
    assert G.grpo_last_device_error(ws)[0] == 0

    counts = oracle.valid_counts(mask)
    assert np.array_equal(f["valid_count"].cpu().numpy(), counts)
    adv_o = oracle.group_advantages(b.rewards.cpu().numpy(), b.group_offsets.cpu().numpy())
    np.testing.assert_allclose(adv.cpu().numpy(), adv_o, rtol=1e-5, atol=2e-6)
    assert np.all(adv.cpu().numpy()[adv_o == 0] == 0)

    for k in ("logp", "lse", "entropy"):
        e = np.abs(f[k].cpu().numpy()[si, ti] - sc[k]).max()
        assert e <= LOGP_ATOL, (k, e)
    am = f["argmax"].cpu().numpy()[si, ti]
    for j in np.flatnonzero(am != sc["argmax"]):
        a, c = sc["argmax"][j], am[j]
        bound = 2.0 * d * 2.0 ** -24 * (np.abs(Hs[j]) @ (np.abs(W64[a]) + np.abs(W64[c])))
        assert abs(Hs[j] @ W64[a] - Hs[j] @ W64[c]) <= bound

    t = oracle.token_objective(sc["logp"], old_s, ref_s, adv_o[si], w.eps, w.eps, w.beta)
    _, g_s, _ = oracle.aggregate(t["ell"], t["dell"], si, counts, S)
    dH_o = np.concatenate([
        oracle.param_grads(Hs[c0:c0 + CHUNK], W64, y[c0:c0 + CHUNK], sc["lse"][c0:c0 + CHUNK],
                           g_s[c0:c0 + CHUNK], vocab_rows=np.array([], int))[0]
        for c0 in range(0, len(si), CHUNK)])
    dH_g = r["dH"][idx].double().cpu().numpy()
    err = rel_fro(dH_g, dH_o)
    assert err <= GRAD_RTOL, err

    mask_t = b.mask.bool()
    assert bool(torch.all(r["dH"][~mask_t] == 0))
    dW = r["dW"]
    assert bool(torch.isfinite(dW).all()) and np.isfinite(float(r["loss"].item()))
    row_sum = dW.double().sum(0).norm().item()
    row_mass = dW.double().abs().sum(0).norm().item()
    assert row_sum <= 1e-2 * row_mass, (row_sum, row_mass)
    ip_h = (r["dH"].double() * b.H.double()).sum().item()
    ip_w = (dW.double() * b.W.double()).sum().item()
    assert abs(ip_h - ip_w) <= 5e-3 * max(abs(ip_h), abs(ip_w)), (ip_h, ip_w)
    print(name, "sampled", len(si), "dH rel", err, "<dH,H>", ip_h, "<dW,W>", ip_w)
    del b, ws, f0, f, r, old, ref, W64
    gc.collect()
    torch.cuda.empty_cache()
