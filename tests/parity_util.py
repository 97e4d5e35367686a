"""Helpers shared by the parity tests: run one batch through the CUDA path (C ABI) and through
the CPU oracle on identical inputs, and compare with the tolerances of the parity bar.

Tolerances (BF16 inputs, f32 accumulation): counts and argmax bit-exact (argmax modulo near-ties
within the f32 accumulation bound), logp within 2e-3 absolute (also used for lse and entropy),
loss within 1e-3 relative (see check_loss), dH and dW within 1e-2 relative Frobenius norm.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle

LOGP_ATOL = 2e-3
LOSS_RTOL = 1e-3
GRAD_RTOL = 1e-2


def oracle_inputs(batch, old_scale=1.0):
    """old/ref log-probs = oracle log-prob of the sampled token + the batch's noise (float32)."""
    mask = batch.mask.cpu().numpy()
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    H = batch.H.cpu().double().numpy()
    W = batch.W.cpu().double().numpy()
    y = batch.tokens.cpu().numpy()[si, ti]
    sc = oracle.score_tokens(H[si, ti], W, y)
    base = np.zeros(mask.shape)
    base[si, ti] = sc["logp"]
    old = (base + old_scale * batch.noise_old.cpu().numpy()).astype(np.float32)
    ref = (base + batch.noise_ref.cpu().numpy()).astype(np.float32)
    return old, ref


def run_oracle(batch, old, ref, eps_low, eps_high, beta, agg="seq_mean", std_mode="unbiased",
               std_eps=1e-4, with_grads=True, vocab_rows=None, norm=None):
    return oracle.grpo_step(batch.H.cpu().double().numpy(), batch.W.cpu().double().numpy(),
                            batch.tokens.cpu().numpy(), batch.mask.cpu().numpy(),
                            batch.rewards.cpu().numpy(), batch.group_offsets.cpu().numpy(),
                            old.astype(np.float64), ref.astype(np.float64), eps_low, eps_high, beta,
                            agg, std_mode, std_eps, norm=norm, with_grads=with_grads,
                            vocab_rows=vocab_rows)


def run_gpu(batch, old, ref, eps_low, eps_high, beta, agg="seq_mean", std_mode="unbiased",
            std_eps=1e-4, vocab_chunk=0, ref_none=False, device="cuda", norm=0.0):
    from paper_2510_17158_gb300 import grpo as G
    dev = torch.device(device)
    H, W = batch.H.to(dev), batch.W.to(dev)
    tok, mask = batch.tokens.to(dev), batch.mask.to(dev)
    S, T, d = H.shape
    V = W.shape[0]
    ws = G.Workspace.for_problem(S, T, d, V, H.dtype, vocab_chunk=vocab_chunk)
    adv = G.group_advantages(batch.rewards.to(dev), batch.group_offsets.to(dev), ws,
                             std_mode=std_mode, std_eps=std_eps)
    f = G.grpo_score_fwd(H, W, tok, mask, ws)
    old_t = torch.from_numpy(old).to(dev)
    ref_t = None if ref_none else torch.from_numpy(ref).to(dev)
    r = G.grpo_loss_bwd(H, W, tok, mask, f["logp"], f["lse"], old_t, ref_t, adv,
                        f["valid_count"], ws, eps_low=eps_low, eps_high=eps_high, beta=beta,
                        agg=agg, norm=norm)
    torch.cuda.synchronize()
    st, where = G.grpo_last_device_error(ws)
    out = {k: v.cpu() for k, v in f.items()}
    out.update({"adv": adv.cpu(), "loss": float(r["loss"].cpu()[0]), "dH": r["dH"].float().cpu(),
                "dW": r["dW"].cpu(), "status": st, "where": where})
    return out


def rel_fro(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))


def check_loss(loss_gpu, loss_oracle, mass, rep):
    """The loss bar. L sums terms w_t l_t whose advantages cancel within each group, so |L| can
    be far below the magnitude of what is summed (mass = sum_t |w_t l_t|) and a relative error
    against |L| alone is unbounded as L -> 0. Asserted: |dL| <= 1e-3 max(|L|, mass) always, and
    the plain |dL| / |L| <= 1e-3 wherever |L| >= 1e-2 mass (L not dominated by cancellation)."""
    err = abs(loss_gpu - loss_oracle)
    scale = max(abs(loss_oracle), mass)
    rep["loss_err_rel_mass"] = err / scale if scale > 0 else 0.0
    rep["loss_err_rel"] = err / abs(loss_oracle) if loss_oracle else 0.0
    rep["loss_over_mass"] = abs(loss_oracle) / mass if mass > 0 else 0.0
    assert rep["loss_err_rel_mass"] <= LOSS_RTOL, (loss_gpu, loss_oracle, rep)
    if abs(loss_oracle) >= 1e-2 * mass:
        assert rep["loss_err_rel"] <= LOSS_RTOL, (loss_gpu, loss_oracle, rep)


def compare(batch, g, o, check_grads=True):
    """Asserts the parity bar; returns a dict of the measured errors."""
    mask = batch.mask.cpu().numpy() != 0
    rep = {}
    assert g["status"] == 0, ("device status", g["status"], g["where"])
    assert np.array_equal(g["valid_count"].numpy(), o["counts"]), "valid counts differ"
    np.testing.assert_allclose(g["adv"].numpy(), o["adv"], rtol=1e-5, atol=2e-6)
    assert np.all(g["adv"].numpy()[o["adv"] == 0.0] == 0.0), "degenerate advantages not exactly 0"
    for k in ("logp", "lse", "entropy"):
        e = float(np.abs(g[k].numpy()[mask] - o[k][mask]).max()) if mask.any() else 0.0
        rep[k] = e
        assert e <= LOGP_ATOL, f"{k} max abs error {e}"
        assert np.all(g[k].numpy()[~mask] == 0.0), f"{k} not zero at unscored positions"
    am_g = g["argmax"].numpy()
    assert np.all(am_g[~mask] == -1)
    # argmax: bit-exact, except where the top-2 logits are closer than the f32 accumulation bound
    H = batch.H.cpu().double().numpy()
    W = batch.W.cpu().double().numpy()
    d = H.shape[-1]
    diff = np.argwhere(mask & (am_g != o["argmax"]))
    near = 0
    for s, t in diff:
        a, b = o["argmax"][s, t], am_g[s, t]
        bound = 2.0 * d * 2.0 ** -24 * (np.abs(H[s, t]) @ (np.abs(W[a]) + np.abs(W[b])))
        z = H[s, t] @ W.T
        assert abs(z[a] - z[b]) <= bound, f"argmax mismatch at {(s, t)}: {a} vs {b}"
        near += 1
    rep["argmax_near_ties"] = near
    check_loss(g["loss"], o["loss"], o["loss_abs_mass"], rep)
    if check_grads:
        rep["dH"] = rel_fro(g["dH"].numpy(), o["dH"])
        rep["dW"] = rel_fro(g["dW"].numpy(), o["dW"])
        assert rep["dH"] <= GRAD_RTOL, rep
        assert rep["dW"] <= GRAD_RTOL, rep
        assert np.all(g["dH"].numpy()[~mask] == 0.0), "dH not zero at unscored positions"
    return rep
