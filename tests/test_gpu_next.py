"""Widened rows: the distillation (SFT) loss of Sec. 6.2 through the same tensor-core path, and
the rewards of Eqs. 2-4 feeding the group advantages, against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy
from tests.parity_util import GRAD_RTOL, LOGP_ATOL, rel_fro

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,over,agg", [
    ("g8_t1k_d2048_v32k", dict(T=300, len_lo=64, len_hi=300, holes=True), "token_mean"),
    ("g8_t4k_d4096_v152k", dict(group_sizes=(3,), T=150, len_lo=40, len_hi=150), "seq_mean"),
    ("tiny_f32", {}, "token_mean"),
])
def test_sft_distillation_parity(name, over, agg):
    b = make_batch_numpy(WORKLOADS[name].scaled(**over))
    H, W, tok, mask = (t.cuda() for t in (b.H, b.W, b.tokens, b.mask))
    S, T, d = H.shape
    ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
    f = G.grpo_score_fwd(H, W, tok, mask, ws)
    r = G.grpo_sft_loss_bwd(H, W, tok, mask, f["logp"], f["lse"], f["valid_count"], ws, agg=agg)
    torch.cuda.synchronize()
    assert G.grpo_last_device_error(ws)[0] == 0
    o = oracle.sft_step(b.H.double().numpy(), b.W.double().numpy(), b.tokens.numpy(),
                        b.mask.numpy(), agg=agg)
    m = b.mask.numpy() != 0
    assert np.abs(f["logp"].cpu().numpy()[m] - o["logp"][m]).max() <= LOGP_ATOL
    loss = float(r["loss"].item())
    assert abs(loss - o["loss"]) <= 1e-3 * abs(o["loss"]), (loss, o["loss"])
    e_h = rel_fro(r["dH"].float().cpu().numpy(), o["dH"])
    e_w = rel_fro(r["dW"].cpu().numpy(), o["dW"])
    assert e_h <= GRAD_RTOL and e_w <= GRAD_RTOL, (e_h, e_w)
    print(name, "loss", loss, o["loss"], "dH", e_h, "dW", e_w)


def _reward_inputs(n, seed):
    rng = np.random.default_rng(seed)
    correct = (rng.random(n) < 0.7).astype(np.uint8)
    t_base = rng.uniform(0.1, 5.0, n).astype(np.float32)
    speed = np.exp(rng.uniform(np.log(0.3), np.log(40.0), n)).astype(np.float32)
    t_new = (t_base / speed).astype(np.float32)
    t_new[::17] = t_base[::17]                       # exactly unchanged time: reward 0
    avail = rng.integers(4, 7, n).astype(np.int32)    # 4-6 tools offered (Sec. 6.1)
    used = rng.integers(0, 7, n).astype(np.int32)
    used = np.minimum(used, avail).astype(np.int32)
    return correct, t_base, t_new, used, avail


def test_rewards_parity_and_boundaries():
    c, tb, tn, u, a = _reward_inputs(4099, 3)
    r = G.grpo_rewards(*(torch.from_numpy(x).cuda() for x in (c, tb, tn, u, a))).cpu().numpy()
    o = oracle.reward(c, tb.astype(np.float64), tn.astype(np.float64), u, a)
    rp = oracle.perf_reward(c, tb.astype(np.float64), tn.astype(np.float64))
    # the branch (incorrect / slower / speedup) is decided on the same f32 inputs on both sides
    for lab in (-2.0, -1.0):
        assert np.array_equal(np.isclose(r - oracle.tool_reward(u, a), lab, atol=1e-6), rp == lab)
    np.testing.assert_allclose(r, o, rtol=2e-6, atol=2e-6)
    keep = c[::17] == 1
    want = (np.float32(0.5) * u[::17][keep].astype(np.float32)) / a[::17][keep].astype(np.float32)
    assert np.array_equal(r[::17][keep], want.astype(np.float32))   # unchanged time: r_perf = 0
    bad = G.grpo_rewards(*(torch.from_numpy(x).cuda() for x in (
        c[:3], tb[:3], tn[:3], np.array([1, 5, -1], np.int32), np.array([0, 4, 4], np.int32))))
    assert torch.isnan(bad).all()


def test_rewards_feed_group_advantages():
    c, tb, tn, u, a = _reward_inputs(12 * 16, 4)           # 16 prompts x K = 12 (Sec. 6.1)
    go = np.arange(0, 12 * 17, 12, dtype=np.int32)
    ws = G.Workspace.create(256)
    r = G.grpo_rewards(*(torch.from_numpy(x).cuda() for x in (c, tb, tn, u, a)))
    adv = G.group_advantages(r, torch.from_numpy(go).cuda(), ws).cpu().numpy()
    r_o = oracle.reward(c, tb.astype(np.float64), tn.astype(np.float64), u, a)
    adv_o = oracle.group_advantages(r.cpu().numpy(), go)
    np.testing.assert_allclose(r.cpu().numpy(), r_o, rtol=2e-6, atol=2e-6)
    np.testing.assert_allclose(adv, adv_o, rtol=1e-5, atol=2e-6)


@pytest.mark.parametrize("name,over", [
    ("g8_t1k_d2048_v32k", dict(prompts=1, group_sizes=(4,), T=260, len_lo=60, len_hi=260)),
    ("g16_t16k_d5120_v152k", dict(group_sizes=(3,), prompts=1, T=140, len_lo=30, len_hi=140)),
])
def test_exact_kl_parity(name, over):
    """Eq. 1's KL taken exactly over the vocabulary against a frozen reference model."""
    from paper_2510_17158_gb300.synthetic import reference_model_inputs
    from tests.parity_util import oracle_inputs
    b = make_batch_numpy(WORKLOADS[name].scaled(**over))
    w = b.workload
    Hr, Wr = reference_model_inputs(b)
    H, W, tok, mask = (t.cuda() for t in (b.H, b.W, b.tokens, b.mask))
    S, T, d = H.shape
    ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype, kl=True)
    old, _ = oracle_inputs(b, old_scale=2.0)
    adv = G.group_advantages(b.rewards.cuda(), b.group_offsets.cuda(), ws)
    f = G.grpo_score_fwd_kl(H, W, Hr.cuda(), Wr.cuda(), tok, mask, ws)
    r = G.grpo_loss_bwd_kl(H, W, Hr.cuda(), Wr.cuda(), tok, mask, f, torch.from_numpy(old).cuda(),
                           adv, ws, eps_low=w.eps, eps_high=w.eps, beta=0.5)
    torch.cuda.synchronize()
    assert G.grpo_last_device_error(ws)[0] == 0
    o = oracle.grpo_step_exact_kl(b.H.double().numpy(), b.W.double().numpy(),
                                  Hr.double().numpy(), Wr.double().numpy(), b.tokens.numpy(),
                                  b.mask.numpy(), b.rewards.numpy(), b.group_offsets.numpy(),
                                  old.astype(np.float64), w.eps, w.eps, 0.5)
    m = b.mask.numpy() != 0
    for k in ("logp", "lse", "entropy", "lse_ref", "kl"):
        e = np.abs(f[k].cpu().numpy()[m] - o[k][m]).max()
        assert e <= LOGP_ATOL, (k, e)
    loss = float(r["loss"].item())
    assert abs(loss - o["loss"]) <= 1e-3 * max(abs(o["loss"]), o["loss_abs_mass"]), (loss, o["loss"])
    e_h = rel_fro(r["dH"].float().cpu().numpy(), o["dH"])
    e_w = rel_fro(r["dW"].cpu().numpy(), o["dW"])
    assert e_h <= GRAD_RTOL and e_w <= GRAD_RTOL, (e_h, e_w)
    print(name, "kl mean", float(o["kl"][m].mean()), "loss", loss, o["loss"], "dH", e_h, "dW", e_w)
