"""Pins of the CPU oracle to facts outside itself (no GPU).

Each pin takes the oracle module as an argument so that ``test_oracle_mutations.py`` can run the
same pins against copies of the oracle with a planted mistake and check that some pin fails.
The pins: closed forms (uniform logits, hand-derived surrogate/KL/advantage values in
``tests/golden/closed_forms.json``), library routines (scipy ``log_softmax``/``logsumexp``,
``scipy.stats.entropy``, ``scipy.stats.zscore``, torch float64 autograd), invariants (advantages
sum to zero, dW rows sum to zero) and central finite differences in float64.
"""
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle.grpo_oracle as O
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "closed_forms.json")


def _num(x):
    if isinstance(x, str):
        return math.log(float(x[2:]))
    return float(x)


# ---------------------------------------------------------------------------------------------
# pins, written against a module argument
# ---------------------------------------------------------------------------------------------

def pin_uniform_logits(o):
    """W = 0 (and W with identical rows) gives uniform logits: logp = -log V, lse = log V +
    const, entropy = log V, argmax = 0."""
    rng = np.random.default_rng(1)
    for V in (2, 7, 512):
        d, n = 16, 5
        h = rng.normal(size=(n, d))
        y = rng.integers(0, V, size=n)
        sc = o.score_tokens(h, np.zeros((V, d)), y)
        np.testing.assert_allclose(sc["logp"], -math.log(V), rtol=0, atol=1e-12)
        np.testing.assert_allclose(sc["lse"], math.log(V), rtol=0, atol=1e-12)
        np.testing.assert_allclose(sc["entropy"], math.log(V), rtol=0, atol=1e-12)
        assert np.all(sc["argmax"] == 0)
        row = rng.normal(size=d)
        sc = o.score_tokens(h, np.tile(row, (V, 1)), y)
        np.testing.assert_allclose(sc["logp"], -math.log(V), atol=1e-12)
        np.testing.assert_allclose(sc["entropy"], math.log(V), atol=1e-12)
        np.testing.assert_allclose(sc["lse"], h @ row + math.log(V), atol=1e-12)


def pin_scipy_log_softmax(o):
    """logp and lse equal scipy's log_softmax / logsumexp of the logits W h."""
    rng = np.random.default_rng(2)
    n, d, V = 40, 24, 300
    h = rng.normal(size=(n, d))
    W = rng.normal(scale=0.3, size=(V, d))
    y = rng.integers(0, V, size=n)
    sc = o.score_tokens(h, W, y)
    Z = h @ W.T
    np.testing.assert_allclose(sc["lse"], scipy.special.logsumexp(Z, axis=1), rtol=1e-13)
    ls = scipy.special.log_softmax(Z, axis=1)
    np.testing.assert_allclose(sc["logp"], ls[np.arange(n), y], rtol=1e-12, atol=1e-12)


def pin_scipy_entropy(o):
    """entropy = scipy.stats.entropy(softmax(z)) in nats."""
    rng = np.random.default_rng(3)
    n, d, V = 30, 16, 257
    h = rng.normal(size=(n, d))
    W = rng.normal(scale=0.5, size=(V, d))
    y = rng.integers(0, V, size=n)
    sc = o.score_tokens(h, W, y)
    P = scipy.special.softmax(h @ W.T, axis=1)
    np.testing.assert_allclose(sc["entropy"], scipy.stats.entropy(P, axis=1), rtol=1e-11)


def pin_argmax_ties(o):
    """Ties go to the lowest vocabulary index; otherwise argmax is numpy's first maximum."""
    rng = np.random.default_rng(4)
    d, V = 8, 64
    W = rng.normal(size=(V, d))
    h = rng.normal(size=(6, d))
    best = (h @ W.T).argmax(axis=1)
    W2 = W.copy()
    for j, b in enumerate(best):
        W2[(b + 17 + j) % V] = W2[b]             # duplicate the winning row at another index
    sc = o.score_tokens(h, W2, np.zeros(6, int))
    Z = h @ W2.T
    for j in range(6):
        cands = np.flatnonzero(Z[j] == Z[j].max())
        assert sc["argmax"][j] == cands.min()


def pin_golden_objective(o):
    cases = json.load(open(GOLDEN))["token_objective"]
    for c in cases:
        old = 0.0 - _num(c["logp_minus_old"])
        ref = 0.0 + _num(c["ref_minus_logp"])
        t = o.token_objective(np.array([0.0]), np.array([old]), np.array([ref]), np.array([c["A"]]),
                              c["eps_low"], c["eps_high"], c["beta"])
        for k in ("surr", "kl", "ell", "dell"):
            assert abs(float(t[k][0]) - c[k]) <= 1e-12, (c["why"], k, float(t[k][0]), c[k])


def pin_golden_advantages(o):
    for c in json.load(open(GOLDEN))["group_advantages"]:
        a = o.group_advantages(np.array(c["rewards"], np.float32), np.array(c["offsets"]),
                               c["std_mode"], c["std_eps"])
        np.testing.assert_allclose(a, c["adv"], rtol=1e-6, atol=1e-7, err_msg=c["why"])
        for v, want in zip(a, c["adv"]):
            if want == 0.0:
                assert v == 0.0, c["why"]              # degenerate groups: exactly zero


def pin_advantages_scipy_and_invariants(o):
    """z-score per group equals scipy.stats.zscore (ddof 1 unbiased / 0 population) when
    std_eps = 0; with std_eps > 0, sum A = 0 and sum A^2 = dof sigma^2 / (sigma + eps)^2."""
    rng = np.random.default_rng(5)
    sizes = [4, 8, 12, 16, 1, 5]
    go = np.concatenate([[0], np.cumsum(sizes)])
    r = rng.normal(size=go[-1]).astype(np.float32)
    for mode, ddof in (("unbiased", 1), ("population", 0)):
        a = o.group_advantages(r, go, mode, 0.0)
        for g in range(len(sizes)):
            lo, hi = go[g], go[g + 1]
            if hi - lo <= 1:
                assert np.all(a[lo:hi] == 0.0)
                continue
            np.testing.assert_allclose(a[lo:hi], scipy.stats.zscore(r[lo:hi].astype(np.float64),
                                                                    ddof=ddof), rtol=1e-10)
        eps = 1e-4
        a = o.group_advantages(r, go, mode, eps)
        for g in range(len(sizes)):
            lo, hi = go[g], go[g + 1]
            G = hi - lo
            if G <= 1:
                continue
            rg = r[lo:hi].astype(np.float64)
            sig = rg.std(ddof=ddof)
            assert abs(a[lo:hi].sum()) < 1e-10
            np.testing.assert_allclose((a[lo:hi] ** 2).sum(), (G - ddof) * sig**2 / (sig + eps) ** 2,
                                       rtol=1e-10)


def _loss_of(o, h, W, y, old, ref, adv_tok, seq, counts, S, eps_lo, eps_hi, beta, agg):
    sc = o.score_tokens(h, W, y)
    t = o.token_objective(sc["logp"], old, ref, adv_tok, eps_lo, eps_hi, beta)
    L, g, _ = o.aggregate(t["ell"], t["dell"], seq, counts, S, agg)
    return L, g, sc


def _tiny_problem(seed=6, V=8, d=4, S=3, T=5):
    rng = np.random.default_rng(seed)
    mask = (rng.random((S, T)) < 0.8).astype(np.uint8)
    mask[:, 0] = 1
    H = rng.normal(size=(S, T, d))
    W = rng.normal(scale=0.7, size=(V, d))
    tokens = rng.integers(0, V, size=(S, T))
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    adv = rng.normal(size=S)
    # keep the ratio away from the clip kinks so that central differences see one branch
    old = rng.normal(scale=0.6, size=(S, T))
    ref = rng.normal(scale=0.5, size=(S, T))
    return H, W, tokens, mask, si, ti, adv, old, ref


def pin_finite_differences(o, agg=O.SEQ_MEAN):
    """Central differences (float64, h = 1e-6) of the loss built from the oracle's forward
    agree with its dH and dW on every entry of a V=8, d=4 problem."""
    H, W, tokens, mask, si, ti, adv, old0, ref0 = _tiny_problem()
    S = H.shape[0]
    counts = o.valid_counts(mask)
    y = tokens[si, ti]
    # old/ref are fixed numbers (detached), as in a GRPO step
    sc0 = o.score_tokens(H[si, ti], W, y)
    old = sc0["logp"] + old0[si, ti]
    ref = sc0["logp"] + ref0[si, ti]
    args = (y, old, ref, adv[si], si, counts, S, 0.2, 0.3, 0.05, agg)

    def L_of(Hv, Wv):
        return _loss_of(o, Hv, Wv, *args)[0]

    h = H[si, ti]
    _, g, sc = _loss_of(o, h, W, *args)
    dH, dW = o.param_grads(h, W, y, sc["lse"], g)
    step = 1e-6
    num_dH = np.zeros_like(h)
    for idx in np.ndindex(*h.shape):
        hp, hm = h.copy(), h.copy()
        hp[idx] += step
        hm[idx] -= step
        num_dH[idx] = (L_of(hp, W) - L_of(hm, W)) / (2 * step)
    num_dW = np.zeros_like(W)
    for idx in np.ndindex(*W.shape):
        Wp, Wm = W.copy(), W.copy()
        Wp[idx] += step
        Wm[idx] -= step
        num_dW[idx] = (L_of(h, Wp) - L_of(h, Wm)) / (2 * step)
    np.testing.assert_allclose(dH, num_dH, rtol=1e-5, atol=1e-9)
    np.testing.assert_allclose(dW, num_dW, rtol=1e-5, atol=1e-9)


def pin_on_policy_reinforce(o):
    """old = logp (rho = 1) and beta = 0 reduce the GRPO loss to Eq. 1's first term: per token
    g_t = -A_i / (S n_i) (seq_mean) or -A_i / N (token_mean), and L = -(1/S) sum_i A_i which is 0
    when the advantages of each group sum to zero."""
    b = make_batch_numpy(WORKLOADS["tiny_f32"])
    mask = b.mask.numpy()
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    H, W, y = b.H.double().numpy(), b.W.double().numpy(), b.tokens.numpy()[si, ti]
    sc = o.score_tokens(H[si, ti], W, y)
    adv = o.group_advantages(b.rewards.numpy(), b.group_offsets.numpy())
    counts = o.valid_counts(mask)
    S = mask.shape[0]
    t = o.token_objective(sc["logp"], sc["logp"], sc["logp"], adv[si], 0.2, 0.2, 0.0)
    L, g, _ = o.aggregate(t["ell"], t["dell"], si, counts, S, O.SEQ_MEAN)
    np.testing.assert_allclose(g, -adv[si] / (S * counts[si]), rtol=1e-12)
    assert abs(L - (-adv.sum() / S)) < 1e-12 and abs(L) < 1e-9
    L2, g2, _ = o.aggregate(t["ell"], t["dell"], si, counts, S, O.TOKEN_MEAN)
    np.testing.assert_allclose(g2, -adv[si] / counts.sum(), rtol=1e-12)
    # beta = 0.04 with ref = logp adds nothing; the KL term vanishes with its gradient
    t4 = o.token_objective(sc["logp"], sc["logp"], sc["logp"], adv[si], 0.2, 0.2, 0.04)
    np.testing.assert_allclose(t4["dell"], t["dell"], rtol=0, atol=0)
    assert np.all(t4["kl"] == 0)


def pin_torch_autograd(o):
    """torch float64 autograd of the same definitions (log_softmax + gather + min/clamp ratio +
    e^d - d - 1) gives the oracle's loss, dH and dW on the tiny FP32 workload."""
    b = make_batch_numpy(WORKLOADS["tiny_f32"])
    mask = b.mask.numpy()
    S = mask.shape[0]
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    H, W = b.H.double().numpy(), b.W.double().numpy()
    y = b.tokens.numpy()[si, ti]
    base = o.score_tokens(H[si, ti], W, y)["logp"]
    old = base + b.noise_old.numpy()[si, ti] * 6.0            # wide noise: exercise clipping
    ref = base + b.noise_ref.numpy()[si, ti]
    adv = o.group_advantages(b.rewards.numpy(), b.group_offsets.numpy())
    counts = o.valid_counts(mask)
    eps_lo, eps_hi, beta = 0.2, 0.28, 0.04
    L, g, sc = _loss_of(o, H[si, ti], W, y, old, ref, adv[si], si, counts, S, eps_lo, eps_hi,
                        beta, O.SEQ_MEAN)
    dH, dW = o.param_grads(H[si, ti], W, y, sc["lse"], g)

    th = torch.tensor(H[si, ti], requires_grad=True)
    tW = torch.tensor(W, requires_grad=True)
    lp = torch.log_softmax(th @ tW.T, dim=1).gather(1, torch.tensor(y)[:, None])[:, 0]
    rho = torch.exp(lp - torch.tensor(old))
    A = torch.tensor(adv[si])
    surr = torch.minimum(rho * A, torch.clamp(rho, 1 - eps_lo, 1 + eps_hi) * A)
    dl = torch.tensor(ref) - lp
    ell = -surr + beta * (torch.exp(dl) - dl - 1)
    w = torch.tensor(1.0 / (S * counts[si]))
    Lt = (w * ell).sum()
    Lt.backward()
    assert abs(Lt.item() - L) < 1e-12
    np.testing.assert_allclose(dH, th.grad.numpy(), rtol=1e-9, atol=1e-15)
    np.testing.assert_allclose(dW, tW.grad.numpy(), rtol=1e-9, atol=1e-15)


def pin_dW_rows_sum_to_zero(o):
    """sum_v dz_tv = g_t (1 - sum_v p_tv) = 0, so the rows of dW sum to the zero vector and
    dH_t = g_t (W[y_t] - sum_v p_tv W_v)."""
    H, W, tokens, mask, si, ti, adv, old0, ref0 = _tiny_problem(seed=9, V=50, d=6, S=4, T=7)
    h = H[si, ti]
    y = tokens[si, ti]
    sc = o.score_tokens(h, W, y)
    g = np.random.default_rng(0).normal(size=len(y))
    dH, dW = o.param_grads(h, W, y, sc["lse"], g)
    scale = np.abs(dW).sum(axis=0)
    assert np.all(np.abs(dW.sum(axis=0)) <= 1e-12 * np.maximum(scale, 1.0))
    P = scipy.special.softmax(h @ W.T, axis=1)
    np.testing.assert_allclose(dH, g[:, None] * (W[y] - P @ W), rtol=1e-10, atol=1e-14)


def pin_vocab_row_subset(o):
    H, W, tokens, mask, si, ti, adv, _, _ = _tiny_problem(seed=10, V=40, d=5)
    h, y = H[si, ti], tokens[si, ti]
    sc = o.score_tokens(h, W, y)
    g = np.linspace(-1, 1, len(y))
    _, dW = o.param_grads(h, W, y, sc["lse"], g)
    rows = np.array([0, 3, 39, 17])
    _, dWr = o.param_grads(h, W, y, sc["lse"], g, vocab_rows=rows)
    np.testing.assert_array_equal(dWr, dW[rows])


def pin_counts(o):
    rng = np.random.default_rng(11)
    mask = (rng.random((7, 33)) < 0.5).astype(np.uint8)
    mask[3] = 0
    brute = [sum(1 for t in range(33) if mask[i, t]) for i in range(7)]
    assert list(o.valid_counts(mask)) == brute


def pin_sft_torch_cross_entropy(o):
    """Sec. 6.2 distillation loss = torch's cross_entropy (mean over target tokens), and its
    gradients through the LM head equal torch float64 autograd; uniform logits give log V."""
    b = make_batch_numpy(WORKLOADS["tiny_f32"])
    H, W = b.H.double().numpy(), b.W.double().numpy()
    mask = b.mask.numpy()
    tok = b.tokens.numpy()
    out = o.sft_step(H, W, tok, mask)
    idx = np.argwhere(mask != 0)
    th = torch.tensor(H[idx[:, 0], idx[:, 1]], requires_grad=True)
    tW = torch.tensor(W, requires_grad=True)
    L = torch.nn.functional.cross_entropy(th @ tW.T, torch.tensor(tok[idx[:, 0], idx[:, 1]]).long())
    L.backward()
    assert abs(L.item() - out["loss"]) < 1e-12
    np.testing.assert_allclose(out["dH"][idx[:, 0], idx[:, 1]], th.grad.numpy(), rtol=1e-9,
                               atol=1e-15)
    np.testing.assert_allclose(out["dW"], tW.grad.numpy(), rtol=1e-9, atol=1e-15)
    u = o.sft_step(H, np.zeros_like(W), tok, mask, with_grads=False)
    assert abs(u["loss"] - math.log(W.shape[0])) < 1e-12


def pin_golden_rewards(o):
    for c in json.load(open(GOLDEN))["rewards"]:
        rp = o.perf_reward(np.array([c["correct"]]), np.array([c["t_base"]]), np.array([c["t_new"]]))
        rt = o.tool_reward(np.array([c["tools_used"]]), np.array([c["tools_avail"]]))
        r = o.reward(np.array([c["correct"]]), np.array([c["t_base"]]), np.array([c["t_new"]]),
                     np.array([c["tools_used"]]), np.array([c["tools_avail"]]))
        assert abs(rp[0] - c["r_perf"]) < 1e-12 and abs(rt[0] - c["r_tools"]) < 1e-12, c["why"]
        assert abs(r[0] - c["r"]) < 1e-12, c["why"]


def pin_vocab_shards_merge_to_full_vocab(o):
    """For any partition of the vocabulary into shards (uneven, tiny, with exact ties across
    shards) the merged shard statistics equal the whole-vocabulary scoring."""
    rng = np.random.default_rng(13)
    n, d, V = 25, 12, 103
    h = rng.normal(size=(n, d))
    W = rng.normal(scale=0.4, size=(V, d))
    a = int((h @ W.T).argmax(axis=1)[0])
    b = (a + 51) % V
    W[b] = W[a]                                      # exact tie for token 0, in another shard
    cut = (min(a, b) + max(a, b)) // 2 + 1
    y = rng.integers(0, V, size=n)
    full = o.score_tokens(h, W, y)
    for cuts in ([0, V], [0, 50, V], [0, 1, 40, 41, 90, V], [0, cut, V]):
        st = [o.shard_stats(h, W[a:b], y, a) for a, b in zip(cuts[:-1], cuts[1:])]
        mg = o.merge_shard_stats(st)
        for k in ("lse", "logp", "entropy"):
            np.testing.assert_allclose(mg[k], full[k], rtol=1e-12, atol=1e-12)
        assert np.array_equal(mg["argmax"], full["argmax"])


def pin_exact_kl_torch_and_finite_differences(o):
    """The exact per-token KL equals torch.distributions.kl_divergence of the two categorical
    distributions, is 0 when the reference equals the policy, and the GRPO loss with the exact
    KL has dH / dW equal to central finite differences (V = 9, d = 5)."""
    rng = np.random.default_rng(17)
    n, d, V = 7, 5, 9
    h, hr = rng.normal(size=(n, d)), rng.normal(size=(n, d))
    W, Wr = rng.normal(scale=0.6, size=(V, d)), rng.normal(scale=0.6, size=(V, d))
    ek = o.exact_kl(h, W, hr, Wr)
    tk = torch.distributions.kl_divergence(
        torch.distributions.Categorical(logits=torch.tensor(h @ W.T)),
        torch.distributions.Categorical(logits=torch.tensor(hr @ Wr.T))).numpy()
    np.testing.assert_allclose(ek["kl"], tk, rtol=1e-10, atol=1e-13)
    assert np.all(ek["kl"] >= 0)
    np.testing.assert_allclose(o.exact_kl(h, W, h, W)["kl"], 0.0, atol=1e-13)
    S, T = 2, 4
    H = rng.normal(size=(S, T, d))
    Hr = rng.normal(size=(S, T, d))
    mask = np.ones((S, T), np.uint8)
    mask[1, 3] = 0
    tok = rng.integers(0, V, size=(S, T))
    rew = np.array([0.3, 1.1], np.float32)
    go = np.array([0, 2])
    old = rng.normal(-2.2, 0.7, size=(S, T))
    beta = 0.3
    base = o.grpo_step_exact_kl(H, W, Hr, Wr, tok, mask, rew, go, old, 0.2, 0.2, beta)
    step = 1e-6

    def L_of(Hx, Wx):
        return o.grpo_step_exact_kl(Hx, Wx, Hr, Wr, tok, mask, rew, go, old, 0.2, 0.2, beta,
                                    with_grads=False)["loss"]
    for idx in np.ndindex(*H.shape):
        if not mask[idx[0], idx[1]]:
            continue
        Hp, Hm = H.copy(), H.copy()
        Hp[idx] += step
        Hm[idx] -= step
        num = (L_of(Hp, W) - L_of(Hm, W)) / (2 * step)
        assert abs(num - base["dH"][idx]) <= 1e-6 * max(1e-3, abs(num)), (idx, num, base["dH"][idx])
    for idx in np.ndindex(*W.shape):
        Wp, Wm = W.copy(), W.copy()
        Wp[idx] += step
        Wm[idx] -= step
        num = (L_of(H, Wp) - L_of(H, Wm)) / (2 * step)
        assert abs(num - base["dW"][idx]) <= 1e-6 * max(1e-3, abs(num)), (idx, num, base["dW"][idx])


PINS = [pin_uniform_logits, pin_scipy_log_softmax, pin_scipy_entropy, pin_argmax_ties,
        pin_golden_objective, pin_golden_advantages, pin_advantages_scipy_and_invariants,
        pin_finite_differences, pin_on_policy_reinforce, pin_torch_autograd,
        pin_dW_rows_sum_to_zero, pin_vocab_row_subset, pin_counts, pin_sft_torch_cross_entropy,
        pin_golden_rewards, pin_vocab_shards_merge_to_full_vocab,
        pin_exact_kl_torch_and_finite_differences]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_oracle_pin(pin):
    pin(O)


def test_finite_differences_token_mean():
    pin_finite_differences(O, agg=O.TOKEN_MEAN)


def test_finite_differences_sampled_entries_tiny_workload():
    """Central differences on a seeded sample of dH and dW entries of the 1 x 4 x 64, d=64,
    V=512 workload with the full GRPO objective (eps=0.2, beta=0.04)."""
    b = make_batch_numpy(WORKLOADS["tiny_f32"])
    mask = b.mask.numpy()
    S = mask.shape[0]
    H, W = b.H.double().numpy(), b.W.double().numpy()
    base = O.grpo_step(H, W, b.tokens.numpy(), mask, b.rewards.numpy(), b.group_offsets.numpy(),
                       np.zeros_like(mask, float), np.zeros_like(mask, float), with_grads=False)
    old = base["logp"] + b.noise_old.numpy()
    ref = base["logp"] + b.noise_ref.numpy()
    args = (b.tokens.numpy(), mask, b.rewards.numpy(), b.group_offsets.numpy(), old, ref)
    full = O.grpo_step(H, W, *args)
    rng = np.random.default_rng(12)
    idx = np.argwhere(mask != 0)
    step = 1e-6
    for _ in range(12):
        s, t = idx[rng.integers(len(idx))]
        k = rng.integers(H.shape[2])
        Hp, Hm = H.copy(), H.copy()
        Hp[s, t, k] += step
        Hm[s, t, k] -= step
        num = (O.grpo_step(Hp, W, *args, with_grads=False)["loss"]
               - O.grpo_step(Hm, W, *args, with_grads=False)["loss"]) / (2 * step)
        assert abs(num - full["dH"][s, t, k]) <= 1e-6 * max(1e-3, abs(num)), (num, full["dH"][s, t, k])
    for _ in range(12):
        v, k = rng.integers(W.shape[0]), rng.integers(W.shape[1])
        Wp, Wm = W.copy(), W.copy()
        Wp[v, k] += step
        Wm[v, k] -= step
        num = (O.grpo_step(H, Wp, *args, with_grads=False)["loss"]
               - O.grpo_step(H, Wm, *args, with_grads=False)["loss"]) / (2 * step)
        assert abs(num - full["dW"][v, k]) <= 1e-6 * max(1e-3, abs(num)), (num, full["dW"][v, k])
    assert S == 4
