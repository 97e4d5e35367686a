"""Plain CPU float64 oracle of one GRPO update's token-scoring, loss and backward path.

TEST INFRASTRUCTURE. Only the test suite, ``__graft_entry__.smoke()`` and the ``cpu_baseline``
leg of ``bench.py`` may import or run this module. It shares no code with the CUDA path and
imports nothing from the package: callers hand it plain numpy arrays.

What it computes (arxiv 2510.17158):

* Eq. 1 (Sec. 2.1) is the GRPO objective
  ``L = E_{x~pi}[-w(x) log pi(x|c)] + beta KL(pi || pi_ref)``, where ``w(x)`` is the reward of
  ``x`` normalised within its group of K completions (Sec. 2.1; Alg. 1).
* Sec. 6.1 keeps the standard GRPO policy update of DeepSeekMath, i.e. the
  per-token probability ratio with a clipped surrogate; Alg. 1 computes the KL to a frozen
  reference and takes a gradient step on L.
* ``log pi(x|c)`` is the sum over the completion's sampled tokens of the log-softmax of the
  LM-head logits ``z_t = W h_t`` at the sampled token.

Readings of points the paper leaves open (each one is a documented choice):

* advantage = z-score within the group, ``(r - mean) / (std + std_eps)``; std unbiased by
  default (population on request); a group of one, or whose rewards are all equal, gets 0;
* ratio ``rho = exp(logp - old)``; surrogate ``min(rho A, clip(rho, 1-eps_lo, 1+eps_hi) A)``;
* KL per sampled token with the non-negative estimator ``e^delta - delta - 1``,
  ``delta = ref - logp``;
* per-token loss ``l = -surr + beta kl``; aggregation "seq_mean" ``(1/S) sum_i (1/n_i) sum_t l``
  (default; a sequence with no scored token adds 0 and still counts in S) or "token_mean"
  ``sum l / sum n``; masked tokens (padding, tool-result text) are not scored;
* the subgradient of the clipped surrogate takes the unclipped branch when it is active with
  inclusive boundaries: active iff (A >= 0 and rho <= 1+eps_hi) or (A < 0 and rho >= 1-eps_lo);
* argmax ties go to the lowest vocabulary index; entropy is in nats;
* distillation (Sec. 6.2) is token cross-entropy with the same aggregation choices;
* the performance reward's branch for a correct but slower kernel is t > t_base.

Every input is converted exactly to float64 (bf16 and fp32 values are exactly representable).
"""
from __future__ import annotations

import numpy as np

SEQ_MEAN = "seq_mean"
TOKEN_MEAN = "token_mean"


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def valid_counts(mask):
    """n_i = number of scored tokens of completion i (Eq. 1 takes its expectation over sampled
    completion tokens; tool-result text appended inside a completion (Sec. 5) is not sampled
    from the policy and is masked out)."""
    m = np.asarray(mask)
    return (m != 0).sum(axis=1).astype(np.int64)


def group_advantages(rewards, group_offsets, std_mode="unbiased", std_eps=1e-4):
    """w(x_k) of Eq. 1: the reward of completion k normalised within its group, which Alg. 1
    turns into the advantages (Sec. 2.1; Alg. 1).

    ``group_offsets[g] .. group_offsets[g+1]`` are the completions of prompt g (contiguous).
    """
    r = _f64(rewards)
    go = np.asarray(group_offsets, dtype=np.int64)
    adv = np.zeros_like(r)
    for g in range(len(go) - 1):
        lo, hi = int(go[g]), int(go[g + 1])
        G = hi - lo
        if G <= 1:
            continue
        rg = r[lo:hi]
        if np.all(np.asarray(rewards)[lo:hi] == np.asarray(rewards)[lo]):
            continue                      # degenerate group: no relative signal, advantage 0
        mu = rg.sum() / G
        dof = G - 1 if std_mode == "unbiased" else G
        sigma = np.sqrt(((rg - mu) ** 2).sum() / dof)
        adv[lo:hi] = (rg - mu) / (sigma + std_eps)
    return adv


def score_tokens(h, W, y):
    """Per-token scoring of Eq. 1's log pi(x|c): for each row h_t and sampled token y_t,
    z_t = W h_t over the whole vocabulary, lse_t = log sum_v exp(z_tv), logp_t = z_t[y_t] - lse_t,
    entropy_t = -sum_v p_tv log p_tv = lse_t - sum_v p_tv z_tv, argmax_t = first v with the
    largest z_tv.

    h: [n, d]; W: [V, d]; y: [n] ints in [0, V).
    """
    h = _f64(h)
    W = _f64(W)
    y = np.asarray(y, dtype=np.int64)
    n = h.shape[0]
    Z = h @ W.T                                   # logits, [n, V]
    m = Z.max(axis=1)
    lse = m + np.log(np.exp(Z - m[:, None]).sum(axis=1))
    logp = Z[np.arange(n), y] - lse
    P = np.exp(Z - lse[:, None])
    entropy = lse - (P * Z).sum(axis=1)
    rows = np.arange(n)
    argmax = Z.argmax(axis=1)                     # numpy returns the first maximal index
    # runner-up (tie diagnostics only): the best logit once the argmax entry is removed
    Z[rows, argmax] = -np.inf
    second = Z.argmax(axis=1)
    Z[rows, argmax] = m
    gap = m - Z[rows, second] if Z.shape[1] > 1 else np.full(n, np.inf)
    return {"logp": logp, "lse": lse, "entropy": entropy, "argmax": argmax, "top_gap": gap,
            "second": second}


def shard_stats(h, W_shard, y, v_offset):
    """Vocabulary-parallel scoring (the paper shards the policy with tensor parallelism, Sec. 6.3):
    statistics of one vocabulary shard [v_offset, v_offset + V_shard) per token: m = max_v z_v,
    s = sum_v e^{z_v - m}, u = sum_v e^{z_v - m} z_v, the first global index of the maximum, and
    z at the sampled token if the shard owns it (else -inf)."""
    h, W_shard = _f64(h), _f64(W_shard)
    y = np.asarray(y, dtype=np.int64)
    Z = h @ W_shard.T
    m = Z.max(axis=1)
    E = np.exp(Z - m[:, None])
    yl = y - v_offset
    own = (yl >= 0) & (yl < W_shard.shape[0])
    zy = np.full(len(y), -np.inf)
    zy[own] = Z[np.flatnonzero(own), yl[own]]
    return {"m": m, "s": E.sum(axis=1), "u": (E * Z).sum(axis=1),
            "argmax": Z.argmax(axis=1) + v_offset, "zy": zy}


def merge_shard_stats(stats):
    """Combines the per-shard statistics of all shards (any partition of the vocabulary) into
    lse, logp, entropy and argmax: M = max m_p, S = sum s_p e^{m_p - M}, U = sum u_p e^{m_p - M},
    lse = M + log S, entropy = lse - U / S, logp = z_y - lse, argmax = lowest index attaining M."""
    m = np.stack([st["m"] for st in stats])
    M = m.max(axis=0)
    sc = np.exp(m - M)
    S_ = sum(st["s"] * sc[p] for p, st in enumerate(stats))
    U = sum(st["u"] * sc[p] for p, st in enumerate(stats))
    lse = M + np.log(S_)
    zy = np.max(np.stack([st["zy"] for st in stats]), axis=0)
    cand = np.stack([np.where(m[p] == M, st["argmax"], np.iinfo(np.int64).max)
                     for p, st in enumerate(stats)])
    return {"lse": lse, "logp": zy - lse, "entropy": lse - U / S_, "argmax": cand.min(axis=0)}


def exact_kl(h, W, h_ref, W_ref):
    """Eq. 1's KL(pi_theta(.|c) || pi_ref(.|c)) at each scored position, over the whole
    vocabulary: KL_t = sum_v p_tv (log p_tv - log q_tv), p = softmax(W h_t) (policy),
    q = softmax(W_ref h_ref_t) (the frozen reference model of Alg. 1, its own hidden state and
    LM head). The KL of the completion is the sum of KL_t over its tokens (chain rule)."""
    Z = _f64(h) @ _f64(W).T
    Zr = _f64(h_ref) @ _f64(W_ref).T
    lse = Z.max(axis=1) + np.log(np.exp(Z - Z.max(axis=1)[:, None]).sum(axis=1))
    lser = Zr.max(axis=1) + np.log(np.exp(Zr - Zr.max(axis=1)[:, None]).sum(axis=1))
    logP = Z - lse[:, None]
    logQ = Zr - lser[:, None]
    P = np.exp(logP)
    return {"kl": (P * (logP - logQ)).sum(axis=1), "lse_ref": lser, "logP": logP, "logQ": logQ}


def exact_kl_logit_grads(h, W, y, lse, g, h_ref, W_ref, c):
    """dL/dz_t for a loss sum_t [g-weighted log-prob term + c_t KL_t]: g_t (onehot(y_t) - p_t)
    + c_t p_t (log p_t - log q_t - KL_t), the second term being d KL_t / d z_t."""
    ek = exact_kl(h, W, h_ref, W_ref)
    P = np.exp(ek["logP"])
    dZ = logit_grads(h, W, y, lse, g)
    return dZ + _f64(c)[:, None] * P * (ek["logP"] - ek["logQ"] - ek["kl"][:, None])


def token_objective(logp, old, ref, adv_tok, eps_low, eps_high, beta):
    """Per-token GRPO terms (Sec. 6.1 clipped-ratio surrogate; Eq. 1 KL term with the
    per-token estimator) and their derivative with respect to logp.

    Returns rho, surr, kl, ell = -surr + beta*kl, and dell = d ell / d logp.
    """
    logp, old, ref, A = _f64(logp), _f64(old), _f64(ref), _f64(adv_tok)
    rho = np.exp(logp - old)
    unclipped = rho * A
    clipped = np.clip(rho, 1.0 - eps_low, 1.0 + eps_high) * A
    surr = np.minimum(unclipped, clipped)
    delta = ref - logp
    kl = np.exp(delta) - delta - 1.0
    ell = -surr + beta * kl
    active = ((A >= 0) & (rho <= 1.0 + eps_high)) | ((A < 0) & (rho >= 1.0 - eps_low))
    dsurr = np.where(active, A * rho, 0.0)        # d(rho A)/dlogp = A rho where unclipped is taken
    dkl = 1.0 - np.exp(delta)                     # d(e^delta - delta - 1)/dlogp
    dell = -dsurr + beta * dkl
    return {"rho": rho, "surr": surr, "kl": kl, "ell": ell, "dell": dell, "active": active}


def aggregate(ell, dell, seq_of_token, counts, num_seqs, agg=SEQ_MEAN, norm=None):
    """Loss L over the scored tokens and g_t = dL/dlogp_t (Eq. 1's expectation). Also returns
    sum_t |w_t l_t|, the magnitude against which L's rounding error is measured.

    seq_mean:   L = (1/S) sum_i (1/n_i) sum_t l_t        (S = norm or num_seqs)
    token_mean: L = sum_t l_t / N                          (N = norm or sum_i n_i)
    """
    ell, dell = _f64(ell), _f64(dell)
    seq = np.asarray(seq_of_token, dtype=np.int64)
    n = np.asarray(counts, dtype=np.float64)
    if agg == SEQ_MEAN:
        S = float(norm) if norm else float(num_seqs)
        w_tok = 1.0 / (S * n[seq])
    elif agg == TOKEN_MEAN:
        N = float(norm) if norm else float(n.sum())
        w_tok = np.full(ell.shape, 1.0 / N)
    else:
        raise ValueError(agg)
    L = float((w_tok * ell).sum())
    g = w_tok * dell
    mass = float(np.abs(w_tok * ell).sum())      # sum of |terms|: the scale of L's rounding
    return L, g, mass


def sft_objective(logp):
    """Sec. 6.2 (reasoning distillation): the small model is fine-tuned with supervised learning
    on the large model's filtered traces, tool-call tokens and arguments kept in the targets, i.e.
    token cross-entropy l_t = -log pi(y_t) over the target tokens. Returns l_t and dl/dlogp = -1."""
    logp = _f64(logp)
    return {"ell": -logp, "dell": -np.ones_like(logp)}


def perf_reward(correct, t_base, t_new):
    """Eq. 3: -2 if the edit is incorrect, -1 if correct but slower than the baseline, else
    min{10, t_base / t - 1}. "Slower" is read as t > t_base (an unchanged time earns 0)."""
    correct = np.asarray(correct) != 0
    t_base, t_new = _f64(t_base), _f64(t_new)
    out = np.empty(np.broadcast(correct, t_base, t_new).shape)
    for i in np.ndindex(out.shape):
        if not correct[i]:
            out[i] = -2.0
        elif t_new[i] > t_base[i]:
            out[i] = -1.0
        else:
            out[i] = min(10.0, t_base[i] / t_new[i] - 1.0)
    return out


def tool_reward(tools_used, tools_avail, lam=0.5):
    """Eq. 4: lambda_tools * |UniqueToolsUsed(x)| / |T_avail| with lambda_tools = 0.5."""
    return lam * _f64(tools_used) / _f64(tools_avail)


def reward(correct, t_base, t_new, tools_used, tools_avail, lam=0.5):
    """Eq. 2: r(x) = r_perf(x) + r_tools(x)."""
    return perf_reward(correct, t_base, t_new) + tool_reward(tools_used, tools_avail, lam)


def logit_grads(h, W, y, lse, g):
    """dL/dz_t = g_t (onehot(y_t) - softmax(z_t)) for each scored token (chain rule through
    logp_t = z_t[y_t] - lse_t)."""
    h, W, lse, g = _f64(h), _f64(W), _f64(lse), _f64(g)
    y = np.asarray(y, dtype=np.int64)
    Z = h @ W.T
    P = np.exp(Z - lse[:, None])
    onehot = np.zeros_like(P)
    onehot[np.arange(len(y)), y] = 1.0
    return g[:, None] * (onehot - P)


def param_grads(h, W, y, lse, g, vocab_rows=None):
    """dL/dh_t = W^T dz_t and dL/dW = sum_t dz_t h_t^T (Alg. 1's gradient step on L, for the
    LM head and its input). ``vocab_rows`` restricts dW to a subset of rows (exact, since a row
    of dW needs only its own column of dz)."""
    dZ = logit_grads(h, W, y, lse, g)
    dH = dZ @ _f64(W)
    if vocab_rows is None:
        dW = dZ.T @ _f64(h)
    else:
        dW = dZ[:, vocab_rows].T @ _f64(h)
    return dH, dW


def sft_step(H, W, tokens, mask, agg=TOKEN_MEAN, norm=None, vocab_rows=None, with_grads=True):
    """The distillation (SFT) path of Sec. 6.2 on a padded batch: per-position logp etc. as in
    grpo_step, L = mean token cross-entropy, dH [S,T,d] and dW [V,d]."""
    H = _f64(H)
    S, T, d = H.shape
    mask = np.asarray(mask)
    counts = valid_counts(mask)
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    h = H[si, ti]
    y = np.asarray(tokens)[si, ti]
    sc = score_tokens(h, W, y)
    ob = sft_objective(sc["logp"])
    L, g_tok, mass = aggregate(ob["ell"], ob["dell"], si, counts, S, agg, norm)
    out = {"counts": counts, "loss": L, "loss_abs_mass": mass}
    lp = np.zeros((S, T))
    lp[si, ti] = sc["logp"]
    out["logp"] = lp
    if with_grads:
        dHv, dW = param_grads(h, W, y, sc["lse"], g_tok, vocab_rows)
        dH = np.zeros((S, T, d))
        dH[si, ti] = dHv
        out["dH"] = dH
        out["dW"] = dW
    return out


def grpo_step_exact_kl(H, W, H_ref, W_ref, tokens, mask, rewards, group_offsets, old,
                       eps_low=0.2, eps_high=0.2, beta=0.04, agg=SEQ_MEAN, std_mode="unbiased",
                       std_eps=1e-4, norm=None, with_grads=True):
    """GRPO with Eq. 1's KL term taken exactly over the vocabulary: l_t = -surr_t + beta KL_t;
    dH, dW through dz = g (onehot - p) + beta w p (log p - log q - KL)."""
    H = _f64(H)
    S, T, d = H.shape
    mask = np.asarray(mask)
    counts = valid_counts(mask)
    adv = group_advantages(rewards, group_offsets, std_mode, std_eps)
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    h, hr = H[si, ti], _f64(H_ref)[si, ti]
    y = np.asarray(tokens)[si, ti]
    sc = score_tokens(h, W, y)
    ek = exact_kl(h, W, hr, W_ref)
    tob = token_objective(sc["logp"], _f64(old)[si, ti], sc["logp"], adv[si], eps_low, eps_high,
                          0.0)
    ell = tob["ell"] + beta * ek["kl"]
    L, g_tok, mass = aggregate(ell, tob["dell"], si, counts, S, agg, norm)
    _, w_tok, _ = aggregate(np.zeros_like(ell), np.ones_like(ell), si, counts, S, agg, norm)
    out = {"counts": counts, "adv": adv, "loss": L, "loss_abs_mass": mass}
    for k, v in (("logp", sc["logp"]), ("lse", sc["lse"]), ("kl", ek["kl"]),
                 ("lse_ref", ek["lse_ref"]), ("entropy", sc["entropy"])):
        a = np.zeros((S, T))
        a[si, ti] = v
        out[k] = a
    if with_grads:
        dZ = exact_kl_logit_grads(h, W, y, sc["lse"], g_tok, hr, W_ref, beta * w_tok)
        dH = np.zeros((S, T, d))
        dH[si, ti] = dZ @ _f64(W)
        out["dH"] = dH
        out["dW"] = dZ.T @ h
    return out


def grpo_step(H, W, tokens, mask, rewards, group_offsets, old, ref, eps_low=0.2, eps_high=0.2,
              beta=0.04, agg=SEQ_MEAN, std_mode="unbiased", std_eps=1e-4, norm=None,
              adv=None, vocab_rows=None, with_grads=True):
    """The whole path on a padded batch: H [S,T,d], W [V,d], tokens/mask/old/ref [S,T],
    rewards [S]. Returns per-position outputs ([S,T], zeros at unscored positions, argmax -1),
    per-sequence counts and advantages, the loss, g, dH [S,T,d] and dW [V,d] (or its rows)."""
    H = _f64(H)
    S, T, d = H.shape
    mask = np.asarray(mask)
    counts = valid_counts(mask)
    if adv is None:
        adv = group_advantages(rewards, group_offsets, std_mode, std_eps)
    idx = np.argwhere(mask != 0)
    si, ti = idx[:, 0], idx[:, 1]
    h = H[si, ti]
    y = np.asarray(tokens)[si, ti]
    sc = score_tokens(h, W, y)
    out = {"counts": counts, "adv": adv}
    for k in ("logp", "lse", "entropy"):
        a = np.zeros((S, T))
        a[si, ti] = sc[k]
        out[k] = a
    am = np.full((S, T), -1, dtype=np.int64)
    am[si, ti] = sc["argmax"]
    out["argmax"] = am
    gap = np.full((S, T), np.inf)
    gap[si, ti] = sc["top_gap"]
    out["top_gap"] = gap
    tob = token_objective(sc["logp"], _f64(old)[si, ti], _f64(ref)[si, ti], adv[si],
                          eps_low, eps_high, beta)
    L, g_tok, mass = aggregate(tob["ell"], tob["dell"], si, counts, S, agg, norm)
    out["loss"] = L
    out["loss_abs_mass"] = mass
    g = np.zeros((S, T))
    g[si, ti] = g_tok
    out["g"] = g
    if with_grads:
        dHv, dW = param_grads(h, W, y, sc["lse"], g_tok, vocab_rows)
        dH = np.zeros((S, T, d))
        dH[si, ti] = dHv
        out["dH"] = dH
        out["dW"] = dW
    return out
