"""Planted mistakes in copies of the oracle (CPU only): each mutation must make some pin fail.

A mutation replaces one fragment of the oracle source with a plausible error (dropped term, wrong
sign or index, transposed operand, wrong degrees of freedom); the mutated module is executed
from text, so the real oracle is untouched.
"""
import inspect
import types

import pytest

import oracle.grpo_oracle as O
import tests.test_oracle_pins as P

MUTATIONS = [
    ("kl gradient sign", "dkl = 1.0 - np.exp(delta)", "dkl = np.exp(delta) - 1.0"),
    ("kl drops the -1", "kl = np.exp(delta) - delta - 1.0", "kl = np.exp(delta) - delta"),
    ("clip upper bound uses eps_low", "(rho <= 1.0 + eps_high)", "(rho <= 1.0 + eps_low)"),
    ("clip lower branch sign", "(A < 0) & (rho >= 1.0 - eps_low)", "(A < 0) & (rho <= 1.0 - eps_low)"),
    ("surrogate uses max", "surr = np.minimum(unclipped, clipped)", "surr = np.maximum(unclipped, clipped)"),
    ("entropy drops lse", "entropy = lse - (P * Z).sum(axis=1)", "entropy = -(P * Z).sum(axis=1)"),
    ("lse drops the max shift", "lse = m + np.log(", "lse = np.log("),
    ("logp sign", "logp = Z[np.arange(n), y] - lse", "logp = lse - Z[np.arange(n), y]"),
    ("advantage std dof", "dof = G - 1 if std_mode", "dof = G if std_mode"),
    ("advantage not centred", "adv[lo:hi] = (rg - mu) /", "adv[lo:hi] = rg /"),
    ("std_eps inside the sqrt", "(rg - mu) / (sigma + std_eps)",
     "(rg - mu) / np.sqrt(sigma**2 + std_eps)"),
    ("onehot dropped from dz", "return g[:, None] * (onehot - P)", "return g[:, None] * (-P)"),
    ("dz sign", "return g[:, None] * (onehot - P)", "return g[:, None] * (P - onehot)"),
    ("seq_mean weight ignores n_i", "w_tok = 1.0 / (S * n[seq])", "w_tok = np.full(ell.shape, 1.0 / S)"),
    ("argmax last index", "argmax = Z.argmax(axis=1) ", "argmax = Z.shape[1] - 1 - Z[:, ::-1].argmax(axis=1) "),
    ("ratio inverted", "rho = np.exp(logp - old)", "rho = np.exp(old - logp)"),
    ("counts of zeros", "return (m != 0).sum(axis=1)", "return (m == 0).sum(axis=1)"),
    ("sft gradient sign", "return {\"ell\": -logp, \"dell\": -np.ones_like(logp)}",
     "return {\"ell\": -logp, \"dell\": np.ones_like(logp)}"),
    ("reward cap", "out[i] = min(10.0, t_base[i] / t_new[i] - 1.0)",
     "out[i] = min(10.0, t_base[i] / t_new[i])"),
    ("slower penalty", "out[i] = -1.0", "out[i] = -2.0"),
    ("shard argmax keeps the highest index", "\"argmax\": cand.min(axis=0)}",
     "\"argmax\": np.where(cand == np.iinfo(np.int64).max, -1, cand).max(axis=0)}"),
    ("shard merge forgets the rescale", "U = sum(st[\"u\"] * sc[p] for p, st in enumerate(stats))",
     "U = sum(st[\"u\"] for p, st in enumerate(stats))"),
    ("exact-KL gradient drops -KL", "* P * (ek[\"logP\"] - ek[\"logQ\"] - ek[\"kl\"][:, None])",
     "* P * (ek[\"logP\"] - ek[\"logQ\"])"),
    ("exact KL reversed", "\"kl\": (P * (logP - logQ)).sum(axis=1)",
     "\"kl\": (np.exp(logQ) * (logQ - logP)).sum(axis=1)"),
    ("tool reward ratio inverted", "return lam * _f64(tools_used) / _f64(tools_avail)",
     "return lam * _f64(tools_avail) / _f64(tools_used)"),
]


def _mutant(src_old, src_new):
    src = inspect.getsource(O)
    assert src_old in src, src_old
    mod = types.ModuleType("oracle_mutant")
    exec(compile(src.replace(src_old, src_new, 1), "oracle_mutant", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_some_pin_catches(name, old, new):
    mod = _mutant(old, new)
    caught = []
    for pin in P.PINS:
        try:
            pin(mod)
        except Exception as e:  # noqa: BLE001  (assertion or shape error both count)
            caught.append((pin.__name__, type(e).__name__))
    assert caught, f"no pin caught the planted mistake: {name}"
