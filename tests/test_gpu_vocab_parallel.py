"""Vocabulary-parallel (tensor-parallel) LM head, emulated on one GPU: each shard's forward and
backward run as separate calls (no kernel waits on another), the statistics are stacked as an
all-gather would leave them, merged, and the dH partials summed. Checked against the oracle and
against the unsharded path."""
import numpy as np
import pytest
import torch

from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.dp import vocab_shard_bounds
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy
from tests.parity_util import GRAD_RTOL, LOGP_ATOL, oracle_inputs, rel_fro, run_oracle

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,over,bounds", [
    ("g8_t1k_d2048_v32k", dict(prompts=1, group_sizes=(4,), T=200, len_lo=50, len_hi=200), None),
    ("g8_t4k_d4096_v152k", dict(group_sizes=(3,), T=130, len_lo=30, len_hi=130),
     [0, 777, 50000, 50001, 151936]),
])
def test_vocab_parallel_matches_oracle_and_unsharded(name, over, bounds):
    b = make_batch_numpy(WORKLOADS[name].scaled(**over))
    w = b.workload
    H, W, tok, mask = (t.cuda() for t in (b.H, b.W, b.tokens, b.mask))
    S, T, d = H.shape
    V = W.shape[0]
    if bounds is None:
        bounds = [vocab_shard_bounds(V, 3, r)[0] for r in range(3)] + [V]
    shards = list(zip(bounds[:-1], bounds[1:]))
    stats, zys = [], []
    for v0, v1 in shards:
        ws = G.Workspace.for_problem(S, T, d, v1 - v0, H.dtype)
        o = G.grpo_score_fwd_shard(H, W[v0:v1], tok, mask, v0, V, ws)
        stats.append(o["stats"])
        zys.append(o["zy"])
    ws_m = G.Workspace.create(256 + 4 * S + 256)
    f = G.grpo_merge_shard_stats(torch.stack(stats), torch.stack(zys), tok, mask, V, ws_m)
    ws_full = G.Workspace.for_problem(S, T, d, V, H.dtype)
    f_full = G.grpo_score_fwd(H, W, tok, mask, ws_full)
    old, ref = oracle_inputs(b)
    o = run_oracle(b, old, ref, w.eps, w.eps, w.beta)
    m = b.mask.numpy() != 0
    for k in ("logp", "lse", "entropy"):
        assert np.abs(f[k].cpu().numpy()[m] - o[k][m]).max() <= LOGP_ATOL, k
        assert float((f[k] - f_full[k]).abs().max()) <= 1e-4, k
    assert torch.equal(f["argmax"], f_full["argmax"])
    assert torch.equal(f["valid_count"], f_full["valid_count"])

    adv = G.group_advantages(b.rewards.cuda(), b.group_offsets.cuda(), ws_full)
    old_t, ref_t = torch.from_numpy(old).cuda(), torch.from_numpy(ref).cuda()
    dH = torch.zeros((S, T, d), dtype=torch.float32, device="cuda")
    dW = torch.empty((V, d), dtype=torch.float32, device="cuda")
    losses = []
    for v0, v1 in shards:
        ws = G.Workspace.for_problem(S, T, d, v1 - v0, H.dtype)
        r = G.grpo_loss_bwd_shard(H, W[v0:v1], tok, mask, v0, V, f["logp"], f["lse"], old_t,
                                  ref_t, adv, f["valid_count"], ws, eps_low=w.eps,
                                  eps_high=w.eps, beta=w.beta)
        dH += r["dH_partial"]                 # the all-reduce of dH
        dW[v0:v1] = r["dW_shard"]
        losses.append(float(r["loss"].item()))
        assert G.grpo_last_device_error(ws)[0] == 0
    torch.cuda.synchronize()
    assert max(losses) == min(losses)
    scale = max(abs(o["loss"]), o["loss_abs_mass"])
    assert abs(losses[0] - o["loss"]) <= 1e-3 * scale
    e_h, e_w = rel_fro(dH.cpu().numpy(), o["dH"]), rel_fro(dW.cpu().numpy(), o["dW"])
    assert e_h <= GRAD_RTOL and e_w <= GRAD_RTOL, (e_h, e_w)
    assert bool(torch.all(dH[~b.mask.cuda().bool()] == 0))
    print(name, len(shards), "shards: dH", e_h, "dW", e_w)
