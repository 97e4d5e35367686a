"""Failure detection without a GPU fault: device-detected errors land in the workspace status
word, a stalled pipeline ends by its bounded wait (GRPO_ERR_TIMEOUT) instead of hanging, and the
CUDA context stays usable afterwards."""
import numpy as np
import pytest
import torch

from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy

pytestmark = pytest.mark.gpu

TIMEOUT, TOKEN_RANGE, GROUPS = -6, -5, -7


def _small():
    b = make_batch_numpy(WORKLOADS["g8_t1k_d2048_v32k"].scaled(prompts=1, group_sizes=(3,), T=130,
                                                               len_lo=30, len_hi=130))
    return b, [t.cuda() for t in (b.H, b.W, b.tokens, b.mask)]


def test_stalled_pipeline_times_out_and_context_survives():
    """Single-CTA tiles (mode 0): CTA 0 leaves its first pipeline stage unfilled, its MMA wait
    runs out, and the next call on the same context is bitwise correct."""
    b, (H, W, tok, mask) = _small()
    S, T, d = H.shape
    ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
    G.grpo_set_tile_mode(G.TILE_SINGLE)
    try:
        good = G.grpo_score_fwd(H, W, tok, mask, ws)
        torch.cuda.synchronize()
        good = {k: v.clone() for k, v in good.items()}
        assert G.grpo_last_device_error(ws)[0] == 0
        G.grpo_debug_inject_stall(True)
        try:
            G.grpo_score_fwd(H, W, tok, mask, ws)
            st, where = G.grpo_last_device_error(ws)       # synchronises; the kernel gave up
        finally:
            G.grpo_debug_inject_stall(False)
        assert st == TIMEOUT, (st, where)
        assert where // 16 == 3                              # recorded by a GEMM wait
        again = G.grpo_score_fwd(H, W, tok, mask, ws)
        torch.cuda.synchronize()
        assert G.grpo_last_device_error(ws)[0] == 0
        for k in ("logp", "lse", "entropy", "argmax", "valid_count"):
            assert torch.equal(again[k], good[k]), k
    finally:
        G.grpo_set_tile_mode(G.TILE_DEFAULT)


def test_token_out_of_range_sets_status():
    b, (H, W, tok, mask) = _small()
    S, T, d = H.shape
    V = W.shape[0]
    ws = G.Workspace.for_problem(S, T, d, V, H.dtype)
    bad = tok.clone()
    bad[1, 5] = V                     # a scored position (lengths >= 30)
    assert int(mask[1, 5]) == 1
    out = G.grpo_score_fwd(H, W, bad, mask, ws)
    st, where = G.grpo_last_device_error(ws)
    assert st == TOKEN_RANGE, (st, where)
    assert torch.isnan(out["logp"][1, 5])
    out = G.grpo_score_fwd(H, W, tok, mask, ws)
    assert G.grpo_last_device_error(ws)[0] == 0


def test_bad_group_offsets_set_status():
    ws = G.Workspace.create(256)
    r = torch.randn(8, device="cuda")
    go = torch.tensor([0, 4, 7], dtype=torch.int32, device="cuda")   # ends at 7, not S = 8
    a = G.group_advantages(r, go, ws)
    st, _ = G.grpo_last_device_error(ws)
    assert st == GROUPS
    assert torch.isnan(a[4:7]).all() and not torch.isnan(a[:4]).any()
    go = torch.tensor([0, 4, 8], dtype=torch.int32, device="cuda")
    a = G.group_advantages(r, go, ws)
    assert G.grpo_last_device_error(ws)[0] == 0
    assert np.isfinite(a.cpu().numpy()).all()


def test_stalled_pipeline_times_out_in_cta_pair_tiles():
    """The same injected stall with CTA pairs (mode 1, every GEMM role): the leader's MMA wait
    runs out, its peer's producer wait runs out after it, both leave through their bounded waits
    and the final cluster barrier, and the next call is correct."""
    b, (H, W, tok, mask) = _small()
    S, T, d = H.shape
    ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
    G.grpo_set_tile_mode(G.TILE_CTA_PAIR)
    try:
        good = {k: v.clone() for k, v in G.grpo_score_fwd(H, W, tok, mask, ws).items()}
        assert G.grpo_last_device_error(ws)[0] == 0
        G.grpo_debug_inject_stall(True)
        try:
            G.grpo_score_fwd(H, W, tok, mask, ws)
            st, where = G.grpo_last_device_error(ws)
        finally:
            G.grpo_debug_inject_stall(False)
        assert st == TIMEOUT, (st, where)
        again = G.grpo_score_fwd(H, W, tok, mask, ws)
        torch.cuda.synchronize()
        assert G.grpo_last_device_error(ws)[0] == 0
        for k in ("logp", "lse", "entropy", "argmax"):
            assert torch.equal(again[k], good[k]), k
    finally:
        G.grpo_set_tile_mode(G.TILE_DEFAULT)


def test_stalled_backward_times_out_in_wide_pair_tiles():
    """The injected stall in a backward whose dH and dW GEMMs run 256 x 512 CTA-pair tiles (the
    default): every GEMM of the call (dz recompute, dH, dW) gives up through its bounded waits and
    records GRPO_ERR_TIMEOUT, and the next backward on the same context gives bitwise the
    gradients of one made before the stall."""
    b, (H, W, tok, mask) = _small()
    S, T, d = H.shape
    ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
    G.grpo_set_tile_mode(G.TILE_DEFAULT)
    assert [G.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 0, 2, 2]
    dev = H.device
    adv = G.group_advantages(b.rewards.to(dev), b.group_offsets.to(dev), ws)
    f = G.grpo_score_fwd(H, W, tok, mask, ws)
    old = (f["logp"] + b.noise_old.to(dev)).contiguous()
    ref = (f["logp"] + b.noise_ref.to(dev)).contiguous()

    def backward():
        r = G.grpo_loss_bwd(H, W, tok, mask, f["logp"], f["lse"], old, ref, adv,
                            f["valid_count"], ws)
        return {k: v.clone() for k, v in r.items()}

    good = backward()
    assert G.grpo_last_device_error(ws)[0] == 0
    G.grpo_debug_inject_stall(True)
    try:
        backward()
        st, where = G.grpo_last_device_error(ws)
    finally:
        G.grpo_debug_inject_stall(False)
    assert st == TIMEOUT, (st, where)
    again = backward()
    torch.cuda.synchronize()
    assert G.grpo_last_device_error(ws)[0] == 0
    for k in ("loss", "dH", "dW"):
        assert torch.equal(again[k], good[k]), k
