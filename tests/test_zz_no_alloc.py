"""The allocation-free forward entry point, grpo_score_fwd_static.

Some callers cannot allocate device memory at all: a plugin whose host framework owns every
device allocation and forbids extensions from making their own, or code in a latency-critical
section where an allocation (which can synchronise the device) is not allowed. For them the
library offers a forward pass whose scratch is a fixed 64 MiB device array inside the library.
This file checks, through the C ABI, that two calls in a row give the results of the workspace
entry point grpo_score_fwd on the same inputs (bf16 and f32), that a batch whose scratch ends just
below the array's size runs and one 128-row tile larger is refused, that a device-detected error
is reported through the status word and cleared by the next call, and that a stalled GEMM ends by
its bounded wait. It is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy, make_batch_torch

pytestmark = pytest.mark.gpu

LOGP_ATOL = 2e-3


def _inputs(seed, **over):
    w = WORKLOADS["g8_t1k_d2048_v32k"].scaled(seed=seed, **over)
    b = make_batch_numpy(w)
    return [t.cuda() for t in (b.H, b.W, b.tokens, b.mask)]


def test_static_scratch_forward_matches_workspace_forward_twice():
    batches = [_inputs(11, prompts=1, T=260, len_lo=60, len_hi=260),
               _inputs(12, prompts=1, group_sizes=(5,), T=140, len_lo=20, len_hi=140),
               _inputs(13, prompts=1, group_sizes=(3,), T=100, len_lo=20, len_hi=100, d=320,
                       V=1000)]                       # d a multiple of 64, not of 256
    for H, W, tok, mask in batches:                   # calls in a row, different shapes
        S, T, d = H.shape
        ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
        ref = G.grpo_score_fwd(H, W, tok, mask, ws)
        got = G.grpo_score_fwd_static(H, W, tok, mask)
        torch.cuda.synchronize()
        assert int(got["status"].item()) == 0
        assert G.grpo_last_device_error(ws)[0] == 0
        m = mask.cpu().numpy() != 0
        for k in ("logp", "lse", "entropy"):
            e = np.abs(got[k].cpu().numpy() - ref[k].cpu().numpy())
            assert float(e.max()) <= LOGP_ATOL, (k, float(e.max()))
        assert torch.equal(got["argmax"], ref["argmax"])
        assert torch.equal(got["valid_count"], ref["valid_count"])
        assert np.all(got["argmax"].cpu().numpy()[~m] == -1)


def test_static_scratch_rejects_batches_larger_than_the_array():
    lib = G._lib()
    fake = ctypes.c_void_p(1 << 20)       # never dereferenced: the size check fails first
    st = lib.grpo_score_fwd_static(fake, fake, G.GRPO_BF16, fake, fake, 32, 16384, 5120, 151936,
                                   fake, fake, fake, fake, fake, ctypes.c_void_p(0),
                                   ctypes.c_void_p(0))
    assert st == -4, G.grpo_status_string(st)


def _static_bytes(S, T, d, V):
    """Scratch the bf16 path of grpo_score_fwd_static lays out (256-byte aligned regions):
    header, sequence bases, packed-row map, position map, target logits, per-strip statistics
    (16 bytes per packed row and 256-column vocabulary strip) and the packed hidden states."""
    up = lambda x: (x + 255) // 256 * 256            # noqa: E731
    P = S * T
    R = (P + 127) // 128 * 128
    strips = (V + 255) // 256
    return (256 + up(4 * (S + 1)) + up(4 * R) + up(4 * P) + up(4 * P) + up(16 * strips * R) +
            up(2 * R * d))


def _same_as_workspace_forward(H, W, tok, mask, got):
    S, T, d = H.shape
    ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
    ref = G.grpo_score_fwd(H, W, tok, mask, ws)
    torch.cuda.synchronize()
    assert G.grpo_last_device_error(ws)[0] == 0
    for k in ("logp", "lse", "entropy"):
        e = np.abs(got[k].cpu().numpy() - ref[k].cpu().numpy())
        assert float(e.max()) <= LOGP_ATOL, (k, float(e.max()))
    assert torch.equal(got["argmax"], ref["argmax"])
    assert torch.equal(got["valid_count"], ref["valid_count"])


def test_static_scratch_f32_forward_matches_workspace_forward():
    w = WORKLOADS["tiny_f32"]
    b = make_batch_numpy(w)
    H, W, tok, mask = [t.cuda() for t in (b.H, b.W, b.tokens, b.mask)]
    for _ in range(2):
        got = G.grpo_score_fwd_static(H, W, tok, mask)
        torch.cuda.synchronize()
        assert int(got["status"].item()) == 0
        _same_as_workspace_forward(H, W, tok, mask, got)


def test_static_scratch_batch_just_below_the_array_size():
    """At d = 2048, V = 32000 one completion of T = T_max tokens (the largest multiple of 128
    whose scratch fits the 64 MiB array) runs and matches the workspace path; T_max + 1 rounds up
    to one more 128-row tile and is refused before anything is enqueued."""
    d, V = 2048, 32000
    t_max = 128
    while _static_bytes(1, t_max + 128, d, V) <= G.STATIC_SCRATCH_BYTES:
        t_max += 128
    assert _static_bytes(1, t_max, d, V) <= G.STATIC_SCRATCH_BYTES < _static_bytes(1, t_max + 1, d, V)
    assert G.STATIC_SCRATCH_BYTES - _static_bytes(1, t_max, d, V) < 128 * 6200
    w = WORKLOADS["g8_t1k_d2048_v32k"].scaled(seed=14, prompts=1, group_sizes=(1,), T=t_max,
                                             len_lo=t_max - 300, len_hi=t_max)
    b = make_batch_torch(w, "cuda")
    H, W, tok, mask = b.H, b.W, b.tokens, b.mask
    got = G.grpo_score_fwd_static(H, W, tok, mask)
    torch.cuda.synchronize()
    assert int(got["status"].item()) == 0
    _same_as_workspace_forward(H, W, tok, mask, got)
    # one token more: real buffers of the right size, so that nothing could be read out of
    # bounds even if the size check let the call through
    H2 = torch.zeros((1, t_max + 1, d), dtype=torch.bfloat16, device="cuda")
    tok2 = torch.zeros((1, t_max + 1), dtype=torch.int32, device="cuda")
    mask2 = torch.ones((1, t_max + 1), dtype=torch.uint8, device="cuda")
    with pytest.raises(G.GrpoError) as err:
        G.grpo_score_fwd_static(H2, W, tok2, mask2)
    assert err.value.status == -4, err.value


def test_static_scratch_reports_a_bad_token_and_the_next_call_clears_it():
    """A scored token id equal to V: the call returns GRPO_OK (the fault is only visible on the
    device), *status_out reads GRPO_ERR_TOKEN_RANGE and that position's log-prob is NaN; the next
    call with valid tokens reads 0 and is bitwise equal to a call made before the bad one."""
    H, W, tok, mask = _inputs(15, prompts=1, T=200, len_lo=80, len_hi=200)
    V = W.shape[0]
    good = {k: v.clone() for k, v in G.grpo_score_fwd_static(H, W, tok, mask).items()}
    torch.cuda.synchronize()
    assert int(good["status"].item()) == 0
    bad_tok = tok.clone()
    bad_tok[0, 3] = V
    assert int(mask[0, 3]) == 1
    bad = G.grpo_score_fwd_static(H, W, bad_tok, mask)
    torch.cuda.synchronize()
    assert int(bad["status"].item()) == -5
    assert bool(torch.isnan(bad["logp"][0, 3]))
    again = G.grpo_score_fwd_static(H, W, tok, mask)
    torch.cuda.synchronize()
    assert int(again["status"].item()) == 0
    for k in ("logp", "lse", "entropy", "argmax", "valid_count"):
        assert torch.equal(again[k], good[k]), k


def test_static_scratch_stalled_gemm_times_out_and_next_call_is_correct():
    """The injected pipeline stall (single-CTA forward tiles): the forward GEMM's bounded wait
    runs out, *status_out reads GRPO_ERR_TIMEOUT, and the next call is bitwise equal to one made
    before the stall."""
    H, W, tok, mask = _inputs(16, prompts=1, group_sizes=(3,), T=130, len_lo=30, len_hi=130)
    assert G.grpo_get_role_tile_mode(G.ROLE_FWD) == G.TILE_SINGLE
    good = {k: v.clone() for k, v in G.grpo_score_fwd_static(H, W, tok, mask).items()}
    torch.cuda.synchronize()
    G.grpo_debug_inject_stall(True)
    try:
        stalled = G.grpo_score_fwd_static(H, W, tok, mask)
        torch.cuda.synchronize()
    finally:
        G.grpo_debug_inject_stall(False)
    assert int(stalled["status"].item()) == -6
    again = G.grpo_score_fwd_static(H, W, tok, mask)
    torch.cuda.synchronize()
    assert int(again["status"].item()) == 0
    for k in ("logp", "lse", "entropy", "argmax", "valid_count"):
        assert torch.equal(again[k], good[k]), k
