"""The allocation-free forward entry point, grpo_score_fwd_static.

Some callers cannot allocate device memory at all: a plugin whose host framework owns every
device allocation and forbids extensions from making their own, or code in a latency-critical
section where an allocation (which can synchronise the device) is not allowed. For them the
library offers a forward pass whose scratch is a fixed 64 MiB device array inside the library.
This file checks, through the C ABI, that two calls in a row give the results of the workspace
entry point grpo_score_fwd on the same inputs, and that a batch too large for the array is
refused. It is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy

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
