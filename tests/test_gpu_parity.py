"""Parity of the CUDA path (through the C ABI) with the CPU float64 oracle on seeded inputs.

Oracle-sized cases keep each workload's hidden size d, vocabulary V, dtype and value laws but
fewer / shorter completions, so that they still span several 128-token tiles, many 256-column
vocabulary tiles and the ragged tails (V % 256 = 128 for V = 151936; T % 128 != 0).
"""
import numpy as np
import pytest
import torch

from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy
from tests.parity_util import compare, oracle_inputs, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

CASES = {
    # name: (workload, overrides)
    "tiny_f32": ("tiny_f32", {}),
    "d2048_v32k": ("g8_t1k_d2048_v32k", dict(T=300, len_lo=64, len_hi=300)),
    "d4096_v152k": ("g8_t4k_d4096_v152k", dict(group_sizes=(4,), T=160, len_lo=40, len_hi=160)),
    "d5120_v152k_temp": ("g16_t16k_d5120_v152k",
                         dict(group_sizes=(4,), prompts=1, T=144, len_lo=36, len_hi=144)),
    "d3584_v152k_deg": ("g8_t512_d3584_v152k",
                        dict(prompts=2, T=72, len_lo=16, len_hi=72, degenerate_frac=0.5)),
}


def _batch(name):
    wname, over = CASES[name]
    return make_batch_numpy(WORKLOADS[wname].scaled(**over))


@pytest.mark.parametrize("name", list(CASES))
def test_parity_workload(name):
    b = _batch(name)
    w = b.workload
    old, ref = oracle_inputs(b)
    g = run_gpu(b, old, ref, w.eps, w.eps, w.beta)
    o = run_oracle(b, old, ref, w.eps, w.eps, w.beta)
    rep = compare(b, g, o)
    print(name, rep)


def test_parity_interior_holes_and_wide_ratio_noise():
    """Tool-result spans masked inside completions; old-logp noise sigma 0.3 so that ~30% of
    the tokens sit outside the clip range (both clip branches exercised)."""
    w = WORKLOADS["g8_t1k_d2048_v32k"].scaled(T=200, len_lo=64, len_hi=200, holes=True)
    b = make_batch_numpy(w)
    old, ref = oracle_inputs(b, old_scale=6.0)
    g = run_gpu(b, old, ref, 0.2, 0.28, 0.04)
    o = run_oracle(b, old, ref, 0.2, 0.28, 0.04)
    print(compare(b, g, o))


def test_parity_token_mean_population_std():
    b = _batch("d2048_v32k")
    old, ref = oracle_inputs(b)
    g = run_gpu(b, old, ref, 0.2, 0.2, 0.04, agg="token_mean", std_mode="population")
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04, agg="token_mean", std_mode="population")
    print(compare(b, g, o))


def test_parity_chunked_backward_matches_single_chunk():
    """A workspace that holds only 4096 vocabulary columns of dz runs the backward in chunks with
    an f32 dH accumulator; results match the oracle and the one-chunk run."""
    b = _batch("d2048_v32k")
    old, ref = oracle_inputs(b)
    g1 = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
    gc = run_gpu(b, old, ref, 0.2, 0.2, 0.04, vocab_chunk=4096)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    print(compare(b, gc, o))
    assert np.array_equal(g1["dW"].numpy(), gc["dW"].numpy())


@pytest.mark.parametrize("eps,beta", [(0.1, 0.0), (0.1, 0.04), (0.2, 0.0), (0.2, 0.04),
                                      (0.3, 0.0), (0.3, 0.04)])
def test_parity_eps_beta_grid(eps, beta):
    b = make_batch_numpy(WORKLOADS["g8_t512_d3584_v152k"].scaled(prompts=1, T=48, len_lo=16,
                                                                   len_hi=48))
    old, ref = oracle_inputs(b, old_scale=2.0)
    g = run_gpu(b, old, ref, eps, eps, beta, ref_none=(beta == 0.0))
    o = run_oracle(b, old, ref, eps, eps, beta)
    print(compare(b, g, o))


def test_group_advantages_mixed_group_sizes():
    """64 prompts with G cycling {4, 8, 12, 16} and 10% degenerate groups (advantages only)."""
    from paper_2510_17158_gb300 import grpo as G
    import oracle
    w = WORKLOADS["mixed_t512_d3584_v152k"]
    rng = np.random.default_rng(7)
    sizes = [w.group_sizes[p % 4] for p in range(w.prompts)]
    go = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    r = rng.uniform(-1, 3, size=go[-1]).astype(np.float32)
    for g in rng.choice(len(sizes), size=6, replace=False):
        r[go[g]:go[g + 1]] = r[go[g]]
    ws = G.Workspace.create(256)
    for mode in ("unbiased", "population"):
        a = G.group_advantages(torch.from_numpy(r).cuda(), torch.from_numpy(go).cuda(), ws,
                               std_mode=mode).cpu().numpy()
        o = oracle.group_advantages(r, go, mode, 1e-4)
        np.testing.assert_allclose(a, o, rtol=1e-5, atol=2e-6)
        assert np.all(a[o == 0] == 0)
    assert G.grpo_last_device_error(ws)[0] == 0


def test_deterministic_bitwise():
    b = _batch("d2048_v32k")
    old, ref = oracle_inputs(b)
    g1 = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
    g2 = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
    for k in ("logp", "lse", "entropy", "argmax", "dH", "dW"):
        assert torch.equal(g1[k], g2[k]), k
    assert g1["loss"] == g2["loss"]


MODE_KEYS_FWD = ("logp", "lse", "entropy", "argmax", "valid_count")


def _set_roles(G, modes):
    for role, m in enumerate(modes):
        G.grpo_set_role_tile_mode(role, m)
    assert [G.grpo_get_role_tile_mode(r) for r in range(4)] == list(modes)


@pytest.mark.parametrize("name", ["d4096_v152k", "d2048_v32k"])
def test_tile_modes_match_oracle(name):
    """Every tile mode meets the parity bar: 0 (one CTA per 128 x 256 tile), 1 (CTA pairs,
    M = 256 MMAs with cta_group::2, 256 x 256 tiles) for all four GEMMs, and the library's
    default mix (forward and dz in mode 0, dH and dW in mode 2: CTA pairs on 256 x 512 tiles).
    The d2048 case packs into 85 row tiles (odd), so the second CTA of the last pair has no tile
    of its own and stages a copy of its leader's rows; d = 2048 gives 4 column units of 512 in
    mode 2, d = 4096 gives 8."""
    from paper_2510_17158_gb300 import grpo as G
    b = _batch(name)
    old, ref = oracle_inputs(b)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    assert [G.grpo_get_role_tile_mode(r) for r in range(4)] == [0, 0, 2, 2]
    assert G.grpo_get_tile_mode() == G.TILE_DEFAULT
    try:
        for modes in ((0, 0, 0, 0), (1, 1, 1, 1), (0, 0, 2, 2), (1, 1, 2, 2), (2, 2, 2, 2)):
            _set_roles(G, modes)
            g = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
            print("modes", modes, compare(b, g, o))
    finally:
        G.grpo_set_tile_mode(G.TILE_DEFAULT)


@pytest.mark.parametrize("name", ["d2048_v32k"])
def test_tile_mode_mixes_bitwise_relations(name):
    """Each GEMM role runs in its own tile mode (grpo_set_role_tile_mode). Results that must be
    bitwise equal: the forward statistics and the loss between the pair modes 1 and 2 of the
    forward role, and whenever the forward role's mode is the same (they do not depend on the
    backward roles); dz and hence dH, dW between modes 1 and 2 of the dz role; dH, dW between
    modes 1 and 2 of the backward roles on the same dz (modes 1 and 2 issue the same M = 256,
    N = 256 MMAs for every output element, in the same k order). Mode 0 against the pair modes
    agrees within the parity bar."""
    from paper_2510_17158_gb300 import grpo as G
    b = _batch(name)
    old, ref = oracle_inputs(b)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    outs = {}
    try:
        for modes in ((0, 0, 0, 0), (0, 0, 1, 1), (0, 0, 2, 2), (0, 0, 1, 2), (0, 0, 2, 1),
                      (1, 1, 1, 1), (1, 1, 2, 2), (0, 1, 2, 2), (2, 2, 2, 2), (2, 1, 1, 2)):
            _set_roles(G, modes)
            outs[modes] = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
            print("roles", modes, compare(b, outs[modes], o))
    finally:
        G.grpo_set_tile_mode(G.TILE_DEFAULT)
    for modes, g in outs.items():   # forward in mode 1 or 2: the same M = 256, N = 256 MMAs
        ref_fwd = outs[(0, 0, 0, 0)] if modes[0] == 0 else outs[(1, 1, 1, 1)]
        for k in MODE_KEYS_FWD:
            assert torch.equal(g[k], ref_fwd[k]), (modes, k)
        assert g["loss"] == ref_fwd["loss"], modes
    same_dz = [((0, 0, 1, 1), (0, 0, 2, 2), (0, 0, 1, 2), (0, 0, 2, 1)),
               ((1, 1, 1, 1), (1, 1, 2, 2), (2, 2, 2, 2), (2, 1, 1, 2))]
    for group in same_dz:
        for modes in group[1:]:
            for k in ("dH", "dW"):
                assert torch.equal(outs[modes][k], outs[group[0]][k]), (modes, k)


def test_tile_mode_rejects_unknown_modes():
    from paper_2510_17158_gb300 import grpo as G
    prev = G.grpo_get_tile_mode()
    for bad in (-2, 3, 5):
        with pytest.raises(G.GrpoError):
            G.grpo_set_tile_mode(bad)
    assert G.grpo_get_tile_mode() == prev
    with pytest.raises(G.GrpoError):
        G.grpo_set_role_tile_mode(G.ROLE_FWD, 3)


def test_chunked_backward_full_vocabulary_partial_last_chunk():
    """V = 151936 in vocabulary chunks of 40960 (the last one 29056 wide, not a multiple of
    256): the f32 dH accumulator path across four chunks meets the parity bar."""
    from paper_2510_17158_gb300 import grpo as G
    b = _batch("d4096_v152k")
    old, ref = oracle_inputs(b)
    S, T, d = b.H.shape
    need = G.grpo_workspace_bytes(S, T, d, b.W.shape[0], b.H.dtype, 40960)
    full = G.grpo_workspace_bytes(S, T, d, b.W.shape[0], b.H.dtype, 0)
    assert need < full
    g = run_gpu(b, old, ref, 0.2, 0.2, 0.04, vocab_chunk=40960)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    print(compare(b, g, o))


def test_progress_window_changes_nothing_and_resets_its_counters():
    """The progress window of the dH and dW GEMMs only delays TMA issue: outputs with it off, at
    16 k-blocks with lag 4, at a tight setting (1 k-block, lag 1, so that the producers wait at
    every k-block), with checkpoints at every work unit's start (-1, lag 1: a barrier between
    waves of units) and at the default (a barrier every 256 k-blocks) are bitwise equal, and the
    last CTA of every launch resets the window's counters in the workspace header (arrivals at
    byte 24, CTAs left at byte 32) to 0."""
    from paper_2510_17158_gb300 import grpo as G
    b = _batch("d4096_v152k")
    old, ref = oracle_inputs(b)
    outs = []
    try:
        for check, lag in ((0, 0), (16, 4), (1, 1), (-1, 1), G.GEMM_WINDOW_DEFAULT):
            G.grpo_set_gemm_window(check, lag)
            outs.append(run_gpu(b, old, ref, 0.2, 0.2, 0.04))
            dev = torch.device("cuda")
            H, W = b.H.to(dev), b.W.to(dev)
            S, T, d = H.shape
            ws = G.Workspace.for_problem(S, T, d, W.shape[0], H.dtype)
            tok, mask = b.tokens.to(dev), b.mask.to(dev)
            f = G.grpo_score_fwd(H, W, tok, mask, ws)
            adv = G.group_advantages(b.rewards.to(dev), b.group_offsets.to(dev), ws)
            G.grpo_loss_bwd(H, W, tok, mask, f["logp"], f["lse"], torch.from_numpy(old).to(dev),
                            torch.from_numpy(ref).to(dev), adv, f["valid_count"], ws)
            torch.cuda.synchronize()
            hdr = ws.buf[:64].cpu().numpy()
            assert int(hdr[24:32].view(np.uint64)[0]) == 0
            assert int(hdr[32:36].view(np.uint32)[0]) == 0
    finally:
        G.grpo_set_gemm_window(*G.GEMM_WINDOW_DEFAULT)
    for g in outs[1:]:
        for k in ("logp", "lse", "entropy", "argmax", "valid_count", "dH", "dW"):
            assert torch.equal(g[k], outs[0][k]), k
        assert g["loss"] == outs[0]["loss"]
    with pytest.raises(G.GrpoError):
        G.grpo_set_gemm_window(16, 0)
