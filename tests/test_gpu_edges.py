"""Edge cases of the CUDA path against the oracle: a single token, V < 256 and V not a multiple
of 32, T just past a tile boundary, the smallest bf16 hidden size, hidden sizes that are not a
multiple of 256, a completion with no scored token, an all-masked batch, groups of one, and a
data-parallel normaliser override."""
import numpy as np
import pytest
import torch

from paper_2510_17158_gb300.synthetic import Workload, make_batch_numpy
from tests.parity_util import compare, oracle_inputs, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


def W_(name, prompts, G, T, lo, hi, d, V, dtype="bf16", **kw):
    return Workload(name, prompts, G, T, lo, hi, d, V, dtype, "speedup", **kw)


EDGES = {
    "single_token": W_("single_token", 1, (1,), 1, 1, 1, 256, 512),
    "v200_d256": W_("v200_d256", 1, (3,), 70, 1, 70, 256, 200),
    "v1000_t129": W_("v1000_t129", 2, (2,), 129, 100, 129, 512, 1000),
    "v257_t257_g1": W_("v257_t257_g1", 3, (1, 2), 257, 1, 257, 768, 257),
    # hidden sizes that are multiples of 64 but not of 256: the last 256-column tile of dH and
    # dW is partial (64 and 128 valid columns)
    "d320_v1000": W_("d320_v1000", 2, (3,), 150, 20, 150, 320, 1000),
    "d896_v3001": W_("d896_v3001", 1, (4,), 140, 40, 140, 896, 3001),
    "f32_v33": W_("f32_v33", 2, (2,), 9, 1, 9, 48, 33, dtype="f32"),
}


@pytest.mark.parametrize("name", list(EDGES))
def test_edge_shapes(name):
    b = make_batch_numpy(EDGES[name])
    old, ref = oracle_inputs(b)
    g = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    print(name, compare(b, g, o))


def test_sequence_without_scored_tokens():
    b = make_batch_numpy(W_("empty_seq", 1, (4,), 150, 20, 150, 256, 777))
    b.mask[2] = 0
    old, ref = oracle_inputs(b)
    g = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    assert int(g["valid_count"][2]) == 0
    print(compare(b, g, o))


def test_all_masked_batch():
    b = make_batch_numpy(W_("all_masked", 1, (2,), 40, 5, 40, 256, 300))
    b.mask.zero_()
    old = np.zeros(b.mask.shape, np.float32)
    g = run_gpu(b, old, old, 0.2, 0.2, 0.04)
    assert g["status"] == 0
    assert torch.all(g["valid_count"] == 0) and torch.all(g["argmax"] == -1)
    assert torch.all(g["logp"] == 0) and g["loss"] == 0.0
    assert torch.all(g["dH"] == 0) and torch.all(g["dW"] == 0)


@pytest.mark.parametrize("agg", ["seq_mean", "token_mean"])
def test_normaliser_override_for_data_parallel_shards(agg):
    """A shard passes the global count (S' or N'); its loss and gradients scale accordingly."""
    b = make_batch_numpy(W_("shard", 1, (4,), 100, 30, 100, 256, 1000))
    old, ref = oracle_inputs(b)
    norm = 3.0 * (b.S if agg == "seq_mean" else float(b.mask.sum()))
    g = run_gpu(b, old, ref, 0.2, 0.2, 0.04, agg=agg, norm=norm)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04, agg=agg, norm=norm)
    print(compare(b, g, o))


def test_partial_hidden_tile_chunked_backward_and_every_tile_mode():
    """d = 576 = 2*256 + 64: three output column tiles of dH and dW, the last with 64 valid
    columns; in the wide pair mode (2) two column units of 512, the second with 64 valid
    columns, and 2600 / 128 = 21 vocabulary row tiles of dW (odd: the second CTA of the last
    pair stages a copy). A 3-chunk backward (V = 2600 in chunks of 1024) accumulates dH across
    chunks through the partial tile in every mode. Every mode meets the parity bar; dH and dW of
    mode 2 are bitwise equal to mode 1's on the same dz, and with every role in mode 2 (forward
and dz units of two vocabulary tiles; V = 2600 has 11 tiles, so the last unit's second tile
lies past the vocabulary) every output is bitwise equal to mode 1's."""
    from paper_2510_17158_gb300 import grpo as G
    b = make_batch_numpy(W_("d576_v2600", 1, (4,), 160, 40, 160, 576, 2600))
    old, ref = oracle_inputs(b)
    o = run_oracle(b, old, ref, 0.2, 0.2, 0.04)
    outs = {}
    try:
        for modes in ((0, 0, 0, 0), (1, 1, 1, 1), (1, 1, 2, 2), (0, 0, 2, 2), (2, 2, 2, 2)):
            for role, m in enumerate(modes):
                G.grpo_set_role_tile_mode(role, m)
            outs[modes] = run_gpu(b, old, ref, 0.2, 0.2, 0.04)
            print("modes", modes, compare(b, outs[modes], o))
            print("chunked", modes,
                  compare(b, run_gpu(b, old, ref, 0.2, 0.2, 0.04, vocab_chunk=1024), o))
    finally:
        G.grpo_set_tile_mode(G.TILE_DEFAULT)
    for k in ("dH", "dW"):
        assert torch.equal(outs[(1, 1, 2, 2)][k], outs[(1, 1, 1, 1)][k]), k
    for k in ("logp", "lse", "entropy", "argmax", "dH", "dW"):   # the same M = 256 MMAs
        assert torch.equal(outs[(2, 2, 2, 2)][k], outs[(1, 1, 1, 1)][k]), k
