"""Data-parallel sharding over whole groups, checked with two gloo ranks on CPU against the
single-process oracle: summed losses and dW, and each shard's dH rows, equal the whole-batch
result when every rank uses the global normaliser. The sums go through bench.py's per-step
exchange (`dp_exchange`), the one its multi-GPU runs issue over NCCL."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import oracle
from paper_2510_17158_gb300.dp import global_norm, shard_groups
from paper_2510_17158_gb300.synthetic import Workload, make_batch_numpy

WORLD = 2


def _batch():
    w = Workload("dp", 3, (4, 2, 3), 24, 4, 24, 16, 40, "f32", "speedup", seed=21)
    return make_batch_numpy(w)


def _inputs(b):
    mask = b.mask.numpy()
    idx = np.argwhere(mask != 0)
    H, W = b.H.double().numpy(), b.W.double().numpy()
    sc = oracle.score_tokens(H[idx[:, 0], idx[:, 1]], W, b.tokens.numpy()[idx[:, 0], idx[:, 1]])
    base = np.zeros(mask.shape)
    base[idx[:, 0], idx[:, 1]] = sc["logp"]
    return H, W, base + 3 * b.noise_old.numpy(), base + b.noise_ref.numpy()


def _worker(rank, port, agg, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    b = _batch()
    H, W, old, ref = _inputs(b)
    lo, hi, go_local = shard_groups(b.group_offsets.numpy(), WORLD, rank)
    mask = b.mask.numpy()[lo:hi]

    def allsum(x):
        t = torch.tensor([x], dtype=torch.float64)
        dist.all_reduce(t)
        return float(t.item())

    norm = global_norm(agg, hi - lo, int((mask != 0).sum()), allsum)
    o = oracle.grpo_step(H[lo:hi], W, b.tokens.numpy()[lo:hi], mask, b.rewards.numpy()[lo:hi],
                         go_local, old[lo:hi], ref[lo:hi], 0.2, 0.2, 0.04, agg=agg, norm=norm)
    dH = torch.from_numpy(o["dH"].copy())
    out = bench.dp_exchange({"loss": torch.tensor([o["loss"]], dtype=torch.float64),
                             "dW": torch.from_numpy(o["dW"].copy()), "dH": dH.clone()}, WORLD)
    assert torch.equal(out["dH"], dH)   # dH rows stay with the rank that owns them
    q.put((rank, lo, hi, float(out["loss"].item()), out["dW"].numpy(), o["dH"]))
    dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("agg", ["seq_mean", "token_mean"])
def test_two_gloo_ranks_reproduce_single_process(agg):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, port, agg, q)) for r in range(WORLD)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(WORLD)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    b = _batch()
    H, W, old, ref = _inputs(b)
    full = oracle.grpo_step(H, W, b.tokens.numpy(), b.mask.numpy(), b.rewards.numpy(),
                            b.group_offsets.numpy(), old, ref, 0.2, 0.2, 0.04, agg=agg)
    for rank, lo, hi, loss, dW, dH in res:
        assert abs(loss - full["loss"]) <= 1e-12 * max(1.0, abs(full["loss"]))
        np.testing.assert_allclose(dW, full["dW"], rtol=1e-10, atol=1e-14)
        np.testing.assert_allclose(dH, full["dH"][lo:hi], rtol=1e-10, atol=1e-14)
    assert sorted((lo, hi) for _, lo, hi, *_ in res) == [(0, 4), (4, 9)]


def test_shard_groups_covers_whole_groups():
    go = np.array([0, 4, 8, 12, 16, 28])
    parts = [shard_groups(go, 3, r) for r in range(3)]
    assert [p[:2] for p in parts] == [(0, 4), (4, 12), (12, 28)]
    for lo, hi, local in parts:
        assert local[0] == 0 and local[-1] == hi - lo

