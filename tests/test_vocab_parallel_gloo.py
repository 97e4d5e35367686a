"""Vocabulary-parallel exchange with two gloo ranks on CPU and the oracle: each rank scores its
rows of the LM head, the per-token statistics are all-gathered and merged, the dz of each rank's
columns gives a dH partial that is all-reduced, and each rank keeps its rows of dW. The result
equals the single-process oracle."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2510_17158_gb300.dp import vocab_shard_bounds

WORLD = 2


def _problem():
    rng = np.random.default_rng(31)
    n, d, V = 30, 16, 600
    h = rng.normal(size=(n, d))
    W = rng.normal(scale=0.3, size=(V, d))
    y = rng.integers(0, V, size=n)
    g = rng.normal(size=n)
    return h, W, y, g


def _worker(rank, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    h, W, y, g = _problem()
    v0, v1 = vocab_shard_bounds(W.shape[0], WORLD, rank)
    st = oracle.shard_stats(h, W[v0:v1], y, v0)
    packed = torch.from_numpy(np.stack([st["m"], st["s"], st["u"], st["argmax"], st["zy"]]))
    gathered = [torch.empty_like(packed) for _ in range(WORLD)]
    dist.all_gather(gathered, packed)                  # the one forward exchange
    stats = [{"m": t[0].numpy(), "s": t[1].numpy(), "u": t[2].numpy(),
              "argmax": t[3].numpy().astype(np.int64), "zy": t[4].numpy()} for t in gathered]
    mg = oracle.merge_shard_stats(stats)
    # backward: this rank's columns of dz, its dH partial (all-reduced) and its rows of dW
    Z = h @ W[v0:v1].T
    P = np.exp(Z - mg["lse"][:, None])
    onehot = np.zeros_like(P)
    own = (y >= v0) & (y < v1)
    onehot[np.flatnonzero(own), y[own] - v0] = 1.0
    dZ = g[:, None] * (onehot - P)
    dH = torch.from_numpy(dZ @ W[v0:v1])
    dist.all_reduce(dH)
    q.put((rank, v0, v1, mg, dH.numpy(), dZ.T @ h))
    dist.destroy_process_group()


def test_two_gloo_ranks_vocab_parallel_equal_single_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    procs = [ctx.Process(target=_worker, args=(r, port, q)) for r in range(WORLD)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(WORLD)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    h, W, y, g = _problem()
    full = oracle.score_tokens(h, W, y)
    dH_full, dW_full = oracle.param_grads(h, W, y, full["lse"], g)
    for rank, v0, v1, mg, dH, dW_rows in res:
        for k in ("lse", "logp", "entropy"):
            np.testing.assert_allclose(mg[k], full[k], rtol=1e-12, atol=1e-12)
        assert np.array_equal(mg["argmax"], full["argmax"])
        np.testing.assert_allclose(dH, dH_full, rtol=1e-10, atol=1e-13)
        np.testing.assert_allclose(dW_rows, dW_full[v0:v1], rtol=1e-10, atol=1e-13)
    assert sorted((v0, v1) for _, v0, v1, *_ in res) == [(0, 256), (256, 600)]
