"""Multi-rank host logic on CPU (gloo, world_size 2): row sharding, the
all-reduce of the update's partial sums and counts, the global RabitQ mean
and the global fixed-point exponent give the single-process result.  The
partial sums here are plain numpy per shard (the same quantities skm_update
writes with `partial`); the mean protocol runs with the oracle's fixed-point
arithmetic and must give the single-process mean bit for bit."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2608_14648_gb300 import dist as skd


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _partials(X, a, k, d):
    S = np.zeros((k, d), np.float64)
    np.add.at(S, a, X.astype(np.float64))
    return S, np.bincount(a, minlength=k).astype(np.int64)


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        rng = np.random.default_rng(0)
        n, d, k = 1001, 9, 7
        X = rng.standard_normal((n, d)).astype(np.float32)
        a = rng.integers(0, k, n)
        lo, hi = skd.shard_bounds(n, rank, world)
        S, c = _partials(X[lo:hi], a[lo:hi], k, d)
        St, ct = torch.from_numpy(S), torch.from_numpy(c)
        skd.allreduce_partials(St, ct)
        import oracle

        Xs = X[lo:hi]
        mean = skd.global_mean_fixed(float(np.abs(Xs).max()), hi - lo,
                                     lambda sc: torch.from_numpy(oracle.column_sums_fixed(Xs, sc)),
                                     lambda S, nt, sc: torch.from_numpy(oracle.mean_from_sums(S.numpy(), nt, sc)),
                                     "cpu")
        e = skd.global_exponent(30 + rank, "cpu")
        q.put((rank, St.numpy(), ct.numpy(), mean.numpy(), e, lo, hi))
    finally:
        dist.destroy_process_group()


def test_shard_bounds_cover_rows_once():
    for n in (0, 1, 7, 1000, 1001):
        for world in (1, 2, 3, 8):
            spans = [skd.shard_bounds(n, r, world) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == n
            assert all(spans[i][1] == spans[i + 1][0] for i in range(world - 1))
            sizes = [hi - lo for lo, hi in spans]
            assert max(sizes) - min(sizes) <= 1


def test_two_rank_merge_equals_single_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(2)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    rng = np.random.default_rng(0)
    n, d, k = 1001, 9, 7
    X = rng.standard_normal((n, d)).astype(np.float32)
    a = rng.integers(0, k, n)
    S, c = _partials(X, a, k, d)
    for rank, St, ct, mean, e, lo, hi in out:
        np.testing.assert_allclose(St, S, rtol=1e-12, atol=1e-12)
        np.testing.assert_array_equal(ct, c)
        np.testing.assert_array_equal(mean, oracle.rbq1_mean(X))  # the single-process bits
        assert e == 30
    assert sorted((lo, hi) for _, _, _, _, _, lo, hi in out) == [(0, 501), (501, 1001)]
