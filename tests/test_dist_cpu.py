"""Multi-rank host logic on the CPU with the gloo backend (world size 2): the
bench's rank plumbing (set-up from the launcher's environment, barrier, the
max over ranks of the step time), the token sharding of the boundary, and the
one exchange of the subspace update (the sum of the replicas' Grassmann
accumulations), checked against the fp64 oracle over the whole batch."""
import importlib.util
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2506_01260_gb300.shard import token_shard  # noqa: E402


def _load(name, path):
    spec = importlib.util.spec_from_file_location(name, path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, outdir):
    # CPU ranks (gloo) even on a machine with a GPU: the bench's set-up picks
    # NCCL whenever CUDA is visible
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world),
                      RANK=str(rank), LOCAL_RANK=str(rank), CUDA_VISIBLE_DEVICES="")
    sys.path.insert(0, ROOT)
    import torch
    bench = _load("bench_under_test", os.path.join(ROOT, "bench.py"))
    g = _load("oracle_grassmann", os.path.join(ROOT, "oracle", "grassmann.py"))
    from paper_2506_01260_gb300.shard import allreduce_grassmann, token_shard as ts
    w, r, local, pg = bench.dist_setup(type("A", (), {})())
    assert (w, r, local) == (world, rank, rank) and pg is not None
    bench.barrier(pg)
    # the step time every rank reports is the slowest rank's
    t_max = bench.max_over_ranks(pg, 1.5 + rank)
    # each replica accumulates its own token rows; the sum is the whole batch's
    rng = np.random.default_rng(0)
    T, d, k = 37, 12, 3
    G = rng.standard_normal((T, d))
    U = g.retract(rng.standard_normal((d, k)))
    a, b = ts(T, world, rank)
    M = torch.from_numpy(g.accumulate(np.zeros((d, k)), G[a:b], U))
    allreduce_grassmann(M)
    U1 = g.step(U, M.numpy(), 1, 0.05)
    np.savez(os.path.join(outdir, "rank%d.npz" % rank), t_max=t_max, M=M.numpy(), U1=U1)
    torch.distributed.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_two_gloo_ranks(tmp_path, world):
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    g = _load("oracle_grassmann_main", os.path.join(ROOT, "oracle", "grassmann.py"))
    rng = np.random.default_rng(0)
    T, d, k = 37, 12, 3
    G = rng.standard_normal((T, d))
    U = g.retract(rng.standard_normal((d, k)))
    M_all = g.accumulate(np.zeros((d, k)), G, U)
    res = [np.load(tmp_path / ("rank%d.npz" % r)) for r in range(world)]
    for r in res:
        assert float(r["t_max"]) == 1.5 + (world - 1)
        assert np.allclose(r["M"], M_all, rtol=1e-12, atol=1e-12)
    assert np.array_equal(res[0]["U1"], res[1]["U1"])       # every replica takes the same step


@pytest.mark.parametrize("T", [0, 1, 7, 64, 1001])
@pytest.mark.parametrize("world", [1, 2, 3, 8])
def test_token_shards_cover_every_row_once(T, world):
    spans = [token_shard(T, world, r) for r in range(world)]
    assert spans[0][0] == 0 and spans[-1][1] == T
    assert all(spans[i][1] == spans[i + 1][0] for i in range(world - 1))
    sizes = [b - a for a, b in spans]
    assert max(sizes) - min(sizes) <= 1
