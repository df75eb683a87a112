"""The multi-GPU decomposition on CPU with two gloo ranks: each rank routes its own request range
(bench.rank_requests) against the same trees, with no data-path collective; the job time is the max over
ranks (bench.max_over_ranks).  Routing is done with the CPU oracle here (no GPU), and the union of the
ranks' results must equal routing the whole two-rank job at once."""
import os
import socket

import numpy as np
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    import oracle
    import workload as wl
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    prm = wl.preset(0)
    prm.update(B=300)
    W = wl.Workload(params=prm, seed=9)
    trees = oracle.build_trees([W.tree(p) for p in range(W.P)], n_threads=2)
    b0, b1 = bench.rank_requests(rank, W.B)
    tok, off = W.requests(b0, b1, n_threads=2)
    m, peer, _ = oracle.route(trees, tok, off, W.load(), W.alpha, n_threads=2)
    np.save(os.path.join(out_dir, f"m{rank}.npy"), m)
    np.save(os.path.join(out_dir, f"p{rank}.npy"), peer)
    slowest = bench.max_over_ranks(10.0 * (rank + 1), dist)
    np.save(os.path.join(out_dir, f"t{rank}.npy"), np.array([slowest]))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_weak_scaling_decomposition(tmp_path):
    import oracle
    import workload as wl
    import bench
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    assert bench.rank_requests(0, 300) == (0, 300) and bench.rank_requests(1, 300) == (300, 600)
    prm = wl.preset(0)
    prm.update(B=300)
    W = wl.Workload(params=prm, seed=9)
    trees = oracle.build_trees([W.tree(p) for p in range(W.P)], n_threads=2)
    tok, off = W.requests(0, 600, n_threads=2)
    m_all, p_all, _ = oracle.route(trees, tok, off, W.load(), W.alpha, n_threads=2)
    m = np.concatenate([np.load(tmp_path / f"m{r}.npy") for r in range(world)])
    p = np.concatenate([np.load(tmp_path / f"p{r}.npy") for r in range(world)])
    assert np.array_equal(m, m_all) and np.array_equal(p, p_all)
    assert all(float(np.load(tmp_path / f"t{r}.npy")[0]) == 20.0 for r in range(world))
