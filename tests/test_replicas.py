"""The multi-rank path on CPU (gloo, world size 2): token shards cover the batch,
max-over-ranks timing, and the layer splits over tokens with no collective (each
rank's oracle output on its shard equals that slice of the whole-layer output)."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2608_17402_gb300.replicas import max_over_ranks, token_shard


def test_token_shard_covers_batch():
    for T in (0, 1, 7, 300, 8192):
        for world in (1, 2, 3, 8):
            ranges = [token_shard(T, r, world) for r in range(world)]
            assert ranges[0][0] == 0 and ranges[-1][1] == T
            assert all(a[1] == b[0] for a, b in zip(ranges, ranges[1:]))
            sizes = [b - a for a, b in ranges]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        token_shard(10, 2, 2)


def test_max_over_ranks_single_process():
    assert max_over_ranks([1.5, 2.0]) == [1.5, 2.0]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, outdir):
    import torch.distributed as dist
    import oracle
    import workloads
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        cfg = workloads.small_config(T=37, d=32, E=6, k=2, h=16, h_s=16, seed=3)
        lay = workloads.make_layer(cfg)
        a, b = token_shard(cfg.T, rank, world)
        y, idx, _, _ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k, lay.Ws1,
                                             lay.Ws2, cfg.lam, tokens=np.arange(a, b, dtype=np.int32),
                                             nthreads=1)
        np.save(os.path.join(outdir, f"y{rank}.npy"), y)
        np.save(os.path.join(outdir, f"idx{rank}.npy"), idx)
        got = max_over_ranks([float(rank), 10.0 - rank])
        np.save(os.path.join(outdir, f"max{rank}.npy"), np.array(got))
    finally:
        dist.destroy_process_group()


def test_gloo_two_ranks_shard_tokens_without_collective(tmp_path):
    import oracle
    import workloads
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    cfg = workloads.small_config(T=37, d=32, E=6, k=2, h=16, h_s=16, seed=3)
    lay = workloads.make_layer(cfg)
    y_all, idx_all, _, _ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k,
                                                 lay.Ws1, lay.Ws2, cfg.lam, nthreads=1)
    y = np.concatenate([np.load(tmp_path / f"y{r}.npy") for r in range(world)])
    idx = np.concatenate([np.load(tmp_path / f"idx{r}.npy") for r in range(world)])
    assert np.array_equal(idx, idx_all)
    assert np.array_equal(y, y_all)
    for r in range(world):
        assert list(np.load(tmp_path / f"max{r}.npy")) == [1.0, 10.0]
