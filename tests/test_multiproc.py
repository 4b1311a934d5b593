"""The bench's multi-rank logic on CPU with the gloo backend (world size 2):
each rank times its own replica of the workload; rank 0 reports the maximum
elapsed time over ranks, and a barrier brackets the timed region."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, results):
    import torch.distributed as dist

    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        assert bench.dist_env() == (rank, world, rank)
        bench.barrier()
        local = 10.0 + 5.0 * rank  # rank 1 is the slow one
        results[rank] = bench.max_over_ranks(local)
        bench.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, results)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
        assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
        assert dict(results) == {0: 15.0, 1: 15.0}


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    bench.barrier()


@pytest.mark.parametrize("argv", [["--warmup", "2"]])
def test_bench_rejects_short_warmup(argv):
    import bench
    with pytest.raises(SystemExit):
        bench.main(argv)


def test_oracle_rows_parallel_matches_oracle():
    """The all-cores CPU baseline: the oracle's server MVM with the rows of W
    split over spawned processes gives the single-process oracle's result."""
    import numpy as np

    import bench
    import oracle
    rng = np.random.default_rng(5)
    W = rng.integers(-128, 128, size=(37, 96), dtype=np.int8)
    X = rng.integers(0, oracle.Q, size=(3, 96)).astype(np.uint32)
    macs, dt, y = bench.oracle_rows_parallel(W, X, 2)
    assert macs == 3 * 37 * 96 and dt > 0
    assert np.array_equal(y, oracle.server_mvm(W, X[-1]))
    info = bench.host_cpu()
    assert info["cpu_count"] >= 1 and info["model"]
