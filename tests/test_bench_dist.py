"""The N > 1 host logic of bench.py on CPU with gloo (world size 2): rank set-up,
barrier, max-over-ranks timing, per-rank batches, and the reference arm running
on rank 0 only."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    import torch.distributed as dist
    r, w = bench.init_dist("gloo")
    bench.barrier()
    m = bench.max_over_ranks(10.0 + rank)
    # The reference arm: only rank 0 produces a line.
    class A:
        steps, warmup = 1, 0
    from paper_2606_29563_gb300 import synth
    wl = synth.small_workload(seqlens=(200,), layers=1)
    rr, line = bench.run_reference(A, wl)
    seed = wl.replace(seed=wl.seed + 1000 * rank).seed
    out.put((rank, r, w, m, line is not None, seed))
    dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_rank_gloo_plumbing():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=240) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [x[1] for x in res] == [0, 1] and all(x[2] == 2 for x in res)
    assert all(x[3] == 11.0 for x in res)            # max over ranks
    assert [x[4] for x in res] == [True, False]      # reference line on rank 0 only
    assert res[0][5] != res[1][5]                    # each rank draws its own batch
