"""Multi-GPU = independent replicas (one hyperbatch stream per GPU, no
data-path collective).  The host-side logic bench.py uses for N > 1 runs
here as 2 gloo ranks on the CPU: disjoint targets per rank and the
max-over-ranks time."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    from agnes_inputs import WORKLOADS, target_pool, targets_for_step
    dist.init_process_group("gloo")
    ws, r, local = bench.dist_env()
    assert (ws, r, local) == (world, rank, rank)
    w = WORKLOADS["mini100m"].with_(num_nodes=20000, H=2, B=64, train_frac=0.5)
    pool = target_pool(w, "cpu")
    mine = torch.cat([targets_for_step(w, pool, bench.step_index(r, s)).flatten()
                      for s in range(3)])
    gathered = [torch.zeros_like(mine) for _ in range(world)]
    dist.all_gather(gathered, mine)
    t = bench.reduce_max(10.0 + 5 * r, dist, "cpu")
    out[rank] = (t, [g.tolist() for g in gathered])
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_gloo_ranks_draw_disjoint_hyperbatches_and_agree_on_max_time():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(240)
        assert p.exitcode == 0
    assert out[0][0] == out[1][0] == 15.0
    a, b = out[0][1]
    assert out[0][1] == out[1][1]
    # each step's targets are distinct within a hyperbatch; ranks draw different ones
    assert set(a) != set(b)
    for ids in (a, b):
        assert len(set(ids[:128])) == 128


def test_reduce_max_without_a_process_group_is_identity():
    import bench
    assert bench.reduce_max(3.5, None, "cpu") == 3.5
    assert bench.step_index(0, 7) == 7 and bench.step_index(1, 0) != bench.step_index(0, 0)
