"""The multi-GPU host logic of bench.py on CPU: two gloo ranks, each with its
own batch, the max over ranks and the whole-job aggregate.  The reduction
itself has no collective (images are independent), so nothing else is
exchanged between ranks."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = synth.make("llava576", seed=bench.rank_seed(0, rank), batch=2, n=16, d=64)
        local_ms = 1.0 + rank  # rank 1 is the slow one
        ms = bench.max_over_ranks(local_ms, world)
        value = bench.job_images_per_s(w.batch, world, ms)
        first = w.x[0, :4].float()
        gathered = [torch.zeros(4) for _ in range(world)]
        dist.all_gather(gathered, first)
        out[rank] = (ms, value, [g.tolist() for g in gathered])
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_gloo_ranks_max_and_aggregate():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    ms0, v0, g0 = out[0]
    ms1, v1, g1 = out[1]
    assert ms0 == ms1 == 2.0                      # the slowest rank's step time
    assert v0 == v1 == pytest.approx(2 * 2 / 2e-3)  # all ranks' images / that time
    assert g0[0] != g0[1]                          # each rank drew its own batch


def test_single_rank_is_identity():
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.job_images_per_s(64, 1, 0.25) == pytest.approx(256000.0)


def test_step_bytes():
    # bench.py's byte accounting for one step: the three inputs an
    # end-to-end step copies in, the path's algorithmic traffic, and y plus
    # the int32 indices copied back
    w = synth.make("llava576", seed=0, batch=3, n=40, d=64)
    ks = [8, 8, 8]
    in_b, alg_b, d2h_b = bench.step_bytes(w, ks)
    assert in_b == 3 * 120 * 64 * 2
    assert alg_b == in_b + 2 * 24 * 64 * 2 + 4 * 24
    assert d2h_b == 24 * (64 * 2 + 4)
    w = synth.make("single_clip336", seed=0, n=40)  # fp32
    in_b, alg_b, d2h_b = bench.step_bytes(w, [5])
    assert (in_b, d2h_b) == (3 * 40 * 1024 * 4, 5 * (1024 * 4 + 4))


def test_bench_sweep_and_graph_steps():
    assert bench._sweep_points("k=64,128,192") == ("k", [64, 128, 192])
    assert bench._sweep_points("lam=0/1,1/3") == ("lam", [(0, 1), (1, 3)])
    assert bench._sweep_points("ratio=1/9,2/9") == ("ratio", [(1, 9), (2, 9)])
    assert bench._sweep_points("batch=1,8,64") == ("batch", [1, 8, 64])
    with pytest.raises(SystemExit):
        bench._sweep_points("d=64")
    # replays of a graph of S steps time exactly K steps
    for k in (1, 3, 7, 16, 17, 20, 300, 2000, 4000):
        s = bench.steps_per_graph(k)
        assert 1 <= s <= bench.GRAPH_STEPS and k % s == 0
    assert bench.steps_per_graph(2000) == 16 and bench.steps_per_graph(300) == 15 and bench.steps_per_graph(17) == 1
