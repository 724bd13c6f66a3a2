"""Host-side logic of bench.py: byte/FLOP accounting, the whole-job aggregate, and the
max-over-ranks timing reduction with two gloo ranks on CPU."""
import os
import socket

import pytest

import bench


def test_accounting_matches_the_roofline_table():
    # Llama-2-7B q/k/v/o at M = 16, r = 1.1: n = 4512
    b = bench.layer_bytes(4096, 4096, 4512, 4512, 16)
    assert abs(b / 1e6 - 79.29) < 0.01
    f = bench.layer_flops(4096, 4096, 4512, 4512, 2048)
    assert abs(f / 1e9 - 234.785) < 0.01
    # gate at M = 1: 317.36 MB
    assert abs(bench.layer_bytes(4096, 11008, 4512, 12112, 1) / 1e6 - 317.36) < 0.01


def test_aggregate_is_whole_job():
    assert bench.aggregate(7.0, 100, 7, 1) == pytest.approx(10.0)
    assert bench.aggregate(7.0, 100, 7, 2) == pytest.approx(5.0)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    elapsed = [3.0, 5.0][rank]
    m = bench.max_over_ranks(elapsed, dist, "cpu")
    q.put((rank, m, bench.aggregate(m, 10, 7, world)))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_two_gloo_ranks():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [m for _, m, _ in out] == [5.0, 5.0]
    assert out[0][2] == pytest.approx(5.0 * 1e3 / (10 * 7 * 2))
