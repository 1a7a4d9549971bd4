"""The N > 1 path of bench.py (replicas only: one process per GPU, no
collective on the data path) on the host, as world-size-2 gloo ranks on CPU:
the job's throughput is every rank's tokens over the slowest rank's time, and
every rank translates its own sentences."""
import os
import socket
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import bench

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r: 100 + 50 r ms for its 3 steps of 64 + r tokens each
        value, total_ms, job_toks = bench.aggregate_ranks(100.0 + 50.0 * rank, 64 + rank, 3, dist, device="cpu")
        out[rank] = (value, total_ms, job_toks)
    finally:
        dist.destroy_process_group()


def test_replica_throughput_is_job_tokens_over_slowest_rank():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_rank, args=(world, _free_port(), out), nprocs=world, join=True)
    expect_ms = 150.0                       # the slower rank
    expect_toks = 64.0 + 65.0               # both ranks' tokens per step
    expect = expect_toks * 3 / (expect_ms / 1e3)
    for r in range(world):
        value, total_ms, job_toks = out[r]
        assert total_ms == expect_ms and job_toks == expect_toks
        assert value == pytest.approx(expect, rel=1e-12)


def test_single_rank_needs_no_collective():
    import bench

    value, total_ms, job_toks = bench.aggregate_ranks(200.0, 64, 4)
    assert (total_ms, job_toks) == (200.0, 64.0)
    assert value == pytest.approx(64 * 4 / 0.2)


def test_every_rank_translates_its_own_sentences():
    import bench
    from paper_2306_04235_gb300 import synth

    wl = synth.WORKLOADS[bench.DEFAULT_WORKLOAD]
    cfg = synth.MODELS[wl.model]
    batches = [synth.source_batch(cfg.vocab, wl.batch, wl.src_len[0], wl.src_len[1],
                                  bench.replica_source_seed(wl.src_seed, r))[0] for r in range(4)]
    for i in range(4):
        for j in range(i + 1, 4):
            a, b = batches[i], batches[j]
            assert a.shape != b.shape or not np.array_equal(a, b)
