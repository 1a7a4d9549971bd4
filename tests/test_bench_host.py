"""Host-side pieces of bench.py's roofline: the stamped DRAM traffic of the
batch-1 decode step is reported only while the step kernels' sources are the
ones it was captured on, and the algorithmic bytes per step are the figure
the roofline divides by."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2306_04235_gb300 import synth  # noqa: E402


def test_step_traffic_stamp_matches_the_step_kernel_sources():
    traffic, stamp = bench.STEP_TRAFFIC[(bench.DEFAULT_WORKLOAD, True)]
    assert stamp == bench._source_hash(bench.STEP_SOURCES), "step kernels changed since the traffic capture"
    algo = _mean_step_bytes(bench.DEFAULT_WORKLOAD, 8)
    # every weight, scale and cache byte read once: within a few percent above
    assert algo <= traffic <= 1.05 * algo


def _mean_step_bytes(name, wq, steps=None):
    wl = synth.WORKLOADS[name]
    cfg = synth.MODELS[wl.model]
    ids, _ = synth.source_batch(cfg.vocab, wl.batch, wl.src_len[0], wl.src_len[1], wl.src_seed)
    B, S = ids.shape
    n = steps or wl.max_len
    return sum(bench.decode_step_bytes(cfg, B * wl.beam, B, S, t, wq) for t in range(n)) / n


def test_default_step_bytes():
    # the batch-1 line: S = 46, the mean over 64 greedy steps
    assert int(_mean_step_bytes(bench.DEFAULT_WORKLOAD, 8)) == 10_471_044


def test_step_bytes_grow_with_the_cache_and_shrink_with_4_bit_rows():
    cfg = synth.MODELS["small-12x2-d256-v32k-e128"]
    b = [bench.decode_step_bytes(cfg, 1, 1, 46, t) for t in range(4)]
    # one more self-attention position: a key and a value row of d bytes per decoder layer
    assert all(b[i + 1] - b[i] == 2 * cfg.n_dec * cfg.d_model for i in range(3))
    w8 = bench.decode_step_bytes(cfg, 1, 1, 46, 0, 8)
    w4 = bench.decode_step_bytes(cfg, 1, 1, 46, 0, 4)
    mm = bench.decode_step_bytes(cfg, 1, 1, 46, 0, 4 | 0x100)
    codes = cfg.n_dec * (6 * cfg.d_model ** 2 + 2 * cfg.d_ffn * cfg.d_model)
    assert w8 - w4 == codes // 2
    assert mm - w4 == 4 * cfg.n_dec * (7 * cfg.d_model + cfg.d_ffn)


@pytest.mark.parametrize("name", ["small-b32-s10to80-beam4-t128", "wide-b128-s20to128-beam4-t160"])
def test_batched_step_bytes_include_every_hypothesis_cache(name):
    wl = synth.WORKLOADS[name]
    cfg = synth.MODELS[wl.model]
    R = wl.batch * wl.beam
    one = bench.decode_step_bytes(cfg, R, wl.batch, 0, 0)
    two = bench.decode_step_bytes(cfg, R, wl.batch, 0, 1)
    assert two - one == 2 * cfg.n_dec * R * cfg.d_model
