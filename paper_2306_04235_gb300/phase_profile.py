"""Phase timing of the batch-1 cluster decode step (debug build).

Builds libmnmt_stamps.so (the library with the cluster step compiled with
-DMNMT_DC_STAMPS), translates a workload with it and prints, for decode step
20, how long each of the step's phases spends waiting for its weight slice,
preparing its input (LayerNorm or attention), in its slice GEMV and in the
exchange (its slice stored to every CTA, then the wait until this CTA's copy
of the vector is whole), plus the prologue and the overlap with the previous
step's vocabulary kernel.  Times in ns from %globaltimer at CTA 0.

    python -m paper_2306_04235_gb300.phase_profile [workload]
"""
from __future__ import annotations

import ctypes as C
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))

from paper_2306_04235_gb300 import build, mnmt, synth  # noqa: E402

KINDS = ["qkv", "self-att+O", "q2", "cross-att+O2", "w1", "w2"]


def main(argv):
    import torch

    name = argv[1] if len(argv) > 1 else "small-b1-s10to50-greedy64"
    lib = C.CDLL(build.build(stamps=True))
    mnmt._declare(lib)
    mnmt._lib = lib
    lib.mnmt_dc_stamps.argtypes = [C.c_void_p]
    cfg, blob, ids, lens, beam, T = synth.workload_inputs(name)
    assert beam == 1 and ids.shape[0] <= 4 and T > 20, "a greedy batch-1..4 workload of more than 20 steps"
    tr = mnmt.Translator(blob, ids.shape[0], ids.shape[1], 1, T)
    try:
        for _ in range(3):
            tr.translate(ids, lens, T)
        assert mnmt.mnmt_session_decode_path(tr.session) == 1
    finally:
        tr.close()
    torch.cuda.synchronize()
    ns = np.zeros(128, np.uint64)
    lib.mnmt_dc_stamps(ns.ctypes.data)
    ns = ns.astype(np.int64)
    t0 = ns[0]
    print(f"{name}: S_pad {ids.shape[1]}, decode step 20 (ns from the step kernel's start)")
    print(f"previous vocabulary kernel: start {ns[110] - t0}, wait ends {ns[112] - t0}, ends {ns[113] - t0}")
    print(f"step kernel: grid wait {ns[1] - t0}..{ns[2] - t0}, phase loop starts {ns[3] - t0}")
    print("| phase | kind | ring wait | prep | slice GEMV | exchange |")
    print("|---:|---|---:|---:|---:|---:|")
    prev = ns[3]
    tot = np.zeros(4, np.int64)
    for ph in range(1 + 6 * cfg.n_dec):
        a, b, c, d = ns[4 + 4 * ph:8 + 4 * ph]
        kind = "embedding" if ph == 0 else KINDS[(ph - 1) % 6]
        row = np.array([a - prev, b - a, c - b, d - c])
        tot += row
        prev = d
        print(f"| {ph} | {kind} | {row[0]} | {row[1]} | {row[2]} | {row[3]} |")
    print(f"| all | | {tot[0]} | {tot[1]} | {tot[2]} | {tot[3]} |")
    print(f"final LayerNorm {ns[101] - ns[100]}, output rows {ns[102] - ns[101]}, kernel {ns[102] - t0}")
    return 0


if __name__ == "__main__":
    sys.exit(main(sys.argv))
