"""Benchmark of the INT8 encoder-decoder translation path on GB300.

One step = one translation of one batch of the workload (encoder + every
decoder step until all sentences finish or the step limit), i.e. one pass of
the whole path.  The default workload is the batch-1 latency configuration:
the 12+2-layer d=256 model with a factorised 128-dim embedding and a 32000
vocabulary, source lengths uniform in 10..50, greedy decoding of up to 64
tokens.  Metric: decoded tokens per second (whole job over all GPUs).

  value     inputs already resident in HBM (device pointers through the C ABI),
            CUDA events on the library's stream, L2 flushed between steps (a
            256 MB write, outside the timed events)
  e2e       the same metric through the C ABI with pinned HOST buffers: the
            host->device copy of the source ids and the device->host copy of
            the output ids are inside the timed region
  roofline  the dominant kernel (the fused vocabulary projection + argmax,
            M=1 x N=32000 x K=256) timed with CUDA events on its stream over
            as many launches as the timed region ran, L2 flushed before each
  cpu_baseline  the CPU oracle on a bounded sample of the same workload

--impl reference runs the CPU oracle (the reference of this path) on the host
cores with the same metric and config.  Under torchrun every rank translates
its own replica of the workload (sentences are independent: no collective on
the data path); rank 0 prints the line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2306_04235_gb300 import synth  # noqa: E402

DEFAULT_WORKLOAD = "small-b1-s10to50-greedy64"
METRIC = "decoded tokens/sec"


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def kernels_per_translation(cfg, beam, steps):
    """Kernels the library launches for one translation: encoder (embedding,
    7 per layer, cross K/V per decoder layer), search init, decoder steps
    (embedding, 11 per layer, vocabulary projection, 1 greedy / 2 beam search
    kernels), final backtrack."""
    enc = 1 + 7 * cfg.n_enc + cfg.n_dec
    step = 1 + 11 * cfg.n_dec + 1 + (1 if beam == 1 else 2)
    return enc + 1 + step * steps + 1


def cpu_sample(workload, n_sent, threads):
    """The oracle translating n_sent sentences drawn like the workload's (batch-1
    translations, one per thread at a time)."""
    from oracle import oracle as O

    wl = synth.WORKLOADS[workload]
    cfg = synth.MODELS[wl.model]
    blob = synth.build_blob(cfg, wl.model_seed)
    ids, lens = synth.source_batch(cfg.vocab, n_sent * wl.batch, wl.src_len[0], wl.src_len[1], wl.src_seed + 7)
    O.lib()
    t0 = time.perf_counter()
    out, olen, _ = O.translate(blob, ids, lens, wl.beam, wl.max_len, n_threads=threads)
    dt = time.perf_counter() - t0
    return int(olen.sum()), dt


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    wl = synth.WORKLOADS[args.workload]
    cfg = synth.MODELS[wl.model]
    from oracle import oracle as O

    blob = synth.build_blob(cfg, wl.model_seed)
    ids, lens = synth.source_batch(cfg.vocab, wl.batch, wl.src_len[0], wl.src_len[1], wl.src_seed)
    O.lib()
    threads = min(os.cpu_count() or 1, wl.batch)
    for _ in range(args.warmup):
        O.translate(blob, ids, lens, wl.beam, wl.max_len, n_threads=threads)
    toks, times = 0, []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        out, olen, _ = O.translate(blob, ids, lens, wl.beam, wl.max_len, n_threads=threads)
        times.append(time.perf_counter() - t0)
        toks += int(olen.sum())
    total = sum(times)
    v = toks / total
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int8",
            "data": "synthetic",
            "config": {"workload": args.workload, "model": wl.model, "batch": wl.batch, "beam": wl.beam,
                       "max_len": wl.max_len, "src_len": list(wl.src_len)},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": threads, "kind": "oracle",
                             "sample": f"the full workload batch ({wl.batch} sentence(s)) per step"},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_gpu(args):
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    from paper_2306_04235_gb300 import mnmt

    wl = synth.WORKLOADS[args.workload]
    cfg = synth.MODELS[wl.model]
    blob = synth.build_blob(cfg, wl.model_seed)
    # every rank translates its own replica batch (independent sentences)
    ids, lens = synth.source_batch(cfg.vocab, wl.batch, wl.src_len[0], wl.src_len[1], wl.src_seed + 101 * rank)
    B, S = ids.shape
    stream = torch.cuda.Stream()
    tr = mnmt.Translator(blob, B, S, wl.beam, wl.max_len, stream)
    sess = tr.session
    T = wl.max_len
    d_ids = torch.from_numpy(ids).cuda()
    d_lens = torch.from_numpy(lens).cuda()
    o_ids = torch.zeros((B, T), dtype=torch.int32, device="cuda")
    o_len = torch.zeros(B, dtype=torch.int32, device="cuda")
    o_sc = torch.zeros(B, dtype=torch.float32, device="cuda")
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()

    def step():
        mnmt.mnmt_translate(sess, d_ids, d_lens, B, S, T, mnmt.DEVICE_PTRS, o_ids, o_len, o_sc)

    for _ in range(args.warmup):
        with torch.cuda.stream(stream):
            flush.fill_(1)
        step()
    stream.synchronize()

    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    toks = 0
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for i in range(args.steps):
            with torch.cuda.stream(stream):
                flush.fill_(i & 0xFF)
                evs[i][0].record(stream)
            step()
            with torch.cuda.stream(stream):
                evs[i][1].record(stream)
        torch.cuda.synchronize()
    if dist:
        dist.barrier()
    step_ms = [a.elapsed_time(b) for a, b in evs]
    toks_per_step = int(o_len.sum().item())
    total_ms = sum(step_ms)
    if dist:
        t = torch.tensor([total_ms], dtype=torch.float64, device="cuda")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
        n = torch.tensor([toks_per_step], dtype=torch.float64, device="cuda")
        dist.all_reduce(n, op=dist.ReduceOp.SUM)
        job_toks_per_step = float(n.item())
    else:
        job_toks_per_step = float(toks_per_step)
    value = job_toks_per_step * args.steps / (total_ms / 1e3)

    # per decode-step latency: translation time minus the encoder's, over the steps
    enc_ms = []
    for _ in range(5):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
        mnmt.mnmt_encode(sess, d_ids, d_lens, B, S, mnmt.DEVICE_PTRS)
        with torch.cuda.stream(stream):
            e1.record(stream)
        stream.synchronize()
        enc_ms.append(e0.elapsed_time(e1))
    steps_run = int(o_len.max().item()) if wl.beam == 1 else T
    enc_med = statistics.median(enc_ms)
    step_us = sorted(1e3 * (t - enc_med) / max(steps_run, 1) for t in step_ms)

    # end to end through the C ABI with pinned host buffers
    h_ids = torch.from_numpy(ids).pin_memory()
    h_lens = torch.from_numpy(lens).pin_memory()
    h_out = torch.zeros((B, T), dtype=torch.int32).pin_memory()
    h_olen = torch.zeros(B, dtype=torch.int32).pin_memory()
    h_osc = torch.zeros(B, dtype=torch.float32).pin_memory()
    e2e_times = []
    for i in range(args.warmup + args.steps):
        with torch.cuda.stream(stream):
            flush.fill_(i & 0xFF)
        stream.synchronize()
        t0 = time.perf_counter()
        mnmt.mnmt_translate(sess, h_ids.data_ptr(), h_lens.data_ptr(), B, S, T, 0, h_out.data_ptr(),
                            h_olen.data_ptr(), h_osc.data_ptr())
        if i >= args.warmup:
            e2e_times.append(time.perf_counter() - t0)
    e2e_tok = int(h_olen.sum().item())
    e2e_value = e2e_tok * world * len(e2e_times) / sum(e2e_times)
    assert torch.equal(h_out, o_ids.cpu()), "host and device paths disagree"

    # dominant kernel: fused vocabulary projection + argmax (M=1)
    roof = measure_vocab_kernel(args, cfg, mnmt, torch, stream, flush, n_launch=min(args.steps * steps_run, 640))

    if rank == 0:
        cpu = None
        if not args.no_cpu_baseline and world == 1:
            threads = os.cpu_count() or 1
            n_sent = max(1, min(2 * threads, 32))
            ctoks, cdt = cpu_sample(args.workload, n_sent, threads)
            cpu = {"value": ctoks / cdt, "unit": "tokens/s", "cores": min(threads, n_sent * wl.batch),
                   "kind": "oracle",
                   "sample": f"{n_sent} translation(s) of {wl.batch} sentence(s) drawn like the workload, "
                             f"one per thread ({cdt:.1f} s)"}
        launches = kernels_per_translation(cfg, wl.beam, steps_run) * args.steps
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
            "config": {"workload": args.workload, "model": wl.model, "batch": B, "beam": wl.beam,
                       "max_len": T, "src_len": list(wl.src_len), "s_pad": S, "tokens_per_step": toks_per_step,
                       "l2": "flushed between steps (256 MB write, outside the timed events)",
                       "decode_step_us_p50": step_us[len(step_us) // 2],
                       "decode_step_us_p90": step_us[min(len(step_us) - 1, int(0.9 * len(step_us)))],
                       "encode_ms_p50": enc_med, "parallelism": f"replicas x{world}"},
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": int(ids.nbytes + lens.nbytes),
                    "d2h_bytes_per_step": int(B * T * 4 + B * 8)},
            "roofline": roof,
            "cpu_baseline": cpu,
            "clocks": clk.summary(),
            "gpu_launches": launches,
        }
        print(json.dumps(line), flush=True)
    tr.close()
    if dist:
        dist.destroy_process_group()
    return 0


def measure_vocab_kernel(args, cfg, mnmt, torch, stream, flush, n_launch):
    """The fused vocabulary projection + argmax at batch 1 (the largest weight
    stream of a decode step), timed with CUDA events on its stream, L2 flushed
    before each launch.  Algorithmic bytes: the [V][d] int8 weights, the fp32
    scales and biases, the int8 input row and the 8-byte key."""
    V, d = cfg.vocab, cfg.d_model
    W = torch.from_numpy(synth.uniform_int8(3, "W", (V, d))).cuda()
    s_w = torch.from_numpy(synth.uniform_f32(3, "s", (V,), 1e-4, 2e-4)).cuda()
    b = torch.from_numpy(synth.uniform_f32(3, "b", (V,), -0.1, 0.1)).cuda()
    A = torch.from_numpy(synth.uniform_int8(3, "A", (1, d))).cuda()
    keys = torch.zeros(1, dtype=torch.int64, device="cuda")
    algo_bytes = V * d + V * 8 + d + 8
    ms = []
    for i in range(n_launch + 3):
        with torch.cuda.stream(stream):
            flush.fill_(i & 0xFF)
            keys.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
        mnmt.mnmt_linear_argmax(A, W, s_w, b, 0.01, 1, V, d, keys, stream)
        with torch.cuda.stream(stream):
            e1.record(stream)
        if i >= 3:
            ms.append((e0, e1))
    stream.synchronize()
    avg_ms = sum(a.elapsed_time(b2) for a, b2 in ms) / len(ms)
    peak, kind = _peaks()
    achieved = algo_bytes / (avg_ms * 1e-3) / 1e9
    return {"kernel": "linear_smallm<1,16,2> (vocab projection + argmax, M=1 N=%d K=%d)" % (V, d),
            "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
            "peak_kind": f"{kind} hbm_gbs (burst, kernel timed alone)", "traffic": None,
            "algorithmic_bytes": algo_bytes, "avg_us": avg_ms * 1e3, "launches": len(ms)}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mnmt", choices=["mnmt", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
