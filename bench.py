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
  roofline  the decode step, the unit that dominates the translation time (at
            batch 1 one graph launch of the thread-block-cluster step kernel
            plus the fused vocabulary projection + argmax kernel), timed with
            CUDA events on the library's stream one step at a time with L2
            flushed before each; algorithmic bytes = the weights, scales and
            biases every step must read plus its K/V cache reads
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


def kernels_per_translation(cfg, B, S, beam, steps_launched, cluster):
    """Kernels the library launches for one translation.  Encoder: embedding,
    7 per layer, cross K/V per decoder layer, plus one int8 -> fp16 operand
    copy before each linear of >= 128 rows (4 per layer and the cross K/V).
    Search init and final backtrack.  Per decode step: the cluster step (step
    kernel + vocabulary kernel), or embedding, 11 per layer, vocabulary
    projection, 1 greedy / 2 beam kernels (+ 6 per layer and 1 operand copies
    at >= 128 rows)."""
    tc_enc = B * S >= 128
    enc = 1 + 7 * cfg.n_enc + cfg.n_dec + (4 * cfg.n_enc + cfg.n_dec if tc_enc else 0)
    if cluster:
        step = 2
    else:
        tc_dec = B * beam >= 128
        step = 1 + 11 * cfg.n_dec + 1 + (1 if beam == 1 else 2) + (6 * cfg.n_dec + 1 if tc_dec else 0)
    return enc + 1 + step * steps_launched + 1


def decode_step_bytes(cfg, R, B, S, t):
    """Algorithmic bytes one decode step must move for R hypotheses of B
    sentences (padded source length S) at step t: every decoder weight (int8),
    its per-output-channel scale and bias (fp32) and the requantisation
    constants of its int8 outputs, the LayerNorm vectors, the factorised
    projection, the vocabulary matrix with its scales and biases, the embedding
    rows and the positional row, and the K/V caches read (self [t+1] positions
    per hypothesis, cross [S] per sentence)."""
    d, F, V, E, L = cfg.d_model, cfg.d_ffn, cfg.vocab, cfg.d_embed, cfg.n_dec
    w = L * (6 * d * d + 2 * F * d)
    rows = L * (6 * d + F)
    inv = L * (4 * d + F)
    ln = (3 * L + (1 if cfg.pre_ln else 0)) * 2 * d * 4
    proj = (E * d + 8 * d) if E != d else 0
    vocab = V * d + 8 * V
    emb = R * (E + 4) + d * 4
    kv = 2 * L * R * (t + 1) * d + 2 * L * B * S * d
    return w + 8 * rows + 4 * inv + ln + proj + vocab + emb + kv


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

    # the decode step, one at a time (cold L2) and back to back (warm)
    cluster = mnmt.mnmt_session_decode_path(sess) == 1
    roof = measure_decode_step(cfg, wl, mnmt, torch, stream, flush, sess, d_ids, d_lens, B, S, steps_run, cluster)

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
        # translate queues steps in chunks of 16 with one chunk of look-ahead:
        # a translation that finishes early has one more (no-op) chunk queued
        launched = T if steps_run >= T else min(T, -(-steps_run // 16) * 16 + 16)
        launches = kernels_per_translation(cfg, B, S, wl.beam, launched, cluster) * args.steps
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


# DRAM bytes of one decode step (dram__bytes_read.sum + dram__bytes_write.sum
# of its kernels, one ncu capture of this bench's command); only for the step
# kernels they were taken on -- refresh whenever those kernels change
STEP_TRAFFIC = {("small-b1-s10to50-greedy64", True): 10_582_950}


def measure_decode_step(cfg, wl, mnmt, torch, stream, flush, sess, d_ids, d_lens, B, S, steps_run, cluster):
    """Decode steps of one encoded batch timed with CUDA events on the
    library's stream: one step per event pair with L2 flushed before each
    (cold: the weights come from HBM, as the roofline assumes), then the same
    number of steps back to back (warm: the weights stay in the 129 MB L2)."""
    R = B * wl.beam
    n = max(1, min(steps_run, wl.max_len))
    mnmt.mnmt_encode(sess, d_ids, d_lens, B, S, mnmt.DEVICE_PTRS)
    cold = []
    for t in range(n):
        with torch.cuda.stream(stream):
            flush.fill_(t & 0xFF)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
        mnmt.mnmt_decode_steps(sess, 1)
        with torch.cuda.stream(stream):
            e1.record(stream)
        cold.append((e0, e1))
    mnmt.mnmt_encode(sess, d_ids, d_lens, B, S, mnmt.DEVICE_PTRS)
    with torch.cuda.stream(stream):
        w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0.record(stream)
    mnmt.mnmt_decode_steps(sess, n)
    with torch.cuda.stream(stream):
        w1.record(stream)
    stream.synchronize()
    cold_us = [a.elapsed_time(b) * 1e3 for a, b in cold]
    avg_us = sum(cold_us) / len(cold_us)
    warm_us = w0.elapsed_time(w1) * 1e3 / n
    algo = sum(decode_step_bytes(cfg, R, B, S, t) for t in range(n)) / n
    peak, kind = _peaks()
    achieved = algo / (avg_us * 1e-6) / 1e9
    unit = ("decode_cluster_kernel + vocab_greedy_kernel (one graph launch)" if cluster
            else "multi-kernel decode step (one graph launch)")
    return {"kernel": f"decode step: {unit}, R={R} rows, S={S}", "bound": "hbm", "achieved": achieved, "peak": peak,
            "unit": "GB/s", "frac": achieved / peak, "peak_kind": f"{kind} hbm_gbs (burst)",
            "traffic": STEP_TRAFFIC.get((wl.name, cluster)), "algorithmic_bytes": int(algo), "avg_us": avg_us, "warm_avg_us": warm_us,
            "launches": len(cold_us)}


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
