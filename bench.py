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
  batched   the batched half of the metric on the two batched-beam workloads
            (12+2-layer d=256 model, batch 32 x beam 4; 6+6-layer d=512 model,
            batch 128 x beam 4): tokens/s (device-resident and end to end),
            decode-step p50/p90, encode time, the encoder's operations per
            second as a fraction of the measured dense fp16/bf16 tensor peak
            (the exact int8 route: int8 codes carried as fp16, see the
            tensor-core linear), and the decode step's fraction of HBM
  w4        the batch-1 workload with row-wise 4-bit attention / FFN weights
            (symmetric, and min-max scale + offset), 8-bit embedding
  paper_models  the paper's MobileNMT-10MB / -20MB shapes at its measurement
            setting (src/tgt 30, batch 1, greedy): latency per translation and
            the library's device memory, default and memory-minimal (lean)
  microbench  the int8 linear sweep M in {1..4096} x five (K, N) shapes and
            the wide encoder's linears, each with TOPS and GB/s and its
            fraction of the bounding peak, plus incremental attention over
            caches of 1..512 keys (GB/s)

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


def _tensor_peak():
    """Dense fp16/bf16 tensor peak (TFLOP/s): the measured burst figure, else the fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def _source_hash(files):
    import hashlib
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2306_04235_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


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


def decode_step_bytes(cfg, R, B, S, t, wq=8):
    """Algorithmic bytes one decode step must move for R hypotheses of B
    sentences (padded source length S) at step t: every decoder weight (int8),
    its per-output-channel scale and bias (fp32) and the requantisation
    constants of its int8 outputs, the LayerNorm vectors, the factorised
    projection, the vocabulary matrix with its scales and biases, the embedding
    rows and the positional row, and the K/V caches read (self [t+1] positions
    per hypothesis, cross [S] per sentence)."""
    d, F, V, E, L = cfg.d_model, cfg.d_ffn, cfg.vocab, cfg.d_embed, cfg.n_dec
    w = L * (6 * d * d + 2 * F * d)
    if wq != 8:  # 4-bit attention / FFN codes (+ a row offset per output row in the min-max form)
        w = w // 2 + (4 * L * (7 * d + F) if wq & 0x100 else 0)
    rows = L * (6 * d + F)
    inv = L * (4 * d + F)
    ln = (3 * L + (1 if cfg.pre_ln else 0)) * 2 * d * 4
    proj = (E * d + 8 * d) if E != d else 0
    vocab = V * d + 8 * V
    emb = R * (E + 4) + d * 4
    kv = 2 * L * R * (t + 1) * d + 2 * L * B * S * d
    return w + 8 * rows + 4 * inv + ln + proj + vocab + emb + kv


def encoder_ops(cfg, B, S):
    """Operations (2 per multiply-add) of one encode of B sentences padded to S:
    the factorised embedding projection, every encoder layer's QKV, W_o, FFN1,
    FFN2 linears and its attention (Q K^T and P V over S keys per query row),
    and every decoder layer's cross key/value projection."""
    d, F, E, M = cfg.d_model, cfg.d_ffn, cfg.d_embed, B * S
    ops = 2 * M * d * E if E != d else 0
    ops += cfg.n_enc * (2 * M * (4 * d * d + 2 * d * F) + 4 * B * S * S * d)
    ops += cfg.n_dec * 2 * M * 2 * d * d
    return ops


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


class Workload:
    """One workload's model, session, device buffers and pinned host buffers."""

    def __init__(self, name, mnmt, torch, stream, rank, lean=False, wq=8):
        self.wl = synth.WORKLOADS[name]
        self.cfg = synth.MODELS[self.wl.model]
        self.wq = wq
        self.blob = synth.build_blob(self.cfg, self.wl.model_seed, wq=wq)
        # every rank translates its own replica batch (independent sentences)
        self.ids, self.lens = synth.source_batch(self.cfg.vocab, self.wl.batch, self.wl.src_len[0],
                                                 self.wl.src_len[1], replica_source_seed(self.wl.src_seed, rank))
        self.B, self.S = self.ids.shape
        self.T = self.wl.max_len
        self.mnmt, self.torch, self.stream = mnmt, torch, stream
        self.tr = mnmt.Translator(self.blob, self.B, self.S, self.wl.beam, self.T, stream, lean=lean)
        self.model_bytes = mnmt.mnmt_model_device_bytes(self.tr.model)
        self.session_bytes = mnmt.mnmt_session_device_bytes(self.tr.session)
        self.sess = self.tr.session
        dev = "cuda"
        self.d_ids = torch.from_numpy(self.ids).to(dev)
        self.d_lens = torch.from_numpy(self.lens).to(dev)
        self.o_ids = torch.zeros((self.B, self.T), dtype=torch.int32, device=dev)
        self.o_len = torch.zeros(self.B, dtype=torch.int32, device=dev)
        self.o_sc = torch.zeros(self.B, dtype=torch.float32, device=dev)
        torch.cuda.synchronize()

    def translate(self):
        self.mnmt.mnmt_translate(self.sess, self.d_ids, self.d_lens, self.B, self.S, self.T,
                                 self.mnmt.DEVICE_PTRS, self.o_ids, self.o_len, self.o_sc)

    def close(self):
        self.tr.close()


def _event(torch):
    return torch.cuda.Event(enable_timing=True)


def time_translations(w, flush, steps, warmup, dist=None):
    """`steps` translations timed one by one with CUDA events on the library's
    stream, L2 flushed (outside the events) before each."""
    torch, stream = w.torch, w.stream
    for _ in range(warmup):
        with torch.cuda.stream(stream):
            flush.fill_(1)
        w.translate()
    stream.synchronize()
    evs = [(_event(torch), _event(torch)) for _ in range(steps)]
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    for i in range(steps):
        with torch.cuda.stream(stream):
            flush.fill_(i & 0xFF)
            evs[i][0].record(stream)
        w.translate()
        with torch.cuda.stream(stream):
            evs[i][1].record(stream)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    return [a.elapsed_time(b) for a, b in evs]


def time_encode(w, flush, n=5):
    torch, stream, mnmt = w.torch, w.stream, w.mnmt
    out = []
    for i in range(n):
        e0, e1 = _event(torch), _event(torch)
        with torch.cuda.stream(stream):
            flush.fill_(i & 0xFF)
            e0.record(stream)
        mnmt.mnmt_encode(w.sess, w.d_ids, w.d_lens, w.B, w.S, mnmt.DEVICE_PTRS)
        with torch.cuda.stream(stream):
            e1.record(stream)
        stream.synchronize()
        out.append(e0.elapsed_time(e1))
    return statistics.median(out)


def time_e2e(w, flush, steps, warmup, world):
    """The same translation through the C ABI with pinned host buffers: the
    host->device copy of the sources and the device->host copy of the outputs
    are inside the timed region."""
    torch, stream, mnmt = w.torch, w.stream, w.mnmt
    h_ids = torch.from_numpy(w.ids).pin_memory()
    h_lens = torch.from_numpy(w.lens).pin_memory()
    h_out = torch.zeros((w.B, w.T), dtype=torch.int32).pin_memory()
    h_olen = torch.zeros(w.B, dtype=torch.int32).pin_memory()
    h_osc = torch.zeros(w.B, dtype=torch.float32).pin_memory()
    times = []
    for i in range(warmup + steps):
        with torch.cuda.stream(stream):
            flush.fill_(i & 0xFF)
        stream.synchronize()
        t0 = time.perf_counter()
        mnmt.mnmt_translate(w.sess, h_ids.data_ptr(), h_lens.data_ptr(), w.B, w.S, w.T, 0, h_out.data_ptr(),
                            h_olen.data_ptr(), h_osc.data_ptr())
        if i >= warmup:
            times.append(time.perf_counter() - t0)
    toks = int(h_olen.sum().item())
    assert torch.equal(h_out, w.o_ids.cpu()), "host and device paths disagree"
    return {"value": toks * world * len(times) / sum(times), "unit": "tokens/s",
            "h2d_bytes_per_step": int(w.ids.nbytes + w.lens.nbytes),
            "d2h_bytes_per_step": int(w.B * w.T * 4 + w.B * 8)}


# DRAM bytes of one decode step (dram__bytes_read.sum + dram__bytes_write.sum of
# its kernels, from single-kernel ncu captures of this bench's command), with
# the hash of the step kernels' sources they were taken on: a stale figure
# (sources changed since) is reported as null
STEP_TRAFFIC = {("small-b1-s10to50-greedy64", True): (10_612_800, "e65a24b18aefa0af")}
STEP_SOURCES = ["decode_cluster.cu", "common.cuh", "mbarrier.cuh", "internal.h"]


def measure_decode_step(w, flush, steps_run, cluster):
    """Decode steps of one encoded batch timed with CUDA events on the
    library's stream: one step per event pair with L2 flushed before each
    (cold: the weights come from HBM, as the roofline assumes), then the same
    number of steps back to back (warm: the weights stay in the 129 MB L2)."""
    torch, stream, mnmt, cfg, wl = w.torch, w.stream, w.mnmt, w.cfg, w.wl
    R = w.B * wl.beam
    n = max(1, min(steps_run, wl.max_len))
    mnmt.mnmt_encode(w.sess, w.d_ids, w.d_lens, w.B, w.S, mnmt.DEVICE_PTRS)
    cold = []
    for t in range(n):
        with torch.cuda.stream(stream):
            flush.fill_(t & 0xFF)
            e0, e1 = _event(torch), _event(torch)
            e0.record(stream)
        mnmt.mnmt_decode_steps(w.sess, 1)
        with torch.cuda.stream(stream):
            e1.record(stream)
        cold.append((e0, e1))
    mnmt.mnmt_encode(w.sess, w.d_ids, w.d_lens, w.B, w.S, mnmt.DEVICE_PTRS)
    with torch.cuda.stream(stream):
        w0, w1 = _event(torch), _event(torch)
        w0.record(stream)
    mnmt.mnmt_decode_steps(w.sess, n)
    with torch.cuda.stream(stream):
        w1.record(stream)
    stream.synchronize()
    cold_us = [a.elapsed_time(b) * 1e3 for a, b in cold]
    avg_us = sum(cold_us) / len(cold_us)
    warm_us = w0.elapsed_time(w1) * 1e3 / n
    algo = sum(decode_step_bytes(cfg, R, w.B, w.S, t, w.wq) for t in range(n)) / n
    peak, kind = _peaks()
    achieved = algo / (avg_us * 1e-6) / 1e9
    unit = ("decode_cluster_kernel + vocab_greedy_kernel (one graph launch)" if cluster
            else "multi-kernel decode step (one graph launch)")
    traffic, stamp = STEP_TRAFFIC.get((wl.name, cluster), (None, None))
    if traffic is not None and stamp != _source_hash(STEP_SOURCES):
        traffic = None
    srt = sorted(cold_us)
    return {"kernel": f"decode step: {unit}, R={R} rows, S={w.S}", "bound": "hbm", "achieved": achieved,
            "peak": peak, "unit": "GB/s", "frac": achieved / peak, "peak_kind": f"{kind} hbm_gbs (burst)",
            "traffic": traffic, "algorithmic_bytes": int(algo), "avg_us": avg_us,
            "p50_us": srt[len(srt) // 2], "warm_avg_us": warm_us, "launches": len(cold_us)}


def replica_source_seed(src_seed, rank):
    """Seed of the source batch rank `rank` translates (replicas: independent
    sentences on every rank)."""
    return src_seed + 101 * rank


def aggregate_ranks(total_ms, toks_per_step, steps, dist=None, device="cuda"):
    """Whole-job throughput of N replicas: every rank's tokens (SUM) over the
    slowest rank's time (MAX).  Returns (tokens/s, time in ms, job tokens per
    step)."""
    import torch

    job_toks = float(toks_per_step)
    if dist:
        t = torch.tensor([float(total_ms)], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
        nt = torch.tensor([job_toks], dtype=torch.float64, device=device)
        dist.all_reduce(nt, op=dist.ReduceOp.SUM)
        job_toks = float(nt.item())
    return job_toks * steps / (total_ms / 1e3), total_ms, job_toks


def measure_workload(name, mnmt, torch, stream, flush, steps, warmup, rank=0, world=1, dist=None, lean=False,
                     wq=8):
    """tokens/s (device-resident and end to end), decode-step latency, encode
    time and the decode step's roofline for one workload."""
    w = Workload(name, mnmt, torch, stream, rank, lean, wq)
    try:
        step_ms = time_translations(w, flush, steps, warmup, dist)
        toks_per_step = int(w.o_len.sum().item())
        value, total_ms, _ = aggregate_ranks(sum(step_ms), toks_per_step, steps, dist)
        enc_ms = time_encode(w, flush)
        # decode steps actually executed per translation (greedy stops when
        # every sentence has emitted EOS; the beam workloads run all T)
        steps_run = int(w.o_len.max().item()) if w.wl.beam == 1 else w.T
        step_us = sorted(1e3 * (t - enc_ms) / max(steps_run, 1) for t in step_ms)
        e2e = time_e2e(w, flush, steps, warmup, world)
        cluster = mnmt.mnmt_session_decode_path(w.sess) == 1
        roof = measure_decode_step(w, flush, steps_run, cluster)
        return {"w": w, "value": value, "total_ms": total_ms, "toks_per_step": toks_per_step,
                "steps_run": steps_run, "enc_ms": enc_ms, "step_us": step_us, "e2e": e2e,
                "roofline": roof, "cluster": cluster}
    finally:
        w.close()


def batched_entry(name, mnmt, torch, stream, flush, steps, warmup):
    r = measure_workload(name, mnmt, torch, stream, flush, steps, warmup)
    w = r["w"]
    peak_t, kind_t = _tensor_peak()
    ops = encoder_ops(w.cfg, w.B, w.S)
    enc_tops = ops / (r["enc_ms"] * 1e-3) / 1e12
    su = r["step_us"]
    roof = r["roofline"]
    return {
        "workload": name, "model": w.wl.model, "batch": w.B, "beam": w.wl.beam, "s_pad": w.S, "max_len": w.T,
        "tokens_per_translation": r["toks_per_step"], "translations_timed": steps,
        "value": r["value"], "unit": "tokens/s", "ms_per_translation": r["total_ms"] / steps,
        "e2e": r["e2e"],
        "decode_step_us_p50": su[len(su) // 2], "decode_step_us_p90": su[min(len(su) - 1, int(0.9 * len(su)))],
        "encode_ms_p50": r["enc_ms"],
        "encoder": {"bound": "tensor", "ops": ops, "achieved": enc_tops, "peak": peak_t, "unit": "TOPS",
                    "frac": enc_tops / peak_t,
                    "peak_kind": f"{kind_t} bf16_tflops (burst); int8 codes run as exact fp16 on tcgen05 "
                                 "kind::f16, which has no int8 kind on sm_103a"},
        "decode_step": {"bound": "hbm", "achieved": roof["achieved"], "peak": roof["peak"], "unit": "GB/s",
                        "frac": roof["frac"], "algorithmic_bytes": roof["algorithmic_bytes"],
                        "cold_avg_us": roof["avg_us"], "cold_p50_us": roof["p50_us"],
                        "warm_avg_us": roof["warm_avg_us"], "kernel": roof["kernel"]},
    }


# the paper's on-device figures for its two models (Google Pixel 4 ARM CPU,
# src/tgt length 30, batch 1, greedy): context, not a target
PAPER_PIXEL4 = {"mobilenmt10-b1-s30-greedy30": {"latency_ms": 27.3, "memory_mb": 14.9},
                "mobilenmt20-b1-s30-greedy30": {"latency_ms": 46.3, "memory_mb": 26.0}}


def paper_entry(name, mnmt, torch, stream, flush, steps, warmup):
    """One translation of the paper's measurement shape, default and lean:
    per-translation latency (encode + 30 greedy steps) and the library's
    device memory (model + session)."""
    out = {"workload": name, "paper_pixel4_context": PAPER_PIXEL4[name]}
    for lean in (False, True):
        r = measure_workload(name, mnmt, torch, stream, flush, steps, warmup, lean=lean)
        w = r["w"]
        su = r["step_us"]
        out["lean" if lean else "default"] = {
            "ms_per_translation": r["total_ms"] / steps, "value": r["value"], "unit": "tokens/s",
            "e2e": r["e2e"]["value"], "decode_step_us_p50": su[len(su) // 2], "encode_ms_p50": r["enc_ms"],
            "decode_path": "cluster" if r["cluster"] else "multi-kernel",
            "model_mb": w.model_bytes / 1e6, "session_mb": w.session_bytes / 1e6,
            "device_mb": (w.model_bytes + w.session_bytes) / 1e6}
    return out


def w4_entry(name, wq, mnmt, torch, stream, flush, steps, warmup):
    """The batch-1 workload's model with 4-bit attention / FFN weights."""
    r = measure_workload(name, mnmt, torch, stream, flush, steps, warmup, wq=wq)
    w = r["w"]
    su = r["step_us"]
    roof = r["roofline"]
    return {"workload": name, "weights": "4-bit symmetric rows" if wq == synth.WQ_INT4 else "4-bit min-max rows",
            "value": r["value"], "unit": "tokens/s", "e2e": r["e2e"]["value"],
            "decode_step_us_p50": su[len(su) // 2], "encode_ms_p50": r["enc_ms"],
            "decode_path": "cluster" if r["cluster"] else "multi-kernel",
            "model_mb": w.model_bytes / 1e6, "blob_mb": len(w.blob) / 1e6,
            "decode_step": {"bound": "hbm", "achieved": roof["achieved"], "peak": roof["peak"], "unit": "GB/s",
                            "frac": roof["frac"], "algorithmic_bytes": roof["algorithmic_bytes"],
                            "cold_avg_us": roof["avg_us"], "warm_avg_us": roof["warm_avg_us"]}}


SWEEP_M = [1, 4, 16, 64, 256, 1024, 4096]
SWEEP_KN = [(256, 1024), (1024, 256), (512, 2048), (2048, 512), (256, 32000)]
WIDE_ENCODER_LINEARS = [("qkv", 512, 1536), ("o", 512, 512), ("ffn1", 512, 2048), ("ffn2", 2048, 512)]


def _time_rotating(torch, stream, fns, reps):
    """Per-launch time (us) of `reps` launches cycling through fns (one per
    operand copy; the copies together exceed L2, so every launch reads its
    operands from HBM), captured into one CUDA graph so that host launch
    overhead is not timed; median of 3 replays timed with CUDA events."""
    for f in fns[: min(len(fns), 2)]:
        f()
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(reps):
            fns[i % len(fns)]()
    g.replay()
    stream.synchronize()
    out = []
    for _ in range(3):
        e0, e1 = _event(torch), _event(torch)
        with torch.cuda.stream(stream):
            e0.record(stream)
            g.replay()
            e1.record(stream)
        stream.synchronize()
        out.append(e0.elapsed_time(e1) * 1e3 / reps)
    del g
    return statistics.median(out)


L2_BYTES = 129 << 20


def microbench(mnmt, torch, stream, flush):
    """The int8 linear sweep (E1 epilogue: int8 output) on the kernel the
    translation path uses at each M (<= 16 rows: the int8 GEMV; more: the
    tcgen05 kernel over fp16 copies of the codes), the wide encoder's linears at
    M = 16384, and incremental attention.  Each shape's launches cycle through
    as many copies of its operands as it takes to exceed twice the L2 (inputs
    larger than L2), timed back to back with CUDA events."""
    peak_b, kind_b = _peaks()
    peak_t, kind_t = _tensor_peak()
    ridge = peak_t * 1e12 / (peak_b * 1e9)  # ops per byte where the bounds cross
    dev = "cuda"
    torch.manual_seed(5)
    Nmax = 32000
    s_w = torch.rand(Nmax, device=dev) * 2e-4 + 1e-4
    bias = torch.rand(Nmax, device=dev) - 0.5
    inv = torch.full((Nmax,), 50.0, device=dev)

    def lin_entry(M, K, N, label=None):
        small = M <= 16
        # bytes one launch reads from HBM (the tensor-core kernel reads the fp16 copies)
        per = (M * K + N * K) * (1 if small else 2) + M * N
        copies = max(1, min(1024, -(-2 * L2_BYTES // per)))
        bufs = []
        for _ in range(copies):
            A8 = torch.randint(-127, 128, (M * K,), dtype=torch.int8, device=dev)
            W8 = torch.randint(-127, 128, (N * K,), dtype=torch.int8, device=dev)
            out = torch.empty(M * N, dtype=torch.int8, device=dev)
            if small:
                bufs.append((A8, W8, out))
            else:
                A16 = torch.empty(M * K, dtype=torch.int16, device=dev)
                W16 = torch.empty(N * K, dtype=torch.int16, device=dev)
                mnmt.mnmt_codes_to_f16(A8, A16, A8.numel(), stream)
                mnmt.mnmt_codes_to_f16(W8, W16, W8.numel(), stream)
                bufs.append((A16, W16, out))
        stream.synchronize()
        if small:
            fns = [lambda b=b: mnmt.mnmt_linear(b[0], b[1], s_w, bias, 0.03, inv, 1.0, M, N, K, mnmt.EPI_Q8,
                                                b[2], None, stream) for b in bufs]
            kern = "linear_smallm (int8 dp4a GEMV)"
        else:
            fns = [lambda b=b: mnmt.mnmt_linear_tc(b[0], b[1], s_w, bias, 0.03, inv, 1.0, M, N, K, mnmt.EPI_Q8,
                                                   out_q=b[2], stream=stream) for b in bufs]
            kern = "linear_tc (tcgen05 kind::f16 on exact fp16 codes)"
        us = _time_rotating(torch, stream, fns, max(copies, 20))
        del bufs, fns
        ops = 2 * M * N * K
        byts = M * K + K * N + 8 * N + M * N
        tops = ops / (us * 1e-6) / 1e12
        gbs = byts / (us * 1e-6) / 1e9
        bound = "hbm" if ops / byts < ridge else "tensor"
        frac = gbs / peak_b if bound == "hbm" else tops / peak_t
        e = {"M": M, "K": K, "N": N, "us": round(us, 2), "TOPS": round(tops, 2), "GBps": round(gbs, 1),
             "bound": bound, "frac": round(frac, 4), "kernel": kern, "copies": copies}
        if label:
            e["layer"] = label
        return e

    sweep = [lin_entry(M, K, N) for (K, N) in SWEEP_KN for M in SWEEP_M]
    wide = [lin_entry(16384, K, N, lab) for lab, K, N in WIDE_ENCODER_LINEARS]

    attn = []
    for R, H, T in [(1, 4, 512), (128, 4, 512), (512, 8, 512)]:
        dh = 64
        for t in [1, 16, 64, 256, 512]:
            per = 2 * R * H * t * dh
            copies = max(1, min(1024, -(-2 * L2_BYTES // per)))
            bufs = []
            for _ in range(copies):
                # each copy holds only the first t positions of every (row, head) cache
                Kc = torch.randint(-127, 128, (R * H * t * dh,), dtype=torch.int8, device=dev)
                Vc = torch.randint(-127, 128, (R * H * t * dh,), dtype=torch.int8, device=dev)
                q = torch.randint(-127, 128, (R * H * dh,), dtype=torch.int8, device=dev)
                ctx = torch.empty(R * H * dh, dtype=torch.int8, device=dev)
                bufs.append((q, Kc, Vc, ctx))
            nk = torch.full((R,), t, dtype=torch.int32, device=dev)
            torch.cuda.synchronize()
            fns = [lambda b=b: mnmt.mnmt_attention_decode(b[0], b[1], b[2], nk, R, H, dh, t, 0.001, 0.9, b[3],
                                                          stream) for b in bufs]
            us = _time_rotating(torch, stream, fns, max(copies, 20))
            del bufs, fns
            byts = 2 * R * H * t * dh + 2 * R * H * dh + 4 * R
            gbs = byts / (us * 1e-6) / 1e9
            attn.append({"R": R, "H": H, "dh": dh, "cache": t, "us": round(us, 2), "GBps": round(gbs, 1),
                         "bound": "hbm", "frac": round(gbs / peak_b, 4), "copies": copies})
    return {"linear_sweep": sweep, "wide_encoder_linears_M16384": wide, "attention_decode": attn,
            "peaks": {"hbm_gbs": peak_b, "hbm_kind": kind_b, "tensor_tflops": peak_t, "tensor_kind": kind_t},
            "bytes": "int8 algorithmic bytes M*K + K*N + 8*N + M*N (the tensor-core kernel reads 2-byte "
                     "fp16 copies of the codes)",
            "l2": "operands of each shape rotated over copies totalling >= 2x L2 (129 MB); launches back to back "
                  "in one captured CUDA graph"}


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

    stream = torch.cuda.Stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    with ClockSampler(local) as clk:
        r = measure_workload(args.workload, mnmt, torch, stream, flush, args.steps, args.warmup, rank, world,
                             dist)
    w = r["w"]
    cfg, wl, B, S, T = w.cfg, w.wl, w.B, w.S, w.T
    step_us = r["step_us"]

    batched = micro = None
    if rank == 0 and world == 1 and not args.no_batched:
        with ClockSampler(local) as bclk:
            batched = {"entries": [batched_entry(n, mnmt, torch, stream, flush, 5, 3) for n in BATCHED]}
        batched["clocks"] = bclk.summary()
    paper = w4 = None
    if rank == 0 and world == 1 and not args.no_batched:
        paper = [paper_entry(n, mnmt, torch, stream, flush, 10, 3) for n in PAPER_PIXEL4]
        w4 = [w4_entry(DEFAULT_WORKLOAD, q, mnmt, torch, stream, flush, 10, 3)
              for q in (synth.WQ_INT4, synth.WQ_INT4_MINMAX)]
    if rank == 0 and world == 1 and not args.no_micro:
        with ClockSampler(local) as mclk:
            micro = microbench(mnmt, torch, stream, flush)
        micro["clocks"] = mclk.summary()

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
        steps_run = r["steps_run"]
        # translate queues steps in chunks of 16 with one chunk of look-ahead:
        # a translation that finishes early has one more (no-op) chunk queued
        launched = T if steps_run >= T else min(T, -(-steps_run // 16) * 16 + 16)
        launches = kernels_per_translation(cfg, B, S, wl.beam, launched, r["cluster"]) * args.steps
        line = {
            "metric": METRIC, "value": r["value"], "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": r["total_ms"] / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
            "config": {"workload": args.workload, "model": wl.model, "batch": B, "beam": wl.beam,
                       "max_len": T, "src_len": list(wl.src_len), "s_pad": S,
                       "tokens_per_step": r["toks_per_step"],
                       "l2": "flushed between steps (256 MB write, outside the timed events)",
                       "decode_step_us_p50": step_us[len(step_us) // 2],
                       "decode_step_us_p90": step_us[min(len(step_us) - 1, int(0.9 * len(step_us)))],
                       "encode_ms_p50": r["enc_ms"], "parallelism": f"replicas x{world}"},
            "e2e": r["e2e"],
            "roofline": r["roofline"],
            "cpu_baseline": cpu,
            "clocks": clk.summary(),
            "gpu_launches": launches,
            "device_memory_mb": {"model": w.model_bytes / 1e6, "session": w.session_bytes / 1e6},
            "batched": batched,
            "paper_models": paper,
            "w4": w4,
            "microbench": micro,
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


BATCHED = ["small-b32-s10to80-beam4-t128", "wide-b128-s20to128-beam4-t160"]


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mnmt", choices=["mnmt", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-batched", action="store_true", help="skip the batched-beam workloads")
    ap.add_argument("--no-micro", action="store_true", help="skip the linear / attention sweep")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
