"""Seeded synthetic inputs for the INT8 encoder-decoder translation path.

This module is the ONLY code shared by the CUDA library's callers and the CPU
oracle's tests.  It produces data — int8 weight codes with their fp32 scales,
fp32 biases / LayerNorm parameters / positional table, per-point activation
scales, and source-token batches — and holds none of the inference arithmetic
(no linear layer, attention, LayerNorm, softmax or decoding step lives here).

Everything is drawn from a counter-based splitmix64 stream and shaped with
integer ops and IEEE +,-,*,/,sqrt only, so the same seed gives the same bytes
on x86 and on Arm.  Gaussian draws use the Irwin-Hall sum of four uniforms
scaled to unit variance (bounded at +-3.46 sigma), which is close enough to
N(0, 1) for synthetic weights.

The model blob layout written by :func:`build_blob` is the "MNMT v1" format
documented in ``include/mnmt.h``.
"""
from __future__ import annotations

import dataclasses
import math
import struct

import numpy as np

MASK64 = (1 << 64) - 1
_GOLDEN = 0x9E3779B97F4A7C15

PAD_ID, BOS_ID, EOS_ID = 0, 1, 2


# --------------------------------------------------------------------------
# counter-based random numbers
# --------------------------------------------------------------------------
def _mix64(z: np.ndarray) -> np.ndarray:
    """splitmix64 finaliser on a uint64 array (Steele, Lea, Flood 2014)."""
    z = z.copy()
    z ^= z >> np.uint64(30)
    z *= np.uint64(0xBF58476D1CE4E5B9)
    z ^= z >> np.uint64(27)
    z *= np.uint64(0x94D049BB133111EB)
    z ^= z >> np.uint64(31)
    return z


class Stream:
    """A splitmix64 counter stream keyed by (seed, name)."""

    def __init__(self, seed: int, name: str):
        h = 1469598103934665603  # FNV-1a over the name, then fold in the seed
        for ch in name.encode():
            h = ((h ^ ch) * 1099511628211) & MASK64
        key = (h ^ ((seed * _GOLDEN) & MASK64)) & MASK64
        self.key = int(_mix64(np.array([key], dtype=np.uint64))[0])
        self.ctr = 0

    def u64(self, n: int) -> np.ndarray:
        with np.errstate(over="ignore"):
            idx = np.arange(self.ctr + 1, self.ctr + 1 + n, dtype=np.uint64)
            x = np.uint64(self.key) + idx * np.uint64(_GOLDEN)
            out = _mix64(x)
        self.ctr += n
        return out

    def uniform(self, n: int) -> np.ndarray:
        """Uniform doubles in [0, 1) with 53 random bits."""
        return (self.u64(n) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)

    def normal(self, n: int) -> np.ndarray:
        """Approximate N(0, 1): Irwin-Hall sum of four 16-bit uniforms (one 64-bit
        draw per value), centred and scaled to unit variance."""
        out = np.empty(n, dtype=np.float64)
        chunk = 1 << 14  # small chunks stay in the allocator's heap (no fresh page faults)
        for lo in range(0, n, chunk):
            m = min(chunk, n - lo)
            z = self.u64(m)
            s = np.zeros(m, dtype=np.float64)
            for sh in (0, 16, 32, 48):
                s += ((z >> np.uint64(sh)) & np.uint64(0xFFFF)).astype(np.float64)
            # each field is uniform on {0..65535}; (f + 0.5) / 65536 is uniform in (0, 1)
            out[lo:lo + m] = ((s + 2.0) * (1.0 / 65536.0) - 2.0) * math.sqrt(3.0)
        return out

    def randint(self, lo: int, hi: int, n: int) -> np.ndarray:
        """Integers uniform in [lo, hi] (inclusive), by multiply-shift on 32 bits."""
        span = hi - lo + 1
        r = (self.u64(n) >> np.uint64(32)) * np.uint64(span)
        return (r >> np.uint64(32)).astype(np.int64) + lo


# --------------------------------------------------------------------------
# model and workload descriptions
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class ModelConfig:
    n_enc: int
    n_dec: int
    d_model: int
    n_heads: int
    d_ffn: int
    vocab: int
    d_embed: int
    pre_ln: int
    tied_output: int
    max_pos: int = 512
    pad_id: int = PAD_ID
    bos_id: int = BOS_ID
    eos_id: int = EOS_ID

    def as_ints(self):
        return [self.n_enc, self.n_dec, self.d_model, self.n_heads, self.d_ffn,
                self.vocab, self.d_embed, self.pre_ln, self.tied_output,
                self.max_pos, self.pad_id, self.bos_id, self.eos_id]


MODELS = {
    # 2+1 layers, d=128, post-LN, tied 8000-entry shared vocabulary
    "tiny-2x1-d128-v8k": ModelConfig(2, 1, 128, 4, 512, 8000, 128, 0, 1),
    # deep encoder / shallow decoder, factorised 128-dim embedding, untied output
    "small-12x2-d256-v32k-e128": ModelConfig(12, 2, 256, 4, 1024, 32000, 128, 1, 0),
    # 6+6 layers, d=512, tied 32000-entry vocabulary
    "wide-6x6-d512-v32k": ModelConfig(6, 6, 512, 8, 2048, 32000, 512, 1, 1),
    # the paper's two models (Table "detailed settings of MobileNMT"): 12+2
    # layers, a shared 8000-entry vocabulary tied to the output, no embedding
    # factorisation, pre-LN; 10MB: d=256, 4 heads, FFN 512; 20MB: d=384,
    # 6 heads, FFN 768
    "mobilenmt-10mb": ModelConfig(12, 2, 256, 4, 512, 8000, 256, 1, 1),
    "mobilenmt-20mb": ModelConfig(12, 2, 384, 6, 768, 8000, 384, 1, 1),
}


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    model: str
    model_seed: int
    batch: int
    src_len: tuple
    beam: int
    max_len: int
    src_seed: int


WORKLOADS = {
    w.name: w for w in [
        Workload("tiny-b1-s16-greedy16", "tiny-2x1-d128-v8k", 0, 1, (16, 16), 1, 16, 1000),
        Workload("small-b1-s10to50-greedy64", "small-12x2-d256-v32k-e128", 1, 1, (10, 50), 1, 64, 1001),
        Workload("small-b32-s10to80-beam4-t128", "small-12x2-d256-v32k-e128", 1, 32, (10, 80), 4, 128, 1002),
        Workload("wide-b128-s20to128-beam4-t160", "wide-6x6-d512-v32k", 4, 128, (20, 128), 4, 160, 1004),
        # the paper's own measurement shape: one sentence, source and target length 30
        Workload("small-b1-s30-greedy30", "small-12x2-d256-v32k-e128", 1, 1, (30, 30), 1, 30, 1005),
        # the paper's models at its measurement shape (src/tgt 30, batch 1, greedy)
        Workload("mobilenmt10-b1-s30-greedy30", "mobilenmt-10mb", 10, 1, (30, 30), 1, 30, 1010),
        Workload("mobilenmt20-b1-s30-greedy30", "mobilenmt-20mb", 20, 1, (30, 30), 1, 30, 1020),
    ]
}


# --------------------------------------------------------------------------
# weights
# --------------------------------------------------------------------------
def _f32(x: float) -> float:
    return struct.unpack("<f", struct.pack("<f", float(x)))[0]


# weight formats of the linears (the blob header's wq field): int8 symmetric
# per row, int4 symmetric per row, int4 min-max (scale and offset) per row
WQ_INT8, WQ_INT4, WQ_INT4_MINMAX = 8, 4, 4 | 0x100


def weight_draw(st: Stream, n: int, k: int, std: float = 0.02) -> np.ndarray:
    """The float64 N(0, std) [n][k] matrix a quantised weight is made from."""
    return st.normal(n * k).reshape(n, k) * std


def int4_weight(w: np.ndarray, minmax: bool):
    """Per-row 4-bit codes of a float matrix (row-wise low-bit quantisation):
    symmetric: s = fl32(max|w|/7), v = clip(rint(w/s), -7, 7), stored as v + 8;
    min-max: r = fl32(min w), s = fl32((max w - r)/15), u = clip(rint((w - r)/s), 0, 15).
    Returns (stored codes uint8 [n][k] in 0..15, s f32 [n], r f32 [n] or None)."""
    if not minmax:
        amax = np.abs(w).max(axis=1)
        s = np.where(amax > 0, amax / 7.0, 1.0).astype(np.float32)
        v = np.clip(np.rint(w / s.astype(np.float64)[:, None]), -7, 7)
        return (v + 8).astype(np.uint8), s, None
    r = w.min(axis=1).astype(np.float32)
    span = w.max(axis=1) - r.astype(np.float64)
    s = np.where(span > 0, span / 15.0, 1.0).astype(np.float32)
    s = np.where(s > 0, s, np.float32(1.0)).astype(np.float32)
    u = np.clip(np.rint((w - r.astype(np.float64)[:, None]) / s.astype(np.float64)[:, None]), 0, 15)
    return u.astype(np.uint8), s, r


def pack4(codes: np.ndarray) -> np.ndarray:
    """Pack 4-bit codes [n][k] (k a multiple of 32) two per byte: each run of 32
    codes fills 16 bytes, code j in the low nibble of byte j (j < 16) and code
    16 + j in its high nibble."""
    n, k = codes.shape
    c = codes.reshape(n, k // 32, 2, 16).astype(np.uint8)
    return np.ascontiguousarray((c[:, :, 0, :] | (c[:, :, 1, :] << 4)).reshape(n, k // 2))


def int8_weight(st: Stream, n: int, k: int, std: float = 0.02):
    """Per-row symmetric int8 codes of an N(0, std) [n][k] matrix and the row scales.

    The codes are the row-absmax normalised rounding of the Gaussian draw, which
    is how a per-output-channel quantised checkpoint looks; they are data here.
    """
    w = weight_draw(st, n, k, std)
    amax = np.abs(w).max(axis=1)
    amax = np.where(amax > 0, amax, 1.0)
    s = (amax / 127.0).astype(np.float32)
    q = np.clip(np.rint(w / s.astype(np.float64)[:, None]), -127, 127).astype(np.int8)
    return q, s


def f32_normal(st: Stream, n: int, mean: float, std: float) -> np.ndarray:
    return (mean + std * st.normal(n)).astype(np.float32)


def sinusoid_table(max_pos: int, d: int) -> np.ndarray:
    """Sinusoidal positions in double, rounded once to fp32: even dims sin, odd cos."""
    pos = np.arange(max_pos, dtype=np.float64)[:, None]
    i = np.arange(d // 2, dtype=np.float64)[None, :]
    ang = pos / np.power(10000.0, (2.0 * i) / d)
    pe = np.empty((max_pos, d), dtype=np.float64)
    pe[:, 0::2] = np.sin(ang)
    pe[:, 1::2] = np.cos(ang)
    return pe.astype(np.float32)


def activation_scales(cfg: ModelConfig) -> dict:
    """Per-point activation scales set from the synthetic distributions.

    A LayerNorm output is ~N(0,1) (clip at 4); a linear output on such an input
    with N(0, 0.02) weights has std 0.02*sqrt(K) (clip at 4 std).  The first
    sublayer of a post-LN stack sees the raw embedding plus positions instead.
    """
    d = cfg.d_model
    c_ln = 4.0
    c_lin = 4.0 * 0.02 * math.sqrt(d)
    c_emb = 1.0 + 4.0 * 0.02 * math.sqrt(d)
    return {
        "ln": _f32(c_ln / 127.0),
        "lin": _f32(c_lin / 127.0),
        "emb": _f32(c_emb / 127.0),
    }


class _BlobWriter:
    def __init__(self):
        self.parts = []
        self.size = 0

    def put(self, arr: np.ndarray):
        b = np.ascontiguousarray(arr).tobytes()
        self.parts.append(b)
        self.size += len(b)
        pad = (-self.size) % 16
        if pad:
            self.parts.append(b"\0" * pad)
            self.size += pad

    def bytes(self) -> bytes:
        return b"".join(self.parts)


# Weight-std multipliers of the decoder's cross-attention projections.  With
# every weight drawn N(0, 0.02) the cross-attention scores are ~0.1 (a flat
# softmax) and its output is a small average of source values, so a random
# model decodes almost the same tokens whatever the source (with a tied output
# matrix it repeats its input token).  A translation model's output depends on
# its source through this sublayer, so the synthetic models sharpen it: the
# query and key projections are drawn with std 0.02*qk, the value projection
# 0.02*v, the output projection 0.02*o.  The activation scales of the points
# these weights feed follow the same multipliers.  With these values every
# workload model decodes a different token sequence for each of 8 random
# sources (at most 1 of 8 distinct without them).
CROSS_GAINS = {"qk": 10.0, "v": 3.0, "o": 40.0}
NO_GAINS = {"qk": 1.0, "v": 1.0, "o": 1.0}


def build_blob(cfg: ModelConfig, seed: int, gamma_range=None, out_bias=None, cross_gains=None,
               wq: int = WQ_INT8) -> bytes:
    """Write a seeded synthetic model in the MNMT v1 blob format.

    gamma_range: None for gamma_i = 1 on every sublayer, or (lo, hi) to draw each
    sublayer's residual weight uniformly.  out_bias: optional dict {token: value}
    added to the output bias (used to force e.g. immediate EOS).  cross_gains:
    the cross-attention weight-std multipliers (default CROSS_GAINS; NO_GAINS
    draws every weight N(0, 0.02)).  wq: the weight format of every linear
    (WQ_INT8; WQ_INT4 / WQ_INT4_MINMAX write a version-2 blob whose attention
    and FFN linears hold 4-bit codes; the embedding -- table, factorised
    projection, untied output projection -- stays int8).
    """
    assert wq in (WQ_INT8, WQ_INT4, WQ_INT4_MINMAX)
    d, F, V, E = cfg.d_model, cfg.d_ffn, cfg.vocab, cfg.d_embed
    sc = activation_scales(cfg)
    cg = dict(CROSS_GAINS if cross_gains is None else cross_gains)
    w = _BlobWriter()
    if wq == WQ_INT8:
        hdr = struct.pack("<4sI13i", b"MNMT", 1, *cfg.as_ints())
    else:
        hdr = struct.pack("<4sI13ii", b"MNMT", 2, *cfg.as_ints(), wq)
    hdr += b"\0" * (64 - len(hdr))
    w.parts.append(hdr)
    w.size = 64

    def gamma(st):
        if gamma_range is None:
            return 1.0
        lo, hi = gamma_range
        return _f32(lo + (hi - lo) * st.uniform(1)[0])

    def put_weight(st, n, k, std):
        """codes [+ row offsets] and row scales of one linear's weight, in blob order"""
        if wq == WQ_INT8:
            q, s_ = int8_weight(st, n, k, std)
            return [q, s_]
        u, s_, r = int4_weight(weight_draw(st, n, k, std), wq == WQ_INT4_MINMAX)
        return [pack4(u), s_] + ([r] if r is not None else [])

    def linear(name, n, k, std=0.02, embedding=False):
        st = Stream(seed, name)
        if embedding:  # part of the embedding: 8-bit in every format
            for arr in int8_weight(st, n, k, std):
                w.put(arr)
        else:
            for arr in put_weight(st, n, k, std):
                w.put(arr)
        w.put(f32_normal(Stream(seed, name + ".b"), n, 0.0, 0.02))

    def ln(name):
        w.put(f32_normal(Stream(seed, name + ".g"), d, 1.0, 0.02))
        w.put(f32_normal(Stream(seed, name + ".b"), d, 0.0, 0.02))

    def s_in_for(first_of_stack):
        if cfg.pre_ln:
            return sc["ln"]
        return sc["emb"] if first_of_stack else sc["ln"]

    def self_attn(prefix, first):
        ln(prefix + ".ln")
        g = gamma(Stream(seed, prefix + ".gamma"))
        w.put(np.array([s_in_for(first), sc["lin"], sc["lin"], sc["lin"], sc["lin"], g, 0, 0],
                       dtype=np.float32))
        linear(prefix + ".qkv", 3 * d, d)
        linear(prefix + ".o", d, d)

    def cross_attn(prefix):
        ln(prefix + ".ln")
        g = gamma(Stream(seed, prefix + ".gamma"))
        s_qk = _f32(sc["lin"] * cg["qk"])
        s_v = _f32(sc["lin"] * cg["v"])
        w.put(np.array([sc["ln"], s_qk, s_qk, s_v, s_v, g, 0, 0], dtype=np.float32))
        linear(prefix + ".q", d, d, 0.02 * cg["qk"])
        if cg["qk"] == cg["v"]:
            linear(prefix + ".kv", 2 * d, d, 0.02 * cg["qk"])
        else:  # key rows and value rows drawn with their own std, stored as one [2d][d] linear
            pk = put_weight(Stream(seed, prefix + ".kv"), d, d, 0.02 * cg["qk"])
            pv = put_weight(Stream(seed, prefix + ".kv.v"), d, d, 0.02 * cg["v"])
            for a_, b_ in zip(pk, pv):
                w.put(np.concatenate([a_, b_]))
            w.put(f32_normal(Stream(seed, prefix + ".kv.b"), 2 * d, 0.0, 0.02))
        linear(prefix + ".o", d, d, 0.02 * cg["o"])

    def ffn(prefix):
        ln(prefix + ".ln")
        g = gamma(Stream(seed, prefix + ".gamma"))
        w.put(np.array([sc["ln"], sc["lin"], g, 0], dtype=np.float32))
        linear(prefix + ".w1", F, d)
        linear(prefix + ".w2", d, F)

    eq, es = int8_weight(Stream(seed, "embed"), V, E)
    w.put(eq)
    w.put(es)
    if E != d:
        linear("embed.proj", d, E, embedding=True)
    # emb_scale = fl32(sqrt(d)); s_enc, s_dout: quant scales of the encoder
    # output (cross K/V input) and of the decoder output (vocab input)
    w.put(np.array([_f32(math.sqrt(d)), sc["ln"], sc["ln"], 0], dtype=np.float32))
    w.put(sinusoid_table(cfg.max_pos, d))
    for l in range(cfg.n_enc):
        self_attn(f"enc{l}.self", l == 0)
        ffn(f"enc{l}.ffn")
    if cfg.pre_ln:
        ln("enc.final")
    for l in range(cfg.n_dec):
        self_attn(f"dec{l}.self", l == 0)
        cross_attn(f"dec{l}.cross")
        ffn(f"dec{l}.ffn")
    if cfg.pre_ln:
        ln("dec.final")
    if not cfg.tied_output:  # the output embedding: 8-bit in every format
        oq, os_ = int8_weight(Stream(seed, "out"), V, d)
        w.put(oq)
        w.put(os_)
    ob = f32_normal(Stream(seed, "out.b"), V, 0.0, 0.02)
    if out_bias:
        for tok, val in out_bias.items():
            ob[tok] = np.float32(val)
    w.put(ob)
    return w.bytes()


# --------------------------------------------------------------------------
# source batches
# --------------------------------------------------------------------------
def source_batch(vocab: int, batch: int, len_lo: int, len_hi: int, seed: int):
    """Uniform token ids in [3, vocab) with lengths uniform in [len_lo, len_hi],
    right-padded with PAD to the batch maximum.  Returns (ids int32 [B][S_pad],
    lens int32 [B])."""
    st = Stream(seed, "src")
    lens = st.randint(len_lo, len_hi, batch).astype(np.int32)
    s_pad = int(lens.max())
    ids = st.randint(3, vocab - 1, batch * s_pad).astype(np.int32).reshape(batch, s_pad)
    mask = np.arange(s_pad)[None, :] < lens[:, None]
    ids = np.where(mask, ids, PAD_ID).astype(np.int32)
    return np.ascontiguousarray(ids), lens


def workload_inputs(name: str, batch: int | None = None):
    """(ModelConfig, blob bytes, src ids, src lens, beam, max_len) for a named workload."""
    wl = WORKLOADS[name]
    cfg = MODELS[wl.model]
    blob = build_blob(cfg, wl.model_seed)
    b = wl.batch if batch is None else batch
    ids, lens = source_batch(cfg.vocab, b, wl.src_len[0], wl.src_len[1], wl.src_seed)
    return cfg, blob, ids, lens, wl.beam, wl.max_len


def uniform_int8(seed: int, name: str, shape, lo: int = -127, hi: int = 127) -> np.ndarray:
    """Uniform int8 tensor (microbenchmark and kernel-parity inputs)."""
    n = int(np.prod(shape))
    return Stream(seed, name).randint(lo, hi, n).astype(np.int8).reshape(shape)


def uniform_f32(seed: int, name: str, shape, lo: float, hi: float) -> np.ndarray:
    n = int(np.prod(shape))
    u = Stream(seed, name).uniform(n)
    return (lo + (hi - lo) * u).astype(np.float32).reshape(shape)
