"""Float64 brute-force fake-quantised model: the pin the oracle is checked against.

TEST INFRASTRUCTURE.  A second, independently written reading of the same
model, in numpy float64 with library exp/log and plain softmax instead of the
oracle's fp32 / fixed-point arithmetic.  It quantises at exactly the points
Fig. 5 marks (inputs of every linear, Q/K/V, the attention context, the FFN
hidden layer; softmax, biases, residuals and LayerNorm in full precision), so
its int8 codes agree with the oracle's except where a value lies within
rounding distance of a .5 boundary, and its float outputs agree to ~1e-6.

It also parses the MNMT blob on its own (numpy views), sharing no code
with either the C oracle or the CUDA library.  Every linear is held as its
dequantised float64 weight matrix: s_n * code for int8 and symmetric 4-bit
rows (4-bit codes stored as v + 8), s_n * u + r_n for 4-bit min-max rows
(App. B Eq. quant).
"""
from __future__ import annotations

import math
import struct

import numpy as np


class Blob:
    """numpy views over an MNMT v1 blob."""

    def __init__(self, blob: bytes):
        self.buf = memoryview(blob)
        magic, ver, *cfg = struct.unpack_from("<4sI13i", blob, 0)
        assert magic == b"MNMT" and ver in (1, 2)
        (self.n_enc, self.n_dec, self.d, self.H, self.F, self.V, self.E, self.pre_ln,
         self.tied, self.max_pos, self.pad, self.bos, self.eos) = cfg
        self.wq = struct.unpack_from("<i", blob, 60)[0] if ver == 2 else 8
        assert self.wq in (8, 4, 4 | 0x100)
        self.off = 64
        d, F, V, E = self.d, self.F, self.V, self.E
        self.emb_q = self._arr(np.int8, (V, E))
        self.emb_s = self._arr(np.float32, (V,))
        self.proj = self._lin(d, E, 8) if E != d else None
        g = self._arr(np.float32, (4,))
        self.emb_scale, self.s_enc, self.s_dout = float(g[0]), float(g[1]), float(g[2])
        self.pe = self._arr(np.float32, (self.max_pos, d))
        self.enc = []
        for _ in range(self.n_enc):
            self.enc.append((self._self_attn(), self._ffn()))
        self.enc_final = self._ln() if self.pre_ln else None
        self.dec = []
        for _ in range(self.n_dec):
            self.dec.append((self._self_attn(), self._cross(), self._ffn()))
        self.dec_final = self._ln() if self.pre_ln else None
        if self.tied:
            self.out = self.emb_q.astype(np.float64) * self.emb_s.astype(np.float64)[:, None]
            self.out_b = self._arr(np.float32, (V,))
        else:
            self.out, self.out_b = self._lin(V, d, 8)
        assert self.off == len(blob), (self.off, len(blob))

    def _arr(self, dt, shape):
        n = int(np.prod(shape)) * np.dtype(dt).itemsize
        a = np.frombuffer(self.buf[self.off:self.off + n], dtype=dt).reshape(shape)
        self.off += n
        self.off = (self.off + 15) // 16 * 16
        return a

    def _lin(self, n, k, wq=None):
        """(dequantised weight float64 [n][k], bias [n]); wq: the format (the
        blob's for the attention / FFN linears, 8 for the embedding's)"""
        wq = self.wq if wq is None else wq
        if wq == 8:
            w = self._arr(np.int8, (n, k)).astype(np.float64)
            s_w = self._arr(np.float32, (n,)).astype(np.float64)
            return w * s_w[:, None], self._arr(np.float32, (n,))
        packed = self._arr(np.uint8, (n, k // 2)).reshape(n, k // 32, 16)
        codes = np.concatenate([packed & 15, packed >> 4], axis=2).reshape(n, k).astype(np.float64)
        s_w = self._arr(np.float32, (n,)).astype(np.float64)
        if wq == 4:
            return (codes - 8.0) * s_w[:, None], self._arr(np.float32, (n,))
        r = self._arr(np.float32, (n,)).astype(np.float64)
        return codes * s_w[:, None] + r[:, None], self._arr(np.float32, (n,))

    def _ln(self):
        return (self._arr(np.float32, (self.d,)), self._arr(np.float32, (self.d,)))

    def _self_attn(self):
        ln = self._ln()
        s = self._arr(np.float32, (8,))
        return dict(ln=ln, s_in=s[0], s_q=s[1], s_k=s[2], s_v=s[3], s_ctx=s[4], gamma=s[5],
                    qkv=self._lin(3 * self.d, self.d), o=self._lin(self.d, self.d))

    def _cross(self):
        ln = self._ln()
        s = self._arr(np.float32, (8,))
        return dict(ln=ln, s_in=s[0], s_q=s[1], s_k=s[2], s_v=s[3], s_ctx=s[4], gamma=s[5],
                    q=self._lin(self.d, self.d), kv=self._lin(2 * self.d, self.d),
                    o=self._lin(self.d, self.d))

    def _ffn(self):
        ln = self._ln()
        s = self._arr(np.float32, (4,))
        return dict(ln=ln, s_in=s[0], s_h=s[1], gamma=s[2], w1=self._lin(self.F, self.d),
                    w2=self._lin(self.d, self.F))


def quant(x, s):
    """Codes of x at scale s: round half to even, clamp to [-127, 127]."""
    return np.clip(np.rint(np.asarray(x, np.float64) / float(s)), -127, 127)


def linear(codes, s_x, lin):
    w, b = lin
    return (codes * float(s_x)) @ w.T + b


def layernorm(x, ln, eps=1e-5):
    g, b = ln
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


def attention(qc, kc, vc, s_q, s_k, s_v, s_ctx, mask):
    """qc [n][dh], kc/vc [m][dh] codes; mask [n][m] bool (True = visible)."""
    dh = qc.shape[-1]
    sc = (qc @ kc.T) * (float(s_q) * float(s_k) / math.sqrt(dh))
    sc = np.where(mask, sc, -np.inf)
    sc = sc - sc.max(axis=-1, keepdims=True)
    p = np.exp(sc)
    p = p / p.sum(axis=-1, keepdims=True)
    ctx = (p @ vc) * float(s_v)
    return quant(ctx, s_ctx)


class Model:
    def __init__(self, blob: bytes):
        self.b = Blob(blob)

    def embed(self, ids, pos):
        b = self.b
        rows = b.emb_q[ids].astype(np.float64)
        if b.proj is None:
            x = rows * b.emb_s[ids].astype(np.float64)[:, None]
        else:
            w, bias = b.proj
            x = (rows * b.emb_s[ids].astype(np.float64)[:, None]) @ w.T + bias
        return x * b.emb_scale + b.pe[pos].astype(np.float64)

    def _sub_in(self, r, blk):
        x = layernorm(r, blk["ln"]) if self.b.pre_ln else r
        return quant(x, blk["s_in"])

    def _sub_out(self, r, blk):
        return r if self.b.pre_ln else layernorm(r, blk["ln"])

    def _self_block(self, r, blk, mask):
        d, H = self.b.d, self.b.H
        dh = d // H
        a = self._sub_in(r, blk)
        y = linear(a, blk["s_in"], blk["qkv"])
        q = quant(y[:, :d], blk["s_q"]); k = quant(y[:, d:2 * d], blk["s_k"])
        v = quant(y[:, 2 * d:], blk["s_v"])
        ctx = np.zeros_like(q)
        for h in range(H):
            sl = slice(h * dh, (h + 1) * dh)
            ctx[:, sl] = attention(q[:, sl], k[:, sl], v[:, sl], blk["s_q"], blk["s_k"], blk["s_v"],
                                   blk["s_ctx"], mask)
        y = linear(ctx, blk["s_ctx"], blk["o"])
        return self._sub_out(blk["gamma"] * r + y, blk), (k, v)

    def _ffn_block(self, r, blk):
        a = self._sub_in(r, blk)
        h = quant(np.maximum(linear(a, blk["s_in"], blk["w1"]), 0.0), blk["s_h"])
        y = linear(h, blk["s_h"], blk["w2"])
        return self._sub_out(blk["gamma"] * r + y, blk)

    def encode(self, src, length):
        """Returns (enc codes [S][d], cross K codes [L][S][d], cross V codes [L][S][d])."""
        b = self.b
        S = len(src)
        r = self.embed(np.asarray(src), np.arange(S))
        mask = np.broadcast_to(np.arange(S)[None, :] < length, (S, S))
        for att, ffn in b.enc:
            r, _ = self._self_block(r, att, mask)
            r = self._ffn_block(r, ffn)
        x = layernorm(r, b.enc_final) if b.pre_ln else r
        enc = quant(x, b.s_enc)
        ck, cv = [], []
        for _, cross, _ in b.dec:
            y = linear(enc, b.s_enc, cross["kv"])
            ck.append(quant(y[:, :b.d], cross["s_k"]))
            cv.append(quant(y[:, b.d:], cross["s_v"]))
        return enc, np.stack(ck), np.stack(cv)

    def decode_forced(self, src, length, tgt):
        """Teacher-forced logits [T][V] for target prefix tgt (tgt[0] normally BOS)."""
        b = self.b
        d, H = b.d, b.H
        dh = d // H
        _, ck, cv = self.encode(src, length)
        T = len(tgt)
        r = self.embed(np.asarray(tgt), np.arange(T))
        causal = np.arange(T)[None, :] <= np.arange(T)[:, None]
        src_mask = np.broadcast_to(np.arange(len(src))[None, :] < length, (T, len(src)))
        for l, (att, cross, ffn) in enumerate(b.dec):
            r, _ = self._self_block(r, att, causal)
            a = self._sub_in(r, cross)
            q = quant(linear(a, cross["s_in"], cross["q"]), cross["s_q"])
            ctx = np.zeros_like(q)
            for h in range(H):
                sl = slice(h * dh, (h + 1) * dh)
                ctx[:, sl] = attention(q[:, sl], ck[l][:, sl], cv[l][:, sl], cross["s_q"],
                                       cross["s_k"], cross["s_v"], cross["s_ctx"], src_mask)
            y = linear(ctx, cross["s_ctx"], cross["o"])
            r = self._sub_out(cross["gamma"] * r + y, cross)
            r = self._ffn_block(r, ffn)
        x = layernorm(r, b.dec_final) if b.pre_ln else r
        a = quant(x, b.s_dout)
        return (a * b.s_dout) @ b.out.T + b.out_b
