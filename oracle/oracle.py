"""ctypes front end of the CPU oracle (``mnmt_oracle.c``).

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference leg import this module.  Every function
here only marshals numpy arrays into the C oracle; no arithmetic of the method
is done in Python.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mnmt_oracle.c")
_OUT = os.path.join(_HERE, "_build", "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ENOMEM, EFORMAT, EOVERFLOW = 0, -1, -2, -5, -6


def build(force: bool = False) -> str:
    """Compile the oracle with -ffp-contract=off (part of its definition)."""
    os.makedirs(os.path.dirname(_OUT), exist_ok=True)
    if not force and os.path.exists(_OUT) and os.path.getmtime(_OUT) >= os.path.getmtime(_SRC):
        return _OUT
    tmp = _OUT + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-pthread", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _OUT)
    return _OUT


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = C.CDLL(build())
            _declare(_lib)
    return _lib


_p = C.c_void_p
_i = C.c_int
_f = C.c_float
_d = C.c_double
_sz = C.c_size_t


def _declare(L):
    L.oracle_check_blob.argtypes = [_p, _sz, _p]
    L.oracle_q8.argtypes = [_f, _f]; L.oracle_q8.restype = _f
    L.oracle_exp.argtypes = [_f]; L.oracle_exp.restype = _f
    L.oracle_log.argtypes = [_d]; L.oracle_log.restype = _d
    L.oracle_sigma.argtypes = [_f, _f, _i]; L.oracle_sigma.restype = _f
    L.oracle_gemm_i32.argtypes = [_p, _p, _i, _i, _i, _p]; L.oracle_gemm_i32.restype = None
    L.oracle_linear.argtypes = [_p, _p, _p, _p, _f, _p, _f, _i, _i, _i, _i, _p, _p]
    L.oracle_layernorm.argtypes = [_p, _p, _p, _i, _i, _f, _p, _p]
    L.oracle_attention_decode.argtypes = [_p, _p, _p, _p, _i, _i, _i, _i, _f, _f, _p]
    L.oracle_attention_probs.argtypes = [_p, _p, _i, _i, _f, _p]
    L.oracle_encode.argtypes = [_p, _sz, _p, _i, _i, _p, _p, _p]
    L.oracle_decode_trace.argtypes = [_p, _sz, _p, _i, _i, _p, _i, _p, _p, _p, _p]
    L.oracle_decode_forced.argtypes = [_p, _sz, _p, _i, _i, _p, _i, _p]
    L.oracle_embed.argtypes = [_p, _sz, _p, _p, _i, _p]
    L.oracle_log_softmax.argtypes = [_p, _i, _p]
    L.oracle_log_softmax_norm.argtypes = [_p, _i, _p, _p, _p]
    L.oracle_ln_stats.argtypes = [_p, _i, _i, _p, _p]
    L.oracle_quantise_rows.argtypes = [_p, _i, _i, _i, _i, _p, _p, _p]
    L.oracle_fake_quant.argtypes = [_p, _i, _f, _f, _i, _i, _p, _p]
    L.oracle_fake_quant_backward.argtypes = [_p, _p, _i, _f, _f, _i, _i, _p, _p, _p]
    L.oracle_fake_quant_linear.argtypes = [_p, _p, _f, _p, _p, _i, _i, _i, _i, _p]
    L.oracle_linear_w4.argtypes = [_p, _p, _p, _p, _p, _f, _p, _f, _i, _i, _i, _i, _i, _p, _p]
    L.oracle_translate.argtypes = [_p, _sz, _p, _p, _i, _i, _i, _i, _i, _p, _p, _p]
    for name in ["oracle_check_blob", "oracle_linear", "oracle_layernorm", "oracle_attention_decode",
                 "oracle_attention_probs", "oracle_encode", "oracle_decode_trace",
                 "oracle_decode_forced", "oracle_embed", "oracle_log_softmax", "oracle_log_softmax_norm", "oracle_ln_stats",
                 "oracle_quantise_rows", "oracle_linear_w4", "oracle_fake_quant",
                 "oracle_fake_quant_backward", "oracle_fake_quant_linear",
                 "oracle_translate"]:
        getattr(L, name).restype = _i


class OracleError(RuntimeError):
    pass


def _chk(st):
    if st != OK:
        raise OracleError(f"oracle returned {st}")


def _ptr(a):
    return None if a is None else a.ctypes.data


def _blobbuf(blob: bytes):
    return C.create_string_buffer(blob, len(blob)), len(blob)


def check_blob(blob: bytes):
    buf, n = _blobbuf(blob)
    cfg = np.zeros(13, np.int32)
    st = lib().oracle_check_blob(buf, n, _ptr(cfg))
    return st, cfg


def q8(x: float, inv: float) -> int:
    return int(lib().oracle_q8(float(x), float(inv)))


def exp_own(x: float) -> float:
    return float(lib().oracle_exp(float(x)))


def log_own(z: float) -> float:
    return float(lib().oracle_log(float(z)))


def sigma(s_q: float, s_k: float, dh: int) -> float:
    return float(lib().oracle_sigma(float(s_q), float(s_k), int(dh)))


def gemm_i32(A: np.ndarray, W: np.ndarray) -> np.ndarray:
    A = np.ascontiguousarray(A, np.int8); W = np.ascontiguousarray(W, np.int8)
    M, K = A.shape; N = W.shape[0]
    C_ = np.zeros((M, N), np.int32)
    lib().oracle_gemm_i32(_ptr(A), _ptr(W), M, N, K, _ptr(C_))
    return C_


MODE_Q8, MODE_RELU_Q8, MODE_RESID, MODE_F32 = 0, 1, 2, 3


def linear(A, W, s_w, b, s_x, mode, inv_out=None, gamma=1.0, resid=None):
    A = np.ascontiguousarray(A, np.int8); W = np.ascontiguousarray(W, np.int8)
    s_w = np.ascontiguousarray(s_w, np.float32); b = np.ascontiguousarray(b, np.float32)
    M, K = A.shape; N = W.shape[0]
    out_q = out_f = None
    if mode in (MODE_Q8, MODE_RELU_Q8):
        inv_out = np.ascontiguousarray(np.broadcast_to(np.float32(inv_out) if np.isscalar(inv_out)
                                                       else inv_out, (N,)), np.float32)
        out_q = np.zeros((M, N), np.int8)
    elif mode == MODE_RESID:
        out_f = np.array(resid, dtype=np.float32, copy=True).reshape(M, N)
    else:
        out_f = np.zeros((M, N), np.float32)
    _chk(lib().oracle_linear(_ptr(A), _ptr(W), _ptr(s_w), _ptr(b), float(s_x), _ptr(inv_out),
                             float(gamma), M, N, K, mode, _ptr(out_q), _ptr(out_f)))
    return out_q if out_q is not None else out_f


def layernorm(r, g, b, inv=1.0):
    r = np.ascontiguousarray(r, np.float32)
    M, d = r.shape
    of = np.zeros((M, d), np.float32); oq = np.zeros((M, d), np.int8)
    st = lib().oracle_layernorm(_ptr(r), _ptr(np.ascontiguousarray(g, np.float32)),
                                _ptr(np.ascontiguousarray(b, np.float32)), M, d, float(inv),
                                _ptr(of), _ptr(oq))
    if st != OK:
        raise OracleError(f"oracle returned {st}")
    return of, oq


def quantise_rows(W, bits, asym):
    """Row-wise quantisation (App. B Eq. scale / Eq. quant): (codes int32 [N][K], s [N], m [N])."""
    W = np.ascontiguousarray(W, np.float64)
    N, K = W.shape
    codes = np.zeros((N, K), np.int32); s_ = np.zeros(N, np.float32); m_ = np.zeros(N, np.float32)
    _chk(lib().oracle_quantise_rows(_ptr(W), N, K, int(bits), int(asym), _ptr(codes), _ptr(s_), _ptr(m_)))
    return codes, s_, m_


def linear_w4(A, Wp, s_w, m_w, b, s_x, mode, asym, inv_out=None, gamma=1.0, resid=None):
    """4-bit linear; Wp [N][K/2] packed as in the blob."""
    A = np.ascontiguousarray(A, np.int8); Wp = np.ascontiguousarray(Wp, np.uint8)
    s_w = np.ascontiguousarray(s_w, np.float32); b = np.ascontiguousarray(b, np.float32)
    m_w = None if m_w is None else np.ascontiguousarray(m_w, np.float32)
    M, K = A.shape; N = Wp.shape[0]
    out_q = out_f = None
    if mode in (MODE_Q8, MODE_RELU_Q8):
        inv_out = np.ascontiguousarray(np.broadcast_to(np.float32(inv_out) if np.isscalar(inv_out)
                                                       else inv_out, (N,)), np.float32)
        out_q = np.zeros((M, N), np.int8)
    elif mode == MODE_RESID:
        out_f = np.array(resid, dtype=np.float32, copy=True).reshape(M, N)
    else:
        out_f = np.zeros((M, N), np.float32)
    _chk(lib().oracle_linear_w4(_ptr(A), _ptr(Wp), _ptr(s_w), _ptr(m_w), _ptr(b), float(s_x), _ptr(inv_out),
                                float(gamma), M, N, K, int(asym), mode, _ptr(out_q), _ptr(out_f)))
    return out_q if out_q is not None else out_f


def fake_quant(x, s, bits=8, r_m=0.0, minmax=False):
    """QAT fake quantisation (App. B Eq. quant, scale s, offset r_m): (y f32, codes int32)."""
    x = np.ascontiguousarray(x, np.float32)
    y = np.zeros_like(x); q = np.zeros(x.shape, np.int32)
    _chk(lib().oracle_fake_quant(_ptr(x), x.size, float(s), float(r_m), int(bits), int(minmax), _ptr(y), _ptr(q)))
    return y, q


def fake_quant_backward(x, g, s, bits=8, r_m=0.0, minmax=False):
    """(dL/dx f32, dL/ds, dL/dr_m) of the fake quantiser for upstream gradient g."""
    x = np.ascontiguousarray(x, np.float32); g = np.ascontiguousarray(g, np.float32)
    gx = np.zeros_like(x); gs = np.zeros(1, np.float64); gr = np.zeros(1, np.float64)
    _chk(lib().oracle_fake_quant_backward(_ptr(x), _ptr(g), x.size, float(s), float(r_m), int(bits), int(minmax),
                                          _ptr(gx), _ptr(gs), _ptr(gr)))
    return gx, float(gs[0]), float(gr[0])


def fake_quant_linear(X, W, s_x, s_w, b, wbits=8):
    X = np.ascontiguousarray(X, np.float32); W = np.ascontiguousarray(W, np.float32)
    M, K = X.shape; N = W.shape[0]
    y = np.zeros((M, N), np.float32)
    _chk(lib().oracle_fake_quant_linear(_ptr(X), _ptr(W), float(s_x), _ptr(np.ascontiguousarray(s_w, np.float32)),
                                        _ptr(np.ascontiguousarray(b, np.float32)), M, N, K, int(wbits), _ptr(y)))
    return y


def ln_stats(r):
    """(mean, biased variance) per row as the LayerNorm computes them."""
    r = np.ascontiguousarray(r, np.float32)
    M, d = r.shape
    mu = np.zeros(M, np.float32); var = np.zeros(M, np.float32)
    _chk(lib().oracle_ln_stats(_ptr(r), M, d, _ptr(mu), _ptr(var)))
    return mu, var


def attention_decode(q, Kc, Vc, n_keys, sigma_, rho):
    """q [R][H][dh], Kc/Vc [R][H][T][dh] int8, n_keys [R] -> ctx [R][H][dh]."""
    q = np.ascontiguousarray(q, np.int8); Kc = np.ascontiguousarray(Kc, np.int8)
    Vc = np.ascontiguousarray(Vc, np.int8); n_keys = np.ascontiguousarray(n_keys, np.int32)
    R, H, T, dh = Kc.shape
    out = np.zeros((R, H, dh), np.int8)
    _chk(lib().oracle_attention_decode(_ptr(q), _ptr(Kc), _ptr(Vc), _ptr(n_keys), R, H, dh, T,
                                       float(sigma_), float(rho), _ptr(out)))
    return out


def attention_probs(q, K, sigma_):
    q = np.ascontiguousarray(q, np.int8); K = np.ascontiguousarray(K, np.int8)
    n, dh = K.shape
    P = np.zeros(n, np.float32)
    _chk(lib().oracle_attention_probs(_ptr(q), _ptr(K), n, dh, float(sigma_), _ptr(P)))
    return P


def encode(blob, src, length, cfg):
    buf, n = _blobbuf(blob)
    src = np.ascontiguousarray(src, np.int32)
    S = src.shape[0]
    d, L = cfg.d_model, cfg.n_dec
    enc_q = np.zeros((S, d), np.int8)
    ck = np.zeros((L, S, d), np.int8); cv = np.zeros((L, S, d), np.int8)
    _chk(lib().oracle_encode(buf, n, _ptr(src), int(length), S, _ptr(enc_q), _ptr(ck), _ptr(cv)))
    return enc_q, ck, cv


def decode_trace(blob, src, length, tgt, cfg, want_cache=False):
    buf, n = _blobbuf(blob)
    src = np.ascontiguousarray(src, np.int32); tgt = np.ascontiguousarray(tgt, np.int32)
    S = src.shape[0]; T = tgt.shape[0]
    logits = np.zeros((T, cfg.vocab), np.float32)
    dec_q = np.zeros((T, cfg.d_model), np.int8)
    sk = sv = None
    if want_cache:
        sk = np.zeros((cfg.n_dec, T, cfg.d_model), np.int8)
        sv = np.zeros((cfg.n_dec, T, cfg.d_model), np.int8)
    _chk(lib().oracle_decode_trace(buf, n, _ptr(src), int(length), S, _ptr(tgt), T, _ptr(logits),
                                   _ptr(dec_q), _ptr(sk), _ptr(sv)))
    return (logits, dec_q, sk, sv) if want_cache else (logits, dec_q)


def decode_forced(blob, src, length, tgt, cfg):
    buf, n = _blobbuf(blob)
    src = np.ascontiguousarray(src, np.int32); tgt = np.ascontiguousarray(tgt, np.int32)
    logits = np.zeros((tgt.shape[0], cfg.vocab), np.float32)
    _chk(lib().oracle_decode_forced(buf, n, _ptr(src), int(length), src.shape[0], _ptr(tgt),
                                    tgt.shape[0], _ptr(logits)))
    return logits


def embed(blob, ids, pos, cfg):
    buf, n = _blobbuf(blob)
    ids = np.ascontiguousarray(ids, np.int32); pos = np.ascontiguousarray(pos, np.int32)
    x = np.zeros((ids.shape[0], cfg.d_model), np.float32)
    _chk(lib().oracle_embed(buf, n, _ptr(ids), _ptr(pos), ids.shape[0], _ptr(x)))
    return x


def log_softmax(l):
    l = np.ascontiguousarray(l, np.float32)
    lp = np.zeros_like(l)
    _chk(lib().oracle_log_softmax(_ptr(l), l.shape[0], _ptr(lp)))
    return lp


def log_softmax_norm(l):
    """(m, lambda, Z) of the beam search's log-softmax of one logit row."""
    l = np.ascontiguousarray(l, np.float32)
    m = np.zeros(1, np.float32); lam = np.zeros(1, np.float32); Z = np.zeros(1, np.int64)
    _chk(lib().oracle_log_softmax_norm(_ptr(l), l.shape[0], _ptr(m), _ptr(lam), _ptr(Z)))
    return float(m[0]), float(lam[0]), int(Z[0])


def translate(blob, src, lens, beam, max_len, n_threads=1):
    buf, n = _blobbuf(blob)
    src = np.ascontiguousarray(src, np.int32); lens = np.ascontiguousarray(lens, np.int32)
    B, S = src.shape
    ids = np.zeros((B, max_len), np.int32); ol = np.zeros(B, np.int32); sc = np.zeros(B, np.float32)
    _chk(lib().oracle_translate(buf, n, _ptr(src), _ptr(lens), B, S, int(beam), int(max_len),
                                int(n_threads), _ptr(ids), _ptr(ol), _ptr(sc)))
    return ids, ol, sc
