"""Thin ctypes binding of libmnmt (include/mnmt.h): the same calls, argument
marshalling only.  Every step of the translation path runs in the library's
sm_103a kernels; if the library is missing or fails to load, importing this
module's functions raises — there is no fallback.

Host arrays are numpy arrays; device arrays are torch CUDA tensors (or raw
integer device addresses) — torch is used only for device memory and streams.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

from . import build as _build

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, EFORMAT, EOVERFLOW = 0, -1, -2, -3, -4, -5, -6
DEVICE_PTRS = 1
EPI_Q8, EPI_RELU_Q8, EPI_RESID, EPI_F32, EPI_ARGMAX = 0, 1, 2, 3, 4
(TAP_ENC_OUT, TAP_CROSS_K, TAP_CROSS_V, TAP_SELF_K, TAP_SELF_V, TAP_DEC_OUT, TAP_LOGITS, TAP_RESID,
 TAP_HISTORY, TAP_PARENTS, TAP_ANCESTRY) = range(1, 12)

_lock = threading.Lock()
_lib = None


class MnmtError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"mnmt error {code}: {msg}")
        self.code = code


class _Config(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ["n_enc", "n_dec", "d_model", "n_heads", "d_ffn", "vocab", "d_embed",
                                         "pre_ln", "tied_output", "max_pos", "pad_id", "bos_id", "eos_id"]]


def lib_path() -> str:
    return _build.LIB


def lib():
    """Load libmnmt.so (building it first if its sources are newer)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            if not os.path.exists(path):
                raise RuntimeError(f"libmnmt.so missing at {path}")
            L = C.CDLL(path)
            _declare(L)
            _lib = L
    return _lib


def _declare(L):
    p, i32, sz, f = C.c_void_p, C.c_int32, C.c_size_t, C.c_float
    L.mnmt_blob_check.argtypes = [p, sz, C.POINTER(_Config)]
    L.mnmt_load_weights.argtypes = [p, sz, p, C.POINTER(p)]
    L.mnmt_load_weights_ex.argtypes = [p, sz, p, i32, C.POINTER(p)]
    L.mnmt_session_create_ex.argtypes = [p, i32, i32, i32, i32, i32, C.POINTER(p)]
    L.mnmt_model_device_bytes.argtypes = [p]; L.mnmt_model_device_bytes.restype = C.c_int64
    L.mnmt_session_device_bytes.argtypes = [p]; L.mnmt_session_device_bytes.restype = C.c_int64
    L.mnmt_model_free.argtypes = [p]; L.mnmt_model_free.restype = None
    L.mnmt_model_config.argtypes = [p, C.POINTER(_Config)]
    L.mnmt_session_create.argtypes = [p, i32, i32, i32, i32, C.POINTER(p)]
    L.mnmt_session_free.argtypes = [p]; L.mnmt_session_free.restype = None
    L.mnmt_encode.argtypes = [p, p, p, i32, i32, i32]
    L.mnmt_decode_step.argtypes = [p, p, p, p, p]
    L.mnmt_decode_steps.argtypes = [p, i32]; L.mnmt_decode_steps.restype = C.c_int
    L.mnmt_translate.argtypes = [p, p, p, i32, i32, i32, i32, p, p, p]
    L.mnmt_debug_tap.argtypes = [p, i32, i32, p, sz]; L.mnmt_debug_tap.restype = C.c_int64
    L.mnmt_session_decode_path.argtypes = [p]; L.mnmt_session_decode_path.restype = C.c_int
    L.mnmt_last_error.argtypes = []; L.mnmt_last_error.restype = C.c_char_p
    L.mnmt_linear.argtypes = [p, p, p, p, f, p, f, i32, i32, i32, i32, p, p, p]
    L.mnmt_linear_argmax.argtypes = [p, p, p, p, f, i32, i32, i32, p, p]
    L.mnmt_linear_argmax_ids_noalloc.argtypes = [p, p, p, p, f, i32, i32, i32, p, p]
    L.mnmt_linear_argmax_ids_noalloc.restype = C.c_int
    L.mnmt_attention_decode.argtypes = [p, p, p, p, i32, i32, i32, i32, f, f, p, p]
    L.mnmt_layernorm.argtypes = [p, p, p, i32, i32, f, p, p, p, p]
    L.mnmt_linear_tc.argtypes = [p, p, p, p, f, p, f, i32, i32, i32, i32, p, p, p, p, p]
    L.mnmt_codes_to_f16.argtypes = [p, p, sz, p]
    L.mnmt_linear_w4.argtypes = [p, p, p, p, p, f, p, f, i32, i32, i32, i32, p, p, p, p]
    L.mnmt_linear_w4.restype = C.c_int
    L.mnmt_fake_quant.argtypes = [p, sz, f, f, i32, i32, p, p, p]
    L.mnmt_fake_quant_backward.argtypes = [p, p, sz, f, f, i32, i32, p, p, p, p]
    L.mnmt_fake_quant_linear.argtypes = [p, p, f, p, p, i32, i32, i32, i32, p, p, p]
    for n in ["mnmt_fake_quant", "mnmt_fake_quant_backward", "mnmt_fake_quant_linear"]:
        getattr(L, n).restype = C.c_int
    L.mnmt_wait_timeout_selftest.argtypes = [p, p]
    for n in ["mnmt_blob_check", "mnmt_load_weights", "mnmt_load_weights_ex", "mnmt_session_create_ex",
              "mnmt_model_config", "mnmt_session_create", "mnmt_encode",
              "mnmt_decode_step", "mnmt_translate", "mnmt_linear", "mnmt_linear_argmax", "mnmt_attention_decode", "mnmt_layernorm",
              "mnmt_linear_tc", "mnmt_codes_to_f16", "mnmt_wait_timeout_selftest"]:
        getattr(L, n).restype = C.c_int


def last_error() -> str:
    return lib().mnmt_last_error().decode()


def _chk(code):
    if code != OK:
        raise MnmtError(code, last_error())
    return code


def _ptr(x):
    """Address of a numpy array, a torch tensor, or an integer address."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    return x.data_ptr()


def _stream_handle(stream):
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# --------------------------------------------------------------------------- C calls
def mnmt_blob_check(blob: bytes) -> dict:
    cfg = _Config()
    _chk(lib().mnmt_blob_check(blob, len(blob), C.byref(cfg)))
    return {n: getattr(cfg, n) for n, _ in _Config._fields_}


LOAD_LEAN = 1
SESSION_LEAN = 1


def mnmt_load_weights(blob: bytes, stream=None, flags: int = 0) -> int:
    h = C.c_void_p()
    if flags:
        _chk(lib().mnmt_load_weights_ex(blob, len(blob), _stream_handle(stream), flags, C.byref(h)))
    else:
        _chk(lib().mnmt_load_weights(blob, len(blob), _stream_handle(stream), C.byref(h)))
    return h.value


def mnmt_model_device_bytes(model: int) -> int:
    r = lib().mnmt_model_device_bytes(model)
    if r < 0:
        raise MnmtError(int(r), last_error())
    return int(r)


def mnmt_session_device_bytes(session: int) -> int:
    r = lib().mnmt_session_device_bytes(session)
    if r < 0:
        raise MnmtError(int(r), last_error())
    return int(r)


def mnmt_model_free(model: int):
    lib().mnmt_model_free(model)


def mnmt_model_config(model: int) -> dict:
    cfg = _Config()
    _chk(lib().mnmt_model_config(model, C.byref(cfg)))
    return {n: getattr(cfg, n) for n, _ in _Config._fields_}


def mnmt_session_create(model: int, max_batch: int, max_src_len: int, beam: int, max_len: int,
                        flags: int = 0) -> int:
    h = C.c_void_p()
    if flags:
        _chk(lib().mnmt_session_create_ex(model, max_batch, max_src_len, beam, max_len, flags, C.byref(h)))
    else:
        _chk(lib().mnmt_session_create(model, max_batch, max_src_len, beam, max_len, C.byref(h)))
    return h.value


def mnmt_session_free(session: int):
    lib().mnmt_session_free(session)


def mnmt_encode(session: int, src_ids, src_lens, B: int, S_pad: int, flags: int = 0):
    _chk(lib().mnmt_encode(session, _ptr(src_ids), _ptr(src_lens), B, S_pad, flags))


def mnmt_decode_steps(session: int, n: int) -> int:
    """Queue n decode steps without waiting; returns the number queued."""
    r = lib().mnmt_decode_steps(session, n)
    if r < 0:
        raise MnmtError(r, last_error())
    return r


def mnmt_decode_step(session: int, R: int):
    """One decode step; returns (tokens [R], parents [R], scores [R], all_done)."""
    tok = np.zeros(R, np.int32); par = np.zeros(R, np.int32); sc = np.zeros(R, np.float32)
    done = C.c_int32(0)
    _chk(lib().mnmt_decode_step(session, _ptr(tok), _ptr(par), _ptr(sc), C.byref(done)))
    return tok, par, sc, bool(done.value)


def mnmt_translate(session: int, src_ids, src_lens, B: int, S_pad: int, max_len: int, flags: int,
                   out_ids, out_lens, out_scores):
    _chk(lib().mnmt_translate(session, _ptr(src_ids), _ptr(src_lens), B, S_pad, max_len, flags,
                              _ptr(out_ids), _ptr(out_lens), _ptr(out_scores)))


def mnmt_debug_tap(session: int, tap: int, layer: int = 0, dtype=np.int8, shape=None) -> np.ndarray:
    n = lib().mnmt_debug_tap(session, tap, layer, None, 0)
    if n < 0:
        raise MnmtError(int(n), last_error())
    out = np.zeros(n // np.dtype(dtype).itemsize, dtype)
    _chk(int(lib().mnmt_debug_tap(session, tap, layer, _ptr(out), n)))
    return out.reshape(shape) if shape is not None else out


def mnmt_session_decode_path(session: int) -> int:
    """1 if the session's decode step runs on one thread-block cluster, 0 for the multi-kernel step."""
    r = lib().mnmt_session_decode_path(session)
    if r < 0:
        raise MnmtError(r, last_error())
    return r


def mnmt_linear(A, W, s_w, bias, s_x, inv_out, gamma, M, N, K, mode, out_q, out_f, stream=None):
    _chk(lib().mnmt_linear(_ptr(A), _ptr(W), _ptr(s_w), _ptr(bias), float(s_x), _ptr(inv_out), float(gamma),
                           M, N, K, mode, _ptr(out_q), _ptr(out_f), _stream_handle(stream)))


def mnmt_linear_argmax(A, W, s_w, bias, s_x, M, N, K, keys, stream=None):
    _chk(lib().mnmt_linear_argmax(_ptr(A), _ptr(W), _ptr(s_w), _ptr(bias), float(s_x), M, N, K, _ptr(keys),
                                  _stream_handle(stream)))


def mnmt_linear_argmax_ids_noalloc(A, W, s_w, bias, s_x, M, N, K, ids, stream=None):
    """Greedy vocabulary argmax into int32 ids with library-owned scratch (no allocation)."""
    _chk(lib().mnmt_linear_argmax_ids_noalloc(_ptr(A), _ptr(W), _ptr(s_w), _ptr(bias), float(s_x), M, N, K,
                                              _ptr(ids), _stream_handle(stream)))


def mnmt_linear_tc(A16, W16, s_w, bias, s_x, inv_out, gamma, M, N, K, mode, out_q=None, out_f=None, keys=None,
                   status=None, stream=None):
    """Tensor-core quantised linear over fp16 copies of the int8 codes (see mnmt_codes_to_f16)."""
    _chk(lib().mnmt_linear_tc(_ptr(A16), _ptr(W16), _ptr(s_w), _ptr(bias), float(s_x), _ptr(inv_out), float(gamma),
                              M, N, K, mode, _ptr(out_q), _ptr(out_f), _ptr(keys), _ptr(status),
                              _stream_handle(stream)))


def mnmt_linear_w4(A, Wp, s_w, m_w, bias, s_x, inv_out, gamma, M, N, K, mode, out_q=None, out_f=None, keys=None,
                   stream=None):
    """Quantised linear with row-wise 4-bit weights (m_w None: symmetric rows)."""
    _chk(lib().mnmt_linear_w4(_ptr(A), _ptr(Wp), _ptr(s_w), _ptr(m_w), _ptr(bias), float(s_x), _ptr(inv_out),
                              float(gamma), M, N, K, mode, _ptr(out_q), _ptr(out_f), _ptr(keys),
                              _stream_handle(stream)))


def mnmt_fake_quant(x, n, s, r_m=0.0, bits=8, minmax=False, y=None, codes=None, stream=None):
    """QAT fake quantisation (device buffers): y = Q(x), codes = q (int32)."""
    _chk(lib().mnmt_fake_quant(_ptr(x), n, float(s), float(r_m), bits, int(minmax), _ptr(y), _ptr(codes),
                               _stream_handle(stream)))


def mnmt_fake_quant_backward(x, g, n, s, gx, gs, gr=None, r_m=0.0, bits=8, minmax=False, stream=None):
    """STE gradient gx and the scale / offset gradients gs, gr (device fp64 scalars)."""
    _chk(lib().mnmt_fake_quant_backward(_ptr(x), _ptr(g), n, float(s), float(r_m), bits, int(minmax), _ptr(gx),
                                        _ptr(gs), _ptr(gr), _stream_handle(stream)))


def mnmt_fake_quant_linear(X, W, s_x, s_w, bias, M, N, K, wbits, workspace, y, stream=None):
    """QAT forward of a linear from fp32 input and weights (learnable scales)."""
    _chk(lib().mnmt_fake_quant_linear(_ptr(X), _ptr(W), float(s_x), _ptr(s_w), _ptr(bias), M, N, K, wbits,
                                      _ptr(workspace), _ptr(y), _stream_handle(stream)))


def mnmt_codes_to_f16(src, dst, n, stream=None):
    """dst[i] = fp16(src[i]) for n int8 codes (device buffers)."""
    _chk(lib().mnmt_codes_to_f16(_ptr(src), _ptr(dst), n, _stream_handle(stream)))


def mnmt_wait_timeout_selftest(status, stream=None):
    """Queue one block whose barrier wait runs out (one second): *status -> ETIMEOUT."""
    _chk(lib().mnmt_wait_timeout_selftest(_ptr(status), _stream_handle(stream)))


def argmax_from_keys(keys: np.ndarray) -> np.ndarray:
    """Token ids encoded in mnmt_linear_argmax keys (uint64 viewed as int64 is fine)."""
    k = keys.view(np.uint64)
    return (np.uint64(0xFFFFFFFF) - (k & np.uint64(0xFFFFFFFF))).astype(np.int64)


def mnmt_attention_decode(q, Kc, Vc, n_keys, R, H, dh, T, sigma, rho, ctx, stream=None):
    _chk(lib().mnmt_attention_decode(_ptr(q), _ptr(Kc), _ptr(Vc), _ptr(n_keys), R, H, dh, T, float(sigma),
                                     float(rho), _ptr(ctx), _stream_handle(stream)))


def mnmt_layernorm(r, g, b, M, d, inv, out_f, out_q, status=None, stream=None):
    _chk(lib().mnmt_layernorm(_ptr(r), _ptr(g), _ptr(b), M, d, float(inv), _ptr(out_f), _ptr(out_q),
                              _ptr(status), _stream_handle(stream)))


# --------------------------------------------------------------------------- convenience
class Translator:
    """A loaded model plus one session (owner of both handles)."""

    def __init__(self, blob: bytes, max_batch: int, max_src_len: int, beam: int, max_len: int, stream=None,
                 lean: bool = False):
        """lean=True: memory-minimal model and session (MNMT_LOAD_LEAN, MNMT_SESSION_LEAN)."""
        self.model = mnmt_load_weights(blob, stream, LOAD_LEAN if lean else 0)
        try:
            self.session = mnmt_session_create(self.model, max_batch, max_src_len, beam, max_len,
                                               SESSION_LEAN if lean else 0)
        except Exception:
            mnmt_model_free(self.model)
            raise
        self.cfg = mnmt_model_config(self.model)
        self.beam = beam

    def translate(self, src_ids: np.ndarray, src_lens: np.ndarray, max_len: int):
        """Host arrays in, host arrays out (ids [B][max_len], lens [B], scores [B])."""
        src_ids = np.ascontiguousarray(src_ids, np.int32)
        src_lens = np.ascontiguousarray(src_lens, np.int32)
        B, S = src_ids.shape
        ids = np.zeros((B, max_len), np.int32); lens = np.zeros(B, np.int32); sc = np.zeros(B, np.float32)
        mnmt_translate(self.session, src_ids, src_lens, B, S, max_len, 0, ids, lens, sc)
        return ids, lens, sc

    def close(self):
        if getattr(self, "session", None):
            mnmt_session_free(self.session)
            self.session = None
        if getattr(self, "model", None):
            mnmt_model_free(self.model)
            self.model = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
