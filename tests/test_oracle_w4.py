"""Pins of the oracle's 4-bit row-wise weight formats (no GPU): Sec. 3.3 and
the table "quantizing weights to lower bits" (4-8-8: 4-bit weights, 8-bit
embedding and activations, row-wise scales for low bits), with App. B Eq.
scale / Eq. quant (min-max scale and offset r_m) as the second form."""
import numpy as np
import pytest

from oracle import bruteforce as BF
from oracle import oracle as O
from paper_2306_04235_gb300 import synth


def _w(seed, n, k, std=0.02):
    return synth.weight_draw(synth.Stream(seed, "w4"), n, k, std)


# ---------------------------------------------------------------- quantiser
def test_symmetric_4bit_round_trip_table():
    """Rows that are exact multiples v*s of a scale with max |v| = 7 quantise
    back to v (Eq. quant with zero offset and 2^4 - 1 symmetric levels)."""
    s = np.float32(0.0125)
    v = np.array([[-7, -3, 0, 1, 2, 5, 7, -1], [7, 7, -7, 0, 0, 0, 3, -6]], np.int64)
    W = v.astype(np.float64) * float(s)
    codes, sc, m = O.quantise_rows(W, 4, 0)
    assert np.array_equal(codes, v) and np.all(sc == s) and np.all(m == 0)


def test_minmax_4bit_round_trip_table():
    """Rows r + u*s with u spanning 0..15 quantise back to u, offset r, scale s."""
    s, r = np.float32(0.003), np.float32(-0.021)
    u = np.array([[0, 15, 3, 8, 1, 14, 7, 9], [15, 0, 0, 15, 5, 5, 10, 2]], np.int64)
    W = u.astype(np.float64) * float(s) + float(r)
    codes, sc, m = O.quantise_rows(W, 4, 1)
    assert np.array_equal(codes, u)
    assert np.allclose(sc, s, rtol=1e-6) and np.all(m == r)


@pytest.mark.parametrize("asym", [0, 1])
def test_4bit_quantisation_error_and_extremes(asym):
    """Every dequantised weight is within half a step of the float weight
    (float64 brute force); the row extremes map to the end codes."""
    W = _w(3, 64, 256)
    codes, s, m = O.quantise_rows(W, 4, asym)
    deq = codes * s.astype(np.float64)[:, None] + m.astype(np.float64)[:, None]
    assert np.all(np.abs(deq - W) <= 0.5 * s.astype(np.float64)[:, None] * (1 + 1e-6))
    rows = np.arange(64)
    if asym:
        assert np.all(codes[rows, W.argmin(axis=1)] == 0) and np.all(codes[rows, W.argmax(axis=1)] == 15)
        assert codes.min() >= 0 and codes.max() <= 15
    else:
        big = np.abs(W).argmax(axis=1)
        assert np.all(np.abs(codes[rows, big]) == 7) and np.abs(codes).max() <= 7


@pytest.mark.parametrize("asym", [False, True])
def test_generator_codes_are_the_quantiser_of_its_draw(asym):
    W = _w(4, 33, 128)
    stored, s, r = synth.int4_weight(W, asym)
    codes, s_o, m_o = O.quantise_rows(W, 4, int(asym))
    assert np.array_equal(stored.astype(np.int64) - (0 if asym else 8), codes)
    assert np.array_equal(s, s_o)
    if asym:
        assert np.array_equal(r, m_o)


# ------------------------------------------------------------------- linear
def _case(seed, M, N, K, asym):
    A = synth.uniform_int8(seed, "a", (M, K))
    W = _w(seed, N, K)
    stored, s, r = synth.int4_weight(W, asym)
    b = synth.uniform_f32(seed, "b", (N,), -0.05, 0.05)
    return A, stored, synth.pack4(stored), s, r, b


def test_packing_layout_by_one_hot_rows():
    """a = e_k selects code k of each row: the packed layout (32-code chunks,
    low nibble = first 16) is read back exactly."""
    N, K = 5, 96
    stored = synth.Stream(7, "c").randint(0, 15, N * K).astype(np.uint8).reshape(N, K)
    Wp = synth.pack4(stored)
    A = np.eye(K, dtype=np.int8)
    ones = np.ones(N, np.float32)
    y = O.linear_w4(A, Wp, ones, None, np.zeros(N, np.float32), 1.0, O.MODE_F32, False)
    assert np.array_equal(y.T.astype(np.int64), stored.astype(np.int64) - 8)
    y = O.linear_w4(A, Wp, ones, np.zeros(N, np.float32), np.zeros(N, np.float32), 1.0, O.MODE_F32, True)
    assert np.array_equal(y.T.astype(np.int64), stored.astype(np.int64))


def test_symmetric_4bit_linear_equals_int8_linear_on_the_same_codes():
    """Integer identity: a symmetric 4-bit row is an int8 row with codes in
    [-7, 7]; every epilogue gives the same bits as the int8 linear."""
    A, stored, Wp, s, _, b = _case(5, 6, 40, 256, False)
    W8 = (stored.astype(np.int16) - 8).astype(np.int8)
    inv = np.float32(50.0)
    for mode in (O.MODE_Q8, O.MODE_RELU_Q8, O.MODE_F32):
        iv = None if mode == O.MODE_F32 else inv
        got = O.linear_w4(A, Wp, s, None, b, 0.03, mode, False, inv_out=iv)
        ref = O.linear(A, W8, s, b, 0.03, mode, inv_out=iv)
        assert np.array_equal(got.view(np.uint8) if got.dtype == np.float32 else got,
                              ref.view(np.uint8) if ref.dtype == np.float32 else ref)
    r0 = synth.uniform_f32(5, "r", (6, 40), -2, 2)
    got = O.linear_w4(A, Wp, s, None, b, 0.03, O.MODE_RESID, False, gamma=0.75, resid=r0)
    ref = O.linear(A, W8, s, b, 0.03, O.MODE_RESID, gamma=0.75, resid=r0)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("asym", [False, True])
def test_4bit_linear_vs_float64(asym):
    """y = x Q(W)^T + b with Q(W) the dequantised rows (s (u - 8), or s u + r)
    in float64: within a few fp32 roundings of the terms' magnitude."""
    A, stored, Wp, s, r, b = _case(6, 4, 48, 512, asym)
    s_x = np.float32(0.03)
    deq = (stored.astype(np.float64) - (0 if asym else 8)) * s.astype(np.float64)[:, None]
    if asym:
        deq += r.astype(np.float64)[:, None]
    ref = (A.astype(np.float64) * float(s_x)) @ deq.T + b
    got = O.linear_w4(A, Wp, s, r, b, s_x, O.MODE_F32, asym)
    mag = (np.abs(A.astype(np.float64) * float(s_x)) @ np.abs(deq).T) + np.abs(b)
    assert np.all(np.abs(got - ref) <= 4 * 2.0 ** -24 * mag + 1e-12)


@pytest.mark.parametrize("wq", [synth.WQ_INT4, synth.WQ_INT4_MINMAX])
def test_4bit_model_matches_float64_bruteforce(wq):
    """Encoder codes and decoder logits of a 4-bit model against the float64
    fake-quantised model reading the same blob."""
    cfg = synth.ModelConfig(2, 2, 64, 2, 128, 300, 48, 1, 0, max_pos=64)   # factorised, untied (8-bit)
    blob = synth.build_blob(cfg, 12, gamma_range=(0.5, 1.5), wq=wq)
    ids, lens = synth.source_batch(cfg.vocab, 1, 12, 12, 4)
    enc, ck, cv = O.encode(blob, ids[0], lens[0], cfg)
    benc, bck, bcv = BF.Model(blob).encode(ids[0], lens[0])
    for got, ref in [(enc, benc), (ck, bck), (cv, bcv)]:
        diff = np.abs(got.astype(np.int64) - ref.astype(np.int64))
        assert diff.max() <= 2 and np.mean(diff == 0) > 0.98
    tgt = np.concatenate([[cfg.bos_id], synth.Stream(5, "t").randint(3, cfg.vocab - 1, 7)]).astype(np.int32)
    logits, _ = O.decode_trace(blob, ids[0], lens[0], tgt, cfg)
    ref = BF.Model(blob).decode_forced(ids[0], lens[0], tgt)
    err = np.abs(logits - ref) / np.abs(ref).max(axis=1, keepdims=True)
    assert np.median(err) < 1e-4 and err.max() < 2e-2


def test_4bit_blob_sizes_halve_the_linears():
    """4-8-8: the linears' codes take half the bytes of 8-8-8 (Table
    "quantizing weights to lower bits": 10 MB -> 5 MB for the 10MB model's
    weights); the min-max form adds one fp32 offset per row."""
    cfg = synth.MODELS["mobilenmt-10mb"]
    b8 = len(synth.build_blob(cfg, 10))
    b4 = len(synth.build_blob(cfg, 10, wq=synth.WQ_INT4))
    b4m = len(synth.build_blob(cfg, 10, wq=synth.WQ_INT4_MINMAX))
    d, F, L = cfg.d_model, cfg.d_ffn, cfg
    # attention and FFN linears only: the embedding stays 8-bit
    lin_codes = cfg.n_enc * (4 * d * d + 2 * d * F) + cfg.n_dec * (8 * d * d + 2 * d * F)
    assert b8 - b4 == lin_codes // 2
    rows = cfg.n_enc * (5 * d + F) + cfg.n_dec * (9 * d + F)   # output rows of every linear
    assert b4m - b4 == 4 * rows


@pytest.mark.parametrize("wq", [synth.WQ_INT4, synth.WQ_INT4_MINMAX])
def test_4bit_workload_translates_each_source_differently(wq):
    wl = synth.WORKLOADS["small-b1-s10to50-greedy64"]
    cfg = synth.MODELS[wl.model]
    blob = synth.build_blob(cfg, wl.model_seed, wq=wq)
    ids, lens = synth.source_batch(cfg.vocab, 5, 10, 40, 4243)
    out, olen, _ = O.translate(blob, ids, lens, 1, 8, n_threads=5)
    assert len({tuple(out[b, :olen[b]]) for b in range(5)}) == 5
