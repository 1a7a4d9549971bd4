"""Pins of the oracle's building blocks against closed forms, library routines
and float64 brute force (no GPU).

Quantiser: App. B (Eq. 3/4) with zero point 0, symmetric clamp, ties to even.
Linear: Sec. 3.3 / Fig. 5 (int8 x int8 -> int32, full-precision bias).
LayerNorm: App. A / App. D.  Attention: Eq. 1/2.
"""
import math
import struct

import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import synth


def f32(x):
    return struct.unpack("<f", struct.pack("<f", x))[0]


def ulp32(x):
    x = abs(f32(x))
    if x == 0.0:
        return 2.0 ** -149
    e = math.frexp(x)[1]
    return 2.0 ** (e - 24)


# ----------------------------------------------------------------- quantiser
@pytest.mark.parametrize("x,code", [
    (0.5, 0), (1.5, 2), (2.5, 2), (-0.5, 0), (-1.5, -2), (-2.5, -2),
    (126.5, 126), (127.5, 127), (127.49, 127), (128.0, 127), (1e9, 127),
    (-126.5, -126), (-127.5, -127), (-128.0, -127), (-1e9, -127), (0.49999997, 0),
])
def test_q8_table(x, code):
    assert O.q8(x, 1.0) == code


def test_q8_never_minus_128_and_scale_roundtrip():
    for s in [f32(0.01), f32(4.0 / 127), f32(0.3), f32(1e-3)]:
        inv = f32(1.0 / s)
        for q in range(-127, 128):
            assert O.q8(f32(q * s), inv) == q
    assert O.q8(-3e38, 1.0) == -127


# -------------------------------------------------------------- integer GEMM
def test_gemm_matches_int64_matmul():
    rng = np.random.default_rng(0)
    for M, N, K in [(1, 7, 16), (5, 33, 256), (3, 4, 2048)]:
        A = rng.integers(-127, 128, (M, K), dtype=np.int64).astype(np.int8)
        W = rng.integers(-127, 128, (N, K), dtype=np.int64).astype(np.int8)
        ref = A.astype(np.int64) @ W.astype(np.int64).T
        assert np.array_equal(O.gemm_i32(A, W).astype(np.int64), ref)


def test_gemm_extremes_and_row_sums():
    K = 2048
    A = np.full((2, K), 127, np.int8); A[1] = -127
    W = np.full((3, K), -127, np.int8); W[1] = 127; W[2, ::2] = 1
    C = O.gemm_i32(A, W)
    assert C[0, 0] == -127 * 127 * K and C[1, 0] == 127 * 127 * K   # |acc| < 2^31
    ones = np.ones((1, 300), np.int8)
    W = synth.uniform_int8(3, "w", (9, 300))
    assert np.array_equal(O.gemm_i32(ones, W)[0], W.astype(np.int64).sum(axis=1))


# ------------------------------------------------------------------ epilogues
def _linear_case(seed, M=4, N=40, K=96):
    A = synth.uniform_int8(seed, "a", (M, K))
    W = synth.uniform_int8(seed, "w", (N, K))
    s_w = synth.uniform_f32(seed, "sw", (N,), 1e-4, 3e-4)
    b = synth.uniform_f32(seed, "b", (N,), -0.05, 0.05)
    return A, W, s_w, b


def test_linear_f32_vs_float64():
    A, W, s_w, b = _linear_case(1)
    s_x = f32(0.031)
    y = O.linear(A, W, s_w, b, s_x, O.MODE_F32)
    acc = A.astype(np.float64) @ W.astype(np.float64).T
    y64 = acc * (np.float64(s_x) * s_w.astype(np.float64)) + b
    tol = 4 * 2.0 ** -24 * (np.abs(acc * s_x * s_w) + np.abs(b)) + 1e-30
    assert np.all(np.abs(y - y64) <= tol)


def test_linear_q8_relu_and_residual_vs_float64():
    A, W, s_w, b = _linear_case(2)
    s_x, s_o = f32(0.031), f32(0.05)
    inv = f32(1.0 / s_o)
    acc = A.astype(np.float64) @ W.astype(np.float64).T
    y64 = acc * (np.float64(s_x) * s_w.astype(np.float64)) + b
    for mode, pre in [(O.MODE_Q8, y64), (O.MODE_RELU_Q8, np.maximum(y64, 0.0))]:
        q = O.linear(A, W, s_w, b, s_x, mode, inv_out=inv).astype(np.int64)
        ref = np.clip(np.rint(pre / s_o), -127, 127)
        frac = np.abs(pre / s_o - np.trunc(pre / s_o))
        near_half = np.abs(frac - 0.5) < 1e-4
        assert np.all(np.abs(q - ref) <= near_half), "codes differ away from a rounding tie"
        if mode == O.MODE_RELU_Q8:
            assert np.all(q[y64 < -1e-3] == 0)
    r0 = synth.uniform_f32(5, "r", y64.shape, -3, 3)
    g = f32(0.75)
    r1 = O.linear(A, W, s_w, b, s_x, O.MODE_RESID, gamma=g, resid=r0)
    ref = g * r0.astype(np.float64) + y64
    assert np.allclose(r1, ref, rtol=1e-6, atol=1e-6)


# ------------------------------------------------------------------ LayerNorm
def _ln64(x, g, b):
    x = x.astype(np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + 1e-5) * g + b


def test_layernorm_constant_row_gives_beta():
    d = 256
    g = synth.uniform_f32(1, "g", (d,), 0.5, 1.5)
    b = synth.uniform_f32(1, "b", (d,), -1, 1)
    r = np.full((3, d), 7.25, np.float32); r[1] = -700.5; r[2] = 0.0
    out, _ = O.layernorm(r, g, b)
    assert np.array_equal(out, np.broadcast_to(b, out.shape))


@pytest.mark.parametrize("d,scale", [(128, 1.0), (256, 30.0), (512, 700.0), (384, 1e-3), (2048, 1e6)])
def test_layernorm_vs_float64(d, scale):
    r = (synth.Stream(d, "r").normal(5 * d).reshape(5, d) * scale + scale * 0.3).astype(np.float32)
    g = synth.uniform_f32(d, "g", (d,), 0.5, 1.5)
    b = synth.uniform_f32(d, "b", (d,), -0.2, 0.2)
    out, codes = O.layernorm(r, g, b, inv=f32(127 / 4.0))
    ref = _ln64(r, g, b)
    # a few fp32 roundings of O(1) values; var/(d-1) or another epsilon is far outside this
    assert np.all(np.abs(out - ref) <= 1e-6 + 1e-6 * np.abs(ref))
    assert np.array_equal(codes, np.array([[O.q8(v, f32(127 / 4.0)) for v in row] for row in out]))


def test_layernorm_permutation_invariant_and_overflow():
    d = 256
    r = (synth.Stream(9, "r").normal(d) * 5).astype(np.float32)[None]
    g = np.ones(d, np.float32); b = np.zeros(d, np.float32)
    perm = np.argsort(synth.Stream(9, "p").uniform(d))
    out, _ = O.layernorm(r, g, b)
    out_p, _ = O.layernorm(r[:, perm], g, b)
    assert np.array_equal(out[:, perm], out_p)          # same mean and rstd bit for bit
    bad = r.copy(); bad[0, 3] = 2.0 ** 32
    with pytest.raises(O.OracleError):
        O.layernorm(bad, g, b)


# ------------------------------------------------------------------ exp / log
def test_exp_own_within_2ulp_on_a_grid():
    xs = np.concatenate([-np.linspace(0, 87.0, 40001, dtype=np.float32),
                         -np.logspace(-8, 0, 2001, dtype=np.float32),
                         np.float32([-0.34657359, -0.34657358, -0.6931472, -17.328680])])
    for x in xs:
        x = float(x)
        e = O.exp_own(x)
        assert abs(e - math.exp(x)) <= 2 * ulp32(math.exp(x)), x
    assert O.exp_own(0.0) == 1.0
    assert O.exp_own(-87.5) == 0.0 and O.exp_own(-1e30) == 0.0


def test_log_own_relative_error():
    rng = np.random.default_rng(7)
    zs = list(range(1, 2000)) + [2.0 ** k for k in range(0, 45)] + \
         list(np.exp(rng.uniform(0, 30, 3000)))
    for z in zs:
        z = float(z)
        ref = math.log(z)
        got = O.log_own(z)
        if z == 1.0:
            assert got == 0.0
        else:
            assert abs(got - ref) <= 1e-15 * abs(ref) + 1e-300, z


# ------------------------------------------------------------------ attention
def _att_inputs(seed, n, dh=64, lo=-127, hi=127):
    q = synth.uniform_int8(seed, "q", (dh,), lo, hi)
    K = synth.uniform_int8(seed, "k", (n, dh), lo, hi)
    V = synth.uniform_int8(seed, "v", (n, dh), lo, hi)
    return q, K, V


def _attend(q, K, V, sigma, rho):
    n, dh = K.shape
    Kc = K[None, None]; Vc = V[None, None]
    return O.attention_decode(q[None, None], Kc, Vc, np.array([n], np.int32), sigma, rho)[0, 0]


def test_attention_single_key_returns_value():
    q, K, V = _att_inputs(1, 1)
    out = _attend(q, K, V, f32(0.01), 1.0)
    assert np.array_equal(out, V[0])
    rho = f32(0.6)
    out = _attend(q, K, V, f32(0.01), rho)
    assert np.array_equal(out, np.array([O.q8(float(v), rho) for v in V[0]], np.int8))


def test_attention_equal_scores_average_values():
    n, dh = 12, 64
    q, K, V = _att_inputs(2, n)
    K = np.broadcast_to(K[0], (n, dh)).copy()             # every key identical
    out = _attend(q, K, V, f32(0.02), 1.0)
    mean = V.astype(np.float64).mean(axis=0)
    assert np.array_equal(out, np.clip(np.rint(mean), -127, 127).astype(np.int8))


def test_attention_dominant_key_is_one_hot():
    n, dh = 40, 64
    q, K, V = _att_inputs(3, n, lo=-20, hi=20)
    K[17] = np.sign(q) * 127                                # far larger score than the rest
    out = _attend(q, K, V, f32(0.1), 1.0)
    assert np.array_equal(out, V[17])


@pytest.mark.parametrize("n,sigma", [(5, 0.001), (64, 0.0005), (300, 0.0002), (512, 0.0001)])
def test_attention_vs_float64_softmax(n, sigma):
    q, K, V = _att_inputs(n, n)
    sigma = f32(sigma); rho = f32(0.9)
    s = (K.astype(np.float64) @ q.astype(np.float64)) * sigma
    p = np.exp(s - s.max()); p /= p.sum()
    P = O.attention_probs(q, K, sigma)
    assert np.max(np.abs(P - p)) < 2e-6                     # 2^-24 fixed-point weights
    ctx64 = (p @ V.astype(np.float64)) * rho
    out = _attend(q, K, V, sigma, rho).astype(np.float64)
    assert np.all(np.abs(out - np.clip(np.rint(ctx64), -127, 127)) <= 1)
    assert np.mean(out == np.clip(np.rint(ctx64), -127, 127)) > 0.95


def test_sigma_definition():
    assert O.sigma(f32(0.03), f32(0.05), 64) == f32(0.03 * 0.05 / 8.0) or \
        abs(O.sigma(f32(0.03), f32(0.05), 64) - f32(0.03) * f32(0.05) / 8.0) <= ulp32(0.03 * 0.05 / 8)


def _nearest_f32(fr):
    """Nearest float32 to an exact Fraction, ties to even (brute force over neighbours)."""
    from fractions import Fraction
    x = np.float32(float(fr))
    cands = [np.nextafter(x, np.float32(-np.inf)), x, np.nextafter(x, np.float32(np.inf))]
    best = min(cands, key=lambda c: (abs(Fraction(float(c)) - fr), int(np.float32(c).view(np.uint32)) & 1))
    return np.float32(best)


@pytest.mark.parametrize("n,sigma", [(3, 0.0), (7, 0.001), (64, 0.0004), (500, 0.0001)])
def test_attention_weights_are_nearest_float_of_exact_quotient(n, sigma):
    """P_j = E_j / Z rounded once to fp32 (E_j = rne(exp(s_j - max) 2^24) from the pinned exp)."""
    from fractions import Fraction
    q, K, V = _att_inputs(n + 5, n)
    sigma = f32(sigma)
    s = [f32(float(np.dot(K[j].astype(np.int64), q.astype(np.int64))) * sigma) for j in range(n)]
    m = max(s)
    E = [int(np.rint(np.float32(O.exp_own(f32(sj - m))) * np.float32(16777216.0))) for sj in s]
    Z = sum(E)
    P = O.attention_probs(q, K, sigma)
    for j in range(n):
        assert P[j] == _nearest_f32(Fraction(E[j], Z)), j


# ------------------------------------------------- beam log-softmax normaliser
def _lse64(l):
    l = l.astype(np.float64)
    m = l.max()
    return m + math.log(np.exp(l - m).sum())


def _lp_tolerance(l, lp, Z):
    """Bound of |lp - (l - logsumexp(l))| implied by the definition: the weights
    E_n = rne(exp_own(x) 2^24) carry exp_own's 2-ulp relative error and at most
    1/2 absolute rounding each, so ln Z is within (2^-21 Z + V/2) / Z of the
    exact value; fl32(lambda) adds half an ulp of lambda; fl(l - m) and
    fl(. - lambda) one half-ulp each."""
    V = l.shape[0]
    m = float(l.max())
    dlnz = (2.0 ** -21 * Z + 0.5 * V) / Z + 1e-14
    lam = math.log(Z) - 24 * math.log(2.0)
    return dlnz + 2.0 ** -24 * (abs(lam) + np.abs(l.astype(np.float64) - m) + np.abs(lp.astype(np.float64)))


@pytest.mark.parametrize("V,scale", [(8000, 0.1), (8000, 3.0), (32000, 0.1), (32000, 3.0), (32000, 30.0),
                                     (4, 1.0), (300, 10.0)])
def test_log_softmax_vs_float64(V, scale):
    """lp[n] = fl(fl(l - m) - lambda) against float64 l - logsumexp(l); a wrong
    constant (log2 for ln, a dropped 24 ln 2, a sign) is off by >= 0.3."""
    for row in range(3):
        l = (synth.Stream(V + row, "logit").normal(V) * scale).astype(np.float32)
        lp = O.log_softmax(l)
        ref = l.astype(np.float64) - _lse64(l)
        m, lam, Z = O.log_softmax_norm(l)
        assert m == float(l.max())
        tol = _lp_tolerance(l, lp, Z)
        assert np.all(np.abs(lp - ref) <= tol), float(np.max(np.abs(lp - ref) - tol))
        # probabilities sum to one (to the same bound)
        assert abs(math.log(np.exp(lp.astype(np.float64)).sum())) <= float(np.max(tol)) * 1.01


def test_log_softmax_equal_row_is_minus_ln_v():
    """All logits equal: every weight is exactly 2^24, Z = V 2^24, lambda = ln V."""
    for V in (4, 8000, 32000):
        l = np.full(V, 1.375, np.float32)
        m, lam, Z = O.log_softmax_norm(l)
        assert Z == V * 2 ** 24
        assert abs(lam - math.log(V)) <= ulp32(math.log(V))
        lp = O.log_softmax(l)
        assert np.all(lp == np.float32(-lam))


def test_log_softmax_spikes():
    """One logit far above the rest: Z = 2^24, lambda = 0 (to double rounding),
    lp = 0 at the spike and l - m elsewhere; two equal spikes: lambda = ln 2."""
    l = np.full(32000, -50.0, np.float32); l[123] = 60.0
    m, lam, Z = O.log_softmax_norm(l)
    assert Z == 2 ** 24 and abs(lam) <= 1e-14
    lp = O.log_softmax(l)
    assert abs(float(lp[123])) <= 1e-14 and np.all(lp[np.arange(32000) != 123] == np.float32(-110.0))
    l[9] = 60.0
    m, lam, Z = O.log_softmax_norm(l)
    assert Z == 2 ** 25 and lam == f32(math.log(2.0))
    lp = O.log_softmax(l)
    assert lp[9] == lp[123] == np.float32(-f32(math.log(2.0)))


def test_beam_search_scores_use_the_pinned_log_softmax():
    """The cumulative score of a beam-1 search is the sum of the pinned
    log-probabilities of its own tokens along the teacher-forced trace."""
    cfg = synth.ModelConfig(1, 1, 64, 2, 128, 300, 64, 1, 1, max_pos=32)
    blob = synth.build_blob(cfg, 5)
    ids, lens = synth.source_batch(cfg.vocab, 1, 6, 6, 8)
    T = 6
    out, olen, sc = O.translate(blob, ids, lens, -1, T)
    n = int(olen[0])
    tgt = np.concatenate([[cfg.bos_id], out[0, :n - 1]]).astype(np.int32)
    logits, _ = O.decode_trace(blob, ids[0], lens[0], tgt, cfg)
    cum = np.float32(0.0)
    for t in range(n):
        cum = np.float32(cum + O.log_softmax(logits[t])[out[0, t]])
    ref = sum(float(l[out[0, t]]) - _lse64(l) for t, l in enumerate(logits[:n]))
    assert sc[0] == cum
    assert abs(float(sc[0]) - ref) <= 1e-4 * n


# ------------------------------------------- LayerNorm statistics, any width
def _grid_sum(vals, shift):
    """Exact sum of round-half-even(v * 2^shift) over float32 values v."""
    from fractions import Fraction
    tot = 0
    for v in vals:
        x = Fraction(float(v)) * (Fraction(2) ** shift)
        fl = x.numerator // x.denominator
        rem = x - fl
        if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
            fl += 1
        tot += fl
    return tot


@pytest.mark.parametrize("d", [96, 128, 384, 640, 768, 1152, 1536, 2048])
@pytest.mark.parametrize("scale", [1e-30, 1e-3, 1.0, 700.0, 3e6])
def test_layernorm_statistics_are_nearest_floats_of_exact_sums(d, scale):
    """Mean and biased variance (R5): each the nearest float to its exact
    fixed-point sum over d, for widths with odd factors (d = 384, 768, ... of
    the 20MB model) as well as powers of two; and within half an ulp plus the
    grid's rounding of the exact mean of the row."""
    from fractions import Fraction
    r = (synth.Stream(d, f"ln{scale}").normal(4 * d).reshape(4, d) * scale + scale * 0.25).astype(np.float32)
    r[3, ::7] = np.float32(-scale * 2.5)
    mu, var = O.ln_stats(r)
    for m in range(4):
        row = r[m]
        amax = float(np.max(np.abs(row)))
        ea = math.frexp(amax)[1]
        s1 = _grid_sum(row, 52 - ea)
        exact_mu = Fraction(s1) * Fraction(2) ** (ea - 52) / d
        assert mu[m] == _nearest_f32(exact_mu), (d, scale, m)
        true_mean = sum(Fraction(float(v)) for v in row) / d
        assert abs(Fraction(float(mu[m])) - true_mean) <= Fraction(ulp32(float(mu[m]))) / 2 + \
            Fraction(2) ** (ea - 52)
        c = (row - mu[m]).astype(np.float32)
        c2 = (c * c).astype(np.float32)
        eb = math.frexp(float(np.max(np.abs(c))))[1]
        s2 = _grid_sum(c2, 52 - 2 * eb)
        assert var[m] == _nearest_f32(Fraction(s2) * Fraction(2) ** (2 * eb - 52) / d), (d, scale, m)
