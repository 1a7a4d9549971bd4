"""Pins of the oracle's fake quantisation (QAT forward / backward; App. B "PTQ
and QAT": the quantiser of Eq. quant inserted into the float model, its scale
s learnable) and of the QAT forward of a linear (no GPU)."""
import math

import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import synth


def _x(seed, n, scale=1.0):
    return (synth.Stream(seed, "fq").normal(n) * scale).astype(np.float32)


@pytest.mark.parametrize("bits,minmax", [(8, False), (4, False), (8, True), (4, True), (2, False)])
def test_grid_points_are_fixed_points(bits, minmax):
    """Q(Q(x)) = Q(x), and values already on the grid come back unchanged."""
    s, r = np.float32(0.0375), np.float32(-0.3)
    x = _x(bits, 2000, 0.5)
    y, q = O.fake_quant(x, s, bits, r, minmax)
    y2, q2 = O.fake_quant(y, s, bits, r, minmax)
    assert np.array_equal(q, q2) and np.array_equal(y, y2)


@pytest.mark.parametrize("bits,minmax", [(8, False), (4, False), (8, True), (4, True)])
def test_error_at_most_half_a_step_inside_the_range(bits, minmax):
    """float64 brute force: |Q(x) - x| <= s/2 (plus fp32 rounding) where x is
    inside the representable range; outside, Q(x) is the end of the range."""
    s, r = np.float32(0.02), np.float32(-0.25)
    x = _x(10 + bits, 4000, 0.3)
    y, q = O.fake_quant(x, s, bits, r, minmax)
    lo, hi = (0, 2 ** bits - 1) if minmax else (-(2 ** (bits - 1) - 1), 2 ** (bits - 1) - 1)
    off = float(r) if minmax else 0.0
    v = (x.astype(np.float64) - off) / float(s)
    inside = (v >= lo) & (v <= hi)
    err = np.abs(y.astype(np.float64) - x.astype(np.float64))
    assert np.all(err[inside] <= float(s) / 2 * (1 + 1e-5) + 1e-7)
    assert np.all(q[v < lo - 0.5] == lo) and np.all(q[v > hi + 0.5] == hi)
    assert np.all((q >= lo) & (q <= hi))


def test_symmetric_8bit_equals_the_inference_quantiser():
    """The symmetric 8-bit fake quantiser's codes are the inference q8 codes."""
    s = np.float32(4.0 / 127)
    x = _x(3, 1000, 2.0)
    _, q = O.fake_quant(x, s, 8)
    inv = np.float32(1.0) / s
    assert np.array_equal(q, np.array([O.q8(float(v), float(inv)) for v in x], np.int32))


@pytest.mark.parametrize("minmax", [False, True])
def test_backward_matches_finite_differences_of_the_expression(minmax):
    """dL/ds and dL/dr_m (rounding held fixed, STE) against float64 central
    differences of L = sum g * (s q + r) with q frozen at its code (in range)
    and the clamp's end (out of range); dL/dx is g inside the range, 0 outside."""
    s, r, bits = np.float32(0.05), np.float32(-0.4), 4
    x = _x(7, 3000, 0.4)
    g = _x(8, 3000, 1.0)
    gx, gs, gr = O.fake_quant_backward(x, g, s, bits, r, minmax)
    lo, hi = (0, 15) if minmax else (-7, 7)
    off = float(r) if minmax else 0.0
    inv = np.float32(1.0) / s
    t = ((x - np.float32(off)) * inv).astype(np.float64) if minmax else (x * inv).astype(np.float64)
    inside = (t >= lo) & (t <= hi)
    q = np.clip(np.rint(t), lo, hi)
    assert np.array_equal(gx, np.where(inside, g, np.float32(0)))
    # STE: inside, y = s * (t_exact rounded) with d(round)/dt := 1 -> dy/ds = q - t
    ref_s = float(np.sum(g.astype(np.float64) * np.where(inside, q - t, q)))
    assert abs(gs - ref_s) <= 1e-9 * (1 + abs(ref_s))
    if minmax:
        assert abs(gr - float(np.sum(g.astype(np.float64) * (~inside)))) <= 1e-9 * (1 + abs(gr))
    # finite differences of the frozen-code expression: d/ds sum g (s q_in + ...) matches the clamped part
    eps = 1e-6
    def L(ss):
        tt = (x.astype(np.float64) - off) / ss
        qq = np.where(inside, tt, q)          # STE: the rounding's derivative taken as 1 inside
        return float(np.sum(g.astype(np.float64) * (ss * np.where(inside, q - t + tt, qq) + off)))
    fd = (L(float(s) + eps) - L(float(s) - eps)) / (2 * eps)
    assert abs(fd - ref_s) <= 1e-3 * (1 + abs(ref_s))


@pytest.mark.parametrize("wbits", [8, 4])
def test_fake_quant_linear_equals_float64_of_the_dequantised_operands(wbits):
    M, N, K = 5, 40, 256
    X = _x(1, M * K, 0.8).reshape(M, K)
    W = synth.weight_draw(synth.Stream(2, "w"), N, K, 0.05).astype(np.float32)
    s_x = np.float32(4.0 / 127)
    qmax = 2 ** (wbits - 1) - 1
    s_w = (np.abs(W).max(axis=1) / qmax).astype(np.float32)
    b = synth.uniform_f32(3, "b", (N,), -0.1, 0.1)
    y = O.fake_quant_linear(X, W, s_x, s_w, b, wbits)
    xq, _ = O.fake_quant(X, s_x, 8)
    wq = np.stack([O.fake_quant(W[n], s_w[n], wbits)[0] for n in range(N)])
    ref = xq.astype(np.float64) @ wq.astype(np.float64).T + b
    mag = np.abs(xq.astype(np.float64)) @ np.abs(wq.astype(np.float64)).T + np.abs(b)
    assert np.all(np.abs(y - ref) <= 4 * 2.0 ** -24 * mag + 1e-12)
    # and exactly the inference linear on the same codes
    _, qx = O.fake_quant(X, s_x, 8)
    qw = np.stack([O.fake_quant(W[n], s_w[n], wbits)[1] for n in range(N)])
    y8 = O.linear(qx.astype(np.int8), qw.astype(np.int8), s_w, b, s_x, O.MODE_F32)
    assert np.array_equal(y.view(np.uint32), y8.view(np.uint32))
