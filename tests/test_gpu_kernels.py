"""Kernel-level parity of the sm_103a kernels against the CPU oracle, through the
C ABI (mnmt_linear, mnmt_attention_decode, mnmt_layernorm).  Integer and int8
outputs must match bit for bit; the fp32 outputs are bit-identical too, since
both sides follow the same IEEE operation sequence (Sec. 3.3 / Fig. 5 linear
epilogues, Eq. 1/2 attention, App. A LayerNorm)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def _lin_inputs(seed, M, N, K):
    A = synth.uniform_int8(seed, "A", (M, K))
    W = synth.uniform_int8(seed, "W", (N, K))
    s_w = synth.uniform_f32(seed, "sw", (N,), 1e-4, 3e-4)
    b = synth.uniform_f32(seed, "b", (N,), -0.5, 0.5)
    inv = synth.uniform_f32(seed, "inv", (N,), 0.5, 2.0)
    s_x = np.float32(0.02)
    return A, W, s_w, b, inv, s_x


def _gpu_linear(A, W, s_w, b, inv, s_x, mode, gamma=1.0, resid=None):
    M, K = A.shape
    N = W.shape[0]
    dA, dW, ds, db, di = dev(A), dev(W), dev(s_w), dev(b), dev(inv)
    out_q = out_f = None
    if mode in (mnmt.EPI_Q8, mnmt.EPI_RELU_Q8):
        out_q = torch.zeros((M, N), dtype=torch.int8, device="cuda")
    elif mode == mnmt.EPI_RESID:
        out_f = dev(resid.copy())
    else:
        out_f = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    mnmt.mnmt_linear(dA, dW, ds, db, s_x, di, gamma, M, N, K, mode, out_q, out_f)
    return host(out_q if out_q is not None else out_f)


LIN_SHAPES = [(1, 40, 64), (1, 1000, 256), (2, 33, 2048), (3, 777, 128), (16, 256, 1024), (17, 200, 64),
              (64, 1024, 256), (129, 300, 512), (300, 1100, 2048), (1000, 96, 128)]


@pytest.mark.parametrize("M,N,K", LIN_SHAPES)
@pytest.mark.parametrize("mode", [mnmt.EPI_Q8, mnmt.EPI_RELU_Q8, mnmt.EPI_RESID, mnmt.EPI_F32])
def test_linear_matches_oracle(M, N, K, mode):
    A, W, s_w, b, inv, s_x = _lin_inputs(M * 7 + N + K, M, N, K)
    resid = synth.uniform_f32(5, "r", (M, N), -3, 3) if mode == mnmt.EPI_RESID else None
    gamma = np.float32(0.875)
    got = _gpu_linear(A, W, s_w, b, inv, s_x, mode, gamma, resid)
    ref = O.linear(A, W, s_w, b, s_x, mode, inv_out=inv, gamma=gamma, resid=resid)
    assert got.dtype == ref.dtype
    assert np.array_equal(got.view(np.uint8) if got.dtype == np.int8 else got.view(np.uint32),
                          ref.view(np.uint8) if ref.dtype == np.int8 else ref.view(np.uint32))


def test_linear_extreme_accumulators():
    """|acc| up to 2048 * 127^2 (K = 2048, all +-127): exact int32 on both paths."""
    M, N, K = 40, 64, 2048
    A = np.full((M, K), 127, np.int8); A[1::2] = -127
    W = np.full((N, K), 127, np.int8); W[::3] = -127
    s_w = np.full(N, 1e-6, np.float32); b = np.zeros(N, np.float32)
    for Mx in (M, 8):
        got = _gpu_linear(A[:Mx], W, s_w, b, np.ones(N, np.float32), np.float32(1.0), mnmt.EPI_F32)
        ref = O.linear(A[:Mx], W, s_w, b, 1.0, O.MODE_F32)
        assert np.array_equal(got, ref)


@pytest.mark.parametrize("M", [1, 3, 16, 17, 128, 512])
def test_vocab_argmax_matches_oracle(M):
    """Fused vocabulary projection + greedy argmax (ties to the lowest id)."""
    N, K = 32000, 256
    A, W, s_w, b, inv, s_x = _lin_inputs(M + 99, M, N, K)
    W[7] = W[3]; s_w[7] = s_w[3]; b[7] = b[3]          # an exact tie between ids 3 and 7
    keys = torch.zeros(M, dtype=torch.int64, device="cuda")
    mnmt.mnmt_linear_argmax(dev(A), dev(W), dev(s_w), dev(b), s_x, M, N, K, keys)
    got = mnmt.argmax_from_keys(host(keys))
    logits = O.linear(A, W, s_w, b, s_x, O.MODE_F32)
    assert np.array_equal(got, np.argmax(logits, axis=1))   # numpy: first maximum = lowest id


SWEEP_M = [1, 4, 16, 64, 256, 1024, 4096]
SWEEP_KN = [(256, 1024), (1024, 256), (512, 2048), (2048, 512), (256, 32000)]


@pytest.mark.parametrize("K,N", SWEEP_KN)
def test_linear_sweep_full_size_sampled_rows(K, N):
    """The int8 linear microbenchmark shapes at full size (E1 epilogue), checked
    on sampled rows that the oracle computes one by one."""
    for M in SWEEP_M:
        A, W, s_w, b, inv, s_x = _lin_inputs(M + K, M, N, K)
        got = _gpu_linear(A, W, s_w, b, inv, s_x, mnmt.EPI_Q8)
        rows = sorted({0, M - 1, M // 2, (M * 7) // 11})
        ref = O.linear(A[rows], W, s_w, b, s_x, O.MODE_Q8, inv_out=inv)
        assert np.array_equal(got[rows], ref), (M, K, N)


ATT_CASES = [(1, 4, 64, 1), (1, 4, 64, 64), (3, 4, 32, 37), (5, 8, 64, 160), (2, 2, 128, 512), (4, 16, 64, 1024)]


@pytest.mark.parametrize("R,H,dh,T", ATT_CASES)
def test_attention_decode_matches_oracle(R, H, dh, T):
    seed = R * 1000 + H * 10 + T
    q = synth.uniform_int8(seed, "q", (R, H, dh))
    Kc = synth.uniform_int8(seed, "k", (R, H, T, dh))
    Vc = synth.uniform_int8(seed, "v", (R, H, T, dh))
    n_keys = synth.Stream(seed, "n").randint(1, T, R).astype(np.int32)
    n_keys[0] = T
    sigma, rho = np.float32(3e-5), np.float32(0.7)
    ctx = torch.zeros((R, H, dh), dtype=torch.int8, device="cuda")
    mnmt.mnmt_attention_decode(dev(q), dev(Kc), dev(Vc), dev(n_keys), R, H, dh, T, sigma, rho, ctx)
    ref = O.attention_decode(q, Kc, Vc, n_keys, sigma, rho)
    assert np.array_equal(host(ctx), ref)


def test_attention_decode_full_size_sampled():
    """Cache length 512, 512 rows x 8 heads (the batched-beam shape): rows sampled."""
    R, H, dh, T = 512, 8, 64, 512
    q = synth.uniform_int8(9, "q", (R, H, dh))
    Kc = synth.uniform_int8(9, "k", (R, H, T, dh))
    Vc = synth.uniform_int8(9, "v", (R, H, T, dh))
    n_keys = synth.Stream(9, "n").randint(1, T, R).astype(np.int32)
    sigma, rho = np.float32(2e-5), np.float32(0.9)
    ctx = torch.zeros((R, H, dh), dtype=torch.int8, device="cuda")
    mnmt.mnmt_attention_decode(dev(q), dev(Kc), dev(Vc), dev(n_keys), R, H, dh, T, sigma, rho, ctx)
    got = host(ctx)
    rows = [0, 1, 255, 511]
    ref = O.attention_decode(q[rows], Kc[rows], Vc[rows], n_keys[rows], sigma, rho)
    assert np.array_equal(got[rows], ref)


LN_CASES = [(1, 128, 1.0), (7, 256, 30.0), (33, 512, 700.0), (5, 2048, 1e-3), (100, 1024, 3.0), (1, 64, 1e6),
            # widths with an odd factor (the 20MB model's d = 384), decode and encoder block sizes
            (3, 384, 1.0), (1500, 384, 30.0), (9, 768, 1e-3), (4, 1152, 700.0), (2, 96, 3e6), (5, 1536, 1e-30)]


@pytest.mark.parametrize("M,d,scale", LN_CASES)
def test_layernorm_matches_oracle(M, d, scale):
    r = (synth.Stream(M + d, "r").normal(M * d).reshape(M, d) * scale + scale * 0.1).astype(np.float32)
    r[0, : d // 2] = 7.0  # repeated values
    g = synth.uniform_f32(d, "g", (d,), 0.5, 1.5)
    b = synth.uniform_f32(d, "b", (d,), -0.2, 0.2)
    inv = np.float32(127 / 4.0)
    of = torch.zeros((M, d), dtype=torch.float32, device="cuda")
    oq = torch.zeros((M, d), dtype=torch.int8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    mnmt.mnmt_layernorm(dev(r), dev(g), dev(b), M, d, inv, of, oq, status)
    ref_f, ref_q = O.layernorm(r, g, b, inv)
    assert host(status)[0] == 0
    assert np.array_equal(host(of).view(np.uint32), ref_f.view(np.uint32))
    assert np.array_equal(host(oq), ref_q)


def test_layernorm_wide_magnitude_rows():
    """Rows whose terms land on every branch of the fixed-point conversion: one
    large value sets the grid, the others scale to integers far above 2^23,
    to values just below 2^23 with .5 fractions (rounded half to even), and to
    values under 1/2 (rounded to zero)."""
    M, d = 6, 512
    st = synth.Stream(77, "w")
    r = np.zeros((M, d), np.float32)
    for m in range(M):
        big = np.float32(2.0 ** (20 - 3 * m))
        e = st.randint(-44 - 3 * m, -4 - 3 * m, d)                  # exponents around the 2^23 boundary of the grid
        odd = (2 * st.randint(0, 1 << 22, d) + 1).astype(np.float64)  # odd significands: .5 fractions after scaling
        sign = np.where(st.randint(0, 2, d) == 1, -1.0, 1.0)
        r[m] = (sign * odd * np.exp2(e.astype(np.float64) - 23)).astype(np.float32)
        r[m, 3] = big
        r[m, 100] = -big / 2
    g = synth.uniform_f32(5, "g", (d,), 0.5, 1.5)
    b = synth.uniform_f32(5, "b", (d,), -0.2, 0.2)
    inv = np.float32(127 / 4.0)
    of = torch.zeros((M, d), dtype=torch.float32, device="cuda")
    oq = torch.zeros((M, d), dtype=torch.int8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    mnmt.mnmt_layernorm(dev(r), dev(g), dev(b), M, d, inv, of, oq, status)
    ref_f, ref_q = O.layernorm(r, g, b, inv)
    assert host(status)[0] == 0
    assert np.array_equal(host(of).view(np.uint32), ref_f.view(np.uint32))
    assert np.array_equal(host(oq), ref_q)


def test_layernorm_constant_row_and_overflow_status():
    d = 256
    g = np.ones(d, np.float32); b = synth.uniform_f32(1, "b", (d,), -1, 1)
    r = np.full((2, d), 5.5, np.float32)
    r[1, 7] = 2.0 ** 33                                   # outside the fixed-point domain
    of = torch.zeros((2, d), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    mnmt.mnmt_layernorm(dev(r), dev(g), dev(b), 2, d, 1.0, of, None, status)
    assert np.array_equal(host(of)[0], b)
    assert host(status)[0] == mnmt.EOVERFLOW


@pytest.mark.parametrize("rho", [0.5, 1.0, 0.25])
def test_attention_context_on_rounding_ties(rho):
    """Equal scores make the context an exact mean of the values; with these
    rho the scaled context lands exactly on (or next to) .5 rounding ties, so
    the kernel's approximate-quotient shortcut must defer to the exact
    quotient.  Both must agree with the oracle."""
    R, H, dh, T = 6, 4, 64, 8
    q = np.zeros((R, H, dh), np.int8)                         # all scores 0 -> equal weights
    Kc = synth.uniform_int8(31, "k", (R, H, T, dh))
    Vc = synth.uniform_int8(31, "v", (R, H, T, dh), -9, 9)
    Vc[:, :, 1::2] = Vc[:, :, 0::2] + 1                        # pair sums odd: means at .5 / .25 steps
    n_keys = np.array([2, 4, 8, 6, 1, 3], np.int32)
    sigma = np.float32(1e-3)
    ctx = torch.zeros((R, H, dh), dtype=torch.int8, device="cuda")
    mnmt.mnmt_attention_decode(dev(q), dev(Kc), dev(Vc), dev(n_keys), R, H, dh, T, sigma, np.float32(rho), ctx)
    ref = O.attention_decode(q, Kc, Vc, n_keys, sigma, np.float32(rho))
    assert np.array_equal(host(ctx), ref)
