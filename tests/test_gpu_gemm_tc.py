"""Parity of the tensor-core (tcgen05) quantised linear with the CPU oracle,
through the C ABI (mnmt_codes_to_f16, mnmt_linear_tc).  The int8 codes travel
as fp16 and the fp32 accumulation is exact per chunk of 1024 products, so every
output must equal the oracle's int32-accumulator result bit for bit (Sec. 3.3,
Eq. 3 and the Fig. 5 epilogues)."""
import time

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


def f16_codes(a_dev):
    """fp16 copy of a device int8 tensor, made by the library's converter."""
    out = torch.empty(a_dev.shape, dtype=torch.float16, device="cuda")
    mnmt.mnmt_codes_to_f16(a_dev, out, a_dev.numel())
    return out


def _inputs(seed, M, N, K, lo=-127, hi=127):
    A = synth.uniform_int8(seed, "A", (M, K), lo, hi)
    W = synth.uniform_int8(seed, "W", (N, K), lo, hi)
    s_w = synth.uniform_f32(seed, "sw", (N,), 1e-4, 3e-4)
    b = synth.uniform_f32(seed, "b", (N,), -0.5, 0.5)
    inv = synth.uniform_f32(seed, "inv", (N,), 0.5, 2.0)
    return A, W, s_w, b, inv, np.float32(0.02)


def _tc(A, W, s_w, b, inv, s_x, mode, gamma=1.0, resid=None, keys=None):
    M, K = A.shape
    N = W.shape[0]
    A16, W16 = f16_codes(dev(A)), f16_codes(dev(W))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out_q = out_f = None
    if mode in (mnmt.EPI_Q8, mnmt.EPI_RELU_Q8):
        out_q = torch.zeros((M, N), dtype=torch.int8, device="cuda")
    elif mode == mnmt.EPI_RESID:
        out_f = dev(resid.copy())
    elif mode == mnmt.EPI_F32:
        out_f = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    mnmt.mnmt_linear_tc(A16, W16, dev(s_w), dev(b), s_x, dev(inv), gamma, M, N, K, mode, out_q, out_f, keys, status)
    assert host(status)[0] == 0
    if mode == mnmt.EPI_ARGMAX:
        return None
    return host(out_q if out_q is not None else out_f)


def _same(got, ref):
    assert got.dtype == ref.dtype and got.shape == ref.shape
    v = np.uint8 if got.dtype == np.int8 else np.uint32
    return np.array_equal(got.view(v), ref.view(v))


def test_codes_to_f16_is_exact():
    codes = np.concatenate([np.arange(-128, 128, dtype=np.int8), synth.uniform_int8(3, "c", (4133,), -128, 127)])
    out = torch.empty(codes.size, dtype=torch.float16, device="cuda")
    mnmt.mnmt_codes_to_f16(dev(codes), out, codes.size)
    assert np.array_equal(host(out).view(np.uint16), codes.astype(np.float16).view(np.uint16))


# shapes: partial M tile, exact tiles, ragged N, K tails inside a k-block,
# exactly one 1024-chunk, two chunks (K > 1024), the smallest K
TC_SHAPES = [(1, 40, 64), (128, 128, 64), (129, 300, 512), (300, 1100, 2048), (1000, 96, 128),
             (256, 1000, 1032), (200, 130, 8), (513, 200, 1024), (130, 64, 1040), (384, 2048, 520)]


@pytest.mark.parametrize("M,N,K", TC_SHAPES)
@pytest.mark.parametrize("mode", [mnmt.EPI_Q8, mnmt.EPI_RELU_Q8, mnmt.EPI_RESID, mnmt.EPI_F32])
def test_linear_tc_matches_oracle(M, N, K, mode):
    A, W, s_w, b, inv, s_x = _inputs(M * 13 + N + K, M, N, K)
    resid = synth.uniform_f32(6, "r", (M, N), -3, 3) if mode == mnmt.EPI_RESID else None
    gamma = np.float32(0.875)
    got = _tc(A, W, s_w, b, inv, s_x, mode, gamma, resid)
    ref = O.linear(A, W, s_w, b, s_x, mode, inv_out=inv, gamma=gamma, resid=resid)
    assert _same(got, ref)


@pytest.mark.parametrize("K", [1024, 2048])
def test_linear_tc_extreme_accumulators(K):
    """The largest chunk sums: 1024 products of 127 * 127 (16,516,096) and of
    -128 * -128 (exactly 2^24) must come back exact; K = 2048 adds two chunks."""
    M, N = 256, 192
    for code in (127, -128):
        A = np.full((M, K), code, np.int8)
        A[1::2] = -127
        W = np.full((N, K), code, np.int8)
        W[::3] = -127
        W[5::7, : K // 3] = 3
        s_w = np.full(N, 1e-6, np.float32)
        b = np.zeros(N, np.float32)
        got = _tc(A, W, s_w, b, np.ones(N, np.float32), np.float32(1.0), mnmt.EPI_F32)
        ref = O.linear(A, W, s_w, b, 1.0, O.MODE_F32)
        assert _same(got, ref), code


@pytest.mark.parametrize("M,K", [(128, 256), (512, 512), (1000, 256)])
def test_linear_tc_vocab_argmax(M, K):
    """Fused vocabulary projection + greedy argmax on the tensor cores (ties to the lowest id)."""
    N = 32000
    A, W, s_w, b, inv, s_x = _inputs(M + K + 5, M, N, K)
    W[7] = W[3]
    s_w[7] = s_w[3]
    b[7] = b[3]
    keys = torch.zeros(M, dtype=torch.int64, device="cuda")
    _tc(A, W, s_w, b, inv, s_x, mnmt.EPI_ARGMAX, keys=keys)
    got = mnmt.argmax_from_keys(host(keys))
    logits = O.linear(A, W, s_w, b, s_x, O.MODE_F32)
    assert np.array_equal(got, np.argmax(logits, axis=1))


def test_linear_tc_equals_imma_path():
    """The two GPU paths of the same linear agree bit for bit."""
    M, N, K = 640, 768, 512
    A, W, s_w, b, inv, s_x = _inputs(77, M, N, K)
    got = _tc(A, W, s_w, b, inv, s_x, mnmt.EPI_Q8)
    out = torch.zeros((M, N), dtype=torch.int8, device="cuda")
    mnmt.mnmt_linear(dev(A), dev(W), dev(s_w), dev(b), s_x, dev(inv), 1.0, M, N, K, mnmt.EPI_Q8, out, None)
    assert np.array_equal(got, host(out))


SWEEP_M = [256, 1024, 4096]
SWEEP_KN = [(256, 1024), (1024, 256), (512, 2048), (2048, 512), (256, 32000)]


@pytest.mark.parametrize("K,N", SWEEP_KN)
def test_linear_tc_sweep_full_size_sampled_rows(K, N):
    """The tensor-core shapes of the int8 linear microbenchmark at full size (E1
    epilogue), checked on sampled rows that the oracle computes one by one."""
    for M in SWEEP_M:
        A, W, s_w, b, inv, s_x = _inputs(M + K + 1, M, N, K)
        got = _tc(A, W, s_w, b, inv, s_x, mnmt.EPI_Q8)
        rows = sorted({0, 127, 128, M - 1, M // 2, (M * 7) // 11})
        ref = O.linear(A[rows], W, s_w, b, s_x, O.MODE_Q8, inv_out=inv)
        assert np.array_equal(got[rows], ref), (M, K, N)


def test_linear_tc_rejects_bad_shapes():
    A16 = torch.zeros((256, 24), dtype=torch.float16, device="cuda")
    W16 = torch.zeros((64, 24), dtype=torch.float16, device="cuda")
    s = torch.ones(64, dtype=torch.float32, device="cuda")
    out = torch.zeros((256, 64), dtype=torch.float32, device="cuda")
    for K in (12, 4096):    # not a multiple of 8; above two chunks
        with pytest.raises(mnmt.MnmtError):
            mnmt.mnmt_linear_tc(A16, W16, s, s, 1.0, s, 1.0, 256, 64, K, mnmt.EPI_F32, None, out)
    with pytest.raises(mnmt.MnmtError):
        mnmt.mnmt_linear_tc(A16, W16, s, s, 1.0, s, 1.0, 256, 64, 24, mnmt.EPI_Q8, None, out)


@pytest.mark.parametrize("M,N,K", [(4864, 1024, 1040), (4864, 1000, 520), (19456, 512, 2048)])
@pytest.mark.parametrize("mode", [mnmt.EPI_Q8, mnmt.EPI_RESID])
def test_linear_tc_wide_tiles_sampled(M, N, K, mode):
    """Grids large enough for the 128 x 256 tiles (with one and with two exact
    K chunks, ragged N and K), checked on sampled rows."""
    A, W, s_w, b, inv, s_x = _inputs(M + N + K + 3, M, N, K)
    resid = synth.uniform_f32(9, "r", (M, N), -3, 3) if mode == mnmt.EPI_RESID else None
    got = _tc(A, W, s_w, b, inv, s_x, mode, 0.875, resid)
    rows = sorted({0, 127, 128, 129, 255, 256, M // 3, M - 129, M - 1})
    ref = O.linear(A[rows], W, s_w, b, s_x, mode, inv_out=inv, gamma=np.float32(0.875),
                   resid=None if resid is None else resid[rows])
    assert _same(got[rows], ref)


def test_bounded_wait_gives_up_with_status():
    """The give-up path of the pipelines' barrier waits: a wait that nothing
    completes returns after its one-second limit with MNMT_ETIMEOUT in the
    status word (no fault), and the device keeps working: a linear launched
    afterwards is still exact."""
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    mnmt.mnmt_wait_timeout_selftest(status)
    assert host(status)[0] == mnmt.ETIMEOUT
    assert 0.5 < time.perf_counter() - t0 < 60
    A, W, s_w, b, inv, s_x = _inputs(5, 200, 96, 512)
    got = _tc(A, W, s_w, b, inv, s_x, mnmt.EPI_Q8)
    assert _same(got, O.linear(A, W, s_w, b, s_x, mnmt.EPI_Q8, inv_out=inv))
