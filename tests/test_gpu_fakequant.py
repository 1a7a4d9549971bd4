"""Fake quantisation for quantisation-aware training on the GPU (App. B "PTQ
and QAT": Eq. quant with a learnable scale, symmetric or min-max with offset):
forward values and codes bit-exact against the oracle, the straight-through
gradient exact and the scale / offset gradients to fp64 summation order, and
the QAT forward of a linear bit-exact against the oracle."""
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


def _x(seed, n, scale):
    return (synth.Stream(seed, "gfq").normal(n) * scale).astype(np.float32)


@pytest.mark.parametrize("bits,minmax", [(8, False), (4, False), (2, False), (8, True), (4, True)])
@pytest.mark.parametrize("n", [1, 1000, 1 << 20])
def test_fake_quant_forward_and_backward(bits, minmax, n):
    s, r = np.float32(0.03125 * 1.37), np.float32(-0.2)
    x = _x(n + bits, n, 0.6)
    g = _x(n + 7, n, 1.0)
    y = torch.empty(n, dtype=torch.float32, device="cuda")
    q = torch.empty(n, dtype=torch.int32, device="cuda")
    dx, dg = dev(x), dev(g)
    mnmt.mnmt_fake_quant(dx, n, s, r, bits, minmax, y, q)
    ry, rq = O.fake_quant(x, s, bits, r, minmax)
    assert np.array_equal(host(y).view(np.uint32), ry.view(np.uint32))
    assert np.array_equal(host(q), rq)
    gx = torch.empty(n, dtype=torch.float32, device="cuda")
    gs = torch.empty(1, dtype=torch.float64, device="cuda")
    gr = torch.empty(1, dtype=torch.float64, device="cuda")
    mnmt.mnmt_fake_quant_backward(dx, dg, n, s, gx, gs, gr, r, bits, minmax)
    rgx, rgs, rgr = O.fake_quant_backward(x, g, s, bits, r, minmax)
    assert np.array_equal(host(gx).view(np.uint32), rgx.view(np.uint32))
    scale = float(np.sum(np.abs(g.astype(np.float64)))) * (2 ** bits) + 1.0
    assert abs(float(host(gs)[0]) - rgs) <= 1e-13 * scale
    assert abs(float(host(gr)[0]) - rgr) <= 1e-13 * scale


@pytest.mark.parametrize("M,N,K", [(1, 1024, 256), (5, 300, 512), (40, 768, 256), (130, 512, 1024)])
@pytest.mark.parametrize("wbits", [8, 4])
def test_fake_quant_linear_matches_oracle(M, N, K, wbits):
    X = _x(M * 3 + K, M * K, 0.7).reshape(M, K)
    W = synth.weight_draw(synth.Stream(N, "w"), N, K, 0.05).astype(np.float32)
    qmax = 2 ** (wbits - 1) - 1
    s_w = (np.abs(W).max(axis=1) / qmax * 1.1).astype(np.float32)     # learnable scales: any positive values
    s_x = np.float32(3.5 / 127)
    b = synth.uniform_f32(M, "b", (N,), -0.2, 0.2)
    ws = torch.empty(((M * K + 15) // 16) * 16 + N * K, dtype=torch.int8, device="cuda")
    y = torch.empty((M, N), dtype=torch.float32, device="cuda")
    mnmt.mnmt_fake_quant_linear(dev(X), dev(W), s_x, dev(s_w), dev(b), M, N, K, wbits, ws, y)
    ref = O.fake_quant_linear(X, W, s_x, s_w, b, wbits)
    assert np.array_equal(host(y).view(np.uint32), ref.view(np.uint32))


def test_fake_quant_rejects_bad_scale():
    x = torch.zeros(4, dtype=torch.float32, device="cuda")
    with pytest.raises(mnmt.MnmtError) as ei:
        mnmt.mnmt_fake_quant(x, 4, 0.0, y=x)
    assert ei.value.code == mnmt.EINVAL
