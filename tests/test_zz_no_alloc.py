"""The allocation-free variant of the greedy vocabulary argmax
(mnmt_linear_argmax_ids_noalloc), for callers that cannot allocate device
memory: its ids must equal those of mnmt_linear_argmax (caller-provided keys)
on two calls in a row, since the library-owned scratch is reused and must be
cleared by each call.  Collected last so that a failure here does not stop the
other GPU tests."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _inputs(seed, M, N, K):
    A = torch.from_numpy(synth.uniform_int8(seed, "A", (M, K))).cuda()
    W = torch.from_numpy(synth.uniform_int8(seed, "W", (N, K))).cuda()
    s_w = torch.from_numpy(synth.uniform_f32(seed, "s", (N,), 1e-4, 3e-4)).cuda()
    b = torch.from_numpy(synth.uniform_f32(seed, "b", (N,), -0.5, 0.5)).cuda()
    return A, W, s_w, b


@pytest.mark.parametrize("M", [1, 5, 40])
def test_noalloc_argmax_equals_keyed_argmax_twice(M):
    N, K = 32000, 256
    stream = torch.cuda.current_stream()
    for call, seed in enumerate((M, M + 1000)):          # two calls in a row, different inputs
        A, W, s_w, b = _inputs(seed, M, N, K)
        ids = torch.full((M,), -1, dtype=torch.int32, device="cuda")
        mnmt.mnmt_linear_argmax_ids_noalloc(A, W, s_w, b, 0.02, M, N, K, ids, stream)
        keys = torch.zeros(M, dtype=torch.int64, device="cuda")
        mnmt.mnmt_linear_argmax(A, W, s_w, b, 0.02, M, N, K, keys, stream)
        torch.cuda.synchronize()
        ref = mnmt.argmax_from_keys(keys.cpu().numpy())
        assert np.array_equal(ids.cpu().numpy().astype(np.int64), ref), f"call {call}"


@pytest.mark.parametrize("M,N,K", [(4096, 32000, 256), (3, 8000, 2048), (16, 32000, 512)])
def test_noalloc_argmax_at_the_row_limit_and_long_k(M, N, K):
    """The full 4096-row scratch (tensor-core / IMMA tile path), and the GEMV
    path at K = 2048: two calls in a row equal the keyed call, and sampled rows
    equal the oracle's argmax of its fp32 logits (ties to the lowest id)."""
    stream = torch.cuda.current_stream()
    for call, seed in enumerate((7 * M + K, 7 * M + K + 1)):
        A, W, s_w, b = _inputs(seed, M, N, K)
        ids = torch.full((M,), -1, dtype=torch.int32, device="cuda")
        mnmt.mnmt_linear_argmax_ids_noalloc(A, W, s_w, b, 0.02, M, N, K, ids, stream)
        keys = torch.zeros(M, dtype=torch.int64, device="cuda")
        mnmt.mnmt_linear_argmax(A, W, s_w, b, 0.02, M, N, K, keys, stream)
        torch.cuda.synchronize()
        got = ids.cpu().numpy().astype(np.int64)
        assert np.array_equal(got, mnmt.argmax_from_keys(keys.cpu().numpy())), f"call {call}"
        rows = sorted({0, M // 3, M // 2, M - 1} | set(range(0, M, max(1, M // 12))))
        A_h = A.cpu().numpy()[rows]
        logits = O.linear(A_h, W.cpu().numpy(), s_w.cpu().numpy(), b.cpu().numpy(), 0.02, O.MODE_F32)
        assert np.array_equal(got[rows], np.argmax(logits, axis=1)), f"call {call}"


def test_noalloc_rejects_more_rows_than_its_scratch():
    A, W, s_w, b = _inputs(1, 1, 64, 64)
    ids = torch.zeros(4097, dtype=torch.int32, device="cuda")
    with pytest.raises(mnmt.MnmtError) as ei:
        mnmt.mnmt_linear_argmax_ids_noalloc(A, W, s_w, b, 0.02, 4097, 64, 64, ids)
    assert ei.value.code == mnmt.EINVAL
