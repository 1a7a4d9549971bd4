"""Row-wise 4-bit weights on the GPU (Sec. 3.3 row-wise low-bit weights; table
"quantizing weights to lower bits", 4-8-8), symmetric and min-max (App. B Eq.
scale / Eq. quant) rows: the 4-bit GEMV kernel bit-exact against the oracle
over ragged shapes and every epilogue, and whole translations of 4-bit models
(tokens, scores, intermediate taps) against the oracle."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt, synth
from tap_parity import check_taps

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def _case(seed, M, N, K, minmax):
    A = synth.uniform_int8(seed, "a", (M, K))
    W = synth.weight_draw(synth.Stream(seed, "w"), N, K, 0.05)
    stored, s, r = synth.int4_weight(W, minmax)
    b = synth.uniform_f32(seed, "b", (N,), -0.5, 0.5)
    return A, synth.pack4(stored), s, r, b


SHAPES = [(1, 1024, 256), (3, 33, 32), (4, 1000, 384), (5, 768, 768), (16, 512, 2048), (17, 300, 512),
          (40, 1536, 256), (100, 64, 1024), (2, 32000, 256)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("minmax", [False, True])
def test_linear_w4_matches_oracle(M, N, K, minmax):
    A, Wp, s, r, b = _case(M * 7 + K, M, N, K, minmax)
    s_x, inv, g = np.float32(0.02), synth.uniform_f32(3, "inv", (N,), 2.0, 20.0), np.float32(0.75)
    dA, dW, ds, dr, db, dinv = dev(A), dev(Wp), dev(s), dev(r) if minmax else None, dev(b), dev(inv)
    for mode in (mnmt.EPI_Q8, mnmt.EPI_RELU_Q8):
        out = torch.zeros((M, N), dtype=torch.int8, device="cuda")
        mnmt.mnmt_linear_w4(dA, dW, ds, dr, db, s_x, dinv, 1.0, M, N, K, mode, out_q=out)
        ref = O.linear_w4(A, Wp, s, r, b, s_x, mode, minmax, inv_out=inv)
        assert np.array_equal(host(out), ref), mode
    out = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    mnmt.mnmt_linear_w4(dA, dW, ds, dr, db, s_x, None, 1.0, M, N, K, mnmt.EPI_F32, out_f=out)
    ref = O.linear_w4(A, Wp, s, r, b, s_x, O.MODE_F32, minmax)
    assert np.array_equal(host(out).view(np.uint32), ref.view(np.uint32))
    r0 = synth.uniform_f32(5, "r0", (M, N), -3, 3)
    out = dev(r0)
    mnmt.mnmt_linear_w4(dA, dW, ds, dr, db, s_x, None, g, M, N, K, mnmt.EPI_RESID, out_f=out)
    ref = O.linear_w4(A, Wp, s, r, b, s_x, O.MODE_RESID, minmax, gamma=g, resid=r0)
    assert np.array_equal(host(out).view(np.uint32), ref.view(np.uint32))
    keys = torch.zeros(M, dtype=torch.int64, device="cuda")
    mnmt.mnmt_linear_w4(dA, dW, ds, dr, db, s_x, None, 1.0, M, N, K, mnmt.EPI_ARGMAX, keys=keys)
    logits = O.linear_w4(A, Wp, s, r, b, s_x, O.MODE_F32, minmax)
    assert np.array_equal(mnmt.argmax_from_keys(host(keys)), np.argmax(logits, axis=1))


def test_linear_w4_extreme_codes():
    """Codes 0 and 15 everywhere with activations +-127: the largest exact sums."""
    M, N, K = 4, 64, 2048
    A = np.full((M, K), 127, np.int8); A[1] = -127; A[2, ::2] = -127
    stored = np.full((N, K), 15, np.uint8); stored[::2] = 0; stored[5, ::3] = 7
    Wp = synth.pack4(stored)
    s = synth.uniform_f32(2, "s", (N,), 1e-3, 2e-3); r = synth.uniform_f32(2, "r", (N,), -0.02, 0.0)
    b = synth.uniform_f32(2, "b", (N,), -0.5, 0.5)
    for minmax in (False, True):
        out = torch.zeros((M, N), dtype=torch.float32, device="cuda")
        mnmt.mnmt_linear_w4(dev(A), dev(Wp), dev(s), dev(r) if minmax else None, dev(b), 0.01, None, 1.0, M, N, K,
                            mnmt.EPI_F32, out_f=out)
        ref = O.linear_w4(A, Wp, s, r if minmax else None, b, 0.01, O.MODE_F32, minmax)
        assert np.array_equal(host(out).view(np.uint32), ref.view(np.uint32))


@pytest.fixture(scope="module")
def stream():
    return torch.cuda.Stream()


def _translate(blob, ids, lens, beam, T, stream, lean=False):
    tr = mnmt.Translator(blob, ids.shape[0], ids.shape[1], beam, T, stream, lean=lean)
    try:
        return tr.translate(ids, lens, T)
    finally:
        tr.close()


@pytest.mark.parametrize("wq", [synth.WQ_INT4, synth.WQ_INT4_MINMAX])
def test_w4_batch1_workload_matches_oracle(wq, stream):
    """The batch-1 latency workload's model with 4-bit attention / FFN weights
    (encoder at 10-50 rows, decoder steps of 1 row), full size, plus taps."""
    wl = synth.WORKLOADS["small-b1-s10to50-greedy64"]
    cfg = synth.MODELS[wl.model]
    blob = synth.build_blob(cfg, wl.model_seed, wq=wq)
    ids, lens = synth.source_batch(cfg.vocab, 1, 10, 50, wl.src_seed)
    g = _translate(blob, ids, lens, 1, wl.max_len, stream)
    o = O.translate(blob, ids, lens, 1, wl.max_len)
    assert np.array_equal(g[0], o[0]) and np.array_equal(g[1], o[1])
    kind, _ = check_taps(blob, cfg, ids, lens, 1, wl.max_len, 24, [0], stream)
    assert kind == 1  # the cluster decode step streams the packed 4-bit slices
    gl = _translate(blob, ids, lens, 1, wl.max_len, stream, lean=True)
    assert np.array_equal(gl[0], o[0])


@pytest.mark.parametrize("wq", [synth.WQ_INT4, synth.WQ_INT4_MINMAX])
@pytest.mark.parametrize("beam,B", [(4, 40), (1, 150)])
def test_w4_batched_matches_oracle(wq, beam, B, stream):
    """>= 128 rows: symmetric rows run on the tensor cores from their unpacked
    int8 codes, min-max rows on the 4-bit GEMV in 16-row chunks."""
    cfg = synth.ModelConfig(2, 2, 128, 4, 256, 500, 64, 1, 0, max_pos=64)
    blob = synth.build_blob(cfg, 61, gamma_range=(0.5, 1.5), wq=wq)
    ids, lens = synth.source_batch(cfg.vocab, B, 1, 30, 62)
    T = 12
    g_ids, g_len, g_sc = _translate(blob, ids, lens, beam, T, stream)
    pick = [0, B // 3, B - 1]
    o_ids, o_len, o_sc = O.translate(blob, ids[pick], lens[pick], beam, T, n_threads=3)
    assert np.array_equal(g_ids[pick], o_ids) and np.array_equal(g_len[pick], o_len)
    assert np.array_equal(g_sc[pick].view(np.uint32), o_sc.view(np.uint32))


@pytest.mark.parametrize("wq", [synth.WQ_INT4, synth.WQ_INT4_MINMAX])
def test_w4_paper_20mb_model(wq, stream):
    cfg, _, ids, lens, beam, T = synth.workload_inputs("mobilenmt20-b1-s30-greedy30")
    blob = synth.build_blob(cfg, 20, wq=wq)
    g = _translate(blob, ids, lens, beam, T, stream)
    o = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(g[0], o[0]) and np.array_equal(g[1], o[1])


@pytest.mark.parametrize("wq", [synth.WQ_INT4, synth.WQ_INT4_MINMAX])
@pytest.mark.parametrize("B", [1, 4])
@pytest.mark.parametrize("shape", [(2, 2, 64, 2, 128, 300, 64, 1, 1), (3, 2, 128, 4, 256, 500, 32, 1, 0),
                                   (2, 2, 192, 3, 384, 300, 192, 1, 1), (2, 1, 64, 1, 128, 300, 64, 0, 1)])
def test_w4_cluster_step_matches_oracle(wq, B, shape, stream):
    """Greedy batches of <= 4 run the single-cluster step on 4-bit slices."""
    cfg = synth.ModelConfig(*shape, max_pos=64)
    blob = synth.build_blob(cfg, 71, gamma_range=(0.5, 1.5), wq=wq)
    ids, lens = synth.source_batch(cfg.vocab, B, 1, 40, 72)
    T = 20
    tr = mnmt.Translator(blob, B, ids.shape[1], 1, T, stream)
    try:
        g_ids, g_len, _ = tr.translate(ids, lens, T)
        assert mnmt.mnmt_session_decode_path(tr.session) == 1
    finally:
        tr.close()
    o_ids, o_len, _ = O.translate(blob, ids, lens, 1, T, n_threads=B)
    assert np.array_equal(g_ids, o_ids) and np.array_equal(g_len, o_len)
