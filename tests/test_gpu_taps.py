"""Element-by-element parity of the intermediate tensors of full-size
translations against the CPU oracle (App. A encoder-decoder; Sec. 3.3 / Fig. 5
quantisation points): the quantised encoder output, every decoder layer's cross
keys and values, the self-attention cache along each hypothesis's own path, the
decoder output of the last step and, under beam search, its fp32 logits.

The batch-1 workload runs its decoder as the single thread-block-cluster step
and its encoder linears on the tensor cores (tcgen05, split-K for FFN2); the
batched-beam workloads run every linear on the tensor cores.  A wrong value in
any of them shows up here even where it would not change a token."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stream():
    return torch.cuda.Stream()


def _path(hist, par, r, beam, n):
    """Tokens chosen along final hypothesis r's own path, steps 0..n-1."""
    b0 = (r // beam) * beam
    toks = []
    row = r
    for t in range(n - 1, -1, -1):
        toks.append(int(hist[t, row]))
        if beam > 1:
            row = b0 + int(par[t, row])
    return toks[::-1]


def _check_taps(blob, cfg, ids, lens, beam, T, n_steps, picks, stream):
    B, S = ids.shape
    d, H, L, V = cfg.d_model, cfg.n_heads, cfg.n_dec, cfg.vocab
    dh = d // H
    R = B * beam
    tr = mnmt.Translator(blob, B, S, beam, T, stream)
    try:
        s = tr.session
        mnmt.mnmt_encode(s, ids, lens, B, S)
        assert mnmt.mnmt_decode_steps(s, n_steps) == n_steps
        stream.synchronize()
        path_kind = mnmt.mnmt_session_decode_path(s)
        tap = lambda t, l, dt, shape: mnmt.mnmt_debug_tap(s, t, l, dt, shape)  # noqa: E731
        enc = tap(mnmt.TAP_ENC_OUT, 0, np.int8, (B, S, d))
        ck = [tap(mnmt.TAP_CROSS_K, l, np.int8, (B, H, S, dh)) for l in range(L)]
        cv = [tap(mnmt.TAP_CROSS_V, l, np.int8, (B, H, S, dh)) for l in range(L)]
        sk = [tap(mnmt.TAP_SELF_K, l, np.int8, (R, H, T, dh)) for l in range(L)]
        sv = [tap(mnmt.TAP_SELF_V, l, np.int8, (R, H, T, dh)) for l in range(L)]
        dec = tap(mnmt.TAP_DEC_OUT, 0, np.int8, (R, d))
        hist = tap(mnmt.TAP_HISTORY, 0, np.int32, (T, R))
        par = tap(mnmt.TAP_PARENTS, 0, np.int32, (T, R))
        if beam > 1:
            logits = tap(mnmt.TAP_LOGITS, 0, np.float32, (R, V))
            anc = tap(mnmt.TAP_ANCESTRY, 0, np.int32, (R, T))
    finally:
        tr.close()
    n = n_steps
    checked = 0
    for b in picks:
        ln = int(lens[b])
        e_q, e_k, e_v = O.encode(blob, ids[b], ln, cfg)
        assert np.array_equal(enc[b, :ln], e_q[:ln]), f"encoder output, sentence {b}"
        for l in range(L):
            assert np.array_equal(ck[l][b].transpose(1, 0, 2).reshape(S, d)[:ln], e_k[l][:ln]), (b, l)
            assert np.array_equal(cv[l][b].transpose(1, 0, 2).reshape(S, d)[:ln], e_v[l][:ln]), (b, l)
        for i in range(beam):
            r = b * beam + i
            y = _path(hist, par, r, beam, n)
            tgt = np.array([cfg.bos_id] + y[:n - 1], np.int32)
            o_logits, o_dec, o_sk, o_sv = O.decode_trace(blob, ids[b], ln, tgt, cfg, want_cache=True)
            # the path's tokens are the argmax (greedy) of the oracle's own logits
            if beam == 1:
                assert y == [int(np.argmax(o_logits[t])) for t in range(n)]
            for j in range(n):
                phys = int(anc[r, j]) if beam > 1 else r
                for l in range(L):
                    assert np.array_equal(sk[l][phys, :, j].reshape(d), o_sk[l][j]), (b, i, j, l)
                    assert np.array_equal(sv[l][phys, :, j].reshape(d), o_sv[l][j]), (b, i, j, l)
            last = int(anc[r, n - 1]) if beam > 1 else r
            assert np.array_equal(dec[last], o_dec[n - 1]), (b, i)
            if beam > 1:
                assert np.array_equal(logits[last].view(np.uint32), o_logits[n - 1].view(np.uint32)), (b, i)
            checked += 1
    return path_kind, checked


def test_small_batch1_workload_taps(stream):
    """The bench workload at full size: 64 decode steps of the cluster step."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s10to50-greedy64")
    kind, n = _check_taps(blob, cfg, ids, lens, beam, T, T, [0], stream)
    assert kind == 1 and n == 1


def test_paper_shape_taps(stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s30-greedy30")
    _check_taps(blob, cfg, ids, lens, beam, T, T, [0], stream)


def test_small_batched_beam_workload_taps(stream):
    """Batch 32 x beam 4 (128 decoder rows on the tensor cores), source lengths
    10-80; 3 sentences x 4 hypotheses checked over 24 steps."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b32-s10to80-beam4-t128")
    picks = [0, int(np.argmax(lens)), 31]
    kind, n = _check_taps(blob, cfg, ids, lens, beam, T, 24, picks, stream)
    assert kind == 0 and n == 12


def test_wide_batched_beam_workload_taps(stream):
    """Batch 128 x beam 4 (512 rows), d = 512, source lengths 20-128 (encoder
    M up to 16384 rows); 2 sentences x 4 hypotheses over 12 steps."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("wide-b128-s20to128-beam4-t160")
    picks = [int(np.argmin(lens)), int(np.argmax(lens))]
    kind, n = _check_taps(blob, cfg, ids, lens, beam, T, 12, picks, stream)
    assert kind == 0 and n == 8


def test_greedy_batch_of_four_taps(stream):
    """Four sentences through the cluster step (its largest greedy batch)."""
    cfg = synth.MODELS["small-12x2-d256-v32k-e128"]
    blob = synth.build_blob(cfg, 1)
    ids, lens = synth.source_batch(cfg.vocab, 4, 10, 50, 4711)
    kind, n = _check_taps(blob, cfg, ids, lens, 1, 40, 40, [0, 1, 2, 3], stream)
    assert kind == 1 and n == 4


@pytest.mark.parametrize("name", ["mobilenmt10-b1-s30-greedy30", "mobilenmt20-b1-s30-greedy30"])
def test_paper_models_tokens_and_taps(name, stream):
    """The paper's two models (Table "detailed settings of MobileNMT") at its
    measurement shape: src/tgt 30, batch 1, greedy.  The 20MB model's width
    384 = 3 x 128 exercises the LayerNorm's exact division by a width with an
    odd factor in every kernel that normalises."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs(name)
    _check_taps(blob, cfg, ids, lens, beam, T, T, [0], stream)
    tr = mnmt.Translator(blob, 1, ids.shape[1], beam, T, stream)
    try:
        g_ids, g_len, _ = tr.translate(ids, lens, T)
    finally:
        tr.close()
    o_ids, o_len, _ = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(g_ids, o_ids) and np.array_equal(g_len, o_len)


@pytest.mark.parametrize("beam,B", [(1, 160), (4, 40)])
def test_paper_20mb_model_batched(beam, B, stream):
    """The 20MB model with >= 128 decoder rows (tensor-core linears at K = 384
    and 768) under greedy and beam search; 4 sentences checked."""
    cfg = synth.MODELS["mobilenmt-20mb"]
    blob = synth.build_blob(cfg, 20)
    ids, lens = synth.source_batch(cfg.vocab, B, 10, 40, 2020)
    T = 16
    tr = mnmt.Translator(blob, B, ids.shape[1], beam, T, stream)
    try:
        g_ids, g_len, g_sc = tr.translate(ids, lens, T)
    finally:
        tr.close()
    pick = [0, 1, B // 2, B - 1]
    o_ids, o_len, o_sc = O.translate(blob, ids[pick], lens[pick], beam, T, n_threads=4)
    assert np.array_equal(g_ids[pick], o_ids) and np.array_equal(g_len[pick], o_len)
    assert np.array_equal(g_sc[pick].view(np.uint32), o_sc.view(np.uint32))
    _check_taps(blob, cfg, ids, lens, beam, T, 8, [0, B - 1], stream)
