"""End-to-end parity of the translation path (C ABI, sm_103a kernels) against the
CPU oracle: identical token sequences, lengths and beam scores, and bit-exact
intermediate taps (encoder output, cross-attention keys/values, self-attention
cache, decoder output), on the seeded synthetic workloads at full size (sampled
sentences where the oracle is slow) and on small models that span the
configuration space (pre/post-LN, factorised/tied embedding, greedy/beam)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MINI = {
    "odd": synth.ModelConfig(2, 2, 192, 3, 384, 300, 192, 1, 1, max_pos=64),   # d = 3 x 64: 4-CTA cluster step
    "pre": synth.ModelConfig(2, 2, 64, 2, 128, 300, 64, 1, 1, max_pos=64),
    "post": synth.ModelConfig(2, 1, 64, 1, 128, 300, 64, 0, 1, max_pos=64),
    "fact": synth.ModelConfig(3, 2, 128, 4, 256, 500, 32, 1, 0, max_pos=96),
    "wide-head": synth.ModelConfig(1, 2, 256, 2, 256, 400, 256, 1, 1, max_pos=64),
}


@pytest.fixture(scope="module")
def stream():
    return torch.cuda.Stream()


def _gpu(blob, ids, lens, beam, max_len, stream, max_batch=None, max_src=None):
    tr = mnmt.Translator(blob, max_batch or ids.shape[0], max_src or ids.shape[1], beam, max_len, stream)
    try:
        out = tr.translate(ids, lens, max_len)
    finally:
        tr.close()
    return out


@pytest.mark.parametrize("kind", list(MINI))
@pytest.mark.parametrize("beam", [1, 3])
def test_small_models_match_oracle(kind, beam, stream):
    cfg = MINI[kind]
    blob = synth.build_blob(cfg, 21, gamma_range=(0.5, 1.5))
    ids, lens = synth.source_batch(cfg.vocab, 5, 1, 40, 22)
    T = 24
    g_ids, g_len, g_sc = _gpu(blob, ids, lens, beam, T, stream)
    o_ids, o_len, o_sc = O.translate(blob, ids, lens, beam, T, n_threads=5)
    assert np.array_equal(g_ids, o_ids)
    assert np.array_equal(g_len, o_len)
    assert np.array_equal(g_sc.view(np.uint32), o_sc.view(np.uint32))


@pytest.mark.parametrize("kind,beam", [("fact", 4), ("pre", 3)])
def test_many_sentences_beam_search_matches_oracle(kind, beam, stream):
    """80 sentences: enough that the cross attention serves all beams of a
    sentence from one block (the batched-beam layout)."""
    cfg = MINI[kind]
    blob = synth.build_blob(cfg, 31, gamma_range=(0.5, 1.5))
    ids, lens = synth.source_batch(cfg.vocab, 80, 1, 30, 32)
    T = 12
    g_ids, g_len, g_sc = _gpu(blob, ids, lens, beam, T, stream)
    o_ids, o_len, o_sc = O.translate(blob, ids, lens, beam, T, n_threads=8)
    assert np.array_equal(g_ids, o_ids)
    assert np.array_equal(g_len, o_len)
    assert np.array_equal(g_sc.view(np.uint32), o_sc.view(np.uint32))


def test_tiny_workload_tokens_and_taps(stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("tiny-b1-s16-greedy16")
    d, H, L = cfg.d_model, cfg.n_heads, cfg.n_dec
    dh = d // H
    tr = mnmt.Translator(blob, 1, ids.shape[1], beam, T, stream)
    try:
        out, olen, _ = tr.translate(ids, lens, T)
        S = ids.shape[1]
        enc = mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_ENC_OUT, 0, np.int8, (1, S, d))
        ck = [mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_CROSS_K, l, np.int8, (1, H, S, dh)) for l in range(L)]
        cv = [mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_CROSS_V, l, np.int8, (1, H, S, dh)) for l in range(L)]
        sk = [mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_SELF_K, l, np.int8, (1, H, T, dh)) for l in range(L)]
        sv = [mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_SELF_V, l, np.int8, (1, H, T, dh)) for l in range(L)]
        dec = mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_DEC_OUT, 0, np.int8, (1, d))
    finally:
        tr.close()
    ref, rlen, _ = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(out, ref) and np.array_equal(olen, rlen)
    e_q, e_k, e_v = O.encode(blob, ids[0], lens[0], cfg)
    assert np.array_equal(enc[0], e_q)
    for l in range(L):
        assert np.array_equal(ck[l][0].transpose(1, 0, 2).reshape(S, d), e_k[l])
        assert np.array_equal(cv[l][0].transpose(1, 0, 2).reshape(S, d), e_v[l])
    n = int(olen[0])
    tgt = np.concatenate([[cfg.bos_id], out[0, :n - 1]]).astype(np.int32)
    logits, dec_q, self_k, self_v = O.decode_trace(blob, ids[0], lens[0], tgt, cfg, want_cache=True)
    assert np.array_equal(dec, dec_q[n - 1:n])
    for l in range(L):
        assert np.array_equal(sk[l][0, :, :n].transpose(1, 0, 2).reshape(n, d), self_k[l])
        assert np.array_equal(sv[l][0, :, :n].transpose(1, 0, 2).reshape(n, d), self_v[l])


def test_small_batch1_workload_matches_oracle(stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s10to50-greedy64")
    g = _gpu(blob, ids, lens, beam, T, stream)
    o = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(g[0], o[0]) and np.array_equal(g[1], o[1])


def test_paper_shape_src30_tgt30(stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s30-greedy30")
    g = _gpu(blob, ids, lens, beam, T, stream)
    o = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(g[0], o[0]) and np.array_equal(g[1], o[1])


def test_small_batched_beam_workload_sampled(stream):
    """Batch 32, beam 4, 128 steps at full size; the oracle checks 4 sentences."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b32-s10to80-beam4-t128")
    g_ids, g_len, g_sc = _gpu(blob, ids, lens, beam, T, stream)
    pick = [0, 9, 17, 31]
    o_ids, o_len, o_sc = O.translate(blob, ids[pick], lens[pick], beam, T, n_threads=4)
    assert np.array_equal(g_ids[pick], o_ids)
    assert np.array_equal(g_len[pick], o_len)
    assert np.array_equal(g_sc[pick].view(np.uint32), o_sc.view(np.uint32))


def test_wide_batched_beam_workload_sampled(stream):
    """Batch 128, beam 4, 160 steps at full size; the oracle checks 2 sentences."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("wide-b128-s20to128-beam4-t160")
    g_ids, g_len, g_sc = _gpu(blob, ids, lens, beam, T, stream)
    pick = [5, 127]
    o_ids, o_len, o_sc = O.translate(blob, ids[pick], lens[pick], beam, T, n_threads=2)
    assert np.array_equal(g_ids[pick], o_ids)
    assert np.array_equal(g_len[pick], o_len)
    assert np.array_equal(g_sc[pick].view(np.uint32), o_sc.view(np.uint32))


def test_longest_source(stream):
    cfg = synth.MODELS["small-12x2-d256-v32k-e128"]
    blob = synth.build_blob(cfg, 1)
    ids, lens = synth.source_batch(cfg.vocab, 2, 500, 512, 33)
    ids = np.pad(ids, ((0, 0), (0, 512 - ids.shape[1])))
    g = _gpu(blob, ids, lens, 1, 6, stream)
    o = O.translate(blob, ids, lens, 1, 6, n_threads=2)
    assert np.array_equal(g[0], o[0])


@pytest.mark.parametrize("beam", [1, 4])
def test_forced_eos_stops_at_once(beam, stream):
    cfg = MINI["pre"]
    blob = synth.build_blob(cfg, 3, out_bias={cfg.eos_id: 1000.0})
    ids, lens = synth.source_batch(cfg.vocab, 3, 2, 9, 4)
    g_ids, g_len, _ = _gpu(blob, ids, lens, beam, 20, stream)
    assert np.all(g_len == 1) and np.all(g_ids[:, 0] == cfg.eos_id) and np.all(g_ids[:, 1:] == cfg.pad_id)


@pytest.mark.parametrize("kind", list(MINI))
@pytest.mark.parametrize("batch", [1, 3])
def test_cluster_step_models_match_oracle(kind, batch, stream):
    """Every small model shape (pre- and post-LN, factorised and plain
    embedding, tied and untied output, d_h 64 and 128, d = 3 x 64) through
    the single-cluster step: greedy batches of at most 4 rows."""
    cfg = MINI[kind]
    blob = synth.build_blob(cfg, 41, gamma_range=(0.5, 1.5))
    ids, lens = synth.source_batch(cfg.vocab, batch, 1, 40, 42)
    T = 24
    tr = mnmt.Translator(blob, batch, ids.shape[1], 1, T, stream)
    try:
        g_ids, g_len, g_sc = tr.translate(ids, lens, T)
        assert mnmt.mnmt_session_decode_path(tr.session) == 1
    finally:
        tr.close()
    o_ids, o_len, o_sc = O.translate(blob, ids, lens, 1, T, n_threads=3)
    assert np.array_equal(g_ids, o_ids)
    assert np.array_equal(g_len, o_len)
    assert np.array_equal(g_sc.view(np.uint32), o_sc.view(np.uint32))


@pytest.mark.parametrize("seed,bias,rows,lengths", [
    (3, 0.15, None, [23, 1, 40, 40]),
    (3, 0.2, None, [1, 1, 16, 40]),   # one sentence ends on a 16-step graph boundary
    (5, 0.28, None, [1, 1, 24, 40]),
    (3, 0.1, 0, [31]),
    (3, 0.2, 2, [16]),
])
def test_cluster_step_mixed_lengths_match_oracle(seed, bias, rows, lengths, stream):
    """The single-cluster step (greedy, <= 4 rows) with sentences that finish
    at different steps, inside and at the end of a captured run of 16 steps:
    the greedy selection left pending by the vocabulary kernel is applied by
    the next step kernel or by the greedy update that closes the run."""
    cfg = MINI["pre"]
    blob = synth.build_blob(cfg, seed, out_bias={cfg.eos_id: bias})
    ids, lens = synth.source_batch(cfg.vocab, 4, 2, 30, 4)
    if rows is not None:
        ids, lens = ids[rows:rows + 1], lens[rows:rows + 1]
    T = 40
    tr = mnmt.Translator(blob, ids.shape[0], ids.shape[1], 1, T, stream)
    try:
        g_ids, g_len, g_sc = tr.translate(ids, lens, T)
        assert mnmt.mnmt_session_decode_path(tr.session) == 1
    finally:
        tr.close()
    o_ids, o_len, o_sc = O.translate(blob, ids, lens, 1, T, n_threads=4)
    assert o_len.tolist() == lengths
    assert np.array_equal(g_ids, o_ids)
    assert np.array_equal(g_len, o_len)
    assert np.array_equal(g_sc.view(np.uint32), o_sc.view(np.uint32))


@pytest.mark.parametrize("beam", [1, 3])
def test_decode_step_api_matches_translate(beam, stream):
    cfg = MINI["fact"]
    blob = synth.build_blob(cfg, 8)
    ids, lens = synth.source_batch(cfg.vocab, 2, 3, 20, 9)
    T = 12
    o_ids, o_len, o_sc = O.translate(blob, ids, lens, beam, T, n_threads=2)
    tr = mnmt.Translator(blob, 2, ids.shape[1], beam, T, stream)
    try:
        mnmt.mnmt_encode(tr.session, ids, lens, 2, ids.shape[1])
        toks, pars = [], []
        for t in range(T):
            tok, par, sc, done = mnmt.mnmt_decode_step(tr.session, 2 * beam)
            toks.append(tok); pars.append(par)
            if done:
                break
        with pytest.raises(mnmt.MnmtError):
            for _ in range(T + 1):
                mnmt.mnmt_decode_step(tr.session, 2 * beam)
    finally:
        tr.close()
    # backtrack beam 0 of each sentence through the parents
    for b in range(2):
        r = 0
        seq = []
        for t in range(len(toks) - 1, -1, -1):
            seq.append(toks[t][b * beam + r])
            r = pars[t][b * beam + r] if beam > 1 else 0
        seq = seq[::-1]
        n = int(o_len[b])
        assert seq[:n] == list(o_ids[b, :n])


@pytest.mark.parametrize("beam", [1, 3])
def test_queued_decode_steps_match_stepwise_decode(beam, stream):
    """mnmt_decode_steps queues steps without host round trips: the token and
    parent history equals the one of step-by-step decoding, and steps past the
    length limit are not queued."""
    cfg = MINI["fact"]
    blob = synth.build_blob(cfg, 8)
    ids, lens = synth.source_batch(cfg.vocab, 2, 3, 20, 9)
    T, R = 12, 2 * beam
    tr = mnmt.Translator(blob, 2, ids.shape[1], beam, T, stream)
    try:
        mnmt.mnmt_encode(tr.session, ids, lens, 2, ids.shape[1])
        steps = [mnmt.mnmt_decode_step(tr.session, R) for _ in range(T)]
        mnmt.mnmt_encode(tr.session, ids, lens, 2, ids.shape[1])
        assert mnmt.mnmt_decode_steps(tr.session, 5) == 5
        assert mnmt.mnmt_decode_steps(tr.session, 100) == T - 5
        assert mnmt.mnmt_decode_steps(tr.session, 1) == 0
        hist = mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_HISTORY, 0, np.int32, (T, R))
        par = mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_PARENTS, 0, np.int32, (T, R))
    finally:
        tr.close()
    assert np.array_equal(hist, np.stack([s[0] for s in steps]))
    if beam > 1:
        assert np.array_equal(par, np.stack([s[1] for s in steps]))


def test_cluster_step_graph_serves_changing_source_lengths(stream):
    """One session translating sentences of different padded lengths in turn
    (the cluster step keeps its captured graph and only updates the length)."""
    cfg, blob, _, _, beam, T = synth.workload_inputs("small-b1-s10to50-greedy64")
    tr = mnmt.Translator(blob, 1, 50, 1, T, stream)
    try:
        for i, S in enumerate([37, 12, 50, 12, 29]):
            ids, lens = synth.source_batch(cfg.vocab, 1, S, S, 70 + i)
            g_ids, g_len, _ = tr.translate(ids, lens, T)
            assert mnmt.mnmt_session_decode_path(tr.session) == 1
            o_ids, o_len, _ = O.translate(blob, ids, lens, 1, T, n_threads=1)
            assert np.array_equal(g_ids, o_ids) and np.array_equal(g_len, o_len), S
    finally:
        tr.close()


def test_device_pointer_path_equals_host_path(stream):
    cfg = MINI["pre"]
    blob = synth.build_blob(cfg, 5)
    ids, lens = synth.source_batch(cfg.vocab, 4, 2, 30, 6)
    T = 16
    tr = mnmt.Translator(blob, 4, ids.shape[1], 2, T, stream)
    try:
        h = tr.translate(ids, lens, T)
        d_ids, d_lens = torch.from_numpy(ids).cuda(), torch.from_numpy(lens).cuda()
        o_ids = torch.zeros((4, T), dtype=torch.int32, device="cuda")
        o_len = torch.zeros(4, dtype=torch.int32, device="cuda")
        o_sc = torch.zeros(4, dtype=torch.float32, device="cuda")
        torch.cuda.synchronize()
        mnmt.mnmt_translate(tr.session, d_ids, d_lens, 4, ids.shape[1], T, mnmt.DEVICE_PTRS, o_ids, o_len, o_sc)
        stream.synchronize()
        assert np.array_equal(o_ids.cpu().numpy(), h[0]) and np.array_equal(o_len.cpu().numpy(), h[1])
        assert np.array_equal(o_sc.cpu().numpy(), h[2])
    finally:
        tr.close()


def test_bad_inputs_are_rejected(stream):
    cfg = MINI["pre"]
    blob = synth.build_blob(cfg, 5)
    tr = mnmt.Translator(blob, 2, 10, 1, 8, stream)
    try:
        ids = np.full((2, 10), 5, np.int32)
        with pytest.raises(mnmt.MnmtError) as ei:
            tr.translate(ids, np.array([3, 11], np.int32), 8)       # length beyond S_pad
        assert ei.value.code == mnmt.EINVAL
        bad = ids.copy(); bad[1, 2] = cfg.vocab
        with pytest.raises(mnmt.MnmtError):
            tr.translate(bad, np.array([3, 4], np.int32), 8)         # id outside the vocabulary
        with pytest.raises(mnmt.MnmtError):
            tr.translate(np.full((3, 10), 5, np.int32), np.array([3, 4, 5], np.int32), 8)  # batch > capacity
        out = tr.translate(ids, np.array([3, 4], np.int32), 8)      # session still usable
        assert out[0].shape == (2, 8)
    finally:
        tr.close()


def _with_path(cluster: bool):
    import os
    if cluster:
        os.environ.pop("MNMT_DECODE_CLUSTER", None)
    else:
        os.environ["MNMT_DECODE_CLUSTER"] = "0"


@pytest.mark.parametrize("kind", list(MINI))
@pytest.mark.parametrize("B", [1, 3, 4])
def test_cluster_decode_step_matches_oracle(kind, B, stream):
    """Greedy batches of <= 4 sentences run the single-cluster decode step."""
    cfg = MINI[kind]
    blob = synth.build_blob(cfg, 31, gamma_range=(0.5, 1.5))
    ids, lens = synth.source_batch(cfg.vocab, B, 1, 40, 32)
    T = 24
    _with_path(True)
    tr = mnmt.Translator(blob, B, ids.shape[1], 1, T, stream)
    try:
        g_ids, g_len, _ = tr.translate(ids, lens, T)
        assert mnmt.mnmt_session_decode_path(tr.session) == 1
    finally:
        tr.close()
    o_ids, o_len, _ = O.translate(blob, ids, lens, 1, T, n_threads=B)
    assert np.array_equal(g_ids, o_ids) and np.array_equal(g_len, o_len)


@pytest.mark.parametrize("name", ["tiny-b1-s16-greedy16", "small-b1-s10to50-greedy64"])
def test_cluster_and_kernel_paths_bit_identical(name, stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs(name)
    d, H, L = cfg.d_model, cfg.n_heads, cfg.n_dec
    dh = d // H
    res = {}
    for cluster in (True, False):
        _with_path(cluster)
        tr = mnmt.Translator(blob, 1, ids.shape[1], beam, T, stream)
        try:
            out = tr.translate(ids, lens, T)
            assert mnmt.mnmt_session_decode_path(tr.session) == int(cluster)
            taps = [mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_DEC_OUT, 0, np.int8),
                    mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_RESID, 0, np.float32)]
            for l in range(L):
                taps.append(mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_SELF_K, l, np.int8))
                taps.append(mnmt.mnmt_debug_tap(tr.session, mnmt.TAP_SELF_V, l, np.int8))
            res[cluster] = (out, taps)
        finally:
            tr.close()
    _with_path(True)
    (o1, t1), (o0, t0) = res[True], res[False]
    assert np.array_equal(o1[0], o0[0]) and np.array_equal(o1[1], o0[1])
    for a, b in zip(t1, t0):
        assert np.array_equal(a.view(np.uint8), b.view(np.uint8))
    ref = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(o1[0], ref[0])


def test_bench_workload_uses_cluster_step(stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s10to50-greedy64")
    _with_path(True)
    tr = mnmt.Translator(blob, 1, ids.shape[1], beam, T, stream)
    try:
        mnmt.mnmt_encode(tr.session, ids, lens, 1, ids.shape[1])
        assert mnmt.mnmt_session_decode_path(tr.session) == 1
    finally:
        tr.close()


def _with_tc(on: bool):
    import os
    if on:
        os.environ.pop("MNMT_TC", None)
    else:
        os.environ["MNMT_TC"] = "0"


@pytest.mark.parametrize("kind", list(MINI))
@pytest.mark.parametrize("beam", [1, 4])
def test_tensor_core_rows_match_oracle(kind, beam, stream):
    """Batches of >= 128 decoder rows (and encoder rows) run their linears on
    the tcgen05 kernel: tokens, lengths and scores still equal the oracle's."""
    cfg = MINI[kind]
    blob = synth.build_blob(cfg, 41, gamma_range=(0.5, 1.5))
    B = 160 // beam
    ids, lens = synth.source_batch(cfg.vocab, B, 1, 40, 42)
    T = 20
    _with_tc(True)
    g_ids, g_len, g_sc = _gpu(blob, ids, lens, beam, T, stream)
    o_ids, o_len, o_sc = O.translate(blob, ids, lens, beam, T, n_threads=8)
    assert np.array_equal(g_ids, o_ids)
    assert np.array_equal(g_len, o_len)
    assert np.array_equal(g_sc.view(np.uint32), o_sc.view(np.uint32))


def test_tensor_core_and_imma_paths_bit_identical(stream):
    """The same batched beam workload through the tcgen05 linears and through
    the IMMA linears (MNMT_TC=0): identical outputs."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b32-s10to80-beam4-t128")
    outs = []
    for on in (True, False):
        _with_tc(on)
        try:
            outs.append(_gpu(blob, ids, lens, beam, T, stream))
        finally:
            _with_tc(True)
    for a, b in zip(*outs):
        assert np.array_equal(a.view(np.uint32) if a.dtype == np.float32 else a,
                              b.view(np.uint32) if b.dtype == np.float32 else b)
