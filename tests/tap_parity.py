"""Tap parity helper shared by the GPU test files: runs n decode steps of a
batch through the C ABI and compares the quantised encoder output, the cross
keys/values, the self-attention cache along each hypothesis's own path, the
last step's decoder output and (beam search) logits with the CPU oracle."""
import numpy as np

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt


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


def check_taps(blob, cfg, ids, lens, beam, T, n_steps, picks, stream):
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
