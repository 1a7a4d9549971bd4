"""Memory-minimal operation (Sec. 4 "Memory Optimization": shared activation
buffers; the running-memory column of Table 2): a lean model (int8 blob only)
with a lean session (two shared int8 activation buffers and the fp32
residual) translates exactly like the default model and session, and the
library's device memory is what it reports."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2306_04235_gb300 import mnmt, synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stream():
    return torch.cuda.Stream()


def _translate(blob, ids, lens, beam, T, stream, lean):
    tr = mnmt.Translator(blob, ids.shape[0], ids.shape[1], beam, T, stream, lean=lean)
    try:
        out = tr.translate(ids, lens, T)
        mb = mnmt.mnmt_model_device_bytes(tr.model)
        sb = mnmt.mnmt_session_device_bytes(tr.session)
        path = mnmt.mnmt_session_decode_path(tr.session)
    finally:
        tr.close()
    return out, mb, sb, path


@pytest.mark.parametrize("name", ["mobilenmt10-b1-s30-greedy30", "mobilenmt20-b1-s30-greedy30",
                                  "small-b1-s10to50-greedy64"])
def test_lean_translation_equals_default_and_oracle(name, stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs(name)
    (l_ids, l_len, _), l_mb, l_sb, _ = _translate(blob, ids, lens, beam, T, stream, True)
    (d_ids, d_len, _), d_mb, d_sb, _ = _translate(blob, ids, lens, beam, T, stream, False)
    o_ids, o_len, _ = O.translate(blob, ids, lens, beam, T)
    assert np.array_equal(l_ids, d_ids) and np.array_equal(l_len, d_len)
    assert np.array_equal(l_ids, o_ids) and np.array_equal(l_len, o_len)
    # the lean model holds the blob and its derived constants only (no 2x fp16 copy)
    assert len(blob) <= l_mb < len(blob) * 1.05
    assert d_mb - l_mb == 2 * len(blob)
    assert l_sb <= d_sb


@pytest.mark.parametrize("beam,B", [(3, 60), (1, 150)])
def test_lean_batched_search_equals_oracle(beam, B, stream):
    """>= 128 decoder rows: the default session runs its linears on the tensor
    cores, the lean one on the int8 IMMA kernels; both equal the oracle."""
    cfg = synth.ModelConfig(2, 2, 128, 4, 256, 500, 128, 1, 1, max_pos=64)
    blob = synth.build_blob(cfg, 51, gamma_range=(0.5, 1.5))
    ids, lens = synth.source_batch(cfg.vocab, B, 1, 30, 52)
    T = 14
    (l_ids, l_len, l_sc), _, l_sb, _ = _translate(blob, ids, lens, beam, T, stream, True)
    (d_ids, d_len, d_sc), _, d_sb, _ = _translate(blob, ids, lens, beam, T, stream, False)
    assert np.array_equal(l_ids, d_ids) and np.array_equal(l_len, d_len)
    assert np.array_equal(l_sc.view(np.uint32), d_sc.view(np.uint32))
    pick = [0, B // 2, B - 1]
    o_ids, o_len, o_sc = O.translate(blob, ids[pick], lens[pick], beam, T, n_threads=3)
    assert np.array_equal(l_ids[pick], o_ids) and np.array_equal(l_sc[pick].view(np.uint32), o_sc.view(np.uint32))
    assert l_sb < d_sb


def test_lean_flags_validated(stream):
    cfg = synth.ModelConfig(1, 1, 64, 2, 128, 300, 64, 1, 1, max_pos=32)
    blob = synth.build_blob(cfg, 3)
    with pytest.raises(mnmt.MnmtError) as ei:
        mnmt.mnmt_load_weights(blob, stream, 6)
    assert ei.value.code == mnmt.EINVAL
    m = mnmt.mnmt_load_weights(blob, stream, mnmt.LOAD_LEAN)
    try:
        with pytest.raises(mnmt.MnmtError):
            mnmt.mnmt_session_create(m, 1, 8, 1, 8, 4)
        s = mnmt.mnmt_session_create(m, 1, 8, 1, 8, 0)    # a default session on a lean model: int8 kernels
        mnmt.mnmt_session_free(s)
    finally:
        mnmt.mnmt_model_free(m)
