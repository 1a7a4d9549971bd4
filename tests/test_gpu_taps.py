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
from tap_parity import check_taps

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stream():
    return torch.cuda.Stream()


def test_small_batch1_workload_taps(stream):
    """The bench workload at full size: 64 decode steps of the cluster step."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s10to50-greedy64")
    kind, n = check_taps(blob, cfg, ids, lens, beam, T, T, [0], stream)
    assert kind == 1 and n == 1


def test_paper_shape_taps(stream):
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b1-s30-greedy30")
    check_taps(blob, cfg, ids, lens, beam, T, T, [0], stream)


def test_small_batched_beam_workload_taps(stream):
    """Batch 32 x beam 4 (128 decoder rows on the tensor cores), source lengths
    10-80; 3 sentences x 4 hypotheses checked over 24 steps."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("small-b32-s10to80-beam4-t128")
    picks = [0, int(np.argmax(lens)), 31]
    kind, n = check_taps(blob, cfg, ids, lens, beam, T, 24, picks, stream)
    assert kind == 0 and n == 12


def test_wide_batched_beam_workload_taps(stream):
    """Batch 128 x beam 4 (512 rows), d = 512, source lengths 20-128 (encoder
    M up to 16384 rows); 2 sentences x 4 hypotheses over 12 steps."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs("wide-b128-s20to128-beam4-t160")
    picks = [int(np.argmin(lens)), int(np.argmax(lens))]
    kind, n = check_taps(blob, cfg, ids, lens, beam, T, 12, picks, stream)
    assert kind == 0 and n == 8


def test_greedy_batch_of_four_taps(stream):
    """Four sentences through the cluster step (its largest greedy batch)."""
    cfg = synth.MODELS["small-12x2-d256-v32k-e128"]
    blob = synth.build_blob(cfg, 1)
    ids, lens = synth.source_batch(cfg.vocab, 4, 10, 50, 4711)
    kind, n = check_taps(blob, cfg, ids, lens, 1, 40, 40, [0, 1, 2, 3], stream)
    assert kind == 1 and n == 4


@pytest.mark.parametrize("name", ["mobilenmt10-b1-s30-greedy30", "mobilenmt20-b1-s30-greedy30"])
def test_paper_models_tokens_and_taps(name, stream):
    """The paper's two models (Table "detailed settings of MobileNMT") at its
    measurement shape: src/tgt 30, batch 1, greedy.  The 20MB model's width
    384 = 3 x 128 exercises the LayerNorm's exact division by a width with an
    odd factor in every kernel that normalises."""
    cfg, blob, ids, lens, beam, T = synth.workload_inputs(name)
    kind, _ = check_taps(blob, cfg, ids, lens, beam, T, T, [0], stream)
    assert kind == 1  # the single-cluster decode step (12 CTAs of 32 columns at d = 384)
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
    check_taps(blob, cfg, ids, lens, beam, T, 8, [0, B - 1], stream)


def test_encoder_attention_tensor_core_long_sources(stream):
    """The tensor-core encoder attention at its largest key count: sources of
    130-250 tokens (keys padded to 256, four 64-query blocks per head), d_h =
    64, enough sentences that its grid fills the GPU; encoder output, cross
    keys / values and two decode steps checked for the shortest and longest
    sentence."""
    cfg = synth.ModelConfig(2, 1, 192, 3, 384, 300, 192, 1, 1, max_pos=256)
    blob = synth.build_blob(cfg, 77, gamma_range=(0.5, 1.5))
    ids, lens = synth.source_batch(cfg.vocab, 16, 130, 250, 78)
    assert ids.shape[1] > 128
    picks = [int(np.argmin(lens)), int(np.argmax(lens))]
    check_taps(blob, cfg, ids, lens, 1, 4, 2, picks, stream)
