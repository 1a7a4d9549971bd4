"""Host-only checks of the C-ABI library (no GPU): it loads, exports every
symbol include/mnmt.h declares, and validates blobs on the host."""
import os
import re

import pytest

from paper_2306_04235_gb300 import mnmt, synth

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "mnmt.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mnmt_[a-z_0-9]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    L = mnmt.lib()
    names = _declared()
    assert "mnmt_translate" in names and "mnmt_load_weights" in names
    for n in names:
        assert hasattr(L, n), n


def test_blob_validation_on_host():
    cfg = synth.ModelConfig(2, 2, 64, 2, 128, 300, 64, 1, 1, max_pos=64)
    blob = synth.build_blob(cfg, 3)
    got = mnmt.mnmt_blob_check(blob)
    assert got["d_model"] == 64 and got["vocab"] == 300 and got["pre_ln"] == 1
    for bad in [blob[:-16], blob + b"\0" * 16, b"XNMT" + blob[4:], blob[:40]]:
        with pytest.raises(mnmt.MnmtError) as ei:
            mnmt.mnmt_blob_check(bad)
        assert ei.value.code == mnmt.EFORMAT
    assert "blob" in mnmt.last_error() or "magic" in mnmt.last_error()


def test_unsupported_shapes_are_rejected_on_host():
    # head dim 48 is not one the kernels implement
    cfg = synth.ModelConfig(1, 1, 192, 4, 128, 300, 192, 1, 1, max_pos=64)
    with pytest.raises(mnmt.MnmtError) as ei:
        mnmt.mnmt_blob_check(synth.build_blob(cfg, 3))
    assert ei.value.code == mnmt.EFORMAT


def test_paper_model_shapes_pass_host_validation():
    """d_model = 384 (MobileNMT-20MB, 6 heads of 64) is a supported width."""
    for name in ("mobilenmt-10mb", "mobilenmt-20mb"):
        cfg = synth.MODELS[name]
        got = mnmt.mnmt_blob_check(synth.build_blob(cfg, 1))
        assert got["d_model"] == cfg.d_model and got["n_heads"] == cfg.n_heads and got["vocab"] == 8000
    cfg = synth.ModelConfig(1, 1, 352, 4, 128, 300, 352, 1, 1, max_pos=64)   # not a multiple of 64
    with pytest.raises(mnmt.MnmtError) as ei:
        mnmt.mnmt_blob_check(synth.build_blob(cfg, 3))
    assert ei.value.code == mnmt.EFORMAT
