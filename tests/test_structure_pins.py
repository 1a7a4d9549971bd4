"""Pin the model-structure accounting to the sizes the paper prints
(Table 1, Table 3, Table 4), read from tests/golden/paper_model_sizes.txt."""
import os

import pytest

from oracle import structure

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_model_sizes.txt")


def _rows():
    rows = []
    for line in open(GOLDEN):
        if not line.strip() or line.startswith("#"):
            continue
        f = line.split()
        rows.append(dict(name=f[0], V=int(f[1]), d=int(f[2]), F=int(f[3]), ne=int(f[4]), nd=int(f[5]),
                         params=f[6], no_emb=f[7], flops=f[8], tol=float(f[9])))
    return rows


@pytest.mark.parametrize("row", _rows(), ids=lambda r: r["name"])
def test_printed_sizes(row):
    total, body = structure.params(row["V"], row["d"], row["F"], row["ne"], row["nd"])
    assert abs(total / 1e6 - float(row["params"])) <= row["tol"] * float(row["params"])
    if row["no_emb"] != "-":
        # printed to the shown precision
        digits = len(row["no_emb"].split(".")[1]) if "." in row["no_emb"] else 0
        assert round(body / 1e6, digits) == float(row["no_emb"])
    if row["flops"] != "-":
        macs = structure.macs(row["V"], row["d"], row["F"], row["ne"], row["nd"], 30, 30)
        assert abs(macs / 1e9 - float(row["flops"])) <= 0.05 + 1e-9


def test_synthetic_paper_models_have_the_printed_sizes():
    """The synthetic MobileNMT-10MB / -20MB models have the shapes of the
    paper's table and hence its printed parameter counts (10M / 20M)."""
    from paper_2306_04235_gb300 import synth
    rows = {r["name"]: r for r in _rows()}
    for name in ("mobilenmt-10mb", "mobilenmt-20mb"):
        cfg = synth.MODELS[name]
        row = rows[name]
        assert (cfg.vocab, cfg.d_model, cfg.d_ffn, cfg.n_enc, cfg.n_dec) == \
            (row["V"], row["d"], row["F"], row["ne"], row["nd"])
        assert cfg.tied_output == 1 and cfg.d_embed == cfg.d_model and cfg.pre_ln == 1
        total, _ = structure.params(cfg.vocab, cfg.d_model, cfg.d_ffn, cfg.n_enc, cfg.n_dec)
        assert abs(total / 1e6 - float(row["params"])) <= row["tol"] * float(row["params"])
        # int8 weights: the model's weight bytes are its size in MB (Table 5 "8-8-8")
        blob = synth.build_blob(cfg, 1)
        assert abs(total - float(row["params"]) * 1e6) <= 0.04 * float(row["params"]) * 1e6
        assert len(blob) > total
