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
