"""Pins for the oracle's storage accounting against the paper's printed numbers
(Sec. 4.1 operating point, Table 5 compression column, Table 6 code/eff columns,
Sec. 4.5 measured footprint).  Values live in tests/golden/paper_values.json,
each with its citation."""
import json
import math
import os

import oracle
from conftest import GOLDEN

PV = json.load(open(os.path.join(GOLDEN, "paper_values.json")))


def base_id(name):
    return oracle.BASE_AFFINE if name == "affine" else oracle.BASE_TQ


def test_metadata_bits():
    assert oracle.metadata_bits(oracle.BASE_AFFINE) == PV["metadata_bits"]["affine"]
    assert oracle.metadata_bits(oracle.BASE_TQ) == PV["metadata_bits"]["tq"]


def test_operating_points_sec41():
    op = PV["operating_points"]["affine_r25"]
    nominal = op["r"] * math.log2(op["L_hi"]) + (1 - op["r"]) * math.log2(op["L_lo"])
    assert round(nominal, 2) == op["nominal_bits"]
    eff = oracle.effective_bits(oracle.BASE_AFFINE, op["L_hi"], op["L_lo"], op["r"])
    assert round(eff, 2) == op["effective_bits"]
    assert round(16 / eff, 2) == op["compression"]
    op = PV["operating_points"]["affine_r35"]
    nominal = op["r"] * math.log2(op["L_hi"]) + (1 - op["r"]) * math.log2(op["L_lo"])
    assert round(nominal, 2) == op["nominal_bits"]


def test_table6_columns():
    for row in PV["table6"]["rows"]:
        b = base_id(row["base"])
        code = row["r"] * oracle.paper_code_bits(row["L_hi"]) + \
            (1 - row["r"]) * oracle.paper_code_bits(row["L_lo"])
        assert round(code, 3) == row["code"], row["method"]
        eff = oracle.effective_bits(b, row["L_hi"], row["L_lo"], row["r"])
        assert round(eff, 3) == row["eff"], row["method"]


def test_table5_compression_and_tq_points():
    for row in PV["table5_compression"]["rows"]:
        eff = oracle.effective_bits(oracle.BASE_AFFINE, row["L"], row["L"], 0.0)
        assert round(16 / eff, 1) == row["compression"]
    tq = PV["tq_operating_point"]
    assert round(16 / oracle.effective_bits(oracle.BASE_TQ, 4, 3, 0.75), 1) == tq["mix_compression"]
    assert round(16 / oracle.effective_bits(oracle.BASE_TQ, 4, 4, 0.0), 1) == tq["u2_compression"]


def test_footprint_sec45():
    f = PV["footprint"]
    values = 2 * f["layers"] * f["kv_heads"] * f["head_dim"] * f["tokens"]   # Eq. 1
    assert round(values * 2 / 2**30, 1) == f["fp16_gib"]
    eff = oracle.effective_bits(oracle.BASE_AFFINE, 6, 5, 0.25)
    assert round(values * eff / 8 / 2**30, 2) == f["semkv_gib"]
    # this build's records (whole bytes per quarter-aligned row) stay within 2% of it
    n_high = oracle.high_count_floor(f["tokens"], 25, 100)
    layout = oracle.layout_bytes_per_token_head(oracle.BASE_AFFINE, 6, 5, n_high, f["tokens"])
    layout_gib = layout * f["layers"] * f["kv_heads"] / 2**30
    assert abs(layout_gib / f["semkv_gib"] - 1) < 0.02
