"""Pins for the oracle's fp16 conversion and mixed-radix packing (CPU only).

What pins them (none of it re-types the oracle's own formulas):
  - numpy's IEEE float16 conversion (a library routine) for the hand-written
    binary32->binary16 rounding, on every fp16 midpoint and many random floats;
  - the paper's packing rates (Sec. 4.1, Table 6) and the information bound;
  - exhaustive round trips over every group value of every level count;
  - packed bytes worked out by hand (tests/golden/pack_examples.json).
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from conftest import GOLDEN

LEVELS = [2, 3, 4, 5, 6, 7, 8]


def test_f16_matches_numpy_random():
    rng = np.random.default_rng(1)
    bits = rng.integers(0, 2**32, size=2_000_000, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    x = x[np.isfinite(x)]
    ref = x.astype(np.float16).view(np.uint16)
    got = oracle.f32_to_f16_bits(x)
    assert np.array_equal(got, ref)


def test_f16_matches_numpy_on_every_midpoint_and_neighbour():
    # every finite fp16 value, the midpoints between neighbours, and 1 ulp (fp32)
    # either side of each midpoint: exactly where round-to-nearest-even decides
    h = np.arange(0, 0x7C00, dtype=np.uint16)
    v = h.view(np.float16).astype(np.float64)
    mids = (v[:-1] + v[1:]) / 2
    m32 = mids.astype(np.float32)
    cand = np.concatenate([v.astype(np.float32), m32,
                           np.nextafter(m32, np.float32(np.inf)),
                           np.nextafter(m32, np.float32(0))])
    cand = np.concatenate([cand, -cand, np.float32([65519.0, 65520.0, 65536.0, 1e30])])
    ref = cand.astype(np.float16).view(np.uint16)
    assert np.array_equal(oracle.f32_to_f16_bits(cand), ref)


def test_f16_to_f32_is_exact():
    h = np.arange(0, 0x10000, dtype=np.uint32).astype(np.uint16)
    ref = h.view(np.float16).astype(np.float32)
    got = oracle.f16_bits_to_f32(h)
    fin = np.isfinite(ref)
    assert np.array_equal(got[fin].view(np.uint32), ref[fin].view(np.uint32))
    assert np.array_equal(np.isnan(got), np.isnan(ref))


def test_paper_packing_rates():
    pv = json.load(open(os.path.join(GOLDEN, "paper_values.json")))["packing_rates"]
    for L in (2, 3, 4, 5, 6, 8):
        rate = oracle.paper_code_bits(L)
        assert round(rate, 3) == pv[str(L)]["code_bits"], L
    # Sec. 4.1: +0.49% over log2 5 and +0.58% over log2 6
    assert round(100 * (oracle.paper_code_bits(5) / math.log2(5) - 1), 2) == 0.49
    assert round(100 * (oracle.paper_code_bits(6) / math.log2(6) - 1), 2) == 0.58


@pytest.mark.parametrize("L", LEVELS)
def test_row_bytes_near_information_bound(L):
    rb = oracle.row_bytes(L)
    bound_bits = 128 * math.log2(L)
    assert rb * 8 >= bound_bits
    # layout 1 spends at most a few bits per quarter beyond the paper's rate
    assert rb * 8 <= 128 * oracle.paper_code_bits(L) + 4 * 7 + 7
    # quarter structure: four quarters fit the row
    assert 4 * oracle.quarter_bits(L) <= rb * 8


@pytest.mark.parametrize("L", LEVELS)
def test_exhaustive_group_round_trip(L):
    g = oracle.group_size(L)
    tuples = list(itertools.product(range(L), repeat=g))
    groups_per_row = 4 * (32 // g)
    rows = []
    for start in range(0, len(tuples), groups_per_row):
        chunk = tuples[start:start + groups_per_row]
        codes = np.zeros(128, np.uint8)
        for gi, tup in enumerate(chunk):
            q, s = divmod(gi, 32 // g)
            codes[32 * q + s * g: 32 * q + s * g + g] = tup
        rows.append(codes)
    # tails: every tail tuple in every quarter
    r = oracle.tail_codes(L)
    if r:
        for tup in itertools.product(range(L), repeat=r):
            codes = np.zeros(128, np.uint8)
            for q in range(4):
                codes[32 * q + 32 - r: 32 * q + 32] = tup
            rows.append(codes)
    packed = set()
    for codes in rows:
        row = oracle.pack_row(codes, L)
        assert np.array_equal(oracle.unpack_row(row, L), codes)
        packed.add(row.tobytes())
    assert len(packed) == len({c.tobytes() for c in rows})  # injective


@pytest.mark.parametrize("L", LEVELS)
def test_random_round_trip_and_zero_padding(L):
    rng = np.random.default_rng(L)
    qb = oracle.quarter_bits(L)
    for _ in range(300):
        codes = rng.integers(0, L, 128).astype(np.uint8)
        row = oracle.pack_row(codes, L)
        assert np.array_equal(oracle.unpack_row(row, L), codes)
        bits = np.unpackbits(row, bitorder="little")
        assert not bits[4 * qb:].any()  # padding bits are zero


def test_hand_worked_bytes():
    ex = json.load(open(os.path.join(GOLDEN, "pack_examples.json")))
    for case in ex["cases"]:
        L = case["L"]
        codes = np.zeros(128, np.uint8)
        for d, c in case["nonzero"]:
            codes[d] = c
        want = np.zeros(oracle.row_bytes(L), np.uint8)
        for i, b in case["bytes"]:
            want[i] = b
        assert np.array_equal(oracle.pack_row(codes, L), want), case["why"]
    for L, v in ex["all_max"].items():
        if L.startswith("_"):
            continue
        L = int(L)
        row = oracle.pack_row(np.full(128, L - 1, np.uint8), L)
        assert oracle.row_bytes(L) == v["row_bytes"]
        bits = np.unpackbits(row, bitorder="little")
        assert bits[:v["ones_bits"]].all() and not bits[v["ones_bits"]:].any()


def test_record_sizes():
    # affine: two rows + 4 fp16 parameters; TQ: two rows + 2 fp16 norms
    assert oracle.record_bytes(0, 6) == 92 and oracle.record_bytes(0, 5) == 84
    assert oracle.record_bytes(1, 4) == 68 and oracle.record_bytes(1, 3) == 56
    for L in LEVELS:
        assert oracle.record_bytes(0, L) % 4 == 0 and oracle.record_bytes(1, L) % 4 == 0
