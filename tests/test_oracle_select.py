"""Pins for the oracle's top-r selection and block rule (CPU only).

Top-K (Eq. 4 / Algorithm 1): the rank of token i has a closed form that needs no
sorting, rank_i = #{j : s_j > s_i} + #{j < i : s_j = s_i} (NaN below all numbers),
checked exhaustively on every ordering of small tied score vectors; the selection
depends on the scores only through their ranking (Fig. 2 caption), so it must be
invariant under strictly increasing transforms.  Block rule (Algorithm 2): exactly
round(r n) per block with halves rounded up, values from Sec. 3.7 / Table 2.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle
from conftest import GOLDEN
from paper_2608_28911_gb300 import synthetic


def closed_form_rank(s):
    s = np.asarray(s, np.float64)
    T = len(s)
    out = np.zeros(T, np.int64)
    for i in range(T):
        if np.isnan(s[i]):
            out[i] = np.sum(~np.isnan(s)) + np.sum(np.isnan(s[:i]))
        else:
            better = np.sum(s[~np.isnan(s)] > s[i])
            tied_before = np.sum(s[:i] == s[i])
            out[i] = better + tied_before
    return out


def test_rank_closed_form_exhaustive_small():
    base = [3.0, 1.0, 3.0, np.nan, -0.0, 0.0, 2.0]
    for perm in itertools.permutations(range(len(base))):
        s = np.array([base[p] for p in perm], np.float32)
        for n_high in (0, 1, 3, 7):
            is_high, slot, rank = oracle.rank_assign(s, n_high)
            r = closed_form_rank(s)
            assert np.array_equal(rank, r)
            assert np.array_equal(is_high, (r < n_high).astype(np.uint8))


def test_rank_random_ties_and_slots():
    s = synthetic.scores_zipf(7, 3, 5000)
    s[0, 17] = np.nan
    s[1, :10] = -0.0
    s[1, 10:20] = 0.0
    n_high = oracle.high_count_floor(5000, 26, 100)
    is_high, slot, rank = oracle.rank_assign(s, n_high)
    for b in range(3):
        assert np.array_equal(rank[b], closed_form_rank(s[b]))
        assert is_high[b].sum() == n_high
        # every chosen score >= every unchosen one (NaN counts as lowest)
        x = np.where(np.isnan(s[b]), -np.inf, s[b].astype(np.float64))
        if 0 < n_high < 5000:
            assert x[is_high[b] == 1].min() >= x[is_high[b] == 0].max()
        # slots: 0..count-1 in token order within each class
        for cls in (0, 1):
            sl = slot[b][is_high[b] == cls]
            assert np.array_equal(sl, np.arange(len(sl)))


def test_rank_invariant_under_increasing_transform():
    # Zipf scores clipped to <= 1000 so that every transform below stays strictly
    # increasing after rounding to float32 (no new ties, no overflow)
    s = np.minimum(synthetic.scores_zipf(8, 2, 3000), 1000)
    n_high = 750
    ref = oracle.rank_assign(s, n_high)
    for f in (lambda x: np.exp(x / 50.0), lambda x: 3 * x - 7, lambda x: x ** 3):
        got = oracle.rank_assign(f(s.astype(np.float64)).astype(np.float32), n_high)
        for a, b in zip(ref, got):
            assert np.array_equal(a, b)


def test_high_count_floor_eq4():
    # K = floor(r T): cases of the five workloads, checked by hand
    assert oracle.high_count_floor(1024, 0, 100) == 0
    assert oracle.high_count_floor(32768, 26, 100) == 8519      # 8519.68
    assert oracle.high_count_floor(65536, 26, 100) == 17039     # 17039.36
    assert oracle.high_count_floor(131072, 26, 100) == 34078    # 34078.72
    assert oracle.high_count_floor(4096, 26, 100) == 1064       # 1064.96
    assert oracle.high_count_floor(32768, 3, 4) == 24576
    assert oracle.high_count_floor(7, 1, 1) == 7


def test_block_rule():
    pv = json.load(open(os.path.join(GOLDEN, "paper_values.json")))["block_rule"]
    for c in pv["cases"]:
        assert oracle.block_high_count(c["n"], c["r_num"], c["r_den"]) == c["n_high"]
    assert oracle.block_high_count(10, 35, 100) == 4      # 3.5 rounds up
    assert oracle.block_high_count(2, 1, 4) == 1          # 0.5 rounds up
    assert oracle.block_high_count(128, 26, 100) == 33    # 33.28
    assert oracle.block_high_count(0, 26, 100) == 0
    for n in range(1, 300):
        for num, den in ((25, 100), (26, 100), (35, 100), (3, 4), (1, 3)):
            k = oracle.block_high_count(n, num, den)
            assert abs(k - n * num / den) <= 0.5 + 1e-12  # at most half a token
