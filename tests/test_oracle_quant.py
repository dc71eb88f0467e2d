"""Pins for the oracle's quantizers (CPU only).

Affine (Sec. 4.1 per-row asymmetric quantizer, Eq. 7): round-trip error within
half a step, monotone codes, the extreme values map to 0 and L-1, constant rows,
half-way ties going to even, and agreement with an fp64 nearest-level search.
TurboQuant-MSE (Sec. 4.9): the Walsh-Hadamard transform against scipy's Sylvester
matrix, H H = 128 I, Parseval, the Lloyd-Max codebook against Max (1960) and the
centroid condition by numerical integration, codes = nearest centroid, and the
reconstruction MSE of whole rows against the codebook's theoretical MSE.
"""
import json
import math
import os

import numpy as np
import pytest
from scipy import integrate
from scipy.linalg import hadamard

import oracle
from conftest import GOLDEN
from paper_2608_28911_gb300 import synthetic


def f16(a):
    return synthetic.f16_bits(np.asarray(a, np.float16))


def rows_f16(n, seed=0, outliers=True):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((n, 128)).astype(np.float32)
    if outliers:
        x[:, rng.choice(128, 4, replace=False)] *= 8
    return x.astype(np.float16)


# ------------------------------------------------------------------- affine ---

@pytest.mark.parametrize("L", [2, 3, 4, 5, 6, 8])
def test_affine_round_trip_within_half_step(L):
    for x in rows_f16(200, seed=L):
        codes, s16, z16 = oracle.affine_row(f16(x), L)
        s = float(oracle.f16_bits_to_f32(np.uint16(s16)))
        z = float(oracle.f16_bits_to_f32(np.uint16(z16)))
        xf = x.astype(np.float64)
        assert z == xf.min()                       # offset = row minimum, exact
        s32 = (np.float32(xf.max()) - np.float32(xf.min())) / np.float32(L - 1)
        xhat = z + s * codes.astype(np.float64)
        # half a step, plus the clamp at the top when fp16(s) < s, plus fp32 slack
        slack = (L - 1) * abs(float(s32) - s) + 4 * np.spacing(np.float32(abs(xf).max()))
        assert np.max(np.abs(xf - xhat)) <= s / 2 + slack


@pytest.mark.parametrize("L", [3, 5, 6])
def test_affine_codes_monotone_and_extremes(L):
    for x in rows_f16(100, seed=10 + L):
        codes, _, _ = oracle.affine_row(f16(x), L)
        order = np.argsort(x.astype(np.float64), kind="stable")
        assert np.all(np.diff(codes[order].astype(int)) >= 0)
        assert codes[np.argmin(x)] == 0 and codes[np.argmax(x)] == L - 1


def test_affine_constant_row_and_hand_example():
    codes, s16, z16 = oracle.affine_row(f16(np.full(128, 1.5)), 5)
    assert not codes.any() and s16 == 0 and z16 == int(f16([1.5])[0])
    # range [0, 4] with L = 5 -> s = 1, z = 0; 0.5 -> 0 and 2.5 -> 2 (ties to even),
    # 1.5 -> 2, 3.49 -> 3
    x = np.zeros(128, np.float16)
    x[1], x[2], x[3], x[4], x[5] = 4.0, 0.5, 2.5, 1.5, 3.49
    codes, s16, z16 = oracle.affine_row(f16(x), 5)
    assert s16 == 0x3C00 and z16 == 0
    assert list(codes[:6]) == [0, 4, 0, 2, 2, 3]


def test_affine_signed_zero_offset_is_positive():
    # all-zero rows with either zero sign store offset +0 and scale +0
    x = np.zeros(128, np.float16)
    x[::3] = -0.0
    for row in (x, -x, np.full(128, -0.0, np.float16)):
        codes, s16, z16 = oracle.affine_row(f16(row), 5)
        assert s16 == 0 and z16 == 0 and not codes.any()


@pytest.mark.parametrize("L", [5, 6])
def test_affine_matches_fp64_nearest_level(L):
    # away from half-way points the code is the nearest level z + s*k (fp64 search)
    for x in rows_f16(200, seed=20 + L):
        codes, s16, z16 = oracle.affine_row(f16(x), L)
        s = float(oracle.f16_bits_to_f32(np.uint16(s16)))
        z = float(oracle.f16_bits_to_f32(np.uint16(z16)))
        t = (x.astype(np.float64) - z) / s
        nearest = np.clip(np.floor(t + 0.5), 0, L - 1)
        clear = np.abs((t - np.floor(t)) - 0.5) > 1e-4
        assert np.array_equal(codes[clear], nearest[clear].astype(np.uint8))


# ----------------------------------------------------------------- Hadamard ---

def test_fwht_rows_are_sylvester_rows():
    H = hadamard(128)
    for k in range(128):
        e = np.zeros(128, np.float32)
        e[k] = 1
        assert np.array_equal(oracle.fwht_f32(e), H[k].astype(np.float32))


def test_fwht_involution_and_parseval():
    rng = np.random.default_rng(3)
    for _ in range(20):
        ints = rng.integers(-8, 9, 128).astype(np.float32)
        twice = oracle.fwht_f32(oracle.fwht_f32(ints))
        assert np.array_equal(twice, 128 * ints)          # H H = 128 I, exact here
        x = rng.standard_normal(128).astype(np.float32)
        w = oracle.fwht_f32(x).astype(np.float64)
        assert math.isclose((w ** 2).sum(), 128 * (x.astype(np.float64) ** 2).sum(),
                            rel_tol=1e-5)


def test_row_norm():
    rng = np.random.default_rng(4)
    for _ in range(50):
        x = rng.standard_normal(128).astype(np.float32) * rng.uniform(0.1, 10)
        assert math.isclose(oracle.row_norm_f32(x), float(np.linalg.norm(x.astype(np.float64))),
                            rel_tol=2e-6)


# ---------------------------------------------------------------- Lloyd-Max ---

@pytest.mark.parametrize("L", [2, 3, 4, 8])
def test_lloyd_max_matches_max_1960(L):
    ref = json.load(open(os.path.join(GOLDEN, "lloyd_max_max1960.json")))[str(L)]
    c64, c32, t32, mse = oracle.lloyd_max_gaussian(L)
    pos = sorted(c for c in c64 if c > -1e-12)
    assert np.allclose(pos, ref["centroids_pos"], atol=6e-4)
    tpos = sorted(t for t in t32.astype(np.float64) if t > -1e-7)
    assert np.allclose(tpos, ref["thresholds_pos"], atol=6e-4)
    assert abs(mse - ref["mse"]) < 6e-5
    if L == 2:
        assert math.isclose(c64[1], math.sqrt(2 / math.pi), rel_tol=1e-12)
        assert math.isclose(mse, 1 - 2 / math.pi, rel_tol=1e-10)


@pytest.mark.parametrize("L", [3, 4, 5, 6])
def test_lloyd_max_centroid_condition_by_quadrature(L):
    c64, _, t32, _ = oracle.lloyd_max_gaussian(L)
    edges = [-np.inf] + [(c64[i] + c64[i + 1]) / 2 for i in range(L - 1)] + [np.inf]
    pdf = lambda x: math.exp(-x * x / 2) / math.sqrt(2 * math.pi)
    for i in range(L):
        m0 = integrate.quad(pdf, edges[i], edges[i + 1], epsabs=1e-13)[0]
        m1 = integrate.quad(lambda x: x * pdf(x), edges[i], edges[i + 1], epsabs=1e-13)[0]
        assert abs(m1 / m0 - c64[i]) < 1e-9
    assert np.all(np.diff(c64) > 0) and np.allclose(c64, -c64[::-1], atol=1e-12)


# ---------------------------------------------------------------- TQ codes ----

@pytest.mark.parametrize("L", [3, 4])
def test_tq_codes_are_nearest_centroid(L):
    c64, c32, t32, _ = oracle.lloyd_max_gaussian(L)
    rng = np.random.default_rng(5)
    signs = np.where(rng.random(128) < 0.5, -1, 1).astype(np.int8)
    for x in rows_f16(100, seed=30 + L):
        codes, n16 = oracle.tq_row(f16(x), signs, L, t32)
        n = float(oracle.f16_bits_to_f32(np.uint16(n16)))
        u = hadamard(128) @ (x.astype(np.float64) * signs) / n
        dist = np.abs(u[:, None] - c32.astype(np.float64)[None, :])
        nearest = np.argmin(dist, axis=1)
        clear = np.abs(np.sort(dist, axis=1)[:, 1] - np.sort(dist, axis=1)[:, 0]) > 1e-5
        assert np.array_equal(codes[clear], nearest[clear])


@pytest.mark.parametrize("L", [3, 4])
def test_tq_reconstruction_mse_matches_codebook(L):
    # x^ = (n/128) S H cb[c]; with u ~ N(0,1) the relative MSE of a row equals the
    # codebook's MSE (rotation preserves norms): a wrong sign, transpose or scale
    # in quantize or dequantize breaks this.
    c64, c32, t32, mse = oracle.lloyd_max_gaussian(L)
    rng = np.random.default_rng(6)
    signs = np.where(rng.random(128) < 0.5, -1, 1).astype(np.int8)
    x = rows_f16(2000, seed=40 + L, outliers=False)
    errs, norms = 0.0, 0.0
    recs = []
    for row in x:
        ck, kn = oracle.tq_row(f16(row), signs, L, t32)
        rb = oracle.row_bytes(L)
        rec = np.zeros(oracle.record_bytes(1, L), np.uint8)
        rec[:rb] = oracle.pack_row(ck, L)
        rec[rb:2 * rb] = oracle.pack_row(ck, L)
        rec[2 * rb:2 * rb + 4] = np.array([kn, kn], np.uint16).view(np.uint8)
        recs.append(rec)
    khat, _ = oracle.dequant_records(1, L, np.stack(recs), signs, c32.astype(np.float64))
    xf = x.astype(np.float64)
    errs = ((xf - khat) ** 2).sum()
    norms = (xf ** 2).sum()
    assert abs(errs / norms - mse) < 0.1 * mse


def test_tq_zero_row():
    _, _, t32, _ = oracle.lloyd_max_gaussian(4)
    codes, n16 = oracle.tq_row(np.zeros(128, np.uint16), np.ones(128, np.int8), 4, t32)
    assert n16 == 0 and not codes.any()
