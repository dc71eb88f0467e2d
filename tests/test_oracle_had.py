"""Pins for the oracle's Hadamard-rotated affine base (Sec. 4.1: rows rotated by a
randomized Hadamard transform before the per-row affine quantizer).

Rounding toward -inf: the largest binary16 not above the input, checked against
numpy's binary16 neighbours, with the overflow and signed-zero cases.
1/sqrt(128): the binary32 nearest to 2^-3.5 (checked in 50-digit decimal).
Quantizer: the rotated row u, from scipy's Sylvester matrix in fp64, lies within half
a step of z + s c for every coordinate; each code is the nearest grid point; z is at
most min u; orthogonality carries the error bound to the original row; on rows with
outlier channels the rotated base has lower error than the plain one (the reason the
paper rotates).  Dequantization and fake quantization equal S H (z + s c)/sqrt(128)
from the Sylvester matrix.  Attention over a rotated cache equals fp64 attention over
those rows.
"""
from decimal import Decimal, getcontext

import numpy as np
import pytest
from scipy.linalg import hadamard

import oracle
from paper_2608_28911_gb300 import synthetic

D = 128
HM = hadamard(D).astype(np.float64)


def f16v(bits):
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float64)


# ------------------------------------------------------- rounding toward -inf --

def test_f16_round_down_is_largest_not_above():
    rng = np.random.default_rng(0)
    xs = np.concatenate([
        rng.standard_normal(3000) * 10.0 ** rng.integers(-9, 5, 3000),
        np.array([0.0, -0.0, 1.0, -1.0, 65504.0, -65504.0, 6e-8, -6e-8, 1e-12, -1e-12,
                  65519.0, 65520.0, -65519.0, 5.9604645e-08, -5.9604645e-08]),
    ]).astype(np.float32)
    for x in xs:
        r = oracle.f32_to_f16_rd(x)
        rv = np.uint16(r).view(np.float16)
        if x < -65504.0:
            assert r == 0xFC00, x
            continue
        if x > 65504.0:
            assert r == 0x7BFF, x
            continue
        assert float(rv) <= float(x), (x, rv)
        if r != 0x7BFF:
            up = np.nextafter(rv, np.float16(np.inf))
            assert float(up) > float(x), (x, rv)
    # exact values are unchanged, signs of zero kept
    for v in (np.float16(0.0), np.float16(-0.0), np.float16(3.140625), np.float16(-2.0e-7)):
        assert oracle.f32_to_f16_rd(np.float32(v)) == int(np.array(v).view(np.uint16))
    assert oracle.f32_to_f16_rd(np.float32(-1e-30)) == 0x8001
    assert oracle.f32_to_f16_rd(np.float32(1e-30)) == 0x0000


def test_inv_sqrt_d_is_nearest_binary32():
    getcontext().prec = 50
    exact = Decimal(1) / Decimal(128).sqrt()
    c = np.float32(oracle.inv_sqrt_d())
    for nb in (np.nextafter(c, np.float32(0)), np.nextafter(c, np.float32(1))):
        assert abs(Decimal(float(c)) - exact) < abs(Decimal(float(nb)) - exact)


# ----------------------------------------------------------------- quantizer ---

def rows(n, seed):
    k, _ = synthetic.kv(seed, 1, 1, 1, n)
    return synthetic.f16_bits(k)[0, 0, 0]


@pytest.mark.parametrize("L", [2, 3, 5, 6, 8])
def test_rotated_codes_within_half_step_and_nearest(L):
    X = rows(40, 7 + L)
    sg = synthetic.signs(7, 1, 1)[0, 0]
    for x in X:
        c, s16, z16 = oracle.affine_had_row(x, sg, L)
        s, z = f16v(s16), f16v(z16)
        u = HM @ (f16v(x) * sg) / np.sqrt(D)
        scale = np.abs(u).max()
        slack = 16 * 2.0 ** -24 * np.abs(f16v(x)).sum() + 4 * 2.0 ** -24 * scale
        assert z <= u.min() + slack
        assert z > u.min() - max(abs(u.min()) * 2.0 ** -10, 2.0 ** -24) - slack
        grid = z + s * np.arange(L)
        rec = z + s * c
        assert np.all(np.abs(rec - u) <= 0.5 * s * (1 + 2.0 ** -9) + slack)
        best = np.abs(u[:, None] - grid[None, :]).min(1)
        assert np.all(np.abs(rec - u) <= best + 2 * slack + s * 2.0 ** -20)


@pytest.mark.parametrize("L", [5, 6])
def test_rotation_is_orthonormal_through_dequant(L):
    """x^ from the oracle's dequantization equals S H (z + s c)/sqrt(128) built with the
    Sylvester matrix, and ||x - x^|| = ||u - (z + s c)|| (the rotation is orthonormal)."""
    B, NL, H, T = 1, 1, 2, 12
    k, v = synthetic.kv(13, B, NL, H, T)
    kb, vb = synthetic.f16_bits(k), synthetic.f16_bits(v)
    sg = synthetic.signs(13, NL, H)
    cache = oracle.Cache(base=oracle.BASE_AFFINE_HAD, L_hi=L, L_lo=L, batch=B, layers=NL,
                         kv_heads=H, q_heads=4 * H, block=16, hi_cap=16, lo_cap=16, signs=sg)
    oracle.quantize_prompt(cache, kb, vb, np.arange(T, dtype=np.float32)[None], 1, 2)
    for h in range(H):
        K, V = oracle.dequant_cache_head(cache, 0, 0, h)
        toks = np.concatenate([cache.hi_tok[0, :cache.hi_count], cache.lo_tok[0, :cache.lo_count]])
        for i, t in enumerate(toks):
            for rowbits, rec_row in ((kb[0, 0, h, t], K[i]), (vb[0, 0, h, t], V[i])):
                c, s16, z16 = oracle.affine_had_row(rowbits, sg[0, h], L)
                uh = f16v(z16) + f16v(s16) * c
                want = sg[0, h] * (HM @ uh) / np.sqrt(D)
                assert np.allclose(rec_row, want, rtol=0, atol=1e-12 * np.abs(uh).sum())
                x = f16v(rowbits)
                u = HM @ (x * sg[0, h]) / np.sqrt(D)
                assert abs(np.linalg.norm(x - rec_row) - np.linalg.norm(u - uh)) < 1e-9 * (
                    1 + np.linalg.norm(x))


@pytest.mark.parametrize("L", [3, 5, 6])
def test_rotation_lowers_error_on_outlier_rows(L):
    X = rows(200, 31)
    sg = synthetic.signs(31, 1, 1)[0, 0]
    err_plain = err_rot = 0.0
    for x in X:
        xf = f16v(x)
        c, s16, z16 = oracle.affine_row(x, L)
        err_plain += ((f16v(z16) + f16v(s16) * c - xf) ** 2).sum()
        c, s16, z16 = oracle.affine_had_row(x, sg, L)
        uh = f16v(z16) + f16v(s16) * c
        err_rot += ((sg * (HM @ uh) / np.sqrt(D) - xf) ** 2).sum()
    assert err_rot < 0.7 * err_plain, (err_rot, err_plain)


def test_constant_rotated_row_and_zero_row():
    sg = synthetic.signs(2, 1, 1)[0, 0]
    z = np.zeros(D, np.uint16)
    c, s16, z16 = oracle.affine_had_row(z, sg, 6)
    assert not c.any() and s16 == 0 and z16 == 0
    # x = sign_0 a e_0 rotates to the constant row a/sqrt(128): the offset rounds down
    # below it, so every code is equal and z + s c lands within half a step of it
    x = np.zeros(D, np.float16)
    x[0] = np.float16(sg[0] * 4.0)
    c, s16, z16 = oracle.affine_had_row(synthetic.f16_bits(x), sg, 6)
    u = 4.0 / np.sqrt(D)
    assert np.all(c == c[0])
    assert f16v(z16) <= u
    assert abs(f16v(z16) + f16v(s16) * c[0] - u) <= 0.5 * f16v(s16) + 2.0 ** -24


@pytest.mark.parametrize("L", [3, 6])
def test_rotated_fake_quant_matches_sylvester(L):
    B, NL, H, T = 1, 1, 2, 10
    k, v = synthetic.kv(17, B, NL, H, T)
    kb, vb = synthetic.f16_bits(k), synthetic.f16_bits(v)
    sg = synthetic.signs(17, NL, H)
    ko, vo = oracle.fake_quant(oracle.BASE_AFFINE_HAD, L, L, kb, vb, signs=sg)
    for x, xo in ((kb, ko), (vb, vo)):
        for h in range(H):
            for t in range(T):
                c, s16, z16 = oracle.affine_had_row(x[0, 0, h, t], sg[0, h], L)
                uh = f16v(z16) + f16v(s16) * c
                want = sg[0, h] * (HM @ uh) / np.sqrt(D)
                got = f16v(xo[0, 0, h, t])
                ulp = np.spacing(np.abs(want).astype(np.float16)).astype(np.float64)
                bound = ulp + 10 * 2.0 ** -24 * np.abs(uh).sum() / np.sqrt(D)
                assert np.all(np.abs(got - want) <= bound), (h, t)


def test_rotated_attention_equals_fp64_over_rotated_rows():
    B, NL, H, Hq, T = 1, 1, 2, 8, 40
    k, v = synthetic.kv(19, B, NL, H, T)
    kb, vb = synthetic.f16_bits(k), synthetic.f16_bits(v)
    sg = synthetic.signs(19, NL, H)
    cache = oracle.Cache(base=oracle.BASE_AFFINE_HAD, L_hi=6, L_lo=5, batch=B, layers=NL,
                         kv_heads=H, q_heads=Hq, block=16, hi_cap=48, lo_cap=48, signs=sg)
    scores = synthetic.scores_zipf(19, B, T)
    oracle.quantize_prompt(cache, kb, vb, scores, 26, 100)
    q = synthetic.f16_bits(synthetic.queries(19, B, Hq))
    scale = 1 / np.sqrt(D)
    out = oracle.decode_attention(cache, 0, q, scale)
    ih, _, _ = oracle.rank_assign(scores, oracle.high_count_floor(T, 26, 100))
    for h in range(H):
        Kr = np.zeros((T, D))
        Vr = np.zeros((T, D))
        for t in range(T):
            L = 6 if ih[0, t] else 5
            for x, dst in ((kb, Kr), (vb, Vr)):
                c, s16, z16 = oracle.affine_had_row(x[0, 0, h, t], sg[0, h], L)
                dst[t] = sg[0, h] * (HM @ (f16v(z16) + f16v(s16) * c)) / np.sqrt(D)
        for qh in range(h * 4, h * 4 + 4):
            qv = f16v(q[0, qh])
            lg = Kr @ qv * scale
            p = np.exp(lg - lg.max())
            want = (p[:, None] * Vr).sum(0) / p.sum()
            assert np.allclose(out[0, qh], want, rtol=0, atol=1e-10)
