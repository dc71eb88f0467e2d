"""Pins for the oracle's fake quantization (Sec. 4.1: quantize, reconstruct to fp16).

Affine: the output equals fp16(z + s c) recomputed in numpy's own binary32 from the
pinned row quantizer's codes; every element lies within half a step (plus the fp16
rounding of the output) of its input; codes L-1 and 0 reproduce the row's max and
min up to the rounding of s and z.
TQ: the output equals fp16(sign * (H cb[c]) * n/128) with H scipy's Sylvester
matrix (exact in fp64) to within one fp16 ulp plus the binary32 butterflies' rounding
bound; its squared error over many rows
matches the codebook's distortion; a zero row reconstructs to zeros.
Mixed precision: each token takes exactly the uniform result of its own level.
"""
import numpy as np
import pytest
from scipy.linalg import hadamard

import oracle
from paper_2608_28911_gb300 import synthetic

D = 128


def cache_rows(B=1, NL=2, H=2, T=24, seed=5):
    k, v = synthetic.kv(seed, B, NL, H, T)
    return synthetic.f16_bits(k), synthetic.f16_bits(v)


def f16v(bits):
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float32)


@pytest.mark.parametrize("L", [2, 3, 5, 6, 8])
def test_affine_fake_equals_numpy_reconstruction(L):
    k, v = cache_rows()
    ko, vo = oracle.fake_quant(oracle.BASE_AFFINE, L, L, k, v)
    for x, xo in ((k, ko), (v, vo)):
        rows, outs = x.reshape(-1, D), xo.reshape(-1, D)
        for r, o in zip(rows, outs):
            c, s16, z16 = oracle.affine_row(r, L)
            s = np.float32(f16v(s16))
            z = np.float32(f16v(z16))
            want = (z + s * c.astype(np.float32)).astype(np.float16).view(np.uint16)
            np.testing.assert_array_equal(o, want)


@pytest.mark.parametrize("L", [3, 5, 6])
def test_affine_fake_error_within_half_step(L):
    k, v = cache_rows(T=40, seed=9)
    ko, _ = oracle.fake_quant(oracle.BASE_AFFINE, L, L, k, v)
    x = f16v(k).reshape(-1, D).astype(np.float64)
    xo = f16v(ko).reshape(-1, D).astype(np.float64)
    rng = x.max(1) - x.min(1)
    step = rng / (L - 1)
    # half a step, the fp16 rounding of the step and offset, and the output's rounding
    bound = 0.5 * step * (1 + 2 ** -9) + (L - 1) * step * 2 ** -11 + np.abs(x).max(1) * 2 ** -10
    err = np.abs(xo - x).max(1)
    assert np.all(err <= bound), (err / bound).max()
    # the extremes are reproduced up to the parameters' fp16 rounding
    assert np.all(np.abs(xo.max(1) - x.max(1)) <= 2 * L * step * 2 ** -11 + np.abs(x).max(1) * 2 ** -10)
    assert np.all(np.abs(xo.min(1) - x.min(1)) <= np.abs(x).max(1) * 2 ** -10)


def tq_codebooks(L_hi, L_lo):
    out = []
    for L in (L_hi, L_lo):
        _, cent32, thr32, _ = oracle.lloyd_max_gaussian(L)
        out.append((np.asarray(cent32, np.float32), np.asarray(thr32, np.float32)))
    return out


@pytest.mark.parametrize("L", [2, 3, 4])
def test_tq_fake_matches_sylvester_reconstruction(L):
    k, v = cache_rows(NL=1, H=2, T=16, seed=3)
    sg = synthetic.signs(3, 1, 2)
    (cb, _) = tq_codebooks(L, L)
    ko, vo = oracle.fake_quant(oracle.BASE_TQ, L, L, k, v, signs=sg, cb_hi=cb, cb_lo=cb)
    Hm = hadamard(D).astype(np.float64)
    for x, xo in ((k, ko), (v, vo)):
        for h in range(2):
            for t in range(16):
                r = x[0, 0, h, t]
                c, n16 = oracle.tq_row(r, sg[0, h], L, cb[1])
                y = Hm @ cb[0][c].astype(np.float64)
                n = float(f16v(n16))
                want = sg[0, h] * y * (n / 128.0)
                got = f16v(xo[0, 0, h, t]).astype(np.float64)
                ulp = np.spacing(np.abs(want).astype(np.float16)).astype(np.float64)
                # binary32 butterflies: 7 stages over 128 terms, each rounding within
                # 2^-24 of a partial sum bounded by 128 max|cb|; scaled by n/128
                fwht = 7 * 2.0 ** -24 * np.abs(cb[0]).max() * n * (1 + 2.0 ** -20)
                assert np.all(np.abs(got - want) <= ulp + fwht), (h, t)


@pytest.mark.parametrize("L,slack", [(2, 1.25), (3, 1.25), (4, 1.3)])
def test_tq_fake_distortion_matches_codebook(L, slack):
    """Per coordinate of the rotated, normalised row u ~ N(0,1): E(u - cb[c(u)])^2 is the
    codebook's distortion, and the rotation is orthogonal up to 1/128, so the whole-row
    relative squared error is about that distortion (Sec. 4.9)."""
    k, v = cache_rows(NL=1, H=4, T=64, seed=11)
    sg = synthetic.signs(11, 1, 4)
    (cb, _) = tq_codebooks(L, L)
    ko, _ = oracle.fake_quant(oracle.BASE_TQ, L, L, k, v, signs=sg, cb_hi=cb, cb_lo=cb)
    x = f16v(k).astype(np.float64).reshape(-1, D)
    xo = f16v(ko).astype(np.float64).reshape(-1, D)
    rel = ((xo - x) ** 2).sum(1) / (x ** 2).sum(1)
    # distortion of the Lloyd-Max codebook for N(0,1) by dense quadrature
    u = np.linspace(-9, 9, 400001)
    pdf = np.exp(-u * u / 2) / np.sqrt(2 * np.pi)
    c = (u[:, None] > cb[1][None, :].astype(np.float64)).sum(1)
    dist = np.trapezoid((u - cb[0][c]) ** 2 * pdf, u)
    # ||x||^2 = sum u^2 * n^2 / 128, E sum u^2 = 128, so E rel ~ dist
    assert rel.mean() <= dist * slack and rel.mean() >= dist / slack, (rel.mean(), dist)


def test_tq_fake_zero_row():
    k = np.zeros((1, 1, 1, 2, D), np.uint16)
    sg = synthetic.signs(1, 1, 1)
    (cb, _) = tq_codebooks(3, 3)
    ko, vo = oracle.fake_quant(oracle.BASE_TQ, 3, 3, k, k.copy(), signs=sg, cb_hi=cb, cb_lo=cb)
    assert not np.any(ko & 0x7FFF) and not np.any(vo & 0x7FFF)


@pytest.mark.parametrize("base,L_hi,L_lo", [(0, 6, 5), (0, 5, 3), (1, 4, 3)])
def test_mixed_precision_selects_per_token(base, L_hi, L_lo):
    B, NL, H, T = 2, 2, 2, 20
    k, v = cache_rows(B=B, NL=NL, H=H, T=T, seed=21)
    ih = (np.random.default_rng(4).random((B, T)) < 0.3).astype(np.uint8)
    kw = {}
    if base == oracle.BASE_TQ:
        cbh, cbl = tq_codebooks(L_hi, L_lo)
        kw = dict(signs=synthetic.signs(21, NL, H), cb_hi=cbh, cb_lo=cbl)
        hi_kw = dict(kw, cb_lo=cbh)
        lo_kw = dict(kw, cb_hi=cbl)
    else:
        hi_kw = lo_kw = kw
    ko, vo = oracle.fake_quant(base, L_hi, L_lo, k, v, is_high=ih, **kw)
    kh, vh = oracle.fake_quant(base, L_hi, L_hi, k, v, **hi_kw)
    kl, vl = oracle.fake_quant(base, L_lo, L_lo, k, v, **lo_kw)
    sel = ih.astype(bool)[:, None, None, :, None]
    np.testing.assert_array_equal(ko, np.where(sel, kh, kl))
    np.testing.assert_array_equal(vo, np.where(sel, vh, vl))
    assert 0 < ih.sum() < ih.size
