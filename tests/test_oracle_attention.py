"""Pins for the oracle's cache assembly and fp64 decode attention (CPU only).

Attention: T = 1 returns v exactly; equal keys give the mean of the values; two
tokens follow the logistic closed form; a dominant logit returns its value; a
shift of every logit changes nothing; extended precision (long double) agrees on
small cases; the GQA head map is checked with per-head constant values.
Cache: dequantized rows sit within half a step of the inputs at the token each
slot names (pool placement, Eq. 7); every token is preserved exactly once
(Eqs. 8-9) through prompt quantization and block appends (Algorithm 2).
"""
import math

import numpy as np
import pytest

import oracle
from paper_2608_28911_gb300 import synthetic


def test_attention_single_token():
    rng = np.random.default_rng(0)
    q, k, v = rng.standard_normal((3, 128))
    out = oracle.attention_fp64(q, k[None], v[None], 0.1)
    assert np.array_equal(out, v)


def test_attention_equal_keys_gives_mean():
    rng = np.random.default_rng(1)
    k = np.tile(rng.standard_normal(128), (50, 1))
    V = rng.standard_normal((50, 128))
    out = oracle.attention_fp64(rng.standard_normal(128), k, V, 1 / math.sqrt(128))
    assert np.allclose(out, V.mean(0), atol=1e-14)


def test_attention_two_token_closed_form_and_shift():
    rng = np.random.default_rng(2)
    q = rng.standard_normal(128)
    K = rng.standard_normal((2, 128))
    V = rng.standard_normal((2, 128))
    sc = 0.3
    l1, l2 = sc * K[0] @ q, sc * K[1] @ q
    w1 = 1 / (1 + math.exp(l2 - l1))
    assert np.allclose(oracle.attention_fp64(q, K, V, sc), w1 * V[0] + (1 - w1) * V[1],
                       atol=1e-14)
    # shifting every key along q shifts every logit by the same amount
    K2 = K + 5.0 * q / (q @ q)
    assert np.allclose(oracle.attention_fp64(q, K2, V, sc), oracle.attention_fp64(q, K, V, sc),
                       atol=1e-12)


def test_attention_dominant_logit_and_long_double():
    rng = np.random.default_rng(3)
    q = rng.standard_normal(128)
    K = rng.standard_normal((16, 128))
    V = rng.standard_normal((16, 128))
    K[5] = 40 * q
    assert np.allclose(oracle.attention_fp64(q, K, V, 1.0), V[5], atol=1e-12)
    K = rng.standard_normal((16, 128))
    ql, Kl, Vl = q.astype(np.longdouble), K.astype(np.longdouble), V.astype(np.longdouble)
    lg = (Kl @ ql) * np.longdouble(0.125)
    p = np.exp(lg - lg.max())
    ref = (p @ Vl) / p.sum()
    assert np.allclose(oracle.attention_fp64(q, K, V, 0.125), ref.astype(np.float64), atol=1e-13)


def small_cache(base=0, L_hi=6, L_lo=5, B=2, NL=2, H=2, Hq=8, T=96, block=16, seed=0):
    cap = ((T + 4 * block + 15) // 16) * 16
    c = oracle.Cache(base=base, L_hi=L_hi, L_lo=L_lo, batch=B, layers=NL, kv_heads=H,
                     q_heads=Hq, block=block, hi_cap=cap, lo_cap=cap)
    if base == oracle.BASE_TQ:
        c.signs = synthetic.signs(seed, NL, H)
        _, c32, t32, _ = oracle.lloyd_max_gaussian(L_hi)
        c.cb_hi = (c32, t32)
        _, c32, t32, _ = oracle.lloyd_max_gaussian(L_lo)
        c.cb_lo = (c32, t32)
    return c


def test_prompt_pool_placement_within_half_step():
    B, NL, H, T = 2, 2, 2, 96
    c = small_cache(B=B, NL=NL, H=H, T=T)
    k, v = synthetic.kv(0, B, NL, H, T)
    s = synthetic.scores_zipf(0, B, T)
    is_high, slot = oracle.quantize_prompt(c, synthetic.f16_bits(k), synthetic.f16_bits(v), s, 26, 100)
    nh = oracle.high_count_floor(T, 26, 100)
    assert c.hi_count == nh and c.lo_count == T - nh
    for b in range(B):
        toks = np.concatenate([c.hi_tok[b, :c.hi_count], c.lo_tok[b, :c.lo_count]])
        assert sorted(toks) == list(range(T))                     # Eq. 9
        assert np.array_equal(np.sort(c.hi_tok[b, :c.hi_count]), np.nonzero(is_high[b])[0])
        for l in range(NL):
            for h in range(H):
                kh, vh = oracle.dequant_cache_head(c, b, l, h)
                kx = k[b, l, h, toks].astype(np.float64)
                vx = v[b, l, h, toks].astype(np.float64)
                # step of each row: (max-min)/(L-1), L by precision class
                Ls = np.where(np.arange(T) < c.hi_count, 6, 5)[:, None]
                kstep = (kx.max(1, keepdims=True) - kx.min(1, keepdims=True)) / (Ls - 1)
                vstep = (vx.max(1, keepdims=True) - vx.min(1, keepdims=True)) / (Ls - 1)
                assert np.all(np.abs(kh - kx) <= 0.5 * kstep * (1 + 2e-3) + 1e-6)
                assert np.all(np.abs(vh - vx) <= 0.5 * vstep * (1 + 2e-3) + 1e-6)


def test_blocks_preserve_every_token_and_count_exactly():
    B, NL, H, T, blk = 2, 1, 2, 64, 16
    c = small_cache(B=B, NL=NL, H=H, T=T, block=blk)
    k, v = synthetic.kv(1, B, NL, H, T + 3 * blk + 5)
    s = synthetic.scores_zipf(1, B, T + 3 * blk + 5)
    K16, V16 = synthetic.f16_bits(k), synthetic.f16_bits(v)
    oracle.quantize_prompt(c, K16[:, :, :, :T], V16[:, :, :, :T], s[:, :T], 35, 100)
    hi_before = c.hi_count
    for g in range(T, T + 3 * blk + 5):
        oracle.stage_token(c, K16[:, :, :, g], V16[:, :, :, g], s[:, g])
        if c.stage_n == blk:
            before = c.hi_count
            oracle.append_block(c, 35, 100)
            assert c.hi_count - before == oracle.block_high_count(blk, 35, 100)
    assert c.stage_n == 5 and c.n_tokens == T + 3 * blk
    oracle.append_block(c, 35, 100)   # end-of-turn flush of the residual block
    assert c.stage_n == 0 and c.n_tokens == T + 3 * blk + 5
    assert c.hi_count - hi_before == 3 * oracle.block_high_count(blk, 35, 100) + \
        oracle.block_high_count(5, 35, 100)
    for b in range(B):
        toks = np.concatenate([c.hi_tok[b, :c.hi_count], c.lo_tok[b, :c.lo_count]])
        assert sorted(toks) == list(range(T + 3 * blk + 5))
        # within each block the high tokens are the top scores (ties to earlier)
        for start in (T, T + blk, T + 2 * blk):
            blk_scores = s[b, start:start + blk]
            chosen = np.isin(np.arange(start, start + blk), c.hi_tok[b, :c.hi_count])
            ih, _, _ = oracle.rank_assign(blk_scores, oracle.block_high_count(blk, 35, 100))
            assert np.array_equal(chosen.astype(np.uint8), ih)


def test_decode_attention_gqa_map_and_staged_tail():
    # Each KV head holds a constant value row c_h; every query head of group h must
    # return exactly c_h, so a wrong head map is caught.  Staged fp16 tokens take part.
    B, NL, H, Hq, T, blk = 1, 1, 4, 16, 32, 16
    c = small_cache(B=B, NL=NL, H=H, Hq=Hq, T=T, block=blk)
    rng = np.random.default_rng(5)
    k = rng.standard_normal((B, NL, H, T, 128)).astype(np.float16)
    v = np.zeros((B, NL, H, T, 128), np.float16)
    for h in range(H):
        v[:, :, h] = h + 1.0
    oracle.quantize_prompt(c, synthetic.f16_bits(k), synthetic.f16_bits(v),
                           synthetic.scores_zipf(5, B, T), 26, 100)
    for g in range(3):
        oracle.stage_token(c, synthetic.f16_bits(k[:, :, :, g]), synthetic.f16_bits(v[:, :, :, g]),
                           np.float32([1.0]))
    q = synthetic.f16_bits(synthetic.queries(5, B, Hq))
    out = oracle.decode_attention(c, 0, q, 1 / math.sqrt(128))
    for qh in range(Hq):
        assert np.allclose(out[0, qh], qh // (Hq // H) + 1.0, atol=1e-12)


def grid_rows(rng, n, L):
    """Rows that lie exactly on an L-level affine grid containing both ends, with a
    power-of-two step: the quantizer reproduces them exactly."""
    c = rng.integers(0, L, (n, 128))
    c[:, 0], c[:, 1] = 0, L - 1
    step = 2.0 ** rng.integers(-4, 1, (n, 1))
    z = np.round(rng.standard_normal((n, 1)) * 4) * step
    return (z + step * c).astype(np.float16)


def test_decode_attention_lossless_grid_equals_fp64_attention():
    # With every row on its class's grid, dequantization is exact, so the oracle's
    # attention over hi pool + lo pool + fp16 tail must equal plain fp64 attention
    # over the original rows: any dropped term, wrong slot, scale or head fails.
    B, NL, H, Hq, T, blk = 2, 1, 2, 8, 80, 16
    c = small_cache(B=B, NL=NL, H=H, Hq=Hq, T=T + 8, block=blk)
    rng = np.random.default_rng(9)
    s = synthetic.scores_tiefree(9, B, T)
    n_high = oracle.high_count_floor(T, 26, 100)
    is_high, _, _ = oracle.rank_assign(s, n_high)
    k = np.zeros((B, NL, H, T, 128), np.float16)
    v = np.zeros_like(k)
    for b in range(B):
        for h in range(H):
            for i in range(T):
                L = 6 if is_high[b, i] else 5
                k[b, 0, h, i] = grid_rows(rng, 1, L)[0]
                v[b, 0, h, i] = grid_rows(rng, 1, L)[0]
    oracle.quantize_prompt(c, synthetic.f16_bits(k), synthetic.f16_bits(v), s, 26, 100)
    tail_k = rng.standard_normal((B, NL, H, 5, 128)).astype(np.float16)
    tail_v = rng.standard_normal((B, NL, H, 5, 128)).astype(np.float16)
    for g in range(5):
        oracle.stage_token(c, synthetic.f16_bits(tail_k[:, :, :, g]),
                           synthetic.f16_bits(tail_v[:, :, :, g]), np.float32([1.0, 2.0]))
    q16 = synthetic.queries(9, B, Hq)
    sc = 1 / math.sqrt(128)
    out = oracle.decode_attention(c, 0, synthetic.f16_bits(q16), sc)
    for b in range(B):
        for qh in range(Hq):
            h = qh // (Hq // H)
            K = np.concatenate([k[b, 0, h], tail_k[b, 0, h]]).astype(np.float64)
            V = np.concatenate([v[b, 0, h], tail_v[b, 0, h]]).astype(np.float64)
            logits = sc * K @ q16[b, qh].astype(np.float64)
            p = np.exp(logits - logits.max())
            assert np.allclose(out[b, qh], p @ V / p.sum(), atol=1e-11)
