"""GPU parity of decode attention at the edges of its softmax scheme.

The decode kernels do not track a running maximum per tile: each head keeps a
reference exponent e, moved (with the running sums rescaled) only when a tile would
push p = 2^(logit - e) or P' = p * s_v past its bound, and P' reaches the tensor cores
as an fp16 hi + lo pair.  These tests drive that scheme where it is fragile, each
element by element against the oracle's fp64 attention over the same dequantized cache
(the paper's decoding over C^_KV, Algorithm 1; the staged fp16 tail of Algorithm 2
takes part):

  - sharp softmax: queries scaled x16 and x64 (near one-hot weights);
  - one dominant token late in the low pool: e must move after many tiles;
  - all keys equal: the output is the mean of the dequantized values;
  - value rows with ranges near +-60000 (s_v large, P' at its bound), and rows whose
    step is an fp16 subnormal (s_v tiny);
  - a logit shift (every key plus a constant vector): the output must not change.

Each case runs at T = 4096 (hi + lo pools over several CTAs of the balanced or split
plan, then the combine), on the plain affine 6/5, the Hadamard-rotated affine 6/5 and
the TurboQuant-MSE 4/3 bases, most with a staged fp16 tail.  One more case runs sharp
queries and dominant tokens over 320 (sequence, KV head) pairs, where the affine pools
take equal ranges on 16-warp CTAs that each hold several segments.

Tolerance: max-abs 2e-3 and relative L2 1e-3 at the synthetic scale (|v| below 64).
Binary32 carries a relative, not an absolute, error, so the absolute bound follows the
values' scale: where every value is scaled by a power of two sigma it is 2e-3 * sigma;
where a few rows are far larger it is max(2e-3, 8e-6 * max|v^|).  The tensor cores
round each fp32 accumulation toward zero (at most one binary32 ulp, 2^-23 relative,
per MMA) and a warp chains its PV products over up to ~64 tiles of a segment, so an
output may drift by 64 * 2^-23 = 8e-6 of the largest value it averages.
"""
import numpy as np
import pytest

import oracle
from paper_2608_28911_gb300 import synthetic
from parity import ATOL, RTOL_L2, Pair, attention_errors

pytestmark = pytest.mark.gpu

T = 4096
BASES = [
    (0, 6, 5, (26, 100)),     # plain affine, the 2.585/2.322-bit mix
    (2, 6, 5, (26, 100)),     # Hadamard-rotated affine
    (1, 4, 3, (3, 4)),        # TurboQuant-MSE, 2.0/1.585 bits
]
NSTAGE = 37


def _pair(base, L_hi, L_lo, r, seed, Hq=8, H=2, B=2):
    return Pair(base, L_hi, L_lo, B, 1, H, Hq, T, r[0], r[1], seed=seed, block=64)


def _stage_tail(p, seed, kscale=1.0, vscale=1.0, kfill=None):
    k, v = synthetic.kv(seed, p.B, 1, p.H, NSTAGE)
    if kfill is not None:
        k = np.full_like(k, kfill)
    k = (k.astype(np.float32) * kscale).astype(np.float16)
    v = (v.astype(np.float32) * vscale).astype(np.float16)
    p.stage(k, v, synthetic.scores_zipf(seed, p.B, NSTAGE))


def _value_max(p):
    return max(np.abs(oracle.dequant_cache_head(p.oc, b, 0, h)[1]).max()
               for b in range(p.B) for h in range(p.H))


def _check(p, q, atol=None):
    got, ref = p.decode(q=q)
    if atol is None:
        atol = max(ATOL, 8e-6 * _value_max(p))
    err, rel = attention_errors(got, ref)
    assert err <= atol and rel <= RTOL_L2, (err, rel, atol)
    assert int(p.cache.dev_error.item()) == 0
    return got, ref


# ------------------------------------------------------------ sharp softmax -----

@pytest.mark.parametrize("base,L_hi,L_lo,r", BASES)
@pytest.mark.parametrize("qmul", [16, 64])
def test_sharp_softmax(base, L_hi, L_lo, r, qmul):
    p = _pair(base, L_hi, L_lo, r, seed=500 + qmul + base)
    p.quantize()
    _stage_tail(p, 501 + base)
    q = synthetic.queries(502 + base, p.B, p.Hq).astype(np.float32) * qmul
    got, ref = _check(p, q.astype(np.float16))
    # near one-hot: most heads put almost all weight on one token
    assert np.isfinite(got).all()


@pytest.mark.parametrize("Hq", [2, 16])      # GQA groups of 1 and 8 (the unpacked path)
def test_sharp_softmax_group_sizes(Hq):
    p = _pair(0, 6, 5, (26, 100), seed=510 + Hq, Hq=Hq)
    p.quantize()
    _stage_tail(p, 511)
    q = synthetic.queries(512, p.B, p.Hq).astype(np.float32) * 64
    _check(p, q.astype(np.float16))


# -------------------------------------------- a late dominant token (low pool) -----

@pytest.mark.parametrize("base,L_hi,L_lo,r", BASES)
def test_late_dominant_token_in_low_pool(base, L_hi, L_lo, r):
    p = _pair(base, L_hi, L_lo, r, seed=520 + base)
    q = synthetic.queries(521 + base, p.B, p.Hq)
    # the last low-pool token of every sequence gets a key along query head 0 of KV
    # head 0 (logit about +40 for that head, ~2^58 times the others' weight)
    is_high, _, _ = oracle.rank_assign(p.s, oracle.high_count_floor(T, r[0], r[1]))
    k = p.k.astype(np.float32)
    for b in range(p.B):
        t_star = int(np.nonzero(is_high[b] == 0)[0][-1])
        qv = q[b, 0].astype(np.float32)
        k[b, 0, 0, t_star] = 40.0 * np.sqrt(128.0) * qv / float(qv @ qv)
    p.k = k.astype(np.float16)
    p.quantize()
    _stage_tail(p, 522 + base)
    got, ref = _check(p, q)
    # the dominant token did dominate head 0 of each sequence: the output is its value row
    for b in range(p.B):
        K, V = oracle.dequant_cache_head(p.oc, b, 0, 0)
        lg = K @ q[b, 0].astype(np.float64) / np.sqrt(128.0)
        j = int(np.argmax(lg))
        assert lg[j] - np.partition(lg, -2)[-2] > 20.0
        assert np.max(np.abs(ref[b, 0] - V[j])) < 1e-6


# ---------------------------------------------------------- all keys equal -----

@pytest.mark.parametrize("base,L_hi,L_lo,r", [
    (0, 6, 5, (26, 100)),     # a constant row dequantizes exactly at both level counts
    (2, 5, 5, (0, 100)),      # rotated rows: one level count, so hi and lo rows agree
    (1, 4, 4, (3, 4)),        # TQ: one codebook for both pools
])
def test_all_keys_equal_gives_mean_value(base, L_hi, L_lo, r):
    p = _pair(base, L_hi, L_lo, r, seed=530 + base)
    p.k = np.full_like(p.k, 0.75)
    p.quantize()
    if base == 0:
        _stage_tail(p, 531, kfill=0.75)   # fp16 0.75 rows equal the dequantized ones
    q = synthetic.queries(532 + base, p.B, p.Hq)
    got, ref = _check(p, q)
    for b in range(p.B):
        for h in range(p.H):
            K, V = oracle.dequant_cache_head(p.oc, b, 0, h)
            assert np.all(K == K[0])
            for qh in range(h * (p.Hq // p.H), (h + 1) * (p.Hq // p.H)):
                assert np.max(np.abs(ref[b, qh] - V.mean(axis=0))) < 1e-9


# ------------------------------------------------- value scales at the edges -----

@pytest.mark.parametrize("base,L_hi,L_lo,r", BASES)
def test_few_value_rows_near_fp16_limit(base, L_hi, L_lo, r):
    # every 97th token's value row spans -60000..60000: s_v near 24000-30000, P' = p s_v
    # at its bound for those tokens while the others stay at the synthetic scale
    p = _pair(base, L_hi, L_lo, r, seed=540 + base)
    v = p.v.astype(np.float32)
    rng = np.random.default_rng(541)
    v[:, :, :, ::97] = rng.uniform(-60000, 60000, v[:, :, :, ::97].shape)
    v[:, :, :, ::97, 0] = 60000.0
    v[:, :, :, ::97, 1] = -60000.0
    p.v = v.astype(np.float16)
    p.quantize()
    _stage_tail(p, 542 + base)
    _check(p, synthetic.queries(543 + base, p.B, p.Hq))


@pytest.mark.parametrize("base,L_hi,L_lo,r", BASES)
def test_all_value_rows_scaled_up(base, L_hi, L_lo, r):
    # values x 1024: the rows' ranges reach +-30000..60000 everywhere
    sigma = 1024.0
    p = _pair(base, L_hi, L_lo, r, seed=550 + base)
    p.v = (p.v.astype(np.float32) * sigma).astype(np.float16)
    p.quantize()
    _stage_tail(p, 551 + base, vscale=sigma)
    _check(p, synthetic.queries(552 + base, p.B, p.Hq), atol=ATOL * sigma)


@pytest.mark.parametrize("base,L_hi,L_lo,r", BASES)
def test_subnormal_step_value_rows(base, L_hi, L_lo, r):
    # values x 2^-20: the rows' steps s_v (and most values) are fp16 subnormals
    sigma = 2.0 ** -20
    p = _pair(base, L_hi, L_lo, r, seed=560 + base)
    p.v = (p.v.astype(np.float32) * sigma).astype(np.float16)
    p.quantize()
    _stage_tail(p, 561 + base, vscale=sigma)
    _check(p, synthetic.queries(562 + base, p.B, p.Hq), atol=ATOL * sigma)


# ---------------------------------------------------------------- logit shift -----

def test_logit_shift_leaves_output_unchanged():
    """Integer-valued keys shifted by +64 in every dim: min, max and every code difference
    are exact, so each dequantized key moves by exactly 64*1 and every logit of a head by
    the same 64 * scale * sum(q).  The softmax, and the output, must not change."""
    rng = np.random.default_rng(570)
    keys = None
    outs = []
    for shift in (0.0, 64.0):
        p = _pair(0, 6, 5, (26, 100), seed=571)
        if keys is None:
            keys = rng.integers(-3, 4, size=p.k.shape).astype(np.float32)
            kstage = rng.integers(-3, 4, size=(p.B, 1, p.H, NSTAGE, 128)).astype(np.float32)
        p.k = (keys + shift).astype(np.float16)
        p.quantize()
        _, vs = synthetic.kv(573, p.B, 1, p.H, NSTAGE)
        p.stage((kstage + shift).astype(np.float16), vs, synthetic.scores_zipf(573, p.B, NSTAGE))
        got, ref = _check(p, synthetic.queries(574, p.B, p.Hq))
        outs.append((got.astype(np.float64), ref))
    (g0, r0), (g1, r1) = outs
    assert np.max(np.abs(r0 - r1)) < 1e-9          # the oracle: shift invariant
    err, rel = attention_errors(g1, g0)
    assert err <= ATOL and rel <= RTOL_L2, (err, rel)


# ----------------------------- the equal-range plan: several segments per CTA -----

@pytest.mark.parametrize("base", [0, 2])
def test_sharp_softmax_and_dominant_token_equal_range_plan(base):
    """Many (sequence, KV head) pairs: 320 here, more than the CTAs of one wave, so the
    affine pools run equal weighted ranges on one CTA of 16 warps per SM, each CTA taking
    several segments (hi and lo pools of consecutive pairs) and loading new queries for
    each pair.  Queries scaled x16, and in every fifth sequence the last low-pool token
    dominates query head 0 of KV head 0 (logit 640, the rest below about 200); a staged
    fp16 tail.  Sampled heads, those heads included, against the oracle."""
    B, H, Hq, T_ = 40, 8, 32, 1200
    r = (26, 100)
    p = Pair(base, 6, 5, B, 1, H, Hq, T_, r[0], r[1], seed=560 + base, block=64)
    q = synthetic.queries(561 + base, B, Hq).astype(np.float32) * 16
    is_high, _, _ = oracle.rank_assign(p.s, oracle.high_count_floor(T_, r[0], r[1]))
    k = p.k.astype(np.float32)
    for b in range(0, B, 5):
        t_star = int(np.nonzero(is_high[b] == 0)[0][-1])
        qv = q[b, 0]
        # logit 640: the x16 queries put the other tokens' logits below about 200
        k[b, 0, 0, t_star] = 640.0 * np.sqrt(128.0) * qv / float(qv @ qv)
    p.k = k.astype(np.float16)
    p.quantize()
    _stage_tail(p, 562 + base)
    rng = np.random.default_rng(563 + base)
    heads = [(b, 0) for b in range(0, B, 5)]
    heads += [(int(b), int(qh)) for b, qh in zip(rng.integers(0, B, 24), rng.integers(0, Hq, 24))]
    q16 = q.astype(np.float16)
    got, ref = p.decode(q=q16, heads=heads)
    sel = np.zeros((B, Hq), bool)
    for b, qh in heads:
        sel[b, qh] = True
    err, rel = attention_errors(got[sel], ref[sel])
    assert err <= ATOL and rel <= RTOL_L2, (err, rel)
    assert np.isfinite(got).all()
    assert int(p.cache.dev_error.item()) == 0
    # the dominant tokens did dominate: those heads' outputs are their value rows
    for b in range(0, B, 5):
        K, V = oracle.dequant_cache_head(p.oc, b, 0, 0)
        lg = K @ q16[b, 0].astype(np.float64) / np.sqrt(128.0)
        j = int(np.argmax(lg))
        assert lg[j] - np.partition(lg, -2)[-2] > 20.0
