"""Pins for the oracle's TurboQuant-MSE rows under a dense random rotation (Sec. 4.9:
a random rotation, then the Gaussian Lloyd-Max codebook).

Rotation data: the stored fp16 matrix M is sqrt(128) times an orthogonal matrix to
within its fp16 rounding (M M^T = 128 I within 2e-3 relative); its first column has
Haar-random signs.  The rotated row: the oracle's w equals numpy's fp64 product M x
rounded to binary32.  With M = H S (Sylvester times signs, exact in fp16) the dense
base and the Walsh-Hadamard base reach the same codes except where the two binary32
roundings of w straddle a threshold, and the same dequantized rows for equal codes.
Codes are the nearest centroids of u = w / n; whole-row distortion equals the
codebook's MSE; dequantization equals (n/128) M^T cb[c]; attention over a dense-TQ
cache equals fp64 attention over those rows.
"""
import numpy as np
import pytest
from scipy.linalg import hadamard

import oracle
from paper_2608_28911_gb300 import synthetic

D = 128


def f16v(bits):
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float64)


def codebook(L):
    _, c32, t32, mse = oracle.lloyd_max_gaussian(L)
    return np.asarray(c32, np.float32), np.asarray(t32, np.float32), mse


def test_rotation_data_is_scaled_orthogonal():
    M = f16v(synthetic.rotations(4, 2, 3))
    assert M.shape == (2, 3, D, D)
    for l in range(2):
        for h in range(3):
            G = M[l, h] @ M[l, h].T
            assert np.abs(G - 128 * np.eye(D)).max() < 2e-3 * 128
    # different (layer, head) pairs draw different matrices
    assert np.abs(M[0, 0] - M[0, 1]).max() > 1.0 and np.abs(M[0, 0] - M[1, 0]).max() > 1.0


def test_rotated_row_is_fp64_product_rounded():
    M = synthetic.rotations(5, 1, 1)[0, 0]
    k, _ = synthetic.kv(5, 1, 1, 1, 20)
    for x in synthetic.f16_bits(k)[0, 0, 0]:
        w = oracle.tq_dense_w(x, M)
        ref = (f16v(M) @ f16v(x)).astype(np.float32)
        np.testing.assert_array_equal(w, ref)


@pytest.mark.parametrize("L", [2, 3, 4])
def test_hadamard_matrix_reproduces_the_hadamard_base(L):
    sg = synthetic.signs(8, 1, 1)[0, 0]
    M = (hadamard(D) * sg[None, :]).astype(np.float16).view(np.uint16)   # M x = H S x
    c32, t32, _ = codebook(L)
    k, v = synthetic.kv(8, 1, 1, 1, 60)
    X = np.concatenate([synthetic.f16_bits(k)[0, 0, 0], synthetic.f16_bits(v)[0, 0, 0]])
    same = total = 0
    for x in X:
        cd, nd = oracle.tq_dense_row(x, M, L, t32)
        ch, nh = oracle.tq_row(x, sg, L, t32)
        assert nd == nh
        total += D
        same += int((cd == ch).sum())
        diff = np.nonzero(cd != ch)[0]
        if diff.size:
            # only where u sits at a threshold within the butterflies' rounding
            u = f16v(M).dot(f16v(x)) / f16v(nd)
            gap = np.abs(u[diff, None] - t32[None, :].astype(np.float64)).min(1)
            assert np.all(gap < 1e-4 * (1 + np.abs(u[diff])))
            assert np.all(np.abs(cd[diff].astype(int) - ch[diff].astype(int)) == 1)
    assert same >= total - 3
    # equal codes dequantize to the same rows under both bases
    rec_d = np.zeros((1, oracle.record_bytes(oracle.BASE_TQ_DENSE, L)), np.uint8)
    cd, nd = oracle.tq_dense_row(X[0], M, L, t32)
    rec_d[0, :oracle.row_bytes(L)] = oracle.pack_row(cd, L)
    rec_d[0, 2 * oracle.row_bytes(L):2 * oracle.row_bytes(L) + 2] = np.array([nd], np.uint16).view(np.uint8)
    kd, _ = oracle.dequant_records(oracle.BASE_TQ_DENSE, L, rec_d, None, c32.astype(np.float64), M)
    kh, _ = oracle.dequant_records(oracle.BASE_TQ, L, rec_d, sg, c32.astype(np.float64))
    np.testing.assert_allclose(kd, kh, rtol=0, atol=1e-12)


@pytest.mark.parametrize("L", [2, 3, 4, 8])
def test_dense_codes_are_nearest_centroids(L):
    M = synthetic.rotations(9, 1, 1)[0, 0]
    c32, t32, _ = codebook(L)
    k, _ = synthetic.kv(9, 1, 1, 1, 30)
    for x in synthetic.f16_bits(k)[0, 0, 0]:
        c, n16 = oracle.tq_dense_row(x, M, L, t32)
        n = f16v(n16)
        assert abs(n - np.linalg.norm(f16v(x))) <= 2 ** -10 * n
        u = (f16v(M) @ f16v(x)) / n
        dist = np.abs(u[:, None] - c32[None, :].astype(np.float64))
        best = dist.min(1)
        mine = dist[np.arange(D), c]
        assert np.all(mine <= best + 1e-5 * (1 + np.abs(u)))


@pytest.mark.parametrize("L,slack", [(2, 1.2), (3, 1.2), (4, 1.25)])
def test_dense_distortion_matches_codebook(L, slack):
    B, NL, H, T = 1, 1, 2, 200
    k, v = synthetic.kv(10, B, NL, H, T)
    kb, vb = synthetic.f16_bits(k), synthetic.f16_bits(v)
    rot = synthetic.rotations(10, NL, H)
    c32, t32, mse = codebook(L)
    cache = oracle.Cache(base=oracle.BASE_TQ_DENSE, L_hi=L, L_lo=L, batch=B, layers=NL,
                         kv_heads=H, q_heads=4 * H, block=16, hi_cap=208, lo_cap=16,
                         cb_hi=(c32, t32), cb_lo=(c32, t32), rotation=rot)
    oracle.quantize_prompt(cache, kb, vb, np.ones((1, T), np.float32), 1, 1)
    rel = []
    for h in range(H):
        K, _ = oracle.dequant_cache_head(cache, 0, 0, h)
        toks = cache.hi_tok[0, :cache.hi_count]
        X = f16v(kb[0, 0, h, toks])
        rel.append(((K - X) ** 2).sum(1) / (X ** 2).sum(1))
    rel = np.concatenate(rel)
    assert mse / slack <= rel.mean() <= mse * slack, (rel.mean(), mse)


def test_dense_dequant_and_attention_against_numpy():
    B, NL, H, Hq, T = 1, 1, 2, 8, 48
    k, v = synthetic.kv(12, B, NL, H, T)
    kb, vb = synthetic.f16_bits(k), synthetic.f16_bits(v)
    rot = synthetic.rotations(12, NL, H)
    cbh, cbl = codebook(4), codebook(3)
    cache = oracle.Cache(base=oracle.BASE_TQ_DENSE, L_hi=4, L_lo=3, batch=B, layers=NL,
                         kv_heads=H, q_heads=Hq, block=16, hi_cap=48, lo_cap=48,
                         cb_hi=cbh[:2], cb_lo=cbl[:2], rotation=rot)
    scores = synthetic.scores_zipf(12, B, T)
    oracle.quantize_prompt(cache, kb, vb, scores, 3, 4)
    ih, _, _ = oracle.rank_assign(scores, oracle.high_count_floor(T, 3, 4))
    q = synthetic.f16_bits(synthetic.queries(12, B, Hq))
    out = oracle.decode_attention(cache, 0, q, 1 / np.sqrt(D))
    for h in range(H):
        M = f16v(rot[0, h])
        Kr, Vr = np.zeros((T, D)), np.zeros((T, D))
        for t in range(T):
            L, cb = (4, cbh) if ih[0, t] else (3, cbl)
            for x, dst in ((kb, Kr), (vb, Vr)):
                c, n16 = oracle.tq_dense_row(x[0, 0, h, t], rot[0, h], L, cb[1])
                dst[t] = f16v(n16) / D * (M.T @ cb[0][c].astype(np.float64))
        for qh in range(4 * h, 4 * h + 4):
            lg = Kr @ f16v(q[0, qh]) / np.sqrt(D)
            p = np.exp(lg - lg.max())
            np.testing.assert_allclose(out[0, qh], (p[:, None] * Vr).sum(0) / p.sum(),
                                       rtol=0, atol=1e-10)
