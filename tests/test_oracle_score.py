"""Pins of the oracle's KV-norm importance indicator (Sec. 3.3, KV-norm family:
key-norm ||K_i||_2 and value-norm ||V_i||_2 of the tensor being compressed)."""
import numpy as np

import oracle


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape).astype(np.float16)


def test_matches_the_norm_within_fp32_rounding():
    x = _rand((2, 3, 2, 7, 128), 1)
    s = oracle.score_kv_norm(x.view(np.uint16))
    ref = np.sqrt((x.astype(np.float64) ** 2).sum(axis=(1, 2, 4)))
    # 768 fp32 additions per score: relative error well inside 768 * 2^-24
    assert np.abs(s / ref - 1).max() < 1e-5


def test_constant_rows_and_single_entries_are_exact():
    x = np.ones((1, 2, 4, 3, 128), np.float16)
    s = oracle.score_kv_norm(x.view(np.uint16))
    assert np.all(s == np.float32(np.sqrt(np.float32(2 * 4 * 128))))   # sqrt(1024) = 32
    assert s[0, 0] == 32.0
    y = np.zeros((1, 2, 2, 4, 128), np.float16)
    y[0, 1, 1, 2, 77] = np.float16(-3.5)
    s = oracle.score_kv_norm(y.view(np.uint16))
    assert s[0, 2] == 3.5 and np.all(s[0, [0, 1, 3]] == 0.0)


def test_power_of_two_scaling_is_exact_and_tokens_are_independent():
    x = _rand((1, 2, 3, 9, 128), 2)
    s = oracle.score_kv_norm(x.view(np.uint16))
    s2 = oracle.score_kv_norm((x * np.float16(4)).view(np.uint16))
    assert np.array_equal(s2, 4 * s)
    perm = np.random.default_rng(3).permutation(9)
    sp = oracle.score_kv_norm(np.ascontiguousarray(x[:, :, :, perm]).view(np.uint16))
    assert np.array_equal(sp, s[:, perm])


def test_layer_range_is_the_last_m_layers_restriction():
    x = _rand((2, 5, 2, 4, 128), 4)
    s = oracle.score_kv_norm(x.view(np.uint16), layer_begin=3, layer_end=5)
    s_sliced = oracle.score_kv_norm(np.ascontiguousarray(x[:, 3:5]).view(np.uint16))
    assert np.array_equal(s, s_sliced)
