"""CPU checks of the C-ABI library: it loads, exports every entry point that
include/semkv.h declares, and its host-only logic (sizes, counts, argument
validation, the host Lloyd-Max codebook) behaves as documented.  No kernel runs."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "semkv.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_28911_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"\b(semkv_[a-z_0-9]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 12
    for n in names:
        assert hasattr(lib, n), n


def test_host_sizes_and_counts_match_oracle(lib):
    lib.semkv_record_bytes.restype = ctypes.c_size_t
    lib.semkv_row_bytes.restype = ctypes.c_size_t
    for L in range(2, 9):
        assert lib.semkv_row_bytes(L) == oracle.row_bytes(L)
        for base in (0, 1):
            assert lib.semkv_record_bytes(base, L) == oracle.record_bytes(base, L)
    assert lib.semkv_row_bytes(9) == 0 and lib.semkv_row_bytes(1) == 0
    lib.semkv_high_count_floor.restype = ctypes.c_uint32
    lib.semkv_block_high_count.restype = ctypes.c_uint32
    for T in (0, 1, 7, 128, 1024, 32768, 131072):
        for num, den in ((26, 100), (1, 4), (35, 100), (3, 4), (1, 1), (0, 5)):
            assert lib.semkv_high_count_floor(T, num, den) == oracle.high_count_floor(T, num, den)
            assert lib.semkv_block_high_count(T, num, den) == oracle.block_high_count(T, num, den)


def test_host_lloyd_max_agrees_with_oracle(lib):
    lib.semkv_lloyd_max_gaussian.argtypes = [ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p]
    for L in range(2, 9):
        c = np.zeros(L, np.float32)
        t = np.zeros(L - 1, np.float32)
        assert lib.semkv_lloyd_max_gaussian(L, c.ctypes.data, t.ctypes.data) == 0
        _, oc, ot, _ = oracle.lloyd_max_gaussian(L)
        assert np.array_equal(c, oc) and np.array_equal(t, ot), L


def test_argument_validation_returns_status(lib):
    p = ctypes.c_void_p
    lib.semkv_rank_assign.argtypes = [p, ctypes.c_int32, ctypes.c_int32, ctypes.c_uint32, p, p, p,
                                      p, ctypes.c_size_t, p]
    assert lib.semkv_rank_assign(None, 1, 10, 1, None, None, None, None, 0, None) == 1
    lib.semkv_quantize_pack.argtypes = [p, p, p, ctypes.c_int32, p, p, ctypes.c_uint32, p, p]
    assert lib.semkv_quantize_pack(None, None, None, 10, None, None, 0, None, None) == 1
    lib.semkv_decode_attention.argtypes = [p, p, ctypes.c_int32, p, p, ctypes.c_float, p,
                                           ctypes.c_size_t, p]
    assert lib.semkv_decode_attention(None, None, 0, None, None, 1.0, None, 0, None) == 1
    lib.semkv_status_string.restype = ctypes.c_char_p
    assert lib.semkv_status_string(3) == b"pool or staging capacity exceeded"


def test_rank_workspace_sizing_and_checks(lib):
    p = ctypes.c_void_p
    lib.semkv_rank_workspace_bytes.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    lib.semkv_rank_workspace_bytes.restype = ctypes.c_size_t
    assert lib.semkv_rank_workspace_bytes(2, 100, 1) == 2 * 4 * 100 * 4
    assert lib.semkv_rank_workspace_bytes(2, 100, 0) == 0
    lib.semkv_rank_assign.argtypes = [p, ctypes.c_int32, ctypes.c_int32, ctypes.c_uint32, p, p, p,
                                      p, ctypes.c_size_t, p]
    fake = 4096  # never dereferenced: every call below fails validation before a launch
    # ranks wanted without (enough) workspace -> SEMKV_EWORKSPACE
    assert lib.semkv_rank_assign(fake, 2, 100, 3, fake, fake, fake, None, 0, None) == 6
    assert lib.semkv_rank_assign(fake, 2, 100, 3, fake, fake, fake, fake, 3199, None) == 6
    # misaligned workspace -> SEMKV_EALIGN
    assert lib.semkv_rank_assign(fake, 2, 100, 3, fake, fake, fake, fake + 2, 3200, None) == 2


def test_fake_quant_validation(lib):
    from paper_2608_28911_gb300.semkv import QuantDescStruct
    p, i32 = ctypes.c_void_p, ctypes.c_int32
    lib.semkv_fake_quant.argtypes = [p, p, p, i32, i32, i32, i32, p, p, p, p]
    fake = 4096  # never dereferenced: every call below fails validation before a launch
    d = QuantDescStruct(base=0, levels_hi=6, levels_lo=5, head_dim=128)
    assert lib.semkv_fake_quant(None, fake, fake, 1, 1, 1, 1, None, fake, fake, None) == 1
    assert lib.semkv_fake_quant(ctypes.byref(d), None, fake, 1, 1, 1, 1, None, fake, fake,
                                None) == 1
    assert lib.semkv_fake_quant(ctypes.byref(d), fake, fake, 1, 1, 1, 0, None, fake, fake,
                                None) == 1
    assert lib.semkv_fake_quant(ctypes.byref(d), fake + 4, fake, 1, 1, 1, 1, None, fake, fake,
                                None) == 2
    # rows move in 16-byte chunks: 8-byte aligned buffers are refused too
    assert lib.semkv_fake_quant(ctypes.byref(d), fake, fake, 1, 1, 1, 1, None, fake + 8, fake,
                                None) == 2
    bad = QuantDescStruct(base=0, levels_hi=9, levels_lo=5, head_dim=128)
    assert lib.semkv_fake_quant(ctypes.byref(bad), fake, fake, 1, 1, 1, 1, None, fake, fake,
                                None) == 4
    tq = QuantDescStruct(base=1, levels_hi=4, levels_lo=3, head_dim=128)  # no tables
    assert lib.semkv_fake_quant(ctypes.byref(tq), fake, fake, 1, 1, 1, 1, None, fake, fake,
                                None) == 1


def test_row_alignment_rules_per_base(lib):
    """K/V rows move in 16-byte units (bulk or tensor copies) for every base but the
    affine one, which also takes 8-byte aligned rows; misaligned rows are refused with
    SEMKV_EALIGN before anything is launched."""
    from paper_2608_28911_gb300.semkv import CacheStruct, QuantDescStruct
    p, i32, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint32
    lib.semkv_quantize_pack.argtypes = [p, p, p, i32, p, p, u32, p, p]
    lib.semkv_append_block.argtypes = [p, p, u32, u32, p]
    fake = 1 << 20  # never dereferenced: every call below fails validation before a launch
    c = CacheStruct(batch=1, layers=1, kv_heads=1, q_heads=4, head_dim=128, block=16,
                    hi_pool=fake, lo_pool=fake, hi_cap=16, lo_cap=16, hi_tok=fake,
                    lo_tok=fake, stage_k=fake + 8, stage_v=fake, stage_score=fake,
                    stage_n=4, blk_is_high=fake, blk_slot=fake, dev_error=fake)
    aff = QuantDescStruct(base=0, levels_hi=6, levels_lo=5, head_dim=128)
    tq = QuantDescStruct(base=1, levels_hi=4, levels_lo=3, head_dim=128, signs=fake,
                         centroids_hi=fake, thresholds_hi=fake, centroids_lo=fake,
                         thresholds_lo=fake)
    had = QuantDescStruct(base=2, levels_hi=6, levels_lo=5, head_dim=128, signs=fake)
    for d in (tq, had):
        # rows 8-byte but not 16-byte aligned
        assert lib.semkv_quantize_pack(ctypes.byref(d), fake + 8, fake, 16, fake, fake, 4,
                                       ctypes.byref(c), None) == 2
        assert lib.semkv_quantize_pack(ctypes.byref(d), fake, fake + 8, 16, fake, fake, 4,
                                       ctypes.byref(c), None) == 2
        assert lib.semkv_append_block(ctypes.byref(d), ctypes.byref(c), 1, 4, None) == 2
    # the affine base refuses rows that are not even 8-byte aligned
    assert lib.semkv_quantize_pack(ctypes.byref(aff), fake + 4, fake, 16, fake, fake, 4,
                                   ctypes.byref(c), None) == 2
    c.stage_k = fake + 4
    assert lib.semkv_append_block(ctypes.byref(aff), ctypes.byref(c), 1, 4, None) == 2
