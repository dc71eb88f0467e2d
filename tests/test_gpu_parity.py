"""GPU parity: the CUDA library (through the C ABI) against the CPU oracle.

Bit-exact: top-r flags and slots, every packed record byte, slot->token arrays.
Attention: max-abs error <= 2e-3 and relative L2 error <= 1e-3 against the
oracle's fp64 attention over the same dequantized cache.
Sizes span several 16-token tiles with ragged tails, every level count, both
bases, GQA group sizes 1..8, the fp16 staged tail and the degenerate splits.
"""
import numpy as np
import pytest

import oracle
from paper_2608_28911_gb300 import synthetic
from parity import ATOL, RTOL_L2, Pair, attention_errors

pytestmark = pytest.mark.gpu


# ------------------------------------------------------------------ rank -----

@pytest.mark.parametrize("T", [1, 7, 16, 1000, 4097, 70001])
def test_rank_assign_bit_exact(T):
    import torch
    from paper_2608_28911_gb300 import semkv
    B = 3
    s = synthetic.scores_zipf(T, B, T)
    rng = np.random.default_rng(T)
    if T > 20:
        s[0, rng.choice(T, 5, replace=False)] = np.nan
        s[1, rng.choice(T, 5, replace=False)] = -0.0
        s[1, rng.choice(T, 5, replace=False)] = 0.0
        s[2, rng.choice(T, 3, replace=False)] = np.inf
        s[2, rng.choice(T, 3, replace=False)] = -np.inf
        s[2, rng.choice(T, 10, replace=False)] *= -1
    d = torch.device("cuda:0")
    st = torch.from_numpy(s).to(d)
    for n_high in sorted({0, 1, T // 4, max(T - 1, 0), T}):
        ih = torch.empty((B, T), dtype=torch.uint8, device=d)
        sl = torch.empty((B, T), dtype=torch.int32, device=d)
        rk = torch.empty((B, T), dtype=torch.int32, device=d)
        ws = torch.empty(semkv.semkv_rank_workspace_bytes(B, T) // 4, dtype=torch.int32, device=d)
        semkv.semkv_rank_assign(st, n_high, ih, sl, rank=rk, ws=ws)
        o_ih, o_sl, o_rk = oracle.rank_assign(s, n_high)
        assert np.array_equal(ih.cpu().numpy(), o_ih), n_high
        assert np.array_equal(sl.cpu().numpy().view(np.uint32), o_sl), n_high
        assert np.array_equal(rk.cpu().numpy().view(np.uint32), o_rk), n_high


# -------------------------------------------------------------- quantize -----

@pytest.mark.parametrize("base,L_hi,L_lo,B,NL,H,T,r", [
    (0, 5, 5, 1, 1, 1, 1024, (0, 100)),     # tiny uniform 5-level affine
    (0, 6, 5, 2, 2, 2, 333, (26, 100)),     # mixed 6/5, ragged
    (0, 2, 3, 1, 1, 2, 70, (1, 2)),
    (0, 4, 7, 1, 1, 2, 70, (1, 3)),
    (0, 8, 8, 1, 2, 1, 50, (1, 2)),
    (1, 4, 3, 1, 2, 2, 200, (3, 4)),        # TQ 4/3
    (1, 6, 5, 1, 1, 2, 90, (1, 4)),
    (1, 8, 2, 1, 1, 2, 90, (1, 4)),
    (2, 6, 5, 2, 2, 2, 333, (26, 100)),     # Hadamard-rotated affine 6/5
    (2, 5, 5, 1, 1, 2, 100, (0, 100)),
    (2, 2, 8, 1, 1, 2, 70, (1, 2)),
    (2, 3, 7, 1, 2, 1, 50, (1, 3)),
])
def test_quantize_pack_bit_exact(base, L_hi, L_lo, B, NL, H, T, r):
    p = Pair(base, L_hi, L_lo, B, NL, H, 4 * H, T, r[0], r[1], seed=T + L_hi)
    p.quantize()
    assert np.array_equal(p.is_high.cpu().numpy(), p.o_is_high)
    p.assert_records_equal()
    p.assert_untouched_past_counts()
    assert int(p.cache.dev_error.item()) == 0


@pytest.mark.parametrize("base", [0, 1, 2])
def test_quantize_edge_rows_bit_exact(base):
    # constant rows, signed zeros, tiny (subnormal-step) ranges and huge ranges (for the
    # rotated base the rotated range passes 65504: the offset and scale saturate; for TQ
    # the norm saturates and a zero row has norm 0, all codes 0)
    p = Pair(base, 6, 5, 1, 1, 2, 8, 64, 1, 2, seed=3)
    k = p.k.astype(np.float32)
    v = p.v.astype(np.float32)
    k[0, 0, 0, 0] = 1.5
    k[0, 0, 0, 1] = 0.0
    k[0, 0, 0, 1, ::2] = -0.0
    k[0, 0, 0, 2] = np.linspace(0, 6e-5, 128)
    k[0, 0, 0, 3] = np.linspace(-60000, 60000, 128)
    v[0, 0, 1, 4] = -0.0
    v[0, 0, 1, 5, 0] = 65504.0
    v[0, 0, 1, 5, 1] = -65504.0
    p.k, p.v = k.astype(np.float16), v.astype(np.float16)
    p.quantize()
    p.assert_records_equal()


# TQ rows in which some u = y * fl(1/n) equals a codebook threshold exactly (found by a
# search over seeded inputs: token, dim).  Ties go low (Sec. 4.9's quantizer compares
# strictly), and in the rows marked + the exact product y * fl(1/n) lies above the
# threshold, so a quantizer that fused the multiply into its comparison would round the
# code up there.
@pytest.mark.parametrize("seed,L,row,tok,dim", [
    (21, 4, "v", 1214, 122),     # +
    (27, 4, "v", 866, 73),       # +
    (104, 4, "k", 2720, 122),    # +
    (110, 4, "v", 1758, 125),    # +
    (15, 4, "v", 563, 8),
    (153, 3, "k", 3621, 35),     # +
    (197, 3, "k", 2525, 115),    # +
    (62, 3, "k", 1718, 61),
])
def test_tq_threshold_ties_bit_exact(seed, L, row, tok, dim):
    p = Pair(1, L, L, 1, 1, 1, 4, 4096, 1, 1, seed=seed)
    # the input still holds the tie: u at (tok, dim) equals a threshold
    x = (p.k if row == "k" else p.v)[0, 0, 0, tok].astype(np.float32)
    w = x * synthetic.signs(seed, 1, 1)[0, 0].astype(np.float32)
    hs = 1
    while hs < 128:
        i = np.arange(128)[(np.arange(128) & hs) == 0]
        a, b = w[i].copy(), w[i + hs].copy()
        w[i], w[i + hs] = a + b, a - b
        hs <<= 1
    sq = x * x
    part = sq[0::4].copy()
    for k in range(1, 4):
        part = part + sq[k::4]
    pn = part[:16] + part[16:]
    while len(pn) > 1:
        pn = pn[:len(pn) // 2] + pn[len(pn) // 2:]
    n = np.float32(np.float16(np.sqrt(pn[0])))
    u = np.float32(w[dim] * (np.float32(1) / n))
    _, _, thr, _ = oracle.lloyd_max_gaussian(L)
    assert u in thr.astype(np.float32)
    p.quantize()
    p.assert_records_equal()


# ---------------------------------------------------------------- decode -----

def check_attention(p, layer=0, qseed=0):
    got, ref = p.decode(layer, qseed)
    err, rel = attention_errors(got, ref)
    assert err <= ATOL and rel <= RTOL_L2, (err, rel)
    assert int(p.cache.dev_error.item()) == 0
    return err, rel


@pytest.mark.parametrize("L_hi,L_lo,B,NL,H,Hq,T,r", [
    (5, 5, 1, 1, 1, 4, 1024, (0, 100)),     # tiny uniform 5-level, 4 query heads
    (6, 5, 2, 2, 2, 8, 333, (26, 100)),     # mixed, ragged tiles, layer 1 checked too
    (6, 5, 1, 1, 8, 32, 2048, (26, 100)),   # Llama-3.1-8B layer shape, short context
    (2, 2, 1, 1, 2, 8, 100, (0, 1)),
    (3, 4, 1, 1, 2, 8, 100, (1, 2)),
    (7, 8, 1, 1, 2, 8, 100, (1, 2)),
    (6, 5, 1, 1, 2, 2, 200, (1, 4)),        # GQA group of 1
    (6, 5, 1, 1, 2, 16, 200, (1, 4)),       # GQA group of 8
    (6, 5, 1, 1, 1, 3, 150, (1, 4)),        # GQA group of 3
    (6, 5, 1, 1, 1, 4, 1, (0, 1)),          # a single token
    (6, 5, 1, 1, 1, 4, 40, (1, 1)),         # every token high
])
def test_decode_attention_matches_oracle(L_hi, L_lo, B, NL, H, Hq, T, r):
    p = Pair(0, L_hi, L_lo, B, NL, H, Hq, T, r[0], r[1], seed=7 + T)
    p.quantize()
    for layer in range(NL):
        check_attention(p, layer)


@pytest.mark.parametrize("L", [2, 7, 8])
def test_uniform_grid_points_quantize_and_decode(L):
    """The uniform grid points of the cliff sweep (1.0, 2.807, 3.0 bits per code): every
    token at L levels (r = 0, the high pool empty), records bit-exact, attention within
    tolerance."""
    p = Pair(0, L, L, 1, 1, 2, 8, 300, 0, 100, seed=40 + L)
    p.quantize()
    assert np.array_equal(p.is_high.cpu().numpy(), p.o_is_high)
    p.assert_records_equal()
    check_attention(p)


@pytest.mark.parametrize("base", [0, 2])
def test_decode_attention_with_staged_tail(base):
    p = Pair(base, 6, 5, 2, 1, 2, 8, 300, 26, 100, seed=11, block=32)
    p.quantize()
    k, v = synthetic.kv(12, 2, 1, 2, 20)
    s = synthetic.scores_zipf(12, 2, 20)
    import torch
    for g in range(20):
        kt = torch.from_numpy(np.ascontiguousarray(k[:, :, :, g])).to(p.dev)
        vt = torch.from_numpy(np.ascontiguousarray(v[:, :, :, g])).to(p.dev)
        p.cache.stage_token(kt, vt, torch.from_numpy(np.ascontiguousarray(s[:, g])).to(p.dev))
        oracle.stage_token(p.oc, synthetic.f16_bits(k[:, :, :, g]), synthetic.f16_bits(v[:, :, :, g]),
                           s[:, g])
    check_attention(p)


@pytest.mark.parametrize("base", [0, 2])
def test_append_blocks_and_flush_match_oracle(base):
    import torch
    from paper_2608_28911_gb300 import semkv
    blk, T0, ngen = 32, 200, 2 * 32 + 9
    p = Pair(base, 6, 5, 2, 2, 2, 8, T0, 26, 100, seed=21, block=blk, extra_cap=ngen)
    p.quantize()
    k, v = synthetic.kv(22, 2, 2, 2, ngen)
    s = synthetic.scores_zipf(22, 2, ngen)
    for g in range(ngen):
        kt = torch.from_numpy(np.ascontiguousarray(k[:, :, :, g])).to(p.dev)
        vt = torch.from_numpy(np.ascontiguousarray(v[:, :, :, g])).to(p.dev)
        p.cache.stage_token(kt, vt, torch.from_numpy(np.ascontiguousarray(s[:, g])).to(p.dev))
        oracle.stage_token(p.oc, synthetic.f16_bits(k[:, :, :, g]), synthetic.f16_bits(v[:, :, :, g]),
                           s[:, g])
        if p.cache.stage_n == blk:
            semkv.semkv_append_block(p.desc, p.cache, 26, 100)
            oracle.append_block(p.oc, 26, 100)
            torch.cuda.synchronize()
            p.assert_records_equal()
        if g % 13 == 0:
            check_attention(p, layer=g % 2, qseed=g)
    semkv.semkv_append_block(p.desc, p.cache, 26, 100)   # end-of-turn flush
    oracle.append_block(p.oc, 26, 100)
    torch.cuda.synchronize()
    p.assert_records_equal()
    assert p.cache.stage_n == 0 and p.cache.n_tokens == T0 + ngen
    check_attention(p, layer=1, qseed=99)


@pytest.mark.parametrize("base,blk", [(0, 1024), (0, 1000), (1, 1024), (1, 1000)])
def test_append_large_block_matches_oracle(base, blk):
    """The largest block the cache allows (1024 tokens) and a ragged one: one pass ranks
    the block and writes the pools' slot maps, then the block is packed."""
    import torch
    from paper_2608_28911_gb300 import semkv
    T0, ngen = 64, blk + 3
    p = Pair(base, 4 if base == 1 else 6, 3 if base == 1 else 5, 1, 1, 2, 8, T0, 26, 100,
             seed=23, block=blk, extra_cap=ngen)
    p.quantize()
    k, v = synthetic.kv(24, 1, 1, 2, ngen)
    s = synthetic.scores_zipf(24, 1, ngen)
    for g in range(ngen):
        kt = torch.from_numpy(np.ascontiguousarray(k[:, :, :, g])).to(p.dev)
        vt = torch.from_numpy(np.ascontiguousarray(v[:, :, :, g])).to(p.dev)
        p.cache.stage_token(kt, vt, torch.from_numpy(np.ascontiguousarray(s[:, g])).to(p.dev))
        oracle.stage_token(p.oc, synthetic.f16_bits(k[:, :, :, g]), synthetic.f16_bits(v[:, :, :, g]),
                           s[:, g])
        if p.cache.stage_n == blk:
            semkv.semkv_append_block(p.desc, p.cache, 26, 100)
            oracle.append_block(p.oc, 26, 100)
            torch.cuda.synchronize()
            p.assert_records_equal()
    assert p.cache.stage_n == 3 and int(p.cache.dev_error.item()) == 0
    check_attention(p, layer=0, qseed=7)     # pools + the 3 staged fp16 tokens


# ------------------------------------------- Hadamard-rotated affine decode -----

@pytest.mark.parametrize("L_hi,L_lo,B,NL,H,Hq,T,r", [
    (6, 5, 2, 2, 2, 8, 333, (26, 100)),     # mixed, ragged tiles, layer 1 checked too
    (6, 5, 1, 1, 8, 32, 2048, (26, 100)),   # Llama-3.1-8B layer shape, short context
    (5, 5, 1, 1, 1, 4, 1024, (0, 100)),
    (2, 3, 1, 1, 2, 8, 100, (1, 2)),
    (8, 7, 1, 1, 2, 16, 150, (1, 4)),       # GQA group of 8
    (6, 5, 1, 1, 1, 3, 150, (1, 4)),        # GQA group of 3
])
def test_had_decode_attention_matches_oracle(L_hi, L_lo, B, NL, H, Hq, T, r):
    p = Pair(2, L_hi, L_lo, B, NL, H, Hq, T, r[0], r[1], seed=60 + T)
    p.quantize()
    p.assert_records_equal()
    for layer in range(NL):
        check_attention(p, layer)


# --------------------------------------------- dense-rotation TQ (tcgen05) -----

@pytest.mark.parametrize("L_hi,L_lo,B,NL,H,Hq,T,r", [
    (4, 3, 1, 2, 2, 8, 333, (3, 4)),        # the 2.0/1.585-bit mix at r = 75%, ragged
    (4, 3, 2, 1, 8, 32, 1100, (3, 4)),      # Mistral-7B layer shape, short context
    (2, 2, 1, 1, 2, 4, 64, (0, 1)),         # one full 64-token tile
    (8, 5, 1, 1, 2, 16, 150, (1, 4)),       # CUDA-core decode path, GQA group of 8
    (3, 2, 1, 1, 1, 4, 1, (1, 1)),          # a single token
])
def test_dense_tq_quantize_and_decode(L_hi, L_lo, B, NL, H, Hq, T, r):
    p = Pair(3, L_hi, L_lo, B, NL, H, Hq, T, r[0], r[1], seed=70 + T)
    p.quantize()
    assert np.array_equal(p.is_high.cpu().numpy(), p.o_is_high)
    p.assert_records_equal_up_to_ties()
    assert int(p.cache.dev_error.item()) == 0
    p.adopt_gpu_records()
    for layer in range(NL):
        check_attention(p, layer)


def test_dense_tq_append_blocks_and_staged_tail():
    import torch
    from paper_2608_28911_gb300 import semkv
    blk, T0, ngen = 32, 150, 2 * 32 + 5
    p = Pair(3, 4, 3, 1, 2, 2, 8, T0, 3, 4, seed=81, block=blk, extra_cap=ngen)
    p.quantize()
    p.assert_records_equal_up_to_ties()
    k, v = synthetic.kv(82, 1, 2, 2, ngen)
    s = synthetic.scores_zipf(82, 1, ngen)
    for g in range(ngen):
        kt = torch.from_numpy(np.ascontiguousarray(k[:, :, :, g])).to(p.dev)
        vt = torch.from_numpy(np.ascontiguousarray(v[:, :, :, g])).to(p.dev)
        p.cache.stage_token(kt, vt, torch.from_numpy(np.ascontiguousarray(s[:, g])).to(p.dev))
        oracle.stage_token(p.oc, synthetic.f16_bits(k[:, :, :, g]), synthetic.f16_bits(v[:, :, :, g]),
                           s[:, g])
        if p.cache.stage_n == blk:
            semkv.semkv_append_block(p.desc, p.cache, 3, 4)
            oracle.append_block(p.oc, 3, 4)
            torch.cuda.synchronize()
            allk = np.concatenate([p.k, k], axis=3)
            allv = np.concatenate([p.v, v], axis=3)
            p.assert_records_equal_up_to_ties(allk, allv)
    p.adopt_gpu_records()
    check_attention(p, layer=1, qseed=5)     # pools + the 5 staged fp16 tokens
    assert int(p.cache.dev_error.item()) == 0


# ------------------------------------------------------------ TQ decode -----

@pytest.mark.parametrize("L_hi,L_lo,B,NL,H,Hq,T,r", [
    (4, 3, 1, 2, 2, 8, 333, (3, 4)),        # the 2.0/1.585-bit TQ mix at r = 75%
    (4, 3, 2, 1, 8, 32, 1100, (3, 4)),      # Mistral-7B layer shape, short context
    (2, 2, 1, 1, 2, 4, 100, (0, 1)),
    (6, 5, 1, 1, 2, 16, 150, (1, 4)),
    (8, 7, 1, 1, 1, 1, 64, (1, 2)),
])
def test_tq_decode_attention_matches_oracle(L_hi, L_lo, B, NL, H, Hq, T, r):
    p = Pair(1, L_hi, L_lo, B, NL, H, Hq, T, r[0], r[1], seed=40 + T)
    p.quantize()
    p.assert_records_equal()
    for layer in range(NL):
        check_attention(p, layer)


def test_tq_decode_with_staged_tail():
    import torch
    p = Pair(1, 4, 3, 1, 1, 2, 8, 200, 3, 4, seed=51, block=32)
    p.quantize()
    k, v = synthetic.kv(52, 1, 1, 2, 11)
    s = synthetic.scores_zipf(52, 1, 11)
    for g in range(11):
        kt = torch.from_numpy(np.ascontiguousarray(k[:, :, :, g])).to(p.dev)
        vt = torch.from_numpy(np.ascontiguousarray(v[:, :, :, g])).to(p.dev)
        p.cache.stage_token(kt, vt, torch.from_numpy(np.ascontiguousarray(s[:, g])).to(p.dev))
        oracle.stage_token(p.oc, synthetic.f16_bits(k[:, :, :, g]), synthetic.f16_bits(v[:, :, :, g]),
                           s[:, g])
    check_attention(p)


# ------------------------------------------------------ KV-norm scoring -----

@pytest.mark.parametrize("B,NL,H,T,lb,le", [
    (2, 1, 8, 1000, 0, 1),      # value-norm of one Llama-shaped layer
    (1, 4, 2, 333, 2, 4),       # last-2-layers restriction, ragged T
    (3, 2, 1, 17, 0, 2),
])
def test_score_kv_norm_bit_exact_and_ranks(B, NL, H, T, lb, le):
    import torch
    from paper_2608_28911_gb300 import semkv
    _, v = synthetic.kv(T + NL, B, NL, H, T)
    v[0, 0, 0, 0] = 0.0                       # an all-zero row
    d = torch.device("cuda:0")
    vd = torch.from_numpy(v).to(d)
    sc = torch.empty((B, T), dtype=torch.float32, device=d)
    semkv.semkv_score_kv_norm(vd, sc, lb, le)
    got = sc.cpu().numpy()
    want = oracle.score_kv_norm(synthetic.f16_bits(v), lb, le)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    # the scores drive the top-r selection: identical flags and slots follow
    n_high = (26 * T) // 100
    ih = torch.empty((B, T), dtype=torch.uint8, device=d)
    sl = torch.empty((B, T), dtype=torch.int32, device=d)
    semkv.semkv_rank_assign(sc, n_high, ih, sl)
    o_ih, o_sl, _ = oracle.rank_assign(want, n_high)
    assert np.array_equal(ih.cpu().numpy(), o_ih)
    assert np.array_equal(sl.cpu().numpy().view(np.uint32), o_sl)


# -------------------------------------------------------- fake quantization ---

@pytest.mark.parametrize("base,L_hi,L_lo,B,NL,H,T,mixed", [
    (0, 6, 5, 2, 2, 2, 333, True),
    (0, 5, 5, 1, 3, 2, 70, False),
    (0, 2, 8, 1, 1, 4, 129, True),
    (0, 3, 7, 2, 1, 1, 17, True),
    (1, 4, 3, 2, 2, 2, 200, True),
    (1, 2, 2, 1, 1, 2, 64, False),
    (1, 8, 5, 1, 2, 2, 45, True),
    (2, 6, 5, 2, 2, 2, 150, True),
    (2, 5, 5, 1, 1, 3, 40, False),
    (2, 2, 8, 1, 2, 1, 33, True),
])
def test_fake_quant_bit_exact(base, L_hi, L_lo, B, NL, H, T, mixed):
    import torch
    from paper_2608_28911_gb300 import semkv
    d = "cuda"
    seed = 100 + T + L_hi
    k, v = synthetic.kv(seed, B, NL, H, T)
    k = k.astype(np.float32)
    k[0, 0, 0, 0] = 1.25                     # constant row
    k[0, 0, 0, 1] = 0.0                      # zero row (TQ: norm 0)
    k[-1, -1, -1, -1] = np.linspace(-60000, 60000, 128)
    k = k.astype(np.float16)
    kb, vb = synthetic.f16_bits(k), synthetic.f16_bits(v)
    ih = (np.random.default_rng(seed).random((B, T)) < 0.3).astype(np.uint8) if mixed else None
    sg = synthetic.signs(seed, NL, H) if base != semkv.BASE_AFFINE else None
    desc = semkv.QuantDesc(base, L_hi, L_lo, signs=sg)
    kt = torch.from_numpy(k).to(d)
    vt = torch.from_numpy(v).to(d)
    # outputs between canary regions (fp16 bit pattern 0x7BCD) that must stay untouched
    n, pad, canary = kt.numel(), 64, 0x7BCD
    kbig = torch.full((n + 2 * pad,), canary, dtype=torch.int16, device=d)
    vbig = torch.full((n + 2 * pad,), canary, dtype=torch.int16, device=d)
    ko = kbig[pad:pad + n].view(torch.float16).view(kt.shape)
    vo = vbig[pad:pad + n].view(torch.float16).view(vt.shape)
    iht = torch.from_numpy(ih).to(d) if mixed else None
    semkv.semkv_fake_quant(desc, kt, vt, ko, vo, is_high=iht)
    torch.cuda.synchronize()
    for big in (kbig, vbig):
        g = big.cpu().numpy()
        assert np.all(g[:pad] == canary) and np.all(g[pad + n:] == canary), "wrote past the output"
    kw = {}
    if base == semkv.BASE_TQ:
        cbs = []
        for L in (L_hi, L_lo):
            _, c32, t32, _ = oracle.lloyd_max_gaussian(L)
            cbs.append((c32, t32))
        kw = dict(signs=sg, cb_hi=cbs[0], cb_lo=cbs[1])
    elif base == semkv.BASE_AFFINE_HAD:
        kw = dict(signs=sg)
    o_k, o_v = oracle.fake_quant(base, L_hi, L_lo, kb, vb, is_high=ih, **kw)
    g_k = ko.cpu().numpy().view(np.uint16)
    g_v = vo.cpu().numpy().view(np.uint16)
    assert np.array_equal(g_k, o_k), np.argwhere(g_k != o_k)[:5]
    assert np.array_equal(g_v, o_v), np.argwhere(g_v != o_v)[:5]
