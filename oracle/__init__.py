"""CPU oracle for the SemKV packed mixed-precision KV cache.

TEST INFRASTRUCTURE ONLY.  Only tests/, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The GPU library never imports, links or runs it, and this package
imports nothing from the library: the two share no code, table or constant.
The seeded inputs both sides consume come from
``paper_2608_28911_gb300.synthetic``, which holds none of the method's arithmetic.

The bit-exact binary32 work (quantize, pack, FWHT) is plain C in
``semkv_oracle.c``; ranking, the block rule, attention (fp64), the Lloyd-Max
codebook and the storage accounting are plain numpy / Python below.  Each
function names the passage of the paper it follows.

Parity pins: every function here is checked by the ``-m "not gpu"`` tests in
tests/test_oracle_*.py against values fixed by the paper or by mathematics
(Table 6 columns, Sec. 4.1 rates, textbook Lloyd-Max values, closed forms,
brute force on tiny inputs).  No function is left unpinned.
"""
from __future__ import annotations

import ctypes
import math
from dataclasses import dataclass, field

import numpy as np

from .build import build_oracle

D = 128
BASE_AFFINE, BASE_TQ, BASE_AFFINE_HAD, BASE_TQ_DENSE = 0, 1, 2, 3

_lib = None


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build_oracle())
        p = ctypes.c_void_p
        i32, i64 = ctypes.c_int, ctypes.c_int64
        L.orc_f32_to_f16.argtypes = [ctypes.c_float]
        L.orc_f32_to_f16.restype = ctypes.c_uint16
        L.orc_f16_to_f32.argtypes = [ctypes.c_uint16]
        L.orc_f16_to_f32.restype = ctypes.c_float
        L.orc_f32_to_f16_array.argtypes = [p, p, i64]
        L.orc_f16_to_f32_array.argtypes = [p, p, i64]
        for name in ("orc_group_size", "orc_symbol_bits", "orc_tail_codes",
                     "orc_tail_bits", "orc_quarter_bits", "orc_row_bytes"):
            getattr(L, name).argtypes = [i32]
            getattr(L, name).restype = i32
        L.orc_record_bytes.argtypes = [i32, i32]
        L.orc_record_bytes.restype = i32
        L.orc_pack_row.argtypes = [p, i32, p]
        L.orc_unpack_row.argtypes = [p, i32, p]
        L.orc_affine_row.argtypes = [p, i32, p, p, p]
        L.orc_tq_row.argtypes = [p, p, i32, p, p, p]
        L.orc_affine_had_row.argtypes = [p, p, i32, p, p, p]
        L.orc_f32_to_f16_rd.argtypes = [ctypes.c_float]
        L.orc_f32_to_f16_rd.restype = ctypes.c_uint16
        L.orc_inv_sqrt_d.restype = ctypes.c_float
        L.orc_fwht_f32.argtypes = [p]
        L.orc_row_norm.argtypes = [p]
        L.orc_row_norm.restype = ctypes.c_float
        L.orc_quantize_tokens.argtypes = [i32, i32, i32, p, p, i32, i32, i32, i32, i32,
                                          p, p, i64, i64, i64, p, p, p, p, p, i64, i64,
                                          p, p, p]
        L.orc_quantize_tokens.restype = i32
        L.orc_dequant_records.argtypes = [i32, i32, p, i64, p, p, p, p, p]
        L.orc_tq_dense_row.argtypes = [p, p, i32, p, p, p]
        L.orc_tq_dense_w.argtypes = [p, p, p]
        L.orc_score_kv_norm.argtypes = [p, i32, i32, i32, i32, i32, i32, p]
        L.orc_fake_quant.argtypes = [i32, i32, i32, p, p, i32, i32, i32, i32, p, p, p, p, p, p,
                                     p, p]
        _lib = L
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


# ------------------------------------------------------------------ fp16 ------

def f32_to_f16_bits(x) -> np.ndarray:
    """binary32 -> binary16 bit patterns, round to nearest even (hand-written)."""
    shape = np.shape(x)
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().orc_f32_to_f16_array(_ptr(x), _ptr(out), x.size)
    return out.reshape(shape)


def f16_bits_to_f32(h) -> np.ndarray:
    shape = np.shape(h)
    h = np.ascontiguousarray(h, dtype=np.uint16)
    out = np.empty(h.shape, dtype=np.float32)
    lib().orc_f16_to_f32_array(_ptr(h), _ptr(out), h.size)
    return out.reshape(shape)


# --------------------------------------------------------------- format -------

def group_size(L: int) -> int:
    return lib().orc_group_size(L)


def symbol_bits(L: int) -> int:
    return lib().orc_symbol_bits(L)


def tail_codes(L: int) -> int:
    return lib().orc_tail_codes(L)


def tail_bits(L: int) -> int:
    return lib().orc_tail_bits(L)


def quarter_bits(L: int) -> int:
    return lib().orc_quarter_bits(L)


def row_bytes(L: int) -> int:
    return lib().orc_row_bytes(L)


def record_bytes(base: int, L: int) -> int:
    return lib().orc_record_bytes(base, L)


def pack_row(codes, L: int) -> np.ndarray:
    """Mixed-radix packing of one 128-value row (Sec. 4.1)."""
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    assert c.shape == (D,) and int(c.max(initial=0)) < L
    out = np.zeros(row_bytes(L), dtype=np.uint8)
    lib().orc_pack_row(_ptr(c), L, _ptr(out))
    return out


def unpack_row(row, L: int) -> np.ndarray:
    r = np.ascontiguousarray(row, dtype=np.uint8)
    assert r.shape == (row_bytes(L),)
    out = np.zeros(D, dtype=np.uint8)
    lib().orc_unpack_row(_ptr(r), L, _ptr(out))
    return out


# ----------------------------------------------------------- quantizers -------

def affine_row(x_f16bits, L: int):
    """Per-row asymmetric affine quantizer (Sec. 4.1, Eq. 7).  Returns
    (codes u8[128], scale fp16 bits, offset fp16 bits)."""
    x = np.ascontiguousarray(x_f16bits, dtype=np.uint16)
    codes = np.zeros(D, dtype=np.uint8)
    s = np.zeros(1, dtype=np.uint16)
    z = np.zeros(1, dtype=np.uint16)
    lib().orc_affine_row(_ptr(x), L, _ptr(codes), _ptr(s), _ptr(z))
    return codes, int(s[0]), int(z[0])


def tq_row(x_f16bits, signs, L: int, thresholds):
    """TurboQuant-MSE row quantizer (Sec. 4.9).  Returns (codes, norm fp16 bits)."""
    x = np.ascontiguousarray(x_f16bits, dtype=np.uint16)
    sg = np.ascontiguousarray(signs, dtype=np.int8)
    thr = np.ascontiguousarray(thresholds, dtype=np.float32)
    assert thr.shape == (L - 1,)
    codes = np.zeros(D, dtype=np.uint8)
    n = np.zeros(1, dtype=np.uint16)
    lib().orc_tq_row(_ptr(x), _ptr(sg), L, _ptr(thr), _ptr(codes), _ptr(n))
    return codes, int(n[0])


def affine_had_row(x_f16bits, signs, L: int):
    """Hadamard-rotated affine row quantizer (Sec. 4.1 rotation + per-row affine).
    Returns (codes u8[128], scale fp16 bits, offset fp16 bits)."""
    x = np.ascontiguousarray(x_f16bits, dtype=np.uint16)
    sg = np.ascontiguousarray(signs, dtype=np.int8)
    codes = np.zeros(D, dtype=np.uint8)
    s = np.zeros(1, dtype=np.uint16)
    z = np.zeros(1, dtype=np.uint16)
    lib().orc_affine_had_row(_ptr(x), _ptr(sg), L, _ptr(codes), _ptr(s), _ptr(z))
    return codes, int(s[0]), int(z[0])


def f32_to_f16_rd(x: float) -> int:
    """binary32 -> binary16 bits rounded toward -infinity (hand-written)."""
    return int(lib().orc_f32_to_f16_rd(float(np.float32(x))))


def inv_sqrt_d() -> float:
    """The binary32 constant 1/sqrt(128) of the rotated affine base."""
    return float(lib().orc_inv_sqrt_d())


def tq_dense_row(x_f16bits, rot_f16bits, L: int, thresholds):
    """TurboQuant-MSE row under a dense rotation (fp16 matrix [128][128]).  Returns
    (codes, norm fp16 bits)."""
    x = np.ascontiguousarray(x_f16bits, dtype=np.uint16)
    m = np.ascontiguousarray(rot_f16bits, dtype=np.uint16)
    assert m.shape == (D, D)
    thr = np.ascontiguousarray(thresholds, dtype=np.float32)
    codes = np.zeros(D, dtype=np.uint8)
    n = np.zeros(1, dtype=np.uint16)
    lib().orc_tq_dense_row(_ptr(x), _ptr(m), L, _ptr(thr), _ptr(codes), _ptr(n))
    return codes, int(n[0])


def tq_dense_w(x_f16bits, rot_f16bits) -> np.ndarray:
    """The rotated row w = M x of the dense TQ base (fp64 sum rounded to binary32)."""
    x = np.ascontiguousarray(x_f16bits, dtype=np.uint16)
    m = np.ascontiguousarray(rot_f16bits, dtype=np.uint16)
    w = np.zeros(D, dtype=np.float32)
    lib().orc_tq_dense_w(_ptr(x), _ptr(m), _ptr(w))
    return w


def fwht_f32(w) -> np.ndarray:
    a = np.array(w, dtype=np.float32)
    lib().orc_fwht_f32(_ptr(a))
    return a


def row_norm_f32(x) -> float:
    a = np.ascontiguousarray(x, dtype=np.float32)
    return float(lib().orc_row_norm(_ptr(a)))


# ---------------------------------------------------- selection (Eqs. 4-5) ----

def high_count_floor(T: int, r_num: int, r_den: int) -> int:
    """K = floor(r T) with r = r_num / r_den (Eq. 4), exact in integers."""
    return (int(T) * int(r_num)) // int(r_den)


def block_high_count(n: int, r_num: int, r_den: int) -> int:
    """round(r n), nearest integer with halves up (Algorithm 2; Sec. 3.7)."""
    return (2 * int(r_num) * int(n) + int(r_den)) // (2 * int(r_den))


def rank_assign(scores, n_high: int):
    """Top-K by score (Eq. 4) with ties to the lower token index; NaN below every
    number; -0 == +0.  Returns (is_high u8, slot u32, rank u32), each [B][T].
    rank: position in the (score desc, index asc) order.  slot: number of earlier
    tokens of the same class (the token's place in its pool, Eq. 5)."""
    s = np.asarray(scores, dtype=np.float32)
    squeeze = s.ndim == 1
    s = np.atleast_2d(s)
    B, T = s.shape
    assert 0 <= n_high <= T
    is_high = np.zeros((B, T), np.uint8)
    slot = np.zeros((B, T), np.uint32)
    rank = np.zeros((B, T), np.uint32)
    idx = np.arange(T)
    for b in range(B):
        x = s[b].astype(np.float64)
        nan = np.isnan(x)
        key = np.where(nan, 0.0, -x)             # ascending key = descending score
        order = np.lexsort((idx, key, nan))       # primary: not-NaN first
        rank[b, order] = np.arange(T, dtype=np.uint32)
        is_high[b] = (rank[b] < n_high).astype(np.uint8)
        hi = is_high[b].astype(np.int64)
        slot[b] = np.where(hi == 1, np.cumsum(hi) - hi, np.cumsum(1 - hi) - (1 - hi))
    if squeeze:
        return is_high[0], slot[0], rank[0]
    return is_high, slot, rank


# ----------------------------------------------------- Lloyd-Max (Sec. 4.9) ---

def _phi(x):
    return math.exp(-0.5 * x * x) / math.sqrt(2.0 * math.pi) if math.isfinite(x) else 0.0


def _Phi(x):
    if x == math.inf:
        return 1.0
    if x == -math.inf:
        return 0.0
    return 0.5 * math.erfc(-x / math.sqrt(2.0))


def lloyd_max_gaussian(L: int, iters: int = 200000, tol: float = 1e-15):
    """Lloyd-Max quantizer of N(0,1) with L levels (Sec. 4.9: Gaussian-optimal
    Lloyd-Max codebook, any integer L).  Lloyd iteration: thresholds at centroid
    midpoints; centroid of (a, b] = (phi(a) - phi(b)) / (Phi(b) - Phi(a)).
    Returns (centroids fp64, centroids fp32, thresholds fp32, mse fp64)."""
    c = [(-1.0 + 2.0 * (i + 0.5) / L) * 2.0 for i in range(L)]
    for _ in range(iters):
        t = [-math.inf] + [(c[i] + c[i + 1]) / 2 for i in range(L - 1)] + [math.inf]
        nc = [(_phi(t[i]) - _phi(t[i + 1])) / (_Phi(t[i + 1]) - _Phi(t[i]))
              for i in range(L)]
        delta = max(abs(a - b) for a, b in zip(c, nc))
        c = nc
        if delta < tol:
            break
    # N(0,1) is symmetric, so is its Lloyd-Max codebook: symmetrize the converged
    # centroids exactly (the middle centroid of an odd L, and the middle threshold of
    # an even L, become exactly 0 rather than +-1e-16 of iteration noise)
    c = [0.5 * (c[i] - c[L - 1 - i]) for i in range(L)]
    t = [(c[i] + c[i + 1]) / 2 for i in range(L - 1)]
    edges = [-math.inf] + t + [math.inf]
    # MSE = E[X^2] - sum_l P_l c_l^2 for centroid-condition quantizers
    mse = 1.0 - sum((_Phi(edges[i + 1]) - _Phi(edges[i])) * c[i] ** 2 for i in range(L))
    return (np.array(c, np.float64), np.array(c, np.float32),
            np.array(t, np.float32), mse)


# ------------------------------------------------------------ the cache -------

@dataclass
class Cache:
    """Oracle image of one mixed-precision cache (Algorithm 1 output extended by
    Algorithm 2): two packed pools, their slot->token arrays and the fp16 tail."""
    base: int
    L_hi: int
    L_lo: int
    batch: int
    layers: int
    kv_heads: int
    q_heads: int
    block: int
    hi_cap: int
    lo_cap: int
    hi_pool: np.ndarray = None
    lo_pool: np.ndarray = None
    hi_tok: np.ndarray = None
    lo_tok: np.ndarray = None
    hi_count: int = 0
    lo_count: int = 0
    n_tokens: int = 0
    stage_k: np.ndarray = None
    stage_v: np.ndarray = None
    stage_score: np.ndarray = None
    stage_n: int = 0
    signs: np.ndarray = None          # [layers][kv_heads][128] int8 (TQ, rotated affine)
    cb_hi: tuple = None               # (centroids f32, thresholds f32) (TQ)
    cb_lo: tuple = None
    rotation: np.ndarray = None       # [layers][kv_heads][128][128] fp16 bits (dense TQ)

    def __post_init__(self):
        B, NL, H = self.batch, self.layers, self.kv_heads
        rh, rl = record_bytes(self.base, self.L_hi), record_bytes(self.base, self.L_lo)
        assert rh > 0 and rl > 0
        self.hi_pool = np.zeros((B, NL, H, self.hi_cap, rh), np.uint8)
        self.lo_pool = np.zeros((B, NL, H, self.lo_cap, rl), np.uint8)
        self.hi_tok = np.full((B, self.hi_cap), -1, np.int32)
        self.lo_tok = np.full((B, self.lo_cap), -1, np.int32)
        self.stage_k = np.zeros((B, NL, H, self.block, D), np.uint16)
        self.stage_v = np.zeros((B, NL, H, self.block, D), np.uint16)
        self.stage_score = np.zeros((B, self.block), np.float32)
        if self.signs is None:
            self.signs = np.ones((NL, H, D), np.int8)

    def _rot(self, layer=None, head=None):
        """The dense rotation (fp16 bits) of every (layer, head), or of one, or None."""
        if self.rotation is None:
            return None
        r = np.ascontiguousarray(self.rotation, dtype=np.uint16)
        if layer is not None:
            r = np.ascontiguousarray(r[layer, head])
        self._rot_keep = r
        return _ptr(r)

    def _thr(self, which):
        if self.base not in (BASE_TQ, BASE_TQ_DENSE):
            return np.zeros(1, np.float32)
        return np.ascontiguousarray((self.cb_hi if which == "hi" else self.cb_lo)[1],
                                    dtype=np.float32)


def quantize_tokens(cache: Cache, k, v, n: int, is_high, slot, hi_base, lo_base,
                    tok_base):
    """Eq. 7 over tokens 0..n-1 of k/v [B][NL][H][Tsrc][128] (fp16 bits)."""
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    B, NL, H, Tsrc, d = k.shape
    assert d == D and v.shape == k.shape and n <= Tsrc
    ih = np.ascontiguousarray(np.asarray(is_high, np.uint8).reshape(B, n))
    sl = np.ascontiguousarray(np.asarray(slot, np.uint32).reshape(B, n))
    thr_hi, thr_lo = cache._thr("hi"), cache._thr("lo")
    signs = np.ascontiguousarray(cache.signs, dtype=np.int8)
    rc = lib().orc_quantize_tokens(cache.base, cache.L_hi, cache.L_lo, _ptr(k), _ptr(v),
                                   B, NL, H, Tsrc, n, _ptr(ih), _ptr(sl), hi_base,
                                   lo_base, tok_base, _ptr(signs), _ptr(thr_hi),
                                   _ptr(thr_lo), _ptr(cache.hi_pool), _ptr(cache.lo_pool),
                                   cache.hi_cap, cache.lo_cap, _ptr(cache.hi_tok),
                                   _ptr(cache.lo_tok), cache._rot())
    if rc != 0:
        raise ValueError("pool capacity exceeded")


def quantize_prompt(cache: Cache, k, v, scores, r_num: int, r_den: int):
    """Algorithm 1: K = floor(rT) (Eq. 4), H = TopK, b_i by Eq. 5, quantize every
    token of every layer/head with Q_{b_i} (Eq. 7).  Returns (is_high, slot)."""
    T = k.shape[3]
    n_high = high_count_floor(T, r_num, r_den)
    is_high, slot, _ = rank_assign(np.atleast_2d(scores), n_high)
    quantize_tokens(cache, k, v, T, is_high, slot, 0, 0, 0)
    cache.hi_count, cache.lo_count, cache.n_tokens, cache.stage_n = n_high, T - n_high, T, 0
    return is_high, slot


def stage_token(cache: Cache, k_tok, v_tok, score):
    """Algorithm 2: append a generated token at full precision and record its
    score (no per-token decision).  k_tok/v_tok: [B][NL][H][128] fp16 bits."""
    assert cache.stage_n < cache.block
    cache.stage_k[:, :, :, cache.stage_n] = k_tok
    cache.stage_v[:, :, :, cache.stage_n] = v_tok
    cache.stage_score[:, cache.stage_n] = score
    cache.stage_n += 1


def append_block(cache: Cache, r_num: int, r_den: int):
    """Algorithm 2 when |S| = B, and its end-of-turn flush when 0 < |S| < B:
    H_blk = TopKIndices(S, round(r|S|)); quantize the block with Q_{b_g}; S = {}."""
    n = cache.stage_n
    if n == 0:
        return
    n_high = block_high_count(n, r_num, r_den)
    is_high, slot, _ = rank_assign(cache.stage_score[:, :n], n_high)
    quantize_tokens(cache, cache.stage_k, cache.stage_v, n, is_high, slot,
                    cache.hi_count, cache.lo_count, cache.n_tokens)
    cache.hi_count += n_high
    cache.lo_count += n - n_high
    cache.n_tokens += n
    cache.stage_n = 0


def dequant_records(base: int, L: int, recs, signs_lh, centroids, rot_lh=None):
    """Exact fp64 rows of `count` records: affine z + s c; TQ (n/128) S H cb[c]."""
    recs = np.ascontiguousarray(recs, dtype=np.uint8)
    count = recs.shape[0]
    kout = np.zeros((count, D), np.float64)
    vout = np.zeros((count, D), np.float64)
    sg = np.ascontiguousarray(signs_lh if signs_lh is not None else np.ones(D), np.int8)
    cb = np.ascontiguousarray(centroids if centroids is not None else np.zeros(1),
                              dtype=np.float64)
    rot = None if rot_lh is None else np.ascontiguousarray(rot_lh, dtype=np.uint16)
    lib().orc_dequant_records(base, L, _ptr(recs), count, _ptr(sg), _ptr(cb),
                              _ptr(kout), _ptr(vout), None if rot is None else _ptr(rot))
    return kout, vout


def dequant_cache_head(cache: Cache, b: int, layer: int, h: int):
    """All tokens of (b, layer, h): the high pool, the low pool and the fp16 tail,
    as exact fp64 rows (token order is irrelevant to attention)."""
    cb_hi = cache.cb_hi[0] if cache.cb_hi is not None else None
    cb_lo = cache.cb_lo[0] if cache.cb_lo is not None else None
    sg = cache.signs[layer, h]
    rot = None if cache.rotation is None else cache.rotation[layer, h]
    kh, vh = dequant_records(cache.base, cache.L_hi,
                             cache.hi_pool[b, layer, h, :cache.hi_count], sg, cb_hi, rot)
    kl, vl = dequant_records(cache.base, cache.L_lo,
                             cache.lo_pool[b, layer, h, :cache.lo_count], sg, cb_lo, rot)
    n = cache.stage_n
    ks = f16_bits_to_f32(cache.stage_k[b, layer, h, :n]).astype(np.float64)
    vs = f16_bits_to_f32(cache.stage_v[b, layer, h, :n]).astype(np.float64)
    return np.concatenate([kh, kl, ks]), np.concatenate([vh, vl, vs])


def attention_fp64(q64, K, V, scale: float):
    """softmax(scale * q K^T) V in fp64, two-pass (max subtracted)."""
    logits = scale * (K @ q64)
    m = logits.max()
    p = np.exp(logits - m)
    return (p @ V) / p.sum()


def decode_attention(cache: Cache, layer: int, q_f16bits, scale: float,
                     heads=None):
    """Single-query decode attention over the whole cache of one layer (Algorithm 1
    "use Ĉ_KV for decoding"; the staged fp16 tail takes part, Algorithm 2).
    q: [B][Hq][128] fp16 bits -> out fp64 [B][Hq][128].  `heads`: optional list of
    (b, qh) to compute (others left NaN)."""
    q = f16_bits_to_f32(q_f16bits).astype(np.float64)
    B, Hq, _ = q.shape
    group = Hq // cache.kv_heads
    out = np.full((B, Hq, D), np.nan)
    want = set(heads) if heads is not None else None
    for b in range(B):
        for h in range(cache.kv_heads):
            qhs = [qh for qh in range(h * group, (h + 1) * group)
                   if want is None or (b, qh) in want]
            if not qhs:
                continue
            K, V = dequant_cache_head(cache, b, layer, h)
            for qh in qhs:
                out[b, qh] = attention_fp64(q[b, qh], K, V, scale)
    return out


# ------------------------------------------------ accounting (Sec. 4.1) -------

def paper_code_bits(L: int) -> float:
    """Code bits per value at the paper's packing rate: w / g of a full group
    (Sec. 4.1: 7/3 = 2.333 for 5 levels, 13/5 = 2.600 for 6; Table 6: 1.600 for 3)."""
    return symbol_bits(L) / group_size(L)


def metadata_bits(base: int) -> float:
    """fp16 metadata per value: two per 128-row for affine (0.25), one for TQ."""
    return (1 if base in (BASE_TQ, BASE_TQ_DENSE) else 2) * 16 / D


def effective_bits(base: int, L_hi: int, L_lo: int, r: float) -> float:
    """Token-weighted packed code bits plus metadata (Sec. 4.1, Table 6)."""
    return r * paper_code_bits(L_hi) + (1 - r) * paper_code_bits(L_lo) + metadata_bits(base)


def layout_bytes_per_token_head(base: int, L_hi: int, L_lo: int, n_high: int, T: int) -> int:
    """Bytes of this build's records (K and V of one KV head) for T tokens."""
    return n_high * record_bytes(base, L_hi) + (T - n_high) * record_bytes(base, L_lo)


# ------------------------------------------- KV-norm indicator (Sec. 3.3) -----

def score_kv_norm(x_f16bits, layer_begin: int = 0, layer_end: int | None = None):
    """Key-norm / value-norm importance score of each token (Sec. 3.3, KV-norm family):
    ||x_{b,t}||_2 over layers [layer_begin, layer_end) and every KV head of the fp16
    K or V cache x [B][NL][H][T][128] (bit patterns), in the fixed summation order of
    orc_score_kv_norm.  Returns float32 [B][T]."""
    x = np.ascontiguousarray(x_f16bits, dtype=np.uint16)
    B, NL, H, T, d = x.shape
    assert d == D
    le = NL if layer_end is None else layer_end
    assert 0 <= layer_begin < le <= NL
    out = np.zeros((B, T), np.float32)
    lib().orc_score_kv_norm(_ptr(x), B, NL, H, T, layer_begin, le, _ptr(out))
    return out


# ------------------------------------------ fake quantization (Sec. 4.1) ------

def fake_quant(base: int, L_hi: int, L_lo: int, k, v, is_high=None, signs=None,
               cb_hi=None, cb_lo=None):
    """Quantize every row of K and V at its token's precision (Eq. 7; is_high None puts
    every token at L_hi) and reconstruct to fp16 in binary32 in the order of
    orc_fake_quant.  k, v: fp16 bits [B][NL][H][T][128]; cb_*: (centroids, thresholds)
    fp32 for TQ.  Returns (k_out, v_out) fp16 bits."""
    if base == BASE_TQ_DENSE:
        raise NotImplementedError("fake quantization covers the affine, rotated affine and TQ bases")
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    B, NL, H, T, d = k.shape
    assert d == D and v.shape == k.shape
    ko = np.zeros_like(k)
    vo = np.zeros_like(v)
    ih = None if is_high is None else np.ascontiguousarray(is_high, dtype=np.uint8)
    sg = None if signs is None else np.ascontiguousarray(signs, dtype=np.int8)
    z1 = np.zeros(8, np.float32)
    ch, th = (z1, z1) if cb_hi is None else (np.ascontiguousarray(cb_hi[0], np.float32),
                                             np.ascontiguousarray(cb_hi[1], np.float32))
    cl, tl = (z1, z1) if cb_lo is None else (np.ascontiguousarray(cb_lo[0], np.float32),
                                             np.ascontiguousarray(cb_lo[1], np.float32))
    lib().orc_fake_quant(base, L_hi, L_lo, _ptr(k), _ptr(v), B, NL, H, T,
                         None if ih is None else _ptr(ih), None if sg is None else _ptr(sg),
                         _ptr(ch), _ptr(th), _ptr(cl), _ptr(tl), _ptr(ko), _ptr(vo))
    return ko, vo
