"""Shared set-up for the GPU parity tests: the same seeded inputs are fed to the
CUDA library (through the C ABI) and to the CPU oracle, independently."""
import math

import numpy as np

import oracle
from paper_2608_28911_gb300 import synthetic

ATOL = 2e-3       # attention max-abs error vs the oracle's fp64 result
RTOL_L2 = 1e-3    # attention relative L2 error over the whole output


def attention_errors(got, ref):
    got = np.asarray(got, np.float64)
    mask = ~np.isnan(ref)
    d = got[mask] - ref[mask]
    return float(np.abs(d).max()), float(np.linalg.norm(d) / np.linalg.norm(ref[mask]))


class Pair:
    """A GPU cache and an oracle cache built from the same inputs."""

    def __init__(self, base, L_hi, L_lo, B, NL, H, Hq, T, r_num, r_den, seed, block=128,
                 extra_cap=0, tiefree=False):
        import torch
        from paper_2608_28911_gb300 import semkv
        self.torch, self.semkv = torch, semkv
        self.dev = torch.device("cuda:0")
        self.base, self.B, self.NL, self.H, self.Hq, self.T = base, B, NL, H, Hq, T
        self.r_num, self.r_den, self.seed = r_num, r_den, seed
        self.n_high = oracle.high_count_floor(T, r_num, r_den)
        signs = (synthetic.signs(seed, NL, H)
                 if base in (oracle.BASE_TQ, oracle.BASE_AFFINE_HAD) else None)
        rot = synthetic.rotations(seed, NL, H) if base == oracle.BASE_TQ_DENSE else None
        self.desc = semkv.QuantDesc(base, L_hi, L_lo, signs=signs, device=self.dev,
                                    rotation=rot)
        self.cache = semkv.KVCache(self.desc, B, NL, H, Hq, hi_cap=self.n_high + extra_cap,
                                   lo_cap=T - self.n_high + extra_cap, block=block,
                                   device=self.dev)
        self.oc = oracle.Cache(base=base, L_hi=L_hi, L_lo=L_lo, batch=B, layers=NL, kv_heads=H,
                               q_heads=Hq, block=block, hi_cap=self.cache.s.hi_cap,
                               lo_cap=self.cache.s.lo_cap)
        if signs is not None:
            self.oc.signs = signs
        self.oc.rotation = rot
        if base in (oracle.BASE_TQ, oracle.BASE_TQ_DENSE):
            _, c32, t32, _ = oracle.lloyd_max_gaussian(L_hi)
            self.oc.cb_hi = (c32, t32)
            _, c32, t32, _ = oracle.lloyd_max_gaussian(L_lo)
            self.oc.cb_lo = (c32, t32)
        self.k, self.v = synthetic.kv(seed, B, NL, H, T)
        self.s = (synthetic.scores_tiefree(seed, B, T) if tiefree
                  else synthetic.scores_zipf(seed, B, T))

    def quantize(self):
        torch, semkv = self.torch, self.semkv
        d = self.dev
        scores = torch.from_numpy(self.s).to(d)
        self.is_high = torch.empty((self.B, self.T), dtype=torch.uint8, device=d)
        self.slot = torch.empty((self.B, self.T), dtype=torch.int32, device=d)
        semkv.semkv_rank_assign(scores, self.n_high, self.is_high, self.slot)
        semkv.semkv_quantize_pack(self.desc, torch.from_numpy(self.k).to(d),
                                  torch.from_numpy(self.v).to(d), self.is_high, self.slot,
                                  self.n_high, self.cache)
        torch.cuda.synchronize()
        self.o_is_high, self.o_slot = oracle.quantize_prompt(
            self.oc, synthetic.f16_bits(self.k), synthetic.f16_bits(self.v), self.s,
            self.r_num, self.r_den)

    def assert_records_equal(self):
        c, oc = self.cache, self.oc
        assert c.hi_count == oc.hi_count and c.lo_count == oc.lo_count
        assert c.n_tokens == oc.n_tokens
        hp = c.hi_pool.cpu().numpy()[..., :oc.hi_count, :]
        lp = c.lo_pool.cpu().numpy()[..., :oc.lo_count, :]
        for name, got, want in (("hi", hp, oc.hi_pool[..., :oc.hi_count, :]),
                                ("lo", lp, oc.lo_pool[..., :oc.lo_count, :])):
            if not np.array_equal(got, want):
                bad = np.argwhere(np.any(got != want, axis=-1))
                raise AssertionError(f"{name} pool differs at {len(bad)} records, first {bad[:3]}")
        assert np.array_equal(c.hi_tok.cpu().numpy()[:, :oc.hi_count], oc.hi_tok[:, :oc.hi_count])
        assert np.array_equal(c.lo_tok.cpu().numpy()[:, :oc.lo_count], oc.lo_tok[:, :oc.lo_count])

    def assert_records_equal_up_to_ties(self, k=None, v=None, eps=2e-4):
        """Dense-rotation TQ: the GPU forms w = M x on the tensor cores, the oracle rounds
        the exact product once, so a code may differ by one where u sits within rounding
        of the threshold between them.  Norms, token maps and every other code match.
        eps: the worst case of 8 chained MMAs of 16 products, each MMA truncating its 17
        addends below one binary32 unit of the largest (8 * 17 * 2^-23 * ||M_i|| ||x|| / n,
        about 1.8e-4 with ||M_i|| ~ sqrt(128), n ~ ||x||).  The share of flipped codes is
        bounded by 1e-4, five times its expectation for spread-out truncation errors."""
        c, oc = self.cache, self.oc
        k = self.k if k is None else k
        v = self.v if v is None else v
        assert c.hi_count == oc.hi_count and c.lo_count == oc.lo_count
        assert np.array_equal(c.hi_tok.cpu().numpy()[:, :oc.hi_count], oc.hi_tok[:, :oc.hi_count])
        assert np.array_equal(c.lo_tok.cpu().numpy()[:, :oc.lo_count], oc.lo_tok[:, :oc.lo_count])
        flips = total = 0
        for name, L, cnt, gp, op, tok in (
                ("hi", oc.L_hi, oc.hi_count, c.hi_pool, oc.hi_pool, oc.hi_tok),
                ("lo", oc.L_lo, oc.lo_count, c.lo_pool, oc.lo_pool, oc.lo_tok)):
            if cnt == 0:
                continue
            got = gp.cpu().numpy()[..., :cnt, :]
            want = op[..., :cnt, :]
            rb = oracle.row_bytes(L)
            assert np.array_equal(got[..., 2 * rb:2 * rb + 4], want[..., 2 * rb:2 * rb + 4]), name
            bad = np.argwhere(np.any(got != want, axis=-1))
            thr = (oc.cb_hi if name == "hi" else oc.cb_lo)[1].astype(np.float32)
            for b, l, h, s in bad:
                t = tok[b, s]
                for row, src in ((0, k), (1, v)):
                    cg = oracle.unpack_row(got[b, l, h, s, row * rb:(row + 1) * rb], L)
                    co = oracle.unpack_row(want[b, l, h, s, row * rb:(row + 1) * rb], L)
                    diff = np.nonzero(cg != co)[0]
                    if diff.size == 0:
                        continue
                    x = synthetic.f16_bits(src[b, l, h, t])
                    w = oracle.tq_dense_w(x, oc.rotation[l, h])
                    n16 = want[b, l, h, s, 2 * rb + 2 * row:2 * rb + 2 * row + 2].view(np.uint16)[0]
                    n = np.float32(np.uint16(n16).view(np.float16))
                    u = (w * (np.float32(1) / n)).astype(np.float64)
                    lo = np.minimum(cg[diff], co[diff]).astype(int)
                    assert np.all(np.abs(cg[diff].astype(int) - co[diff].astype(int)) == 1)
                    gap = np.abs(u[diff] - thr[lo].astype(np.float64))
                    assert np.all(gap <= eps * (1 + np.abs(u[diff]))), (name, b, l, h, s, gap.max())
                    flips += diff.size
            total += got.shape[0] * got.shape[1] * got.shape[2] * cnt * 256
        assert flips <= max(4, total * 1e-4), (flips, total)
        return flips

    def adopt_gpu_records(self):
        """Attention parity independent of quantization ties: the oracle takes the GPU's
        pools as they are."""
        oc = self.oc
        oc.hi_pool[..., :oc.hi_count, :] = self.cache.hi_pool.cpu().numpy()[..., :oc.hi_count, :]
        oc.lo_pool[..., :oc.lo_count, :] = self.cache.lo_pool.cpu().numpy()[..., :oc.lo_count, :]

    def decode(self, layer=0, qseed=0, heads=None, q=None):
        """Decode through the C ABI and through the oracle on the same queries (drawn
        from the seeded stream unless `q`, fp16 [B][Hq][128], is given)."""
        torch, semkv = self.torch, self.semkv
        if q is None:
            q = synthetic.queries(self.seed + 100 * qseed, self.B, self.Hq)
        q = np.ascontiguousarray(q, dtype=np.float16)
        # the output sits between two canary regions that must come back untouched
        n, pad, canary = self.B * self.Hq * 128, 64, -1234.5
        big = torch.full((n + 2 * pad,), canary, dtype=torch.float32, device=self.dev)
        out = big[pad:pad + n].view(self.B, self.Hq, 128)
        ws = self.cache.workspace()
        scale = 1.0 / math.sqrt(128)
        semkv.semkv_decode_attention(self.desc, self.cache, layer, torch.from_numpy(q).to(self.dev),
                                     out, scale, ws)
        torch.cuda.synchronize()
        g = big.cpu().numpy()
        assert np.all(g[:pad] == canary) and np.all(g[pad + n:] == canary), "decode wrote past out"
        ref = oracle.decode_attention(self.oc, layer, synthetic.f16_bits(q), scale, heads=heads)
        return g[pad:pad + n].reshape(self.B, self.Hq, 128), ref

    def stage(self, k, v, s):
        """Stage tokens (fp16 k, v [B][NL][H][n][128], scores [B][n]) into the GPU cache
        and the oracle's, one at a time (Algorithm 2's per-token step)."""
        torch = self.torch
        for g in range(k.shape[3]):
            kg = np.ascontiguousarray(k[:, :, :, g], dtype=np.float16)
            vg = np.ascontiguousarray(v[:, :, :, g], dtype=np.float16)
            sg = np.ascontiguousarray(s[:, g], dtype=np.float32)
            self.cache.stage_token(torch.from_numpy(kg).to(self.dev),
                                   torch.from_numpy(vg).to(self.dev),
                                   torch.from_numpy(sg).to(self.dev))
            oracle.stage_token(self.oc, synthetic.f16_bits(kg), synthetic.f16_bits(vg), sg)

    def assert_untouched_past_counts(self):
        """Canaries: the pools were zero-filled and the slot maps filled with -1 when the
        cache was allocated; nothing may be written past the counts."""
        c = self.cache
        hc, lc = c.s.hi_count, c.s.lo_count
        assert not c.hi_pool.cpu().numpy()[..., hc:, :].any()
        assert not c.lo_pool.cpu().numpy()[..., lc:, :].any()
        assert np.all(c.hi_tok.cpu().numpy()[:, hc:] == -1)
        assert np.all(c.lo_tok.cpu().numpy()[:, lc:] == -1)
