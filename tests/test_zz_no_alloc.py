"""semkv_decode_attention_noalloc: decode attention for callers that cannot allocate
device memory (the library keeps its split-K scratch in a static device array).

Checked through the C ABI against the oracle's fp64 attention (sampled heads where the
batch is large) and against semkv_decode_attention (which uses a caller workspace),
with the attention tolerance of the other tests, on two calls in a row (the array keeps
the previous call's contents); on shapes whose split plan has to be reduced to fit the
array, with and without a staged fp16 tail; at the documented limits (672 pairs for the
affine bases, 504 with a staged tail: accepted; one more pair: rejected before anything
is launched).  Collected last on purpose.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2608_28911_gb300 import synthetic
from parity import ATOL, RTOL_L2, Pair, attention_errors

pytestmark = pytest.mark.gpu


def _run_both(p, qseed):
    import torch
    from paper_2608_28911_gb300 import semkv
    q = synthetic.queries(p.seed + qseed, p.B, p.Hq)
    qd = torch.from_numpy(q).to(p.dev)
    scale = 1.0 / math.sqrt(128)
    ref = torch.empty((p.B, p.Hq, 128), dtype=torch.float32, device=p.dev)
    semkv.semkv_decode_attention(p.desc, p.cache, 0, qd, ref, scale, p.cache.workspace())
    outs = []
    for _ in range(2):  # two calls in a row share the static array
        out = torch.full((p.B, p.Hq, 128), float("nan"), dtype=torch.float32, device=p.dev)
        semkv.semkv_decode_attention_noalloc(p.desc, p.cache, 0, qd, out, scale)
        outs.append(out)
    torch.cuda.synchronize()
    return q, ref.cpu().numpy().astype(np.float64), [o.cpu().numpy() for o in outs]


def _check(p, qseed, heads=None):
    q, ws_out, outs = _run_both(p, qseed)
    want = oracle.decode_attention(p.oc, 0, synthetic.f16_bits(q), 1.0 / math.sqrt(128),
                                   heads=heads)
    sel = (np.ones((p.B, p.Hq), bool) if heads is None else
           np.isin(np.arange(p.B * p.Hq), [b * p.Hq + qh for b, qh in heads]).reshape(p.B, p.Hq))
    for got in outs:
        err, rel = attention_errors(got[sel], want[sel])      # against the oracle
        assert err <= ATOL and rel <= RTOL_L2, ("oracle", err, rel)
        err, rel = attention_errors(got, ws_out)              # against the workspace call
        assert err <= ATOL and rel <= RTOL_L2, ("workspace", err, rel)
    assert int(p.cache.dev_error.item()) == 0


def _sample(B, Hq, n, seed):
    rng = np.random.default_rng(seed)
    return [(int(b), int(qh)) for b, qh in zip(rng.integers(0, B, n), rng.integers(0, Hq, n))]


@pytest.mark.parametrize("B,H,Hq,T", [
    (2, 8, 32, 3000),     # plan fits the array as it is
    (40, 8, 32, 1200),    # 320 (sequence, KV head) pairs: the split count is reduced
])
def test_noalloc_matches_oracle_and_workspace_entry_point(B, H, Hq, T):
    p = Pair(0, 6, 5, B, 1, H, Hq, T, 26, 100, seed=300 + B)
    p.quantize()
    heads = None if B <= 2 else _sample(B, Hq, 24, B)
    for qseed in (0, 1):
        _check(p, qseed, heads)


def test_noalloc_reduced_plan_with_staged_tail():
    # 320 pairs and a staged tail: the stage's partial takes the last slot of the
    # reduced stride (6 slots per pair)
    p = Pair(0, 6, 5, 40, 1, 8, 32, 1200, 26, 100, seed=310, block=32)
    p.quantize()
    k, v = synthetic.kv(311, p.B, 1, p.H, 9)
    p.stage(k, v, synthetic.scores_zipf(311, p.B, 9))
    _check(p, 0, _sample(p.B, p.Hq, 24, 312))


@pytest.mark.parametrize("base,L_hi,L_lo", [(1, 4, 3), (2, 6, 5), (3, 4, 3)])
def test_noalloc_rotated_bases(base, L_hi, L_lo):
    # TQ, Hadamard-rotated affine and dense-rotation TQ: the rotated queries live in
    # the library's second static array
    p = Pair(base, L_hi, L_lo, 2, 1, 8, 32, 2000, 3, 4, seed=320 + base)
    p.quantize()
    if base == 3:
        p.adopt_gpu_records()   # tensor-core rotation: codes may differ at threshold ties
    for qseed in (0, 1):
        _check(p, qseed)


@pytest.mark.parametrize("staged,pairs", [(False, 672), (True, 504)])
def test_noalloc_limit_of_the_balanced_plan(staged, pairs):
    """The largest request the affine bases' balanced plan fits in the array (3 partial
    slots per pair, 4 with a staged tail) runs and matches the oracle; one more pair is
    rejected with SEMKV_EWORKSPACE."""
    import torch
    from paper_2608_28911_gb300 import semkv
    p = Pair(0, 6, 5, pairs, 1, 1, 4, 48, 26, 100, seed=330 + pairs, block=16)
    p.quantize()
    if staged:
        k, v = synthetic.kv(331, p.B, 1, p.H, 5)
        p.stage(k, v, synthetic.scores_zipf(331, p.B, 5))
    _check(p, 0, _sample(p.B, p.Hq, 16, pairs))
    desc = semkv.QuantDesc(semkv.BASE_AFFINE, 6, 5, device="cuda:0")
    cache = semkv.KVCache(desc, pairs + 1, 1, 1, 4, hi_cap=16, lo_cap=48, block=16,
                          device="cuda:0")
    cache.s.hi_count, cache.s.lo_count = 12, 36
    if staged:
        cache.s.stage_n = 5
    q = torch.zeros((pairs + 1, 4, 128), dtype=torch.float16, device="cuda:0")
    out = torch.zeros((pairs + 1, 4, 128), dtype=torch.float32, device="cuda:0")
    with pytest.raises(semkv.SemkvError) as e:
        semkv.semkv_decode_attention_noalloc(desc, cache, 0, q, out, 0.1)
    assert e.value.status == 6   # SEMKV_EWORKSPACE


def test_noalloc_rejects_requests_beyond_the_array():
    import torch
    from paper_2608_28911_gb300 import semkv
    # 2200 (sequence, KV head) pairs: beyond 672
    desc = semkv.QuantDesc(semkv.BASE_AFFINE, 6, 5, device="cuda:0")
    cache = semkv.KVCache(desc, 275, 1, 8, 32, hi_cap=16, lo_cap=16, block=16, device="cuda:0")
    cache.s.hi_count, cache.s.lo_count = 8, 8
    q = torch.zeros((275, 32, 128), dtype=torch.float16, device="cuda:0")
    out = torch.zeros((275, 32, 128), dtype=torch.float32, device="cuda:0")
    with pytest.raises(semkv.SemkvError) as e:
        semkv.semkv_decode_attention_noalloc(desc, cache, 0, q, out, 0.1)
    assert e.value.status == 6   # SEMKV_EWORKSPACE
