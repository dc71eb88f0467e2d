"""semkv_decode_attention_noalloc: decode attention for callers that cannot allocate
device memory (the library keeps its split-K scratch in a static device array).

Checked through the C ABI against semkv_decode_attention (which uses a caller
workspace), with the attention tolerance of the other tests, on two calls in a row
(the array keeps the previous call's contents), on a shape whose split plan has to
be reduced to fit the array, and with a request too large for the array, which
must be rejected before anything is launched.  Collected last on purpose.
"""
import math

import numpy as np
import pytest

from paper_2608_28911_gb300 import synthetic
from parity import ATOL, RTOL_L2, Pair, attention_errors

pytestmark = pytest.mark.gpu


def _run_both(p, qseed):
    import torch
    from paper_2608_28911_gb300 import semkv
    q = torch.from_numpy(synthetic.queries(p.seed + qseed, p.B, p.Hq)).to(p.dev)
    scale = 1.0 / math.sqrt(128)
    ref = torch.empty((p.B, p.Hq, 128), dtype=torch.float32, device=p.dev)
    semkv.semkv_decode_attention(p.desc, p.cache, 0, q, ref, scale, p.cache.workspace())
    outs = []
    for _ in range(2):  # two calls in a row share the static array
        out = torch.full((p.B, p.Hq, 128), float("nan"), dtype=torch.float32, device=p.dev)
        semkv.semkv_decode_attention_noalloc(p.desc, p.cache, 0, q, out, scale)
        outs.append(out)
    torch.cuda.synchronize()
    return ref.cpu().numpy().astype(np.float64), [o.cpu().numpy() for o in outs]


@pytest.mark.parametrize("B,H,Hq,T", [
    (2, 8, 32, 3000),     # plan fits the array as it is
    (40, 8, 32, 1200),    # 320 (sequence, KV head) pairs: the split count is reduced
])
def test_noalloc_matches_workspace_entry_point(B, H, Hq, T):
    p = Pair(0, 6, 5, B, 1, H, Hq, T, 26, 100, seed=300 + B)
    p.quantize()
    for qseed in (0, 1):
        ref, outs = _run_both(p, qseed)
        for got in outs:
            err, rel = attention_errors(got, ref)
            assert err <= ATOL and rel <= RTOL_L2, (err, rel)
    assert int(p.cache.dev_error.item()) == 0


@pytest.mark.parametrize("base,L_hi,L_lo", [(1, 4, 3), (2, 6, 5), (3, 4, 3)])
def test_noalloc_rotated_bases(base, L_hi, L_lo):
    # TQ, Hadamard-rotated affine and dense-rotation TQ: the rotated queries live in
    # the library's second static array
    p = Pair(base, L_hi, L_lo, 2, 1, 8, 32, 2000, 3, 4, seed=320 + base)
    p.quantize()
    for qseed in (0, 1):
        ref, outs = _run_both(p, qseed)
        for got in outs:
            err, rel = attention_errors(got, ref)
            assert err <= ATOL and rel <= RTOL_L2, (err, rel)
    assert int(p.cache.dev_error.item()) == 0


def test_noalloc_rejects_requests_beyond_the_array():
    import torch
    from paper_2608_28911_gb300 import semkv
    # 2200 (sequence, KV head) pairs x 2 pools > 2016 partials
    desc = semkv.QuantDesc(semkv.BASE_AFFINE, 6, 5, device="cuda:0")
    cache = semkv.KVCache(desc, 275, 1, 8, 32, hi_cap=16, lo_cap=16, block=16, device="cuda:0")
    cache.s.hi_count, cache.s.lo_count = 8, 8
    q = torch.zeros((275, 32, 128), dtype=torch.float16, device="cuda:0")
    out = torch.zeros((275, 32, 128), dtype=torch.float32, device="cuda:0")
    with pytest.raises(semkv.SemkvError) as e:
        semkv.semkv_decode_attention_noalloc(desc, cache, 0, q, out, 0.1)
    assert e.value.status == 6   # SEMKV_EWORKSPACE
