"""Failure detection on the GPU without a fault: a bounded wait that runs out.

Every kernel that waits on a bulk copy gives up after a bounded number of polls,
writes a timeout code into the device error word and returns.  Through the C ABI a
test runs that same wait on a barrier nothing arrives on, with a short poll limit, and
checks that the call returns, the error word holds the timeout code, and the context
is still usable: a quantize and a decode on the same cache afterwards are bit-exact
and within tolerance against the oracle, with no error recorded."""
import numpy as np
import pytest

from parity import ATOL, RTOL_L2, Pair, attention_errors

pytestmark = pytest.mark.gpu

DEV_WAIT_TIMEOUT = 1


@pytest.mark.parametrize("polls", [1, 1000, 100000])
def test_bounded_wait_runs_out_and_context_stays_usable(polls):
    import torch
    from paper_2608_28911_gb300 import semkv
    p = Pair(0, 6, 5, 1, 1, 2, 8, 700, 26, 100, seed=900 + polls)
    err = p.cache.dev_error
    err.zero_()
    semkv.semkv_debug_wait_timeout(err, polls)
    torch.cuda.synchronize()
    assert int(err.item()) == DEV_WAIT_TIMEOUT
    err.zero_()
    p.quantize()
    p.assert_records_equal()
    got, ref = p.decode()
    e, rel = attention_errors(got, ref)
    assert e <= ATOL and rel <= RTOL_L2, (e, rel)
    assert int(err.item()) == 0


def test_wait_timeout_rejects_bad_arguments():
    import torch
    from paper_2608_28911_gb300 import semkv
    err = torch.zeros(4, dtype=torch.int32, device="cuda:0")
    for polls in (0, (1 << 22) + 1):
        with pytest.raises(semkv.SemkvError) as e:
            semkv.semkv_debug_wait_timeout(err, polls)
        assert e.value.status == 1   # SEMKV_EINVAL: nothing was launched
    torch.cuda.synchronize()
    assert not err.any()
