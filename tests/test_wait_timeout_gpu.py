"""The kernels' bounded waits report a wait that runs out (needs a GB300).

fav_check_wait_timeout runs the kernels' own wait code on an mbarrier that nothing arrives on,
with a 1 ms give-up limit: the wait must give up, the status word must carry
FAV_ERR_DEVICE_TIMEOUT to the host exactly once, and the context must stay usable (the next
calls run and match the oracle).  No GPU fault is involved: the waiting warp simply returns."""
import pytest

import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import check, run_gpu

pytestmark = pytest.mark.gpu

FAV_ERR_DEVICE_TIMEOUT = 5


def test_wait_gives_up_and_reports():
    import time
    import torch
    assert fav.device_status() == 0                      # nothing pending from earlier calls
    t0 = time.perf_counter()
    fav.check_wait_timeout(1000)
    torch.cuda.synchronize()
    took = time.perf_counter() - t0
    assert fav.device_status() == FAV_ERR_DEVICE_TIMEOUT
    assert fav.device_status() == 0                      # read once, then cleared
    assert took < 1.0                                    # gave up after its own limit, not 2 s


@pytest.mark.parametrize("w", [
    I.Workload("after_prefill", I.F16, 1, 4, 2, 300, 300, 128, True, False, 31),
    I.Workload("after_decode", I.BF16, 2, 8, 2, 1, 3000, 128, False, False, 32),
])
def test_calls_after_a_timeout_match_the_oracle(w):
    fav.check_wait_timeout(1000)
    assert fav.device_status() == FAV_ERR_DEVICE_TIMEOUT
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)                               # asserts a clean status itself
    check(w, o, lse, x)
