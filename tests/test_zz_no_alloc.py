"""fav_decode_noalloc: the decode path for callers that cannot let a library allocate device
memory (a server whose pool reserves all device memory at start-up, a latency-critical decode
loop that forbids allocator calls after initialisation).  Its split-KV partials live in a fixed
16 MiB device array instead of a cudaMalloc'd workspace.

Checked through the C ABI against the existing entry point fav_forward, within the parity
tolerances of the other GPU tests, on two calls in a row (the array keeps the previous call's
contents).  This file is collected last so that a failure here cannot stop the other tests.
"""
import ctypes

import numpy as np
import pytest

import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import LSE_TOL, O_TOL, to_device

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 16 * 1024 * 1024


def noalloc_fn():
    f = fav.lib().fav_decode_noalloc
    vp, i = ctypes.c_void_p, ctypes.c_int
    f.argtypes = [vp, vp, vp, vp, vp, i, i, i, i, i, i, ctypes.c_float, i, i, vp]
    f.restype = i
    return f


def call_noalloc(w, q, k, v, o, lse):
    import torch
    return noalloc_fn()(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                        lse.data_ptr() if lse is not None else None, w.B, w.Hq, w.Hkv, w.Nq,
                        w.Nkv, w.D, w.scale, int(w.causal), w.dtype,
                        torch.cuda.current_stream().cuda_stream)


@pytest.fixture(autouse=True)
def _reset():
    fav.set_path(fav.PATH_AUTO)
    fav.set_decode_splits(0)
    yield
    fav.set_decode_splits(0)


CASES = [
    I.Workload("gqa_f16", I.F16, 2, 8, 2, 1, 3000, 128, False, False, 21),
    I.Workload("mqa_bf16", I.BF16, 4, 16, 1, 1, 5000, 64, False, False, 22),
    I.Workload("spec_bf16", I.BF16, 1, 8, 2, 4, 2000, 128, True, False, 23),
    I.WORKLOADS[4],
]


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_noalloc_matches_forward_twice(w):
    import torch
    x = I.make_inputs(w)
    q, k, v = (to_device(x[n + "_bits"], w.dtype) for n in ("q", "k", "v"))
    ref_o, ref_lse = fav.forward(q, k, v, causal=w.causal, scale=w.scale)
    assert fav.last_path() == fav.PATH_DECODE
    torch.cuda.synchronize()
    ref_o = ref_o.float().cpu().numpy()
    ref_lse = ref_lse.cpu().numpy()
    for _ in range(2):
        o = torch.full_like(q, float("nan"))
        lse = torch.full((w.B, w.Hq, w.Nq), float("nan"), device="cuda")
        assert call_noalloc(w, q, k, v, o, lse) == 0
        torch.cuda.synchronize()
        assert fav.device_status() == 0
        oo = o.float().cpu().numpy()
        assert np.isfinite(oo).all()
        assert np.abs(oo - ref_o).max() <= O_TOL[w.dtype]
        assert np.abs(lse.cpu().numpy() - ref_lse).max() <= LSE_TOL


def test_noalloc_rejects_partials_beyond_the_array():
    import torch
    w = I.Workload("big", I.F16, 1, 64, 4, 1, 32768, 128, False, False, 24)
    rows = w.B * w.Hq * w.Nq
    fav.set_decode_splits(1024)                      # partials: 64 * 1024 * 129 * 4 B > 16 MiB
    assert rows * 1024 * (w.D + 1) * 4 > SCRATCH_BYTES
    q = torch.zeros((w.B, w.Hq, w.Nq, w.D), dtype=torch.float16, device="cuda")
    kv = torch.zeros((w.B, w.Hkv, w.Nkv, w.D), dtype=torch.float16, device="cuda")
    o = torch.full_like(q, 7.0)
    assert call_noalloc(w, q, kv, kv, o, None) == 2   # FAV_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert bool((o == 7.0).all())


def test_noalloc_rejects_prefill_shapes():
    import torch
    w = I.Workload("prefill", I.F16, 1, 4, 4, 256, 256, 128, True, False, 25)
    q = torch.zeros((1, 4, 256, 128), dtype=torch.float16, device="cuda")
    assert call_noalloc(w, q, q, q, torch.empty_like(q), None) == 2


# Run in a fresh process: fav_decode_noalloc is the first call of the library there (it sets up
# the device state and looks up the array's address itself), and the device's default memory
# pool -- the one cudaMallocAsync draws from -- must not grow across it.  fav_forward on the same
# decode shape afterwards does allocate its workspace from that pool (the probe can see an
# allocation) and must agree with the two no-allocation calls.
FIRST_CALL_SCRIPT = r"""
import ctypes, json, os, sys
sys.path.insert(0, sys.argv[1])
sys.path.insert(0, os.path.join(sys.argv[1], "tests"))
import numpy as np
import torch
import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import to_device
import test_zz_no_alloc as T

w = I.Workload("first_call", I.BF16, 2, 16, 2, 1, 6000, 128, False, False, 26)
x = I.make_inputs(w)
q, k, v = (to_device(x[n + "_bits"], w.dtype) for n in ("q", "k", "v"))
drv = ctypes.CDLL("libcuda.so.1")
dev = ctypes.c_int()
assert drv.cuDeviceGet(ctypes.byref(dev), torch.cuda.current_device()) == 0
pool = ctypes.c_void_p()
assert drv.cuDeviceGetDefaultMemPool(ctypes.byref(pool), dev) == 0
def reserved():
    val = ctypes.c_uint64()
    assert drv.cuMemPoolGetAttribute(pool, 5, ctypes.byref(val)) == 0   # RESERVED_MEM_CURRENT
    return val.value
outs = []
torch.cuda.synchronize()
r0 = reserved()
for _ in range(2):
    o = torch.full_like(q, float("nan"))
    lse = torch.full((w.B, w.Hq, w.Nq), float("nan"), device="cuda")
    rc = T.call_noalloc(w, q, k, v, o, lse)
    torch.cuda.synchronize()
    outs.append((rc, o.float().cpu().numpy(), lse.cpu().numpy()))
r1 = reserved()
status = fav.device_status()
ref_o, ref_lse = fav.forward(q, k, v, causal=w.causal, scale=w.scale)
torch.cuda.synchronize()
r2 = reserved()
ref_o = ref_o.float().cpu().numpy(); ref_lse = ref_lse.cpu().numpy()
err = max(float(np.abs(o_ - ref_o).max()) for _, o_, _ in outs)
lerr = max(float(np.abs(l_ - ref_lse).max()) for _, _, l_ in outs)
print(json.dumps({"rc": [r for r, _, _ in outs], "reserved": [r0, r1, r2], "status": status,
                  "err": err, "lerr": lerr, "splits": fav.last_decode_splits()}))
"""


def test_noalloc_as_first_call_allocates_nothing():
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", FIRST_CALL_SCRIPT, root], capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    res = json.loads(r.stdout.strip().splitlines()[-1])
    assert res["rc"] == [0, 0] and res["status"] == 0
    r0, r1, r2 = res["reserved"]
    assert r1 == r0, "the default memory pool grew across fav_decode_noalloc: %d -> %d" % (r0, r1)
    assert r2 > r1, "fav_forward's workspace did not show in the pool (probe blind?)"
    assert res["splits"] > 1                     # the partials (and so the array) were used
    assert res["err"] <= O_TOL[I.BF16] and res["lerr"] <= LSE_TOL
