"""fav_forward_nonflash (materialised scores, cuBLAS GEMMs + this library's softmax kernel)
against the fp64 oracle on seeded inputs (needs a GB300), with the library's tolerances (O
within 3e-3 for fp16 and bf16, LSE within 1e-4)."""
import numpy as np
import pytest

import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import check, to_device

pytestmark = pytest.mark.gpu


def W(dtype, B, Hq, Hkv, Nq, Nkv, D, causal=False, outliers=False, seed=7):
    return I.Workload("t", dtype, B, Hq, Hkv, Nq, Nkv, D, causal, outliers, seed)


def run_nonflash(w, x, workspace=None):
    import torch
    q, k, v = (to_device(x[n + "_bits"], w.dtype) for n in ("q", "k", "v"))
    o, lse = fav.forward_nonflash(q, k, v, causal=w.causal, scale=w.scale, workspace=workspace)
    torch.cuda.synchronize()
    return o.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("dtype", [I.F16, I.BF16])
@pytest.mark.parametrize("B,Hq,Hkv,Nq,Nkv,D,causal", [
    (1, 4, 4, 128, 128, 128, True),        # MHA, one tile
    (2, 8, 2, 300, 300, 64, True),         # GQA, ragged length
    (1, 8, 1, 200, 517, 128, True),        # MQA, Nq < Nkv (bottom-right mask)
    (2, 4, 2, 257, 1000, 128, False),
    (1, 2, 2, 1, 333, 64, False),          # one query row
    (1, 4, 2, 1, 1, 128, True),            # one key
    (1, 2, 1, 64, 6000, 64, True),         # row of 8 float4 per thread (registers)
    (1, 2, 2, 16, 9000, 128, False),       # row longer than the register path (shared memory)
])
def test_nonflash_matches_oracle(dtype, B, Hq, Hkv, Nq, Nkv, D, causal):
    """Rows of 1..9000 keys: multiples of 4 up to 8192 take the register softmax, the others
    the shared-memory one."""
    w = W(dtype, B, Hq, Hkv, Nq, Nkv, D, causal, seed=Nq + Nkv + D)
    x = I.make_inputs(w)
    o, lse = run_nonflash(w, x)
    check(w, o, lse, x)


def test_nonflash_outliers_and_caller_workspace():
    """Large-magnitude scores (outlier rows) and a caller-given, oversized workspace."""
    import torch
    w = W(I.BF16, 1, 8, 2, 384, 384, 128, True, outliers=True, seed=3)
    x = I.make_inputs(w)
    ws = torch.empty(fav.nonflash_workspace_size(1, 8, 384, 384) + 4096, dtype=torch.uint8,
                     device="cuda")
    o, lse = run_nonflash(w, x, workspace=ws)
    check(w, o, lse, x)


@pytest.mark.parametrize("idx", [1, 2])
def test_nonflash_prefill_workloads(idx):
    """The measured prefill workloads at full size, every row."""
    w = I.WORKLOADS[idx]
    x = I.make_inputs(w)
    o, lse = run_nonflash(w, x)
    check(w, o, lse, x)
