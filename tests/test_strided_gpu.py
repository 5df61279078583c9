"""fav_forward_strided on the GPU: the heads-interleaved layout [B, N, H, D] (the layout of the
paper's inference engine, Method section), padded token strides, and a strided output, on
every kernel family.  The kernels read the same values whatever the layout, so the strided
results must equal the contiguous call's results exactly, and the oracle within tolerance."""
import numpy as np
import pytest

import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import check, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _reset():
    fav.set_path(fav.PATH_AUTO)
    fav.set_decode_splits(0)
    yield
    fav.set_path(fav.PATH_AUTO)
    fav.set_decode_splits(0)


CASES = [
    ("prefill_f16_d128", I.Workload("t", I.F16, 2, 4, 4, 300, 300, 128, True, False, 71), fav.PATH_PREFILL),
    ("prefill_bf16_d64_gqa", I.Workload("t", I.BF16, 2, 8, 2, 257, 257, 64, True, True, 72), fav.PATH_PREFILL),
    ("decode_f16_gqa", I.Workload("t", I.F16, 3, 8, 2, 1, 1000, 128, False, False, 73), fav.PATH_DECODE),
    ("decode_bf16_mqa", I.Workload("t", I.BF16, 2, 8, 1, 2, 3000, 64, True, False, 74), fav.PATH_DECODE),
    ("simt_f32", I.Workload("t", I.F32, 2, 4, 2, 50, 70, 64, False, False, 75), fav.PATH_SIMT),
]


def _interleaved(t):
    """The same values, stored [B, N, H, D]: returned as a [B, H, N, D] view."""
    return t.transpose(1, 2).contiguous().transpose(1, 2)


def _padded(t, pad):
    """The same values in rows of D + pad elements (a sliced, padded cache)."""
    import torch
    B, H, N, D = t.shape
    buf = torch.full((B, H, N, D + pad), float("nan"), dtype=t.dtype, device=t.device)
    buf[..., :D] = t
    return buf[..., :D]


@pytest.mark.parametrize("name,w,path", CASES, ids=[c[0] for c in CASES])
def test_strided_layouts_match_contiguous(name, w, path):
    import torch
    x = I.make_inputs(w)
    q, k, v = (to_device(x[n + "_bits"], w.dtype) for n in ("q", "k", "v"))
    fav.set_path(path)
    o_ref, l_ref = fav.forward(q, k, v, causal=w.causal, scale=w.scale)
    assert fav.last_path() == path
    torch.cuda.synchronize()
    pad = 8 if w.dtype != I.F32 else 4
    variants = {
        "bnhd": (_interleaved(q), _interleaved(k), _interleaved(v), None),
        "padded": (_padded(q, pad), _padded(k, 2 * pad), _padded(v, pad), None),
        "bnhd_out": (q, _interleaved(k), v, _interleaved(torch.empty_like(q))),
    }
    for tag, (qq, kk, vv, oo) in variants.items():
        assert not all(t.is_contiguous() for t in (qq, kk, vv) + ((oo,) if oo is not None else ()))
        o, l = fav.forward(qq, kk, vv, causal=w.causal, scale=w.scale, out=oo)
        torch.cuda.synchronize()
        assert fav.device_status() == 0
        assert fav.last_path() == path
        assert torch.equal(o, o_ref), tag
        assert torch.equal(l, l_ref), tag
    o64 = o_ref.float().cpu().numpy().astype(np.float64)
    check(w, o64, l_ref.cpu().numpy().astype(np.float64), x)
