"""Helpers for the GPU parity tests: seeded inputs -> CUDA path and fp64 oracle."""
import numpy as np

import oracle
import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I

# Tolerances: max-abs on O of 1e-5 (fp32 I/O) and 3e-3 (fp16/bf16 I/O, fp32 accumulation);
# the natural-log LSE within 1e-4.
O_TOL = {I.F32: 1e-5, I.F16: 3e-3, I.BF16: 3e-3}
LSE_TOL = 1e-4


def to_device(bits, dtype):
    import torch
    if dtype == I.BF16:
        return torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(bits).cuda()


def run_gpu(w, x, return_lse=True):
    import torch
    q, k, v = (to_device(x[n + "_bits"], w.dtype) for n in ("q", "k", "v"))
    o, lse = fav.forward(q, k, v, causal=w.causal, scale=w.scale, return_lse=return_lse)
    torch.cuda.synchronize()
    assert fav.device_status() == 0
    o64 = o.float().cpu().numpy().astype(np.float64)
    l64 = lse.cpu().numpy().astype(np.float64) if lse is not None else None
    return o64, l64


def sample_rows(w, n, seed=0):
    total = w.B * w.Hq * w.Nq
    if total <= n:
        return np.arange(total)
    rng = np.random.Generator(np.random.PCG64(seed))
    rows = rng.choice(total, size=n - 2, replace=False)
    return np.unique(np.concatenate([[0, total - 1], rows]))


def check(w, o, lse, x, rows=None):
    """Compare GPU results with the oracle on all rows (rows=None) or on sampled rows."""
    if rows is None:
        ro, rl = oracle.attention(x["q"], x["k"], x["v"], w.scale, w.causal)
        go = o
        gl = lse
    else:
        ro, rl = oracle.attention_rows(x["q"], x["k"], x["v"], rows, w.scale, w.causal)
        go = o.reshape(-1, w.D)[rows]
        gl = lse.reshape(-1)[rows] if lse is not None else None
    assert np.isfinite(go).all()
    err = np.abs(go - ro).max()
    assert err <= O_TOL[w.dtype], "max |O - oracle| = %.3g > %.3g" % (err, O_TOL[w.dtype])
    if gl is not None:
        lerr = np.abs(gl - rl).max()
        assert lerr <= LSE_TOL, "max |LSE - oracle| = %.3g" % lerr
    return err
