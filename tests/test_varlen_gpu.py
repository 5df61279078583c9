"""fav_prefill_varlen against the fp64 oracle, one sequence at a time (needs a GB300).

Seeded packed inputs (Q, K ~ N(0,1), V ~ U(-1,1), rounded to the I/O type); the expected result
of sequence b is the oracle's attention of its own queries over its own keys."""
import numpy as np
import pytest

import oracle
import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import LSE_TOL, O_TOL, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _reset():
    fav.set_prefill_grid(0)
    yield
    fav.set_prefill_grid(0)


def packed(dtype, lq, lk, Hq, Hkv, D, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    tq, tk = int(sum(lq)), int(sum(lk))
    q = I.round_to_dtype(rng.standard_normal((tq, Hq, D)), dtype)
    k = I.round_to_dtype(rng.standard_normal((tk, Hkv, D)), dtype)
    v = I.round_to_dtype(rng.uniform(-1.0, 1.0, (tk, Hkv, D)), dtype)
    cq = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    ck = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    return q, k, v, cq, ck


def run(dtype, q, k, v, cq, ck, causal, scale):
    import torch
    to = lambda a: to_device(I.to_storage(np.ascontiguousarray(a), dtype), dtype)
    o, lse = fav.prefill_varlen(to(q), to(k), to(v), cq, ck, causal=causal, scale=scale)
    torch.cuda.synchronize()
    assert fav.device_status() == 0
    assert fav.last_path() == fav.PATH_PREFILL
    return o.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64)


def check(q, k, v, cq, ck, o, lse, dtype, causal, scale):
    for b in range(len(cq) - 1):
        if cq[b + 1] == cq[b]:
            continue
        qb = q[cq[b]:cq[b + 1]].transpose(1, 0, 2)[None]      # [1, Hq, lq, D]
        kb = k[ck[b]:ck[b + 1]].transpose(1, 0, 2)[None]
        vb = v[ck[b]:ck[b + 1]].transpose(1, 0, 2)[None]
        ro, rl = oracle.attention(qb, kb, vb, scale, causal)
        err = np.abs(o[cq[b]:cq[b + 1]].transpose(1, 0, 2) - ro[0]).max()
        assert err <= O_TOL[dtype], "sequence %d: max |O - oracle| = %.3g" % (b, err)
        assert np.abs(lse[:, cq[b]:cq[b + 1]] - rl[0]).max() <= LSE_TOL, "sequence %d: LSE" % b


@pytest.mark.parametrize("D", [128, 64])
@pytest.mark.parametrize("dtype", [I.F16, I.BF16])
@pytest.mark.parametrize("causal", [False, True])
def test_varlen_self_attention(dtype, causal, D):
    lens = [1, 64, 127, 128, 129, 300, 513, 7]
    q, k, v, cq, ck = packed(dtype, lens, lens, 8, 2, D, seed=17 + causal + 2 * dtype + D)
    scale = float(np.float32(1.0 / np.sqrt(D)))
    o, lse = run(dtype, q, k, v, cq, ck, causal, scale)
    check(q, k, v, cq, ck, o, lse, dtype, causal, scale)


@pytest.mark.parametrize("D", [128, 64])
@pytest.mark.parametrize("causal", [False, True])
def test_varlen_more_keys_than_queries(causal, D):
    """Chunked prefill: each sequence's new queries attend to a longer key prefix (bottom-right
    causal); a sequence with no queries in the middle of the batch."""
    lq, lk = [100, 0, 250, 33, 128], [500, 40, 250, 1000, 129]
    q, k, v, cq, ck = packed(I.BF16, lq, lk, 4, 4, D, seed=23 + causal + D)
    scale = 0.07
    o, lse = run(I.BF16, q, k, v, cq, ck, causal, scale)
    check(q, k, v, cq, ck, o, lse, I.BF16, causal, scale)


@pytest.mark.parametrize("D,Hq,Hkv", [(128, 6, 3), (64, 6, 3), (64, 8, 2), (64, 3, 1)])
@pytest.mark.parametrize("grid", [1, 5])
def test_varlen_many_units_per_block(grid, D, Hq, Hkv):
    """Few blocks, many units each; at D = 64 both unit pairings (two heads of an even GQA
    group, or two consecutive tiles of one head)."""
    fav.set_prefill_grid(grid)
    lens = [200, 129, 40, 300]
    q, k, v, cq, ck = packed(I.F16, lens, lens, Hq, Hkv, D, seed=31 + grid + D + Hq)
    scale = float(np.float32(1.0 / np.sqrt(D)))
    o, lse = run(I.F16, q, k, v, cq, ck, True, scale)
    check(q, k, v, cq, ck, o, lse, I.F16, True, scale)


@pytest.mark.parametrize("D", [128, 64])
def test_varlen_equals_dense_prefill_bitwise(D):
    """A one-sequence batch runs the dense kernel's arithmetic on the same tiles: equal to
    fav_forward on the same sequence bit for bit (O and LSE)."""
    import torch
    lens = [777]
    q, k, v, cq, ck = packed(I.F16, lens, lens, 8, 2, D, seed=3 + D)
    scale = float(np.float32(1.0 / np.sqrt(D)))
    o, lse = run(I.F16, q, k, v, cq, ck, True, scale)
    to = lambda a: to_device(I.to_storage(np.ascontiguousarray(a), I.F16), I.F16)
    od, ld = fav.forward(to(q.transpose(1, 0, 2)[None]), to(k.transpose(1, 0, 2)[None]),
                         to(v.transpose(1, 0, 2)[None]), causal=True, scale=scale)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(o, od[0].float().cpu().numpy().astype(np.float64).transpose(1, 0, 2))
    np.testing.assert_array_equal(lse, ld[0].cpu().numpy().astype(np.float64))
