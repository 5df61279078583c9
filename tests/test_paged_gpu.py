"""fav_decode_paged against the fp64 oracle, one sequence at a time (needs a GB300).

A page pool is filled with seeded Q/K/V values (Q, K ~ N(0,1), V ~ U(-1,1), rounded to the I/O
type); each sequence's keys are scattered over the pool through a random block table (pages in
random order, unused pool pages and unused table entries holding other values).  The expected
result of sequence b is the oracle's attention over its own keys in order."""
import numpy as np
import pytest

import oracle
import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import LSE_TOL, O_TOL, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _reset():
    fav.set_decode_splits(0)
    yield
    fav.set_decode_splits(0)


def build(dtype, lens, Hq, Hkv, Nq, D, page_size, seed, extra_pages=3, share_prefix=False):
    """Seeded inputs in dense form (per sequence) and in paged form (pool + block table)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    B = len(lens)
    max_pages = max(1, max((n + page_size - 1) // page_size for n in lens))
    need = [(n + page_size - 1) // page_size for n in lens]
    num_pages = sum(need) + extra_pages
    pool_k = I.round_to_dtype(rng.standard_normal((num_pages, page_size, Hkv, D)), dtype)
    pool_v = I.round_to_dtype(rng.uniform(-1.0, 1.0, (num_pages, page_size, Hkv, D)), dtype)
    perm = rng.permutation(num_pages)
    table = rng.integers(0, num_pages, size=(B, max_pages)).astype(np.int32)   # unused: any id
    used = 0
    for b in range(B):
        if share_prefix and b > 0 and need[b] > 0 and need[0] > 0:
            # sequence b starts with sequence 0's first page (a shared prompt prefix)
            table[b, 0] = table[0, 0]
            table[b, 1:need[b]] = perm[used:used + need[b] - 1]
            used += need[b] - 1
        else:
            table[b, :need[b]] = perm[used:used + need[b]]
            used += need[b]
    q = I.round_to_dtype(rng.standard_normal((B, Hq, Nq, D)), dtype)
    dense = []
    for b in range(B):
        pages = table[b, :need[b]]
        k = pool_k[pages].reshape(-1, Hkv, D)[:lens[b]].transpose(1, 0, 2)[None]   # [1,Hkv,n,D]
        v = pool_v[pages].reshape(-1, Hkv, D)[:lens[b]].transpose(1, 0, 2)[None]
        dense.append((k, v))
    return dict(q=q, pool_k=pool_k, pool_v=pool_v, table=table, lens=np.array(lens, np.int32),
                dense=dense, B=B, max_pages=max_pages, num_pages=num_pages)


def run_paged(x, dtype, causal, scale):
    import torch
    q = to_device(I.to_storage(x["q"], dtype), dtype)
    kc = to_device(I.to_storage(x["pool_k"], dtype), dtype)
    vc = to_device(I.to_storage(x["pool_v"], dtype), dtype)
    bt = torch.from_numpy(x["table"]).cuda()
    sl = torch.from_numpy(x["lens"]).cuda()
    o, lse = fav.decode_paged(q, kc, vc, bt, sl, causal=causal, scale=scale)
    torch.cuda.synchronize()
    assert fav.device_status() == 0
    return o.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64)


def check_against_oracle(x, o, lse, dtype, Nq, causal, scale):
    for b, (k, v) in enumerate(x["dense"]):
        n = k.shape[2]
        q = x["q"][b:b + 1]
        # rows that see no key: O = 0, LSE = -inf
        vis = np.array([(n - Nq + i + 1) if causal else n for i in range(Nq)])
        rows = np.nonzero(vis > 0)[0]
        empty = np.nonzero(vis <= 0)[0]
        if len(empty):
            assert (o[b][:, empty] == 0).all(), "sequence %d: rows with no key" % b
            assert np.isneginf(lse[b][:, empty]).all()
        if len(rows) == 0:
            continue
        lo = rows[0]                     # visible rows are a suffix of the query rows
        ro, rl = oracle.attention(q[:, :, lo:], k, v, scale, causal)
        err = np.abs(o[b][:, lo:] - ro[0]).max()
        assert err <= O_TOL[dtype], "sequence %d (n=%d): max |O - oracle| = %.3g" % (b, n, err)
        assert np.abs(lse[b][:, lo:] - rl[0]).max() <= LSE_TOL, "sequence %d: LSE" % b


@pytest.mark.parametrize("dtype,D,Hq,Hkv,Nq,page,lens,causal", [
    (I.F16, 128, 8, 2, 1, 16, [1, 17, 300, 1000], False),
    (I.BF16, 64, 8, 1, 1, 64, [0, 64, 65, 2000], False),
    (I.BF16, 128, 4, 2, 4, 32, [3, 4, 100, 513], True),
    (I.F16, 64, 16, 2, 2, 16, [5, 31, 32, 33, 700], True),
    (I.F16, 128, 32, 8, 1, 256, [4096, 1, 255, 257], False),
    (I.BF16, 128, 16, 1, 1, 128, [9000], False),
])
def test_paged_decode_matches_oracle(dtype, D, Hq, Hkv, Nq, page, lens, causal):
    scale = float(np.float32(1.0 / np.sqrt(D)))
    x = build(dtype, lens, Hq, Hkv, Nq, D, page, seed=sum(lens) + page + D)
    o, lse = run_paged(x, dtype, causal, scale)
    assert fav.last_path() == fav.PATH_DECODE
    check_against_oracle(x, o, lse, dtype, Nq, causal, scale)


@pytest.mark.parametrize("page", [16, 32, 64, 128, 256, 1024])
@pytest.mark.parametrize("D", [64, 128])
def test_paged_page_sizes(page, D):
    """Pages smaller than, equal to and larger than the kernel's key tile."""
    scale = float(np.float32(1.0 / np.sqrt(D)))
    x = build(I.F16, [page - 1, 3 * page + 5, 700], 8, 2, 1, D, page, seed=page + D)
    o, lse = run_paged(x, I.F16, False, scale)
    check_against_oracle(x, o, lse, I.F16, 1, False, scale)


@pytest.mark.parametrize("splits", [1, 2, 7])
def test_paged_split_counts_and_shared_prefix(splits):
    """Forced split counts (one split writes O directly; several leave ranges of the shorter
    sequences empty), and sequences that share their first page."""
    fav.set_decode_splits(splits)
    scale = float(np.float32(1.0 / np.sqrt(128)))
    x = build(I.BF16, [40, 600, 1500, 0], 8, 2, 1, 128, 32, seed=11 + splits, share_prefix=True)
    o, lse = run_paged(x, I.BF16, False, scale)
    check_against_oracle(x, o, lse, I.BF16, 1, False, scale)


def test_paged_equals_dense_decode_bitwise():
    """With one split, the paged call runs the dense decode kernel's arithmetic on the same
    key order: equal to fav_forward on the gathered sequence bit for bit."""
    import torch
    fav.set_decode_splits(1)
    scale = float(np.float32(1.0 / np.sqrt(128)))
    x = build(I.F16, [777], 8, 2, 1, 128, 16, seed=5)
    o, lse = run_paged(x, I.F16, False, scale)
    k, v = x["dense"][0]
    qd = to_device(I.to_storage(x["q"], I.F16), I.F16)
    kd = to_device(I.to_storage(np.ascontiguousarray(k), I.F16), I.F16)
    vd = to_device(I.to_storage(np.ascontiguousarray(v), I.F16), I.F16)
    od, ld = fav.forward(qd, kd, vd, scale=scale)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(o, od.float().cpu().numpy().astype(np.float64))
    np.testing.assert_array_equal(lse, ld.cpu().numpy().astype(np.float64))


@pytest.mark.parametrize("splits", [0, 3])
def test_out_of_range_page_ids_are_reported_and_left_out(splits):
    """Block-table entries outside [0, num_pages) inside a sequence's length: the call reports
    FAV_ERR_BAD_PAGE through the device status word, and the keys of those pages take no part in
    the softmax (every other key is attended as usual)."""
    import torch
    fav.set_decode_splits(splits)
    dtype, D, Hq, Hkv, page = I.BF16, 128, 8, 2, 16
    lens = [100, 70]
    x = build(dtype, lens, Hq, Hkv, 1, D, page, seed=9)
    x["table"][0, 2] = x["num_pages"] + 5      # keys 32..47 of sequence 0
    x["table"][1, 0] = -3                      # keys 0..15 of sequence 1
    scale = float(np.float32(1.0 / np.sqrt(D)))
    q = to_device(I.to_storage(x["q"], dtype), dtype)
    kc = to_device(I.to_storage(x["pool_k"], dtype), dtype)
    vc = to_device(I.to_storage(x["pool_v"], dtype), dtype)
    o, lse = fav.decode_paged(q, kc, vc, torch.from_numpy(x["table"]).cuda(),
                              torch.from_numpy(x["lens"]).cuda(), causal=False, scale=scale)
    torch.cuda.synchronize()
    assert fav.device_status() == 7                     # FAV_ERR_BAD_PAGE
    assert fav.device_status() == 0
    o = o.float().cpu().numpy().astype(np.float64)
    lse = lse.cpu().numpy().astype(np.float64)
    for b, dropped in ((0, range(32, 48)), (1, range(0, 16))):
        k, v = x["dense"][b]
        keep = np.array([j for j in range(k.shape[2]) if j not in dropped])
        ro, rl = oracle.attention(x["q"][b:b + 1], k[:, :, keep], v[:, :, keep], scale, False)
        assert np.abs(o[b] - ro[0]).max() <= O_TOL[dtype]
        assert np.abs(lse[b] - rl[0]).max() <= LSE_TOL
