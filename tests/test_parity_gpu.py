"""Parity of the CUDA path with the fp64 oracle on seeded inputs (needs a GB300)."""
import numpy as np

import oracle
import pytest

import paper_2608_18656_gb300 as fav
from paper_2608_18656_gb300 import inputs as I
from gpu_util import LSE_TOL, O_TOL, check, run_gpu, sample_rows, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _reset():
    fav.set_path(fav.PATH_AUTO)
    fav.set_decode_splits(0)
    fav.set_prefill_grid(0)
    yield
    fav.set_path(fav.PATH_AUTO)
    fav.set_decode_splits(0)
    fav.set_prefill_grid(0)


def W(dtype, B, Hq, Hkv, Nq, Nkv, D, causal=False, outliers=False, seed=7):
    return I.Workload("t", dtype, B, Hq, Hkv, Nq, Nkv, D, causal, outliers, seed)


# ---- the five measured workloads at full size ----

def test_workload0_fp32_mha_full():
    w = I.WORKLOADS[0]
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_SIMT
    check(w, o, lse, x)


@pytest.mark.parametrize("idx", [1, 2])
def test_prefill_workloads_full(idx):
    """The two measured prefill workloads, every row against the oracle."""
    w = I.WORKLOADS[idx]
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_PREFILL
    check(w, o, lse, x)


@pytest.mark.parametrize("idx", [3, 4])
def test_decode_workloads_full(idx):
    w = I.WORKLOADS[idx]
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_DECODE
    assert fav.last_decode_splits() > 1
    check(w, o, lse, x)


# ---- decode path edge cases ----

@pytest.mark.parametrize("dtype", [I.F16, I.BF16])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("G", [1, 2, 4, 8, 16])
def test_decode_group_sizes(dtype, D, G):
    w = W(dtype, 2, 2 * G, 2, 1, 1000, D, seed=G + D)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_DECODE
    check(w, o, lse, x)


@pytest.mark.parametrize("splits", [1, 2, 3, 7, 16, 1000])
def test_decode_split_counts(splits):
    fav.set_decode_splits(splits)
    w = W(I.BF16, 1, 8, 1, 1, 777, 128, seed=splits)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert 1 <= fav.last_decode_splits() <= splits
    check(w, o, lse, x)


def test_decode_split_counts_change_between_calls():
    """Calls that alternate split counts on one shape (and one split in between) reuse the
    split-KV workspace with different partial layouts: every call matches the oracle."""
    w = W(I.BF16, 2, 16, 4, 1, 3000, 128, seed=21)
    x = I.make_inputs(w)
    for splits in (3, 7, 2, 7, 1, 5, 3):
        fav.set_decode_splits(splits)
        o, lse = run_gpu(w, x)
        assert fav.last_path() == fav.PATH_DECODE
        check(w, o, lse, x)


@pytest.mark.parametrize("Nkv", [1, 2, 31, 32, 33, 63, 64, 65, 129])
def test_decode_short_caches(Nkv):
    w = W(I.F16, 1, 4, 1, 1, Nkv, 128, seed=Nkv)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    check(w, o, lse, x)


@pytest.mark.parametrize("Nq,G,causal", [(2, 4, True), (4, 4, True), (3, 1, False),
                                         (4, 8, True), (16, 4, True)])
def test_decode_path_small_nq(Nq, G, causal):
    """Several queries per KV head (speculative-decode shape), bottom-right causal."""
    fav.set_path(fav.PATH_DECODE)
    w = W(I.BF16, 2, 2 * G, 2, Nq, 300, 64, causal=causal, seed=Nq * 10 + G)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_DECODE
    check(w, o, lse, x)


def test_decode_without_lse():
    w = W(I.F16, 1, 8, 2, 1, 500, 128, seed=3)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x, return_lse=False)
    assert lse is None
    check(w, o, None, x)


def test_decode_outliers():
    w = W(I.BF16, 2, 16, 1, 1, 4096, 128, outliers=True, seed=5)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    check(w, o, lse, x)


# ---- CUDA-core path ----

@pytest.mark.parametrize("dtype", [I.F32, I.F16, I.BF16])
@pytest.mark.parametrize("shape", [(1, 2, 2, 1, 1, 64, False), (2, 4, 2, 37, 37, 32, True),
                                   (1, 3, 1, 5, 200, 8, True), (1, 2, 2, 128, 128, 256, False),
                                   (1, 1, 1, 33, 70, 96, False), (1, 2, 1, 6, 300, 4, True),
                                   (3, 4, 2, 130, 130, 64, True)])
def test_simt_path(dtype, shape):
    fav.set_path(fav.PATH_SIMT)
    B, Hq, Hkv, Nq, Nkv, D, causal = shape
    if dtype != I.F32 and D % 8:
        pytest.skip("16-bit rows need D % 8 == 0")
    w = W(dtype, B, Hq, Hkv, Nq, Nkv, D, causal=causal, seed=Nq + D)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_SIMT
    check(w, o, lse, x)


def test_forced_path_that_cannot_run_is_unsupported():
    import torch
    fav.set_path(fav.PATH_DECODE)
    q = torch.zeros(1, 1, 4, 64, device="cuda", dtype=torch.float32)
    with pytest.raises(fav.FavError) as e:
        fav.forward(q, q, q)
    assert e.value.status == 2


def test_error_leaves_outputs_untouched():
    import torch
    q = torch.randn(1, 3, 4, 64, device="cuda", dtype=torch.float16)
    k = torch.randn(1, 2, 4, 64, device="cuda", dtype=torch.float16)
    o = torch.full_like(q, 7.0)
    with pytest.raises(fav.FavError):
        fav.forward(q, k, k, out=o)
    torch.cuda.synchronize()
    assert bool((o == 7.0).all())


# ---- prefill path edge cases ----

@pytest.mark.parametrize("dtype,D,causal", [(I.F16, 128, True), (I.BF16, 64, True),
                                            (I.BF16, 128, False), (I.F16, 64, False)])
def test_prefill_growing_scores(dtype, D, causal):
    """Keys scaled by a ramp along the sequence: the row maximum keeps growing from tile to
    tile, so the lazy rescale and the speculative-exponential redo both run many times."""
    w = W(dtype, 1, 4, 2, 700, 700, D, causal=causal, seed=40 + D)
    x = I.make_inputs(w)
    ramp = np.linspace(1.0, 12.0, w.Nkv)[None, None, :, None]
    k = I.round_to_dtype(x["k"] * ramp, dtype)
    x = dict(x, k=k, k_bits=I.to_storage(k, dtype))
    fav.set_path(fav.PATH_PREFILL)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_PREFILL
    check(w, o, lse, x)


@pytest.mark.parametrize("Nq,Nkv,causal", [(1, 1, False), (5, 5, True), (128, 128, True),
                                           (129, 129, True), (255, 1000, True), (300, 40, False)])
def test_prefill_ragged_shapes(Nq, Nkv, causal):
    fav.set_path(fav.PATH_PREFILL)
    w = W(I.BF16, 1, 2, 1, Nq, Nkv, 128, causal=causal, seed=Nq + Nkv)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    check(w, o, lse, x)


@pytest.mark.parametrize("Hq,Hkv", [(3, 1), (6, 3), (5, 5), (8, 1)])
def test_prefill_head_pairings(Hq, Hkv):
    """Even groups pair two heads per block; odd groups pair two query tiles of one head."""
    fav.set_path(fav.PATH_PREFILL)
    w = W(I.F16, 2, Hq, Hkv, 260, 260, 64, causal=True, seed=Hq * 7 + Hkv)
    x = I.make_inputs(w)
    o, lse = run_gpu(w, x)
    check(w, o, lse, x)


@pytest.mark.parametrize("D", [64, 128])
def test_prefill_bf16_v_range(D):
    """bf16 prefill converts V to fp16 under a power-of-two scale per KV head: heads whose V
    is far above or below fp16's range, a head of zeros, and a head with one large outlier
    must all match the oracle.  Scaling the inputs by 2^k scales the exact output and every
    rounding by 2^k, so the tolerance is the workloads' 3e-3 (which holds for |O| < 1) times
    the power of two that brings the row's magnitude below 1."""
    import torch
    fav.set_path(fav.PATH_PREFILL)
    w = W(I.BF16, 1, 10, 5, 300, 300, D, causal=True, seed=60 + D)
    x = I.make_inputs(w)
    v = x["v"].copy()
    bulk = np.array([2.0 ** 20, 2.0 ** -40, 1000.0, 0.0, 1.0])
    v *= bulk[None, :, None, None]
    v[0, 4, 37, 5] = 2.0 ** 25                     # one outlier in an otherwise U(-1,1) head
    v = I.round_to_dtype(v, I.BF16)
    x = dict(x, v=v, v_bits=I.to_storage(v, I.BF16))
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_PREFILL
    ro, rl = oracle.attention(x["q"], x["k"], x["v"], w.scale, w.causal)
    assert np.isfinite(o).all()
    G = w.Hq // w.Hkv
    for h in range(w.Hq):
        ref = ro[0, h]
        mag = np.maximum(bulk[h // G], np.abs(ref).max(axis=1, keepdims=True))
        tol = np.where(mag > 0, 3e-3 * np.exp2(np.ceil(np.log2(np.maximum(mag, 1e-300)))), 0.0)
        assert (np.abs(o[0, h] - ref) <= tol).all(), "head %d" % h
    assert np.abs(lse - rl).max() <= LSE_TOL


@pytest.mark.parametrize("dtype,B,Hq,Hkv,N", [
    (I.F16, 3, 32, 32, 2048),     # 96 heads of 1 MB of K/V: blocks of 64 heads, the last of 32
    (I.BF16, 4, 32, 8, 8192),     # 32 KV heads of 4 MB: blocks of 16 groups (64 query heads)
])
def test_prefill_head_blocks(dtype, B, Hq, Hkv, N):
    """Heads taken in blocks whose K/V fit in L2 (query tiles of a block before the next
    block): every query tile computed exactly once (output prefilled with NaN) and sampled rows
    equal to the oracle."""
    import torch
    w = W(dtype, B, Hq, Hkv, N, N, 128, causal=True, seed=N + B)
    x = I.make_inputs(w)
    q, k, v = (to_device(x[n + "_bits"], dtype) for n in ("q", "k", "v"))
    o = torch.full_like(q, float("nan"))
    lse = torch.full((B, Hq, N), float("nan"), device="cuda")
    fav.forward(q, k, v, causal=True, scale=w.scale, out=o, lse_out=lse)
    torch.cuda.synchronize()
    assert fav.device_status() == 0
    assert fav.last_path() == fav.PATH_PREFILL
    assert bool(torch.isfinite(o.float()).all()) and bool(torch.isfinite(lse).all())
    o64 = o.float().cpu().numpy().astype(np.float64)
    check(w, o64, lse.cpu().numpy().astype(np.float64), x, rows=sample_rows(w, 2048, seed=N))


@pytest.mark.parametrize("grid", [0, 1, 2])
@pytest.mark.parametrize("Nq,Nkv,causal", [(300, 64, False), (300, 300, True), (257, 257, True)])
def test_prefill_pair_missing_second_tile(grid, Nq, Nkv, causal):
    """D = 64 with an odd GQA group pairs query tiles (2p, 2p+1) of one head; with an odd number
    of query tiles the last pair's second tile lies beyond the sequence (no key tiles, its Q copy
    the zero fill).  Short caches make each unit's last S the first, so the Q buffers are handed
    back to the producer almost at once."""
    fav.set_path(fav.PATH_PREFILL)
    w = W(I.BF16, 2, 3, 1, Nq, Nkv, 64, causal=causal, seed=Nq + Nkv + grid)
    x = I.make_inputs(w)
    fav.set_prefill_grid(grid)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_PREFILL
    check(w, o, lse, x)


@pytest.mark.parametrize("grid", [1, 3, 7])
@pytest.mark.parametrize("dtype,D,causal,Hq,Hkv,N", [(I.F16, 128, True, 4, 2, 700),
                                                     (I.BF16, 64, True, 4, 1, 520),
                                                     (I.F16, 64, False, 2, 2, 300),
                                                     (I.BF16, 128, False, 3, 1, 257)])
def test_prefill_many_tiles_per_block(grid, dtype, D, causal, Hq, Hkv, N):
    """The persistent prefill grid capped to a few blocks: each block works through many
    query tiles of different heads and lengths in turn (score buffers, stage rings, Q buffers
    and barrier phases carried from one tile to the next), and the results equal those of the
    default grid bit for bit (a tile's arithmetic does not depend on which block runs it)."""
    fav.set_path(fav.PATH_PREFILL)
    w = W(dtype, 2, Hq, Hkv, N, N, D, causal=causal, seed=grid * 100 + D + N)
    x = I.make_inputs(w)
    o_ref, lse_ref = run_gpu(w, x)
    fav.set_prefill_grid(grid)
    o, lse = run_gpu(w, x)
    assert fav.last_path() == fav.PATH_PREFILL
    check(w, o, lse, x)
    np.testing.assert_array_equal(o, o_ref)
    np.testing.assert_array_equal(lse, lse_ref)


# ---- end-to-end host-buffer entry point ----

@pytest.mark.parametrize("shape", [(I.F16, 1, 8, 8, 700, 700, 128, True),
                                   (I.BF16, 2, 8, 2, 1, 3000, 128, False),
                                   (I.BF16, 1, 6, 3, 333, 333, 64, False),
                                   (I.F32, 1, 2, 2, 64, 64, 64, False)])
def test_forward_host_matches_device(shape):
    """fav_forward_host (pipelined over KV-head chunks) equals fav_forward: bit for bit on the
    prefill and CUDA-core paths (the per-head arithmetic is the same); within the parity
    tolerances on the decode path (a chunk may get a different split count)."""
    import torch
    dt, B, Hq, Hkv, Nq, Nkv, D, causal = shape
    w = W(dt, B, Hq, Hkv, Nq, Nkv, D, causal=causal, seed=Nq + Hq)
    x = I.make_inputs(w)
    o_dev, lse_dev = run_gpu(w, x)
    bits = {n: np.ascontiguousarray(x[n + "_bits"]) for n in ("q", "k", "v")}
    o_host = np.empty_like(bits["q"])
    lse_host = np.empty((B, Hq, Nq), np.float32)
    fav.forward_host(bits["q"], bits["k"], bits["v"], o_host, lse_host, B, Hq, Hkv, Nq, Nkv, D,
                     w.scale, causal, dt)
    if Nq * (Hq // Hkv) <= 16 and dt != I.F32:
        np.testing.assert_allclose(I.from_storage(o_host, dt), o_dev, rtol=0, atol=O_TOL[dt])
        np.testing.assert_allclose(lse_host.astype(np.float64), lse_dev, rtol=0, atol=LSE_TOL)
    else:
        np.testing.assert_array_equal(I.from_storage(o_host, dt), o_dev)
        np.testing.assert_array_equal(lse_host.astype(np.float64), lse_dev)


def test_forward_host_headline_vs_oracle():
    """The host-buffer call on the headline workload (fp16 MHA causal prefill, B 1, H 32,
    N 2048, D 128), every row of O and LSE against the oracle."""
    w = I.WORKLOADS[1]
    x = I.make_inputs(w)
    bits = {n: np.ascontiguousarray(x[n + "_bits"]) for n in ("q", "k", "v")}
    o_host = np.empty_like(bits["q"])
    lse_host = np.empty((w.B, w.Hq, w.Nq), np.float32)
    fav.forward_host(bits["q"], bits["k"], bits["v"], o_host, lse_host, w.B, w.Hq, w.Hkv, w.Nq,
                     w.Nkv, w.D, w.scale, w.causal, w.dtype)
    assert fav.device_status() == 0
    check(w, I.from_storage(o_host, w.dtype), lse_host.astype(np.float64), x)
