"""The seeded input generator: one correct round-to-nearest-even, determinism, recipe (CPU)."""
import numpy as np
import pytest

from paper_2608_18656_gb300 import inputs as I


def test_f16_rounding_matches_numpy_cast():
    rng = np.random.Generator(np.random.PCG64(0))
    x = np.concatenate([rng.standard_normal(100000) * s for s in (1e-6, 1e-3, 1.0, 50.0)])
    np.testing.assert_array_equal(I.round_to_dtype(x, I.F16), x.astype(np.float16).astype(np.float64))


def test_bf16_rounding_matches_torch_on_fp32_values():
    torch = pytest.importorskip("torch")
    rng = np.random.Generator(np.random.PCG64(1))
    x = (rng.standard_normal(200000) * 10).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(I.round_to_dtype(x.astype(np.float64), I.BF16), ref)


def test_bf16_rounding_is_single_rounding_from_fp64():
    """fp64 -> bf16 directly, not via fp32 (which could double-round a tie)."""
    # 1 + 2**-8 + 2**-40 lies just above the bf16 midpoint 1 + 2**-8: rounds up to 1 + 2**-7.
    x = np.array([1.0 + 2.0 ** -8 + 2.0 ** -40, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8])
    np.testing.assert_array_equal(I.round_to_dtype(x, I.BF16),
                                  [1.0 + 2.0 ** -7, 1.0, 1.0 + 2.0 ** -6])


@pytest.mark.parametrize("dt", [I.F32, I.F16, I.BF16])
def test_storage_round_trip(dt):
    rng = np.random.Generator(np.random.PCG64(2))
    r = I.round_to_dtype(rng.standard_normal(1000), dt)
    np.testing.assert_array_equal(I.from_storage(I.to_storage(r, dt), dt), r)


def test_inputs_are_deterministic_and_follow_recipe():
    w = I.WORKLOADS[2].replace(B=1, Hq=4, Hkv=1, Nq=512, Nkv=512)
    a, b = I.make_inputs(w), I.make_inputs(w)
    for n in ("q", "k", "v"):
        np.testing.assert_array_equal(a[n], b[n])
    assert a["v"].min() >= -1 and a["v"].max() <= 1
    # outliers: about 1% of Q entries are larger than any plain N(0,1) draw would plausibly be
    frac = (np.abs(a["q"]) > 6.0).mean()
    assert 0.002 < frac < 0.01
    plain = I.make_inputs(w.replace(outliers=False))
    assert (np.abs(plain["q"]) > 6.0).mean() < 1e-4


def test_workload_flop_counts():
    w = I.WORKLOADS[1]
    assert w.pairs == 2048 * 2049 // 2
    assert w.flops == 4 * 32 * 128 * w.pairs
    assert abs(w.flops / 1e9 - 34.38) < 0.01
    assert abs(I.WORKLOADS[2].flops / 1e9 - 274.9) < 0.1
    assert I.WORKLOADS[3].replace().flops == 4 * 8 * 32 * 128 * 8192


def test_varlen_workload_recipe():
    """The packed-batch workload: lengths in [lo, hi] from the seed (drawn before Q, K, V),
    offsets consistent with them, inputs of the packed shapes, and the FLOP count of causal
    self-attention summed over the sequences."""
    import numpy as np
    w = I.VARLEN_WORKLOADS[0]
    n = w.lengths
    assert len(n) == w.n_seq and n.min() >= w.lo and n.max() <= w.hi
    x = I.make_varlen_inputs(w)
    cu = x["cu_seqlens"]
    assert (cu == w.cu_seqlens).all() and cu[0] == 0 and (np.diff(cu) == n).all()
    assert x["q"].shape == (cu[-1], w.Hq, w.D) and x["k"].shape == (cu[-1], w.Hkv, w.D)
    assert w.flops == sum(4 * w.Hq * w.D * int(m) * (int(m) + 1) // 2 for m in n)
    assert (np.abs(x["v"]) <= 1.0).all()
