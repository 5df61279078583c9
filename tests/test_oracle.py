"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics (no GPU).

Each test names what pins it.  Together they are chosen so that a plausible slip in the
oracle (a dropped scale, a wrong sign in an exponent, a transposed operand, the wrong GQA
head mapping, top-left instead of bottom-right causal alignment, a missing max subtraction,
a log2 LSE, a missing 1/l) fails at least one of them.
"""
import glob
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import naive_flash

HERE = os.path.dirname(os.path.abspath(__file__))


def rand(shape, seed, lo=None):
    rng = np.random.Generator(np.random.PCG64(seed))
    if lo is None:
        return rng.standard_normal(shape)
    return rng.uniform(lo, -lo, shape)


def qkv(B, Hq, Hkv, Nq, Nkv, D, seed=0):
    return (rand((B, Hq, Nq, D), seed), rand((B, Hkv, Nkv, D), seed + 1),
            rand((B, Hkv, Nkv, D), seed + 2, lo=-1.0))


# --- values printed in small worked examples (tests/golden/*.json, each cites its passage) ---

def golden_cases():
    return sorted(glob.glob(os.path.join(HERE, "golden", "*.json")))


@pytest.mark.parametrize("path", golden_cases(), ids=os.path.basename)
def test_golden_two_pass(path):
    g = json.load(open(path))
    q, k, v = (np.array(g[n], np.float64) for n in ("q", "k", "v"))
    o, lse = oracle.attention(q, k, v, g["scale"], g["causal"])
    np.testing.assert_allclose(o, np.array(g["o"]), rtol=0, atol=g["tol"])
    if g["lse"] != "skip":
        np.testing.assert_allclose(lse, np.array(g["lse"]), rtol=0, atol=g["tol"])


@pytest.mark.parametrize("path", golden_cases(), ids=os.path.basename)
def test_golden_naive_flash(path):
    g = json.load(open(path))
    o, lse = naive_flash(g["q"], g["k"], g["v"], g["scale"], g["causal"])
    np.testing.assert_allclose(np.array(o), np.array(g["o"]), rtol=0, atol=g["tol"])
    if g["lse"] != "skip":
        np.testing.assert_allclose(np.array(lse), np.array(g["lse"]), rtol=0, atol=g["tol"])


# --- closed forms of the definition ---

@pytest.mark.parametrize("D", [1, 7, 64])
def test_single_key_returns_its_value(D):
    """Nkv = 1: the only weight is 1, so O = V[0] and LSE = scale * q.k0."""
    q, k, v = qkv(2, 4, 2, 3, 1, D, seed=11)
    scale = 0.37
    o, lse = oracle.attention(q, k, v, scale)
    G = 2
    for h in range(4):
        np.testing.assert_allclose(o[:, h], np.broadcast_to(v[:, h // G], o[:, h].shape),
                                   rtol=0, atol=1e-15)
        expect = scale * np.einsum("bnd,bd->bn", q[:, h], k[:, h // G, 0])
        np.testing.assert_allclose(lse[:, h], expect, rtol=0, atol=1e-13)


def test_identical_keys_give_mean_value():
    """All keys equal: uniform weights, O = mean(V), LSE = s + ln Nkv."""
    B, H, Nq, Nkv, D = 1, 2, 5, 33, 16
    q, k, v = qkv(B, H, H, Nq, Nkv, D, seed=3)
    k[:] = k[:, :, :1, :]
    scale = 0.25
    o, lse = oracle.attention(q, k, v, scale)
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(axis=2, keepdims=True), o.shape),
                               rtol=0, atol=1e-14)
    s = scale * np.einsum("bhnd,bhd->bhn", q, k[:, :, 0])
    np.testing.assert_allclose(lse, s + math.log(Nkv), rtol=0, atol=1e-13)


def test_zero_query_gives_mean_value():
    q, k, v = qkv(2, 3, 3, 4, 17, 8, seed=5)
    q[:] = 0.0
    o, lse = oracle.attention(q, k, v, 0.5)
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(axis=2, keepdims=True), o.shape),
                               rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse, math.log(17), rtol=0, atol=1e-14)


def test_vanishing_scale_gives_mean_value():
    q, k, v = qkv(1, 2, 1, 3, 9, 8, seed=6)
    o, _ = oracle.attention(q, k, v, 1e-300)
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(axis=2, keepdims=True)[:, [0, 0]],
                                                  o.shape), rtol=0, atol=1e-14)


def test_causal_first_query_returns_first_value():
    """Nq = Nkv causal: row 0 sees only key 0."""
    q, k, v = qkv(2, 2, 2, 12, 12, 8, seed=7)
    o, lse = oracle.attention(q, k, v, 0.3, causal=True)
    np.testing.assert_allclose(o[:, :, 0], v[:, :, 0], rtol=0, atol=1e-15)
    np.testing.assert_allclose(lse[:, :, 0], 0.3 * np.einsum("bhd,bhd->bh", q[:, :, 0],
                                                             k[:, :, 0]), rtol=0, atol=1e-14)


# --- invariants ---

@pytest.mark.parametrize("causal", [False, True])
def test_probs_rows_sum_to_one(causal):
    q, k, v = qkv(1, 4, 2, 6, 9, 8, seed=8)
    o, lse, p = oracle.attention_probs(q, k, v, 0.4, causal)
    np.testing.assert_allclose(p.sum(-1), 1.0, rtol=0, atol=1e-14)
    assert (p >= 0).all()
    vr = np.repeat(v, 2, axis=1)
    np.testing.assert_allclose(o, p @ vr, rtol=0, atol=1e-14)
    if causal:
        Nq, Nkv = 6, 9
        for i in range(Nq):
            assert (p[..., i, Nkv - Nq + i + 1:] == 0).all()
            assert (p[..., i, :Nkv - Nq + i + 1] > 0).all()


def test_output_linear_in_values():
    q, k, v = qkv(1, 2, 2, 4, 10, 8, seed=9)
    v2 = rand(v.shape, 99)
    o1, _ = oracle.attention(q, k, v, 0.3)
    o2, _ = oracle.attention(q, k, v2, 0.3)
    o3, _ = oracle.attention(q, k, 2.0 * v - 3.0 * v2, 0.3)
    np.testing.assert_allclose(o3, 2.0 * o1 - 3.0 * o2, rtol=0, atol=1e-13)


def test_joint_kv_permutation_invariance():
    q, k, v = qkv(2, 2, 1, 3, 20, 8, seed=10)
    perm = np.random.Generator(np.random.PCG64(1)).permutation(20)
    o1, l1 = oracle.attention(q, k, v, 0.2)
    o2, l2 = oracle.attention(q, k[:, :, perm], v[:, :, perm], 0.2)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-14)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-13)


@pytest.mark.parametrize("G", [1, 2, 4, 8])
def test_gqa_equals_mha_with_repeated_kv(G):
    Hkv = 2
    q, k, v = qkv(2, Hkv * G, Hkv, 5, 11, 8, seed=12)
    o1, l1 = oracle.attention(q, k, v, 0.3, causal=True)
    o2, l2 = oracle.attention(q, np.repeat(k, G, axis=1), np.repeat(v, G, axis=1), 0.3,
                              causal=True)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=0)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=0)


def test_decode_equals_last_causal_row():
    """A single query against the whole cache is the last row of a causal prefill."""
    q, k, v = qkv(1, 4, 2, 16, 16, 8, seed=13)
    o1, l1 = oracle.attention(q, k, v, 0.35, causal=True)
    o2, l2 = oracle.attention(q[:, :, -1:], k, v, 0.35, causal=False)
    o3, l3 = oracle.attention(q[:, :, -1:], k, v, 0.35, causal=True)
    np.testing.assert_allclose(o1[:, :, -1:], o2, rtol=0, atol=1e-15)
    np.testing.assert_allclose(l1[:, :, -1:], l2, rtol=0, atol=1e-14)
    np.testing.assert_allclose(o2, o3, rtol=0, atol=0)


def test_causal_rows_equal_prefix_attention():
    """Bottom-right causal row i equals non-causal attention over the first Nkv-Nq+i+1 keys."""
    Nq, Nkv = 5, 12
    q, k, v = qkv(1, 2, 2, Nq, Nkv, 8, seed=14)
    o, lse = oracle.attention(q, k, v, 0.5, causal=True)
    for i in range(Nq):
        n = Nkv - Nq + i + 1
        oi, li = oracle.attention(q[:, :, i:i + 1], k[:, :, :n], v[:, :, :n], 0.5)
        np.testing.assert_allclose(o[:, :, i:i + 1], oi, rtol=0, atol=0)
        np.testing.assert_allclose(lse[:, :, i:i + 1], li, rtol=0, atol=0)


@pytest.mark.parametrize("splits", [2, 3, 7])
def test_split_kv_logsumexp_combine(splits):
    """Partials over disjoint key ranges combine exactly: L = logsumexp_s lse_s and
    O = sum_s exp(lse_s - L) O_s (associativity of the online softmax)."""
    q, k, v = qkv(2, 4, 1, 1, 50, 16, seed=15)
    o, lse = oracle.attention(q, k, v, 0.25)
    edges = np.linspace(0, 50, splits + 1).astype(int)
    parts = [oracle.attention(q, k[:, :, a:b], v[:, :, a:b], 0.25)
             for a, b in zip(edges[:-1], edges[1:])]
    ls = np.stack([p[1] for p in parts])
    L = ls.max(0) + np.log(np.exp(ls - ls.max(0)).sum(0))
    oc = sum(np.exp(l_s - L)[..., None] * o_s for o_s, l_s in parts)
    np.testing.assert_allclose(L, lse, rtol=0, atol=1e-13)
    np.testing.assert_allclose(oc, o, rtol=0, atol=1e-14)


# --- brute force: the independent streaming recurrence of Algorithm "ggml-vec FlashAttention" ---

@pytest.mark.parametrize("shape,causal", [
    ((1, 1, 1, 1, 5, 4), False),
    ((1, 2, 2, 4, 7, 8), False),
    ((2, 4, 2, 3, 9, 8), True),
    ((1, 8, 1, 6, 6, 16), True),
    ((1, 2, 1, 1, 13, 8), False),
])
def test_two_pass_equals_streaming_recurrence(shape, causal):
    B, Hq, Hkv, Nq, Nkv, D = shape
    q, k, v = qkv(B, Hq, Hkv, Nq, Nkv, D, seed=sum(shape))
    q *= 3.0  # spread the scores so that the running maximum moves often
    o1, l1 = oracle.attention(q, k, v, 0.7, causal)
    o2, l2 = naive_flash(q, k, v, 0.7, causal)
    np.testing.assert_allclose(o1, np.array(o2), rtol=0, atol=1e-12)
    np.testing.assert_allclose(l1, np.array(l2), rtol=0, atol=1e-12)


def test_rows_entry_matches_full():
    q, k, v = qkv(2, 4, 2, 9, 9, 8, seed=16)
    o, lse = oracle.attention(q, k, v, 0.3, causal=True)
    rows = np.array([0, 5, 17, 35, 71, 70, 8])
    orow, lrow = oracle.attention_rows(q, k, v, rows, 0.3, causal=True)
    np.testing.assert_array_equal(orow, o.reshape(-1, 8)[rows])
    np.testing.assert_array_equal(lrow, lse.reshape(-1)[rows])


def test_threads_do_not_change_results():
    q, k, v = qkv(1, 3, 3, 40, 40, 8, seed=17)
    o1, l1 = oracle.attention(q, k, v, 0.3, causal=True, nthreads=1)
    o2, l2 = oracle.attention(q, k, v, 0.3, causal=True, nthreads=5)
    np.testing.assert_array_equal(o1, o2)
    np.testing.assert_array_equal(l1, l2)


# --- a library routine as a secondary cross-check ---

def test_cross_check_torch_sdpa_fp64():
    torch = pytest.importorskip("torch")
    q, k, v = qkv(2, 4, 2, 7, 7, 16, seed=18)
    o, _ = oracle.attention(q, k, v, 0.25, causal=True)
    t = lambda a: torch.from_numpy(a)
    ref = torch.nn.functional.scaled_dot_product_attention(
        t(q), t(np.repeat(k, 2, axis=1)), t(np.repeat(v, 2, axis=1)), is_causal=True,
        scale=0.25)
    np.testing.assert_allclose(o, ref.numpy(), rtol=0, atol=1e-13)


def test_rejects_invalid_arguments():
    q, k, v = qkv(1, 3, 2, 2, 2, 4)
    with pytest.raises(ValueError):
        oracle.attention(q, k, v, 1.0)              # Hq % Hkv != 0
    q, k, v = qkv(1, 2, 2, 5, 3, 4)
    with pytest.raises(ValueError):
        oracle.attention(q, k, v, 1.0, causal=True)  # causal with Nq > Nkv
