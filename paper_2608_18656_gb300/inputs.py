"""Seeded synthetic attention inputs, shared by the tests, the bench and smoke().

This module holds no attention arithmetic: it only draws random numbers and rounds them
once to the I/O dtype.  Both the fp64 oracle and the CUDA path consume exactly the values
produced here (the oracle after an exact upcast to fp64).

Recipe (shapes of the paper's model layers, Models section, table of network models:
TinyLlama / Llama 3.2 with D = 64 and 8- or 4-way head sharing, Qwen2.5 with D = 128):
  * numpy ``Generator(PCG64(seed))``, seed = 1234 + workload index;
  * Q, K iid N(0, 1); V iid U(-1, 1), drawn in fp64 in the order Q, K, V;
  * optional outliers: independent Bernoulli(0.01) masks on Q then K, masked entries x 8;
  * one round-to-nearest-even to the I/O dtype (fp32, fp16 or bf16), straight from fp64.
"""
from dataclasses import dataclass

import numpy as np

F32, F16, BF16 = 0, 1, 2
DTYPE_NAMES = {F32: "f32", F16: "f16", BF16: "bf16"}
_MANT = {F16: 10, BF16: 7}       # stored mantissa bits
_EMIN = {F16: -14, BF16: -126}   # smallest normal exponent


@dataclass(frozen=True)
class Workload:
    name: str
    dtype: int
    B: int
    Hq: int
    Hkv: int
    Nq: int
    Nkv: int
    D: int
    causal: bool
    outliers: bool
    seed: int

    @property
    def scale(self):
        """1/sqrt(D) rounded to fp32, the value every caller passes."""
        return float(np.float32(1.0 / np.sqrt(self.D)))

    @property
    def pairs(self):
        """Unmasked (query, key) pairs per head."""
        if self.causal:
            off = self.Nkv - self.Nq
            return self.Nq * off + self.Nq * (self.Nq + 1) // 2
        return self.Nq * self.Nkv

    @property
    def flops(self):
        """Algorithmic FLOPs: 2 for Q.K and 2 for P.V per unmasked pair and head dim."""
        return 4 * self.B * self.Hq * self.D * self.pairs

    @property
    def elem_bytes(self):
        return 4 if self.dtype == F32 else 2

    @property
    def io_bytes(self):
        """Bytes of Q, K, V read plus O (I/O dtype) and LSE (fp32) written, once each."""
        e = self.elem_bytes
        q = self.B * self.Hq * self.Nq * self.D * e
        kv = 2 * self.B * self.Hkv * self.Nkv * self.D * e
        return q + kv + q + self.B * self.Hq * self.Nq * 4

    def replace(self, **kw):
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


# The five workloads of this library's measurement plan (index 0..4).
WORKLOADS = [
    Workload("mha_f32_b1_h2_n128_d64", F32, 1, 2, 2, 128, 128, 64, False, False, 1234),
    Workload("mha_f16_causal_prefill_b1_h32_n2048_d128", F16, 1, 32, 32, 2048, 2048, 128,
             True, False, 1235),
    Workload("gqa_bf16_causal_prefill_b4_hq32_hkv8_n4096_d64_outliers", BF16, 4, 32, 8, 4096,
             4096, 64, True, True, 1236),
    Workload("gqa_f16_decode_b8_hq32_hkv8_nkv8192_d128", F16, 8, 32, 8, 1, 8192, 128, False,
             False, 1237),
    Workload("mqa_bf16_decode_b16_hq16_hkv1_nkv32768_d128", BF16, 16, 16, 1, 1, 32768, 128,
             False, False, 1238),
]


@dataclass(frozen=True)
class VarlenWorkload:
    """A packed batch of prompts of different lengths (the paper's short edge prompts, N from 64
    to 512 tokens): n_seq lengths drawn uniformly from [lo, hi] (seeded), each sequence attending
    to itself; Q [total, Hq, D], K and V [total, Hkv, D] (token-major, cu_seqlens layout)."""
    name: str
    dtype: int
    n_seq: int
    lo: int
    hi: int
    Hq: int
    Hkv: int
    D: int
    causal: bool
    seed: int

    @property
    def scale(self):
        return float(np.float32(1.0 / np.sqrt(self.D)))

    @property
    def lengths(self):
        rng = np.random.Generator(np.random.PCG64(self.seed))
        return rng.integers(self.lo, self.hi + 1, size=self.n_seq)

    @property
    def cu_seqlens(self):
        return np.concatenate([[0], np.cumsum(self.lengths)]).astype(np.int32)

    @property
    def flops(self):
        """Algorithmic FLOPs: 4 * Hq * D per unmasked (query, key) pair of every sequence."""
        n = self.lengths.astype(np.int64)
        pairs = n * (n + 1) // 2 if self.causal else n * n
        return int(4 * self.Hq * self.D * pairs.sum())


# Packed-batch workload of the measurement plan: 64 prompts of 64..512 tokens, GQA, fp16.
VARLEN_WORKLOADS = [
    VarlenWorkload("varlen_f16_causal_64prompts_n64to512_hq32_hkv8_d128", F16, 64, 64, 512, 32,
                   8, 128, True, 1240),
]


def make_varlen_inputs(w):
    """Draw a packed batch: the lengths first (VarlenWorkload.lengths), then Q, K, V as in
    make_inputs, each [total, H, D]."""
    rng = np.random.Generator(np.random.PCG64(w.seed))
    n = rng.integers(w.lo, w.hi + 1, size=w.n_seq)
    total = int(n.sum())
    q = rng.standard_normal((total, w.Hq, w.D))
    k = rng.standard_normal((total, w.Hkv, w.D))
    v = rng.uniform(-1.0, 1.0, (total, w.Hkv, w.D))
    out = {"cu_seqlens": np.concatenate([[0], np.cumsum(n)]).astype(np.int32)}
    for name, x in (("q", q), ("k", k), ("v", v)):
        r = round_to_dtype(x, w.dtype)
        out[name] = r
        out[name + "_bits"] = to_storage(r, w.dtype)
    return out


def round_to_dtype(x, dtype):
    """Round fp64 values once, to nearest-even, to the I/O dtype; returns fp64 values."""
    x = np.asarray(x, dtype=np.float64)
    if dtype == F32:
        return x.astype(np.float32).astype(np.float64)
    mant, emin = _MANT[dtype], _EMIN[dtype]
    _, e = np.frexp(x)                        # |x| = m * 2**e with m in [0.5, 1)
    ex = np.maximum(e - 1, emin)              # exponent of the leading bit (clamped: subnormals)
    quantum = np.ldexp(1.0, ex - mant)        # spacing of representable values near x
    return np.rint(x / quantum) * quantum     # np.rint rounds halves to even


def to_storage(x_rounded, dtype):
    """Exact bit patterns of already-rounded values: float32, float16 or uint16 (bf16)."""
    if dtype == F32:
        return x_rounded.astype(np.float32)
    if dtype == F16:
        return x_rounded.astype(np.float16)
    bits = x_rounded.astype(np.float32).view(np.uint32)
    return (bits >> 16).astype(np.uint16)


def from_storage(a, dtype):
    """Inverse of ``to_storage``: exact fp64 values of stored bits."""
    a = np.asarray(a)
    if dtype == BF16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def make_inputs(w):
    """Draw one workload's inputs.  Returns dict of fp64 rounded values and storage arrays."""
    rng = np.random.Generator(np.random.PCG64(w.seed))
    qs = (w.B, w.Hq, w.Nq, w.D)
    ks = (w.B, w.Hkv, w.Nkv, w.D)
    q = rng.standard_normal(qs)
    k = rng.standard_normal(ks)
    v = rng.uniform(-1.0, 1.0, ks)
    if w.outliers:
        q = np.where(rng.random(qs) < 0.01, q * 8.0, q)
        k = np.where(rng.random(ks) < 0.01, k * 8.0, k)
    out = {}
    for name, x in (("q", q), ("k", k), ("v", v)):
        r = round_to_dtype(x, w.dtype)
        out[name] = r
        out[name + "_bits"] = to_storage(r, w.dtype)
    return out
