"""Planted mistakes in a copy of the C oracle must each fail at least one pin (CPU only).

Every mutation below is a plausible slip in writing the definition of attention out by
hand.  The test compiles the mutated source into a temporary library, swaps it in for the
real one and runs the pins of test_oracle.py; at least one pin must fail for each mutation.
"""
import ctypes
import os
import subprocess

import pytest

import oracle
import test_oracle as T  # noqa: E402

SRC = os.path.join(os.path.dirname(oracle.__file__), "fav_oracle.c")

MUTATIONS = {
    "interleaved_gqa_mapping": ("const int64_t g = h / G;", "const int64_t g = h % J->Hkv;"),
    "top_left_causal": ("return J->Nkv - J->Nq + i + 1;", "return i + 1;"),
    "exp_sign_flipped": ("const double w = exp(s[j] - m);", "const double w = exp(m - s[j]);"),
    "scale_dropped": ("s[j] = J->scale * dot;", "s[j] = dot;"),
    "keys_used_as_values": ("o_out[d] += w * Vh[j * D + d];", "o_out[d] += w * Kh[j * D + d];"),
    "lse_in_log2": ("*lse_out = m + log(l);", "*lse_out = m + log2(l);"),
    "missing_normalisation": ("for (int64_t d = 0; d < D; ++d) o_out[d] /= l;", ""),
    "key_matrix_transposed": ("dot += qr[d] * Kh[j * D + d];", "dot += qr[d] * Kh[d * n + j];"),
    "no_max_subtraction": ("if (s[j] > m) m = s[j];", "m = 0.0;"),
    "last_key_skipped": ("for (int64_t j = 0; j < n; ++j) {\n        const double w",
                         "for (int64_t j = 0; j < n - 1; ++j) {\n        const double w"),
}

PINS = [
    (T.test_golden_two_pass, p) for p in T.golden_cases()
] + [
    (T.test_single_key_returns_its_value, 7),
    (T.test_identical_keys_give_mean_value, None),
    (T.test_zero_query_gives_mean_value, None),
    (T.test_causal_first_query_returns_first_value, None),
    (T.test_probs_rows_sum_to_one, True),
    (T.test_gqa_equals_mha_with_repeated_kv, 4),
    (T.test_causal_rows_equal_prefix_attention, None),
    (T.test_split_kv_logsumexp_combine, 3),
    (T.test_two_pass_equals_streaming_recurrence, ((2, 4, 2, 3, 9, 8), True)),
    (T.test_two_pass_equals_streaming_recurrence, ((1, 2, 2, 4, 7, 8), False)),
]


def _run_pin(fn, arg):
    if arg is None:
        fn()
    elif isinstance(arg, tuple):
        fn(*arg)
    else:
        fn(arg)


def _mutated_lib(tmp_path, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, "mutation anchor not found exactly once: %r" % old
    path = tmp_path / "mut.c"
    path.write_text(src.replace(old, new))
    so = tmp_path / "libmut.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
                           str(path), "-o", str(so), "-lm"])
    return str(so)


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, tmp_path, monkeypatch):
    so = _mutated_lib(tmp_path, *MUTATIONS[name])
    real = oracle._load()
    lib = ctypes.CDLL(so)
    for fn in ("fav_oracle_forward", "fav_oracle_rows", "fav_oracle_probs"):
        getattr(lib, fn).argtypes = getattr(real, fn).argtypes
        getattr(lib, fn).restype = getattr(real, fn).restype
    monkeypatch.setattr(oracle, "_lib", lib)
    failed = []
    for fn, arg in PINS:
        try:
            _run_pin(fn, arg)
        except (AssertionError, ValueError, FloatingPointError):
            failed.append(fn.__name__)
    assert failed, "no pin caught the planted mistake %s" % name


def test_unmutated_oracle_passes_every_pin():
    for fn, arg in PINS:
        _run_pin(fn, arg)
