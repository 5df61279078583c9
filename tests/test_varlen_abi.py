"""fav_prefill_varlen: argument validation before anything is launched (runs without a GPU;
the tensor pointers are aligned fake device addresses, the sequence offsets real host arrays)."""
import ctypes

import numpy as np
import pytest

import paper_2608_18656_gb300 as fav

Q, K, V, O, LSE = 1 << 20, 2 << 20, 3 << 20, 4 << 20, 5 << 20


def call(cq=(0, 5, 9), ck=(0, 5, 9), q=Q, k=K, v=V, o=O, lse=LSE, B=None, Hq=4, Hkv=2, D=128,
         scale=0.088, causal=0, dtype=fav.F16, null_cq=False):
    cq = np.asarray(cq, np.int32)
    ck = np.asarray(ck, np.int32)
    B = len(cq) - 1 if B is None else B
    pq = None if null_cq else cq.ctypes.data
    return fav.lib().fav_prefill_varlen(q, k, v, o, lse, pq, ck.ctypes.data, B, Hq, Hkv, D,
                                        scale, causal, dtype, None)


INVALID = [
    dict(q=None), dict(k=None), dict(v=None), dict(o=None), dict(null_cq=True),
    dict(q=Q + 8), dict(k=K + 2), dict(o=O + 4), dict(lse=LSE + 1),
    dict(B=0), dict(causal=2), dict(Hq=6, Hkv=4), dict(scale=0.0),
    dict(cq=(1, 5, 9)), dict(ck=(2, 5, 9)),                  # not starting at 0
    dict(cq=(0, 5, 4)), dict(ck=(0, 9, 5)),                  # decreasing
    dict(cq=(0, 5, 9), ck=(0, 5, 5)),                        # queries without keys
    dict(cq=(0, 5, 9), ck=(0, 5, 8), causal=1),              # causal: more queries than keys
]


@pytest.mark.parametrize("kw", INVALID)
def test_rejects_invalid_arguments(kw):
    assert call(**kw) == 1


@pytest.mark.parametrize("kw", [dict(D=96), dict(D=256), dict(dtype=fav.F32)])
def test_rejects_unsupported(kw):
    assert call(**kw) == 2


def test_empty_batch_is_a_no_op():
    assert call(cq=(0, 0, 0), ck=(0, 3, 7)) == 0
