"""fav_forward_nonflash: argument validation before anything is launched, and the workspace
size (runs without a GPU; the pointers are aligned fake device addresses)."""
import pytest

import paper_2608_18656_gb300 as fav

Q, K, V, O, LSE, WS = (1 << 20, 2 << 20, 3 << 20, 4 << 20, 5 << 20, 6 << 20)
GOOD = dict(B=2, Hq=8, Hkv=2, Nq=256, Nkv=256, D=128, scale=0.088, causal=1, dtype=fav.F16)
BIG = 1 << 40


def call(q=Q, k=K, v=V, o=O, lse=LSE, ws=WS, ws_bytes=BIG, **kw):
    a = dict(GOOD)
    a.update(kw)
    return fav.lib().fav_forward_nonflash(q, k, v, o, lse, a["B"], a["Hq"], a["Hkv"], a["Nq"],
                                          a["Nkv"], a["D"], a["scale"], a["causal"], a["dtype"],
                                          ws, ws_bytes, None)


def test_workspace_size():
    # fp32 scores of every query row of every head
    assert fav.nonflash_workspace_size(2, 8, 256, 300) == 2 * 8 * 256 * 300 * 4
    assert fav.nonflash_workspace_size(1, 32, 2048, 2048) == 32 * 2048 * 2048 * 4
    assert fav.nonflash_workspace_size(0, 8, 256, 256) == 0


INVALID = [
    dict(q=None), dict(k=None), dict(v=None), dict(o=None), dict(ws=None),
    dict(q=Q + 8), dict(k=K + 2), dict(o=O + 4), dict(lse=LSE + 1), dict(ws=WS + 8),
    dict(B=0), dict(Hq=0), dict(Nq=0), dict(Nkv=0), dict(D=0),
    dict(Hq=6, Hkv=4), dict(scale=0.0), dict(scale=float("nan")), dict(causal=2),
    dict(Nq=300, Nkv=200),                           # causal needs Nq <= Nkv
    dict(ws_bytes=2 * 8 * 256 * 256 * 4 - 1),        # one byte short
]


@pytest.mark.parametrize("kw", INVALID)
def test_rejects_invalid_arguments(kw):
    assert call(**kw) == 1


UNSUPPORTED = [
    dict(dtype=fav.F32), dict(D=4),
    dict(Nkv=40000, Nq=1),                           # a score row above 32768 keys
    dict(Hq=64, Hkv=1, Nq=32768, Nkv=32768, causal=0),   # GEMM rows x keys >= 2^31
]


@pytest.mark.parametrize("kw", UNSUPPORTED)
def test_rejects_unsupported_shapes(kw):
    assert call(**kw) == 2
