"""fav_decode_paged: argument validation before any pointer is touched or anything launched
(runs without a GPU; the pointers are aligned fake device addresses)."""
import pytest

import paper_2608_18656_gb300 as fav

Q, KC, VC, O, LSE, BT, SL = (1 << 20, 2 << 20, 3 << 20, 4 << 20, 5 << 20, 6 << 20, 7 << 20)
GOOD = dict(B=2, Hq=8, Hkv=2, Nq=1, max_pages=4, page_size=16, num_pages=8, D=128,
            scale=0.088, causal=0, dtype=fav.F16)


def call(q=Q, kc=KC, vc=VC, o=O, lse=LSE, bt=BT, sl=SL, **kw):
    a = dict(GOOD)
    a.update(kw)
    return fav.lib().fav_decode_paged(q, kc, vc, o, lse, bt, sl, a["B"], a["Hq"], a["Hkv"],
                                      a["Nq"], a["max_pages"], a["page_size"], a["num_pages"],
                                      a["D"], a["scale"], a["causal"], a["dtype"], None)


INVALID = [
    dict(q=None), dict(kc=None), dict(vc=None), dict(o=None), dict(bt=None), dict(sl=None),
    dict(q=Q + 8), dict(kc=KC + 2), dict(vc=VC + 4), dict(o=O + 1), dict(lse=LSE + 2),
    dict(bt=BT + 2), dict(sl=SL + 1),
    dict(B=0), dict(Hq=0), dict(Hkv=0), dict(Nq=0), dict(D=0),
    dict(max_pages=0), dict(num_pages=0), dict(page_size=0), dict(page_size=-16),
    dict(Hq=6, Hkv=4), dict(scale=0.0), dict(scale=float("inf")), dict(causal=2),
]


@pytest.mark.parametrize("kw", INVALID)
def test_rejects_invalid_arguments(kw):
    assert call(**kw) == 1


UNSUPPORTED = [
    dict(page_size=8), dict(page_size=24), dict(page_size=48), dict(page_size=1 << 17),
    dict(D=96), dict(D=256), dict(dtype=fav.F32),
    dict(Nq=17, Hq=8, Hkv=2),                       # 68 query rows per KV head > 64
    dict(max_pages=1 << 20, page_size=1 << 12),     # longer than the kernel's int range
]


@pytest.mark.parametrize("kw", UNSUPPORTED)
def test_rejects_unsupported_shapes(kw):
    assert call(**kw) == 2
