"""The C-ABI library: it loads, exports every declared entry point, and rejects invalid
arguments before touching any pointer or launching anything (runs without a GPU)."""
import ctypes
import os
import re

import pytest

import paper_2608_18656_gb300 as fav

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in sorted(os.listdir(os.path.join(ROOT, "include")))
           if f.endswith(".h")]


def declared_symbols():
    names = []
    for h in HEADERS:
        names += re.findall(r"FAV_API\s+[\w\s\*]+?\b(\w+)\s*\(", open(h).read())
    return names


def test_header_declares_entry_points():
    names = declared_symbols()
    for n in ("fav_forward", "fav_forward_host", "fav_status_string",
              "fav_get_last_device_status", "fav_release_workspace"):
        assert n in names


def test_library_exports_every_declared_symbol():
    L = ctypes.CDLL(fav.library_path())
    for n in declared_symbols():
        assert hasattr(L, n), n


def test_status_strings():
    L = fav.lib()
    for code in range(8):
        assert L.fav_status_string(code)
    assert L.fav_status_string(99) == b"unknown status"


# Aligned, non-null fake device addresses: validation must reject the call before using them.
Q, K, V, O, LSE = 1 << 20, 2 << 20, 3 << 20, 4 << 20, 5 << 20
GOOD = dict(B=1, Hq=4, Hkv=2, Nq=8, Nkv=8, D=64, scale=0.125, causal=0, dtype=fav.F16)


def call(fn="fav_forward", q=Q, k=K, v=V, o=O, lse=LSE, **kw):
    a = dict(GOOD)
    a.update(kw)
    return getattr(fav.lib(), fn)(q, k, v, o, lse, a["B"], a["Hq"], a["Hkv"], a["Nq"], a["Nkv"],
                                  a["D"], a["scale"], a["causal"], a["dtype"], None)


INVALID = [
    dict(q=None), dict(k=None), dict(v=None), dict(o=None),
    dict(q=Q + 8), dict(k=K + 2), dict(v=V + 4), dict(o=O + 1), dict(lse=LSE + 2),
    dict(B=0), dict(Hq=0), dict(Hkv=0), dict(Nq=0), dict(Nkv=0), dict(D=0),
    dict(B=-1), dict(Nkv=-5), dict(D=-64),
    dict(Hq=6, Hkv=4),
    dict(causal=1, Nq=9, Nkv=8),
    dict(causal=2),
    dict(scale=0.0), dict(scale=-0.125), dict(scale=float("nan")), dict(scale=float("inf")),
    dict(dtype=3), dict(dtype=-1),
]


@pytest.mark.parametrize("kw", INVALID, ids=lambda kw: ",".join("%s=%s" % i for i in kw.items()))
def test_invalid_arguments_rejected(kw):
    assert call(**kw) == 1


@pytest.mark.parametrize("kw", [dict(D=4, dtype=fav.F16), dict(D=2, dtype=fav.F32),
                                dict(D=12, dtype=fav.BF16)])
def test_unaligned_rows_unsupported(kw):
    assert call(**kw) == 2


@pytest.mark.parametrize("kw", [dict(q=None), dict(Hq=3, Hkv=2), dict(scale=-1.0),
                                dict(causal=1, Nq=4, Nkv=3)])
def test_host_entry_rejects_invalid_arguments(kw):
    assert call("fav_forward_host", **kw) == 1


def test_option_setters_validate():
    L = fav.lib()
    assert L.fav_set_path(7) == 1
    assert L.fav_set_path(-1) == 1
    assert L.fav_set_decode_splits(-1) == 1
    assert L.fav_set_decode_splits(5000) == 1
    assert L.fav_set_prefill_grid(-1) == 1
    assert L.fav_set_path(fav.PATH_AUTO) == 0
    assert L.fav_set_decode_splits(0) == 0
    assert L.fav_set_prefill_grid(0) == 0


def test_python_binding_has_no_cpu_path():
    torch = pytest.importorskip("torch")
    q = torch.zeros(1, 1, 4, 64, dtype=torch.float16)
    with pytest.raises(ValueError):
        fav.forward(q, q, q)


@pytest.mark.parametrize("limit_us", [0, -1, 1000001])
def test_wait_self_test_rejects_limits(limit_us):
    assert fav.lib().fav_check_wait_timeout(limit_us, None) == 1   # FAV_ERR_INVALID_ARG
