"""fp64 CPU oracle for exact attention.  TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline / reference leg
may import this package.  The product path (``paper_2608_18656_gb300``) never does, and this
package imports nothing from it.

* ``attention`` / ``attention_rows`` / ``attention_probs`` call the plain C two-pass fp64
  implementation in ``fav_oracle.c`` (the definition of softmax attention from the paper's
  Background section, see that file's header for the readings it takes).
* ``naive_flash`` is the independent pure-Python recurrence of the paper's Algorithm
  "ggml-vec FlashAttention in llama.cpp" (tiny inputs only).

Inputs are numpy arrays of any float dtype; they are upcast exactly to fp64 here.
"""
import ctypes
import os
import subprocess

import numpy as np

from .naive_flash import naive_flash, naive_flash_row  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fav_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lib = None


def build(force=False):
    """Compile fav_oracle.c with gcc into oracle/_build/liboracle.so."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
           "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.check_call(cmd)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        i64 = ctypes.c_int64
        dp = ctypes.c_void_p
        lib.fav_oracle_forward.argtypes = [dp, dp, dp, dp, dp, i64, i64, i64, i64, i64, i64,
                                           ctypes.c_double, ctypes.c_int, ctypes.c_int]
        lib.fav_oracle_forward.restype = ctypes.c_int
        lib.fav_oracle_rows.argtypes = [dp, dp, dp, dp, i64, dp, dp, i64, i64, i64, i64, i64, i64,
                                        ctypes.c_double, ctypes.c_int, ctypes.c_int]
        lib.fav_oracle_rows.restype = ctypes.c_int
        lib.fav_oracle_probs.argtypes = [dp, dp, dp, dp, dp, dp, i64, i64, i64, i64, i64, i64,
                                         ctypes.c_double, ctypes.c_int]
        lib.fav_oracle_probs.restype = ctypes.c_int
        _lib = lib
    return _lib


def default_threads():
    return max(1, len(os.sched_getaffinity(0)))


def _prep(q, k, v):
    q = np.ascontiguousarray(q, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    if q.ndim != 4 or k.ndim != 4 or v.ndim != 4 or k.shape != v.shape:
        raise ValueError("q [B,Hq,Nq,D], k/v [B,Hkv,Nkv,D] expected")
    if q.shape[0] != k.shape[0] or q.shape[3] != k.shape[3]:
        raise ValueError("batch or head dimension mismatch")
    return q, k, v


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def attention(q, k, v, scale, causal=False, nthreads=None):
    """Full attention in fp64: returns (o [B,Hq,Nq,D], lse [B,Hq,Nq])."""
    q, k, v = _prep(q, k, v)
    B, Hq, Nq, D = q.shape
    Hkv, Nkv = k.shape[1], k.shape[2]
    o = np.empty((B, Hq, Nq, D), np.float64)
    lse = np.empty((B, Hq, Nq), np.float64)
    rc = _load().fav_oracle_forward(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse),
                                    B, Hq, Hkv, Nq, Nkv, D, float(scale), int(bool(causal)),
                                    nthreads or default_threads())
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    return o, lse


def attention_rows(q, k, v, rows, scale, causal=False, nthreads=None):
    """Selected query rows (flat indices into [B,Hq,Nq]): returns (o [n,D], lse [n])."""
    q, k, v = _prep(q, k, v)
    B, Hq, Nq, D = q.shape
    Hkv, Nkv = k.shape[1], k.shape[2]
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    o = np.empty((rows.size, D), np.float64)
    lse = np.empty((rows.size,), np.float64)
    rc = _load().fav_oracle_rows(_ptr(q), _ptr(k), _ptr(v), _ptr(rows), rows.size, _ptr(o),
                                 _ptr(lse), B, Hq, Hkv, Nq, Nkv, D, float(scale),
                                 int(bool(causal)), nthreads or default_threads())
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    return o, lse


def attention_probs(q, k, v, scale, causal=False):
    """Tiny cases: returns (o, lse, p [B,Hq,Nq,Nkv]) with p the softmax weights."""
    q, k, v = _prep(q, k, v)
    B, Hq, Nq, D = q.shape
    Hkv, Nkv = k.shape[1], k.shape[2]
    o = np.empty((B, Hq, Nq, D), np.float64)
    lse = np.empty((B, Hq, Nq), np.float64)
    p = np.empty((B, Hq, Nq, Nkv), np.float64)
    rc = _load().fav_oracle_probs(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(p),
                                  B, Hq, Hkv, Nq, Nkv, D, float(scale), int(bool(causal)))
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    return o, lse, p
