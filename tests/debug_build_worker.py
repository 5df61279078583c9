"""Runs small prefill, decode, paged-decode and packed-batch calls through whichever library
FAV_LIBRARY names (the self-checking -DFAV_DEBUG_CHECKS build, for test_debug_build_gpu.py) and
checks each against the fp64 oracle.  Prints one line per case and exits non-zero on the first
failure.  A helper run as a child process, not a test module of its own."""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import paper_2608_18656_gb300 as fav  # noqa: E402
from paper_2608_18656_gb300 import inputs as I  # noqa: E402
import gpu_util  # noqa: E402
import test_paged_gpu as P  # noqa: E402
import test_varlen_gpu as V  # noqa: E402


def dense(name, dtype, B, Hq, Hkv, Nq, Nkv, D, causal, grid=0, splits=0):
    fav.set_prefill_grid(grid)
    fav.set_decode_splits(splits)
    w = I.Workload(name, dtype, B, Hq, Hkv, Nq, Nkv, D, causal, False, B + Hq + Nq + grid)
    x = I.make_inputs(w)
    o, lse = gpu_util.run_gpu(w, x)          # asserts a zero device status (no check fired)
    gpu_util.check(w, o, lse, x)
    return fav.PATH_NAMES[fav.last_path()]


def main():
    assert os.path.abspath(fav.library_path()) == os.path.abspath(os.environ["FAV_LIBRARY"])
    cases = [
        ("prefill d128 f16 causal", lambda: dense("p128", I.F16, 2, 8, 2, 300, 300, 128, True)),
        ("prefill d128 f16 causal, 3 blocks", lambda: dense("p128g", I.F16, 2, 8, 2, 300, 300, 128, True, grid=3)),
        ("prefill d128 bf16 ragged, 2 units per block", lambda: dense("p128r", I.BF16, 16, 8, 2, 200, 200, 128, True)),
        ("prefill d64 bf16 causal", lambda: dense("p64", I.BF16, 2, 8, 2, 300, 300, 64, True)),
        ("prefill d64 bf16 non-causal, 3 blocks", lambda: dense("p64g", I.BF16, 2, 6, 3, 257, 257, 64, False, grid=3)),
        ("decode f16 split 4", lambda: dense("d", I.F16, 2, 16, 2, 1, 5000, 128, False, splits=4)),
        ("decode bf16 d64 small Nq causal", lambda: dense("dn", I.BF16, 2, 8, 2, 4, 700, 64, True)),
    ]
    for name, fn in cases:
        path = fn()
        print("ok  %-45s path=%s" % (name, path), flush=True)
    fav.set_prefill_grid(0)
    fav.set_decode_splits(0)
    # paged decode: 16-row pages in random order
    scale = float(np.float32(1.0 / np.sqrt(128)))
    x = P.build(I.BF16, [700, 33, 1500], 8, 2, 1, 128, 16, seed=5)
    o, lse = P.run_paged(x, I.BF16, False, scale)
    P.check_against_oracle(x, o, lse, I.BF16, 1, False, scale)
    print("ok  %-45s" % "paged decode bf16, 16-row pages", flush=True)
    # packed batch, D = 128 and 64
    for D in (128, 64):
        lens = [200, 130, 1, 256]
        q, k, v, cq, ck = V.packed(I.F16, lens, lens, 8, 2, D, seed=D)
        sc = float(np.float32(1.0 / np.sqrt(D)))
        o, lse = V.run(I.F16, q, k, v, cq, ck, True, sc)
        V.check(q, k, v, cq, ck, o, lse, I.F16, True, sc)
        print("ok  %-45s" % ("packed batch d%d" % D), flush=True)
    print("all cases passed")


if __name__ == "__main__":
    main()
