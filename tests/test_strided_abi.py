"""fav_forward_strided argument rules, checked on the CPU (validation happens before any
CUDA call, so no GPU is needed)."""
import ctypes

import pytest

import paper_2608_18656_gb300 as fav

ADDR = 1 << 20                      # any 16-byte aligned address: nothing is dereferenced


def call(qs, ks, vs, os_, B=1, Hq=2, Hkv=2, Nq=8, Nkv=8, D=64, dtype=fav.F16, lse=None):
    S = fav.Strides
    return fav.lib().fav_forward_strided(ADDR, ADDR, ADDR, ADDR, lse, S(*qs), S(*ks), S(*vs),
                                         S(*os_), B, Hq, Hkv, Nq, Nkv, D, ctypes.c_float(0.125),
                                         0, dtype, None)


C = (2 * 8 * 64, 8 * 64, 64)        # contiguous strides of [1, 2, 8, 64]


@pytest.mark.parametrize("bad", [(-1, 512, 64), (1024, -512, 64), (1024, 512, -64)])
def test_negative_stride_is_invalid(bad):
    assert call(bad, C, C, C) == 1
    assert call(C, C, C, bad) == 1


@pytest.mark.parametrize("bad", [(1024, 512, 65), (1024, 516, 64), (1028, 512, 64)])
def test_stride_not_16_byte_multiple_is_unsupported(bad):
    # 2-byte elements: every stride must be a multiple of 8 elements
    assert call(C, bad, C, C) == 2


def test_fp32_strides_need_multiples_of_four():
    c32 = (2 * 8 * 64, 8 * 64, 64)
    assert call(c32, c32, c32, (1024, 512, 66), dtype=fav.F32) == 2
    assert call(c32, c32, c32, (1024, 512, 68), dtype=fav.F32) != 2


def test_zero_stride_only_on_size_one_axes():
    assert call(C, C, C, (1024, 0, 64)) == 1                 # output heads would coincide
    assert call(C, (1024, 0, 64), C, C) == 2                 # broadcast K heads: unsupported
    assert call(C, C, (0, 512, 64), C, B=2) == 2             # broadcast V batches
    # size-1 axes may carry a zero stride: validation passes (the call then needs a GPU)
    st = call((0, 512, 64), (0, 512, 64), (0, 512, 64), (0, 512, 64), B=1)
    assert st not in (1, 2)


def test_shape_rules_as_fav_forward():
    assert call(C, C, C, C, Hq=3, Hkv=2) == 1                # Hq % Hkv
    assert call(C, C, C, C, Nq=0) == 1
