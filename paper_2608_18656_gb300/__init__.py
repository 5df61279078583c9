"""libfav Python binding: argument marshalling onto the C ABI declared in include/fav.h.

Every step of the attention forward runs in the CUDA kernels of ``libfav.so``; this module
only turns torch CUDA tensors into pointers, sizes and the current stream.  There is no
CPU fallback: without the built library every call raises.
"""
import ctypes
import os

__all__ = ["forward", "forward_nonflash", "nonflash_workspace_size", "forward_host", "decode_paged", "prefill_varlen", "Strides", "set_path", "last_path", "set_decode_splits",
           "last_decode_splits", "set_prefill_grid", "device_status", "check_wait_timeout", "release_workspace", "library_path",
           "FavError", "F32", "F16", "BF16", "PATH_AUTO", "PATH_SIMT", "PATH_DECODE",
           "PATH_PREFILL"]

F32, F16, BF16 = 0, 1, 2
PATH_AUTO, PATH_SIMT, PATH_DECODE, PATH_PREFILL = 0, 1, 2, 3
PATH_NAMES = {PATH_AUTO: "auto", PATH_SIMT: "simt", PATH_DECODE: "decode",
              PATH_PREFILL: "prefill"}
STATUS_NAMES = {0: "FAV_OK", 1: "FAV_ERR_INVALID_ARG", 2: "FAV_ERR_UNSUPPORTED",
                3: "FAV_ERR_CUDA", 4: "FAV_ERR_NO_MEMORY", 5: "FAV_ERR_DEVICE_TIMEOUT",
                6: "FAV_ERR_DEVICE_CHECK", 7: "FAV_ERR_BAD_PAGE"}

_HERE = os.path.dirname(os.path.abspath(__file__))
# FAV_LIBRARY in the environment selects another build of the library (the self-checking
# -DFAV_DEBUG_CHECKS variant, libfav_debug.so); by default the in-tree libfav.so.
_LIB_PATH = os.environ.get("FAV_LIBRARY") or os.path.join(_HERE, "libfav.so")
_lib = None


class Strides(ctypes.Structure):
    """fav_strides: element strides (batch, head, token) of a [B, H, N, D] tensor."""
    _fields_ = [("batch", ctypes.c_longlong), ("head", ctypes.c_longlong),
                ("token", ctypes.c_longlong)]


class FavError(RuntimeError):
    def __init__(self, status, msg=""):
        self.status = status
        super().__init__("%s%s" % (STATUS_NAMES.get(status, status), (": " + msg) if msg else ""))


def library_path():
    return _LIB_PATH


def lib():
    """The loaded libfav.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError("libfav.so is not built; run __graft_entry__.build() "
                               "(or python paper_2608_18656_gb300/build.py)")
        L = ctypes.CDLL(_LIB_PATH)
        vp, i = ctypes.c_void_p, ctypes.c_int
        sig = [vp, vp, vp, vp, vp, i, i, i, i, i, i, ctypes.c_float, i, i, vp]
        for fn in ("fav_forward", "fav_forward_host"):
            getattr(L, fn).argtypes = sig
            getattr(L, fn).restype = i
        S = Strides
        L.fav_forward_strided.argtypes = [vp, vp, vp, vp, vp, S, S, S, S, i, i, i, i, i, i,
                                          ctypes.c_float, i, i, vp]
        L.fav_forward_strided.restype = i
        L.fav_decode_paged.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, i, i, i,
                                       ctypes.c_float, i, i, vp]
        L.fav_decode_paged.restype = i
        L.fav_prefill_varlen.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, ctypes.c_float,
                                         i, i, vp]
        L.fav_prefill_varlen.restype = i
        L.fav_nonflash_workspace_size.argtypes = [i, i, i, i]
        L.fav_nonflash_workspace_size.restype = ctypes.c_size_t
        L.fav_forward_nonflash.argtypes = [vp, vp, vp, vp, vp, i, i, i, i, i, i, ctypes.c_float,
                                           i, i, vp, ctypes.c_size_t, vp]
        L.fav_forward_nonflash.restype = i
        L.fav_status_string.argtypes = [i]
        L.fav_status_string.restype = ctypes.c_char_p
        L.fav_get_last_device_status.argtypes = []
        L.fav_get_last_device_status.restype = i
        L.fav_release_workspace.argtypes = []
        L.fav_release_workspace.restype = None
        L.fav_set_path.argtypes = [i]
        L.fav_set_path.restype = i
        L.fav_last_path.argtypes = []
        L.fav_last_path.restype = i
        L.fav_set_decode_splits.argtypes = [i]
        L.fav_set_decode_splits.restype = i
        L.fav_last_decode_splits.argtypes = []
        L.fav_last_decode_splits.restype = i
        L.fav_set_prefill_grid.argtypes = [i]
        L.fav_set_prefill_grid.restype = i
        L.fav_check_wait_timeout.argtypes = [i, vp]
        L.fav_check_wait_timeout.restype = i
        _lib = L
    return _lib


def _check(st):
    if st != 0:
        raise FavError(st, lib().fav_status_string(st).decode())


def _dtype_code(t):
    import torch
    codes = {torch.float32: F32, torch.float16: F16, torch.bfloat16: BF16}
    if t.dtype not in codes:
        raise TypeError("unsupported dtype %s" % t.dtype)
    return codes[t.dtype]


def forward(q, k, v, causal=False, scale=None, return_lse=True, out=None, lse_out=None,
            stream=None):
    """Attention forward on torch CUDA tensors q [B,Hq,Nq,D], k/v [B,Hkv,Nkv,D].

    The tensors may be any strided views whose last axis is contiguous (for example
    ``x.transpose(1, 2)`` of a [B, N, H, D] tensor): those go through fav_forward_strided.
    Returns (o, lse) with lse [B,Hq,Nq] fp32 (None if return_lse is False); o is allocated
    contiguous unless ``out`` is given.  Runs on the current torch stream unless ``stream``
    (a torch.cuda.Stream) is given.
    """
    import torch
    for t in (q, k, v):
        if not t.is_cuda:
            raise ValueError("tensors must live on a CUDA device")
        if t.dim() != 4 or t.stride(-1) != 1:
            raise ValueError("tensors must be 4-D with a contiguous last axis")
    if k.dtype != q.dtype or v.dtype != q.dtype:
        raise TypeError("q, k and v must share a dtype")
    B, Hq, Nq, D = q.shape
    Bk, Hkv, Nkv, Dk = k.shape
    if tuple(v.shape) != tuple(k.shape) or Bk != B or Dk != D:
        raise ValueError("shape mismatch between q, k and v")
    if scale is None:
        import numpy as np
        scale = float(np.float32(1.0 / np.sqrt(D)))
    o = out if out is not None else torch.empty(q.shape, dtype=q.dtype, device=q.device)
    if o.dim() != 4 or o.stride(-1) != 1:
        raise ValueError("out must be 4-D with a contiguous last axis")
    lse = None
    if return_lse:
        lse = lse_out if lse_out is not None else torch.empty((B, Hq, Nq), device=q.device,
                                                              dtype=torch.float32)
    s = stream if stream is not None else torch.cuda.current_stream(q.device)
    lse_ptr = lse.data_ptr() if lse is not None else None
    with torch.cuda.device(q.device):
        if all(t.is_contiguous() for t in (q, k, v, o)):
            st = lib().fav_forward(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                                   lse_ptr, B, Hq, Hkv, Nq, Nkv, D, float(scale),
                                   int(bool(causal)), _dtype_code(q), s.cuda_stream)
        else:
            sd = [Strides(t.stride(0), t.stride(1), t.stride(2)) for t in (q, k, v, o)]
            st = lib().fav_forward_strided(q.data_ptr(), k.data_ptr(), v.data_ptr(),
                                           o.data_ptr(), lse_ptr, *sd, B, Hq, Hkv, Nq, Nkv, D,
                                           float(scale), int(bool(causal)), _dtype_code(q),
                                           s.cuda_stream)
    _check(st)
    return o, lse


def nonflash_workspace_size(B, Hq, Nq, Nkv):
    """Bytes of device workspace fav_forward_nonflash needs (fp32 scores of every head)."""
    return lib().fav_nonflash_workspace_size(B, Hq, Nq, Nkv)


def forward_nonflash(q, k, v, causal=False, scale=None, out=None, lse_out=None, workspace=None,
                     stream=None):
    """The non-fused attention (fav_forward_nonflash): S = scale Q K^T materialised in a
    workspace, masked row softmax, O = P V.  Contiguous fp16/bf16 tensors q [B,Hq,Nq,D],
    k/v [B,Hkv,Nkv,D].  ``workspace`` is a CUDA uint8 tensor of at least
    nonflash_workspace_size(...) bytes (allocated per call if None).  Returns (o, lse)."""
    import torch
    for t in (q, k, v):
        if not t.is_cuda or t.dim() != 4 or not t.is_contiguous():
            raise ValueError("tensors must be contiguous 4-D CUDA tensors")
    if k.dtype != q.dtype or v.dtype != q.dtype:
        raise TypeError("q, k and v must share a dtype")
    B, Hq, Nq, D = q.shape
    Bk, Hkv, Nkv, Dk = k.shape
    if tuple(v.shape) != tuple(k.shape) or Bk != B or Dk != D:
        raise ValueError("shape mismatch between q, k and v")
    if scale is None:
        import numpy as np
        scale = float(np.float32(1.0 / np.sqrt(D)))
    o = out if out is not None else torch.empty(q.shape, dtype=q.dtype, device=q.device)
    lse = lse_out if lse_out is not None else torch.empty((B, Hq, Nq), device=q.device,
                                                          dtype=torch.float32)
    if not o.is_contiguous() or not lse.is_contiguous():
        raise ValueError("out and lse_out must be contiguous")
    need = nonflash_workspace_size(B, Hq, Nq, Nkv)
    ws = workspace if workspace is not None else torch.empty(need, dtype=torch.uint8,
                                                             device=q.device)
    s = stream if stream is not None else torch.cuda.current_stream(q.device)
    with torch.cuda.device(q.device):
        st = lib().fav_forward_nonflash(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                                        lse.data_ptr(), B, Hq, Hkv, Nq, Nkv, D, float(scale),
                                        int(bool(causal)), _dtype_code(q), ws.data_ptr(),
                                        ws.numel() * ws.element_size(), s.cuda_stream)
    _check(st)
    return o, lse


def decode_paged(q, k_cache, v_cache, block_table, seq_lens, causal=False, scale=None,
                 return_lse=True, out=None, lse_out=None, stream=None):
    """Decode attention over a paged cache (fav_decode_paged).

    q [B,Hq,Nq,D] contiguous; k_cache / v_cache [num_pages, page_size, Hkv, D] contiguous;
    block_table int32 [B, max_pages] and seq_lens int32 [B], all torch CUDA tensors on one
    device.  Returns (o, lse) like forward().
    """
    import torch
    for t in (q, k_cache, v_cache, block_table, seq_lens):
        if not t.is_cuda:
            raise ValueError("tensors must live on a CUDA device")
        if not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
    if k_cache.dtype != q.dtype or v_cache.dtype != q.dtype:
        raise TypeError("q and the caches must share a dtype")
    if block_table.dtype != torch.int32 or seq_lens.dtype != torch.int32:
        raise TypeError("block_table and seq_lens must be int32")
    B, Hq, Nq, D = q.shape
    num_pages, page_size, Hkv, Dk = k_cache.shape
    if tuple(v_cache.shape) != tuple(k_cache.shape) or Dk != D:
        raise ValueError("shape mismatch between q and the caches")
    if block_table.dim() != 2 or block_table.shape[0] != B or tuple(seq_lens.shape) != (B,):
        raise ValueError("block_table must be [B, max_pages] and seq_lens [B]")
    max_pages = block_table.shape[1]
    if scale is None:
        import numpy as np
        scale = float(np.float32(1.0 / np.sqrt(D)))
    o = out if out is not None else torch.empty(q.shape, dtype=q.dtype, device=q.device)
    lse = None
    if return_lse:
        lse = lse_out if lse_out is not None else torch.empty((B, Hq, Nq), device=q.device,
                                                              dtype=torch.float32)
    s = stream if stream is not None else torch.cuda.current_stream(q.device)
    with torch.cuda.device(q.device):
        st = lib().fav_decode_paged(q.data_ptr(), k_cache.data_ptr(), v_cache.data_ptr(),
                                    o.data_ptr(), lse.data_ptr() if lse is not None else None,
                                    block_table.data_ptr(), seq_lens.data_ptr(), B, Hq, Hkv, Nq,
                                    max_pages, page_size, num_pages, D, float(scale),
                                    int(bool(causal)), _dtype_code(q), s.cuda_stream)
    _check(st)
    return o, lse


def prefill_varlen(q, k, v, cu_seqlens_q, cu_seqlens_k, causal=False, scale=None,
                   return_lse=True, out=None, lse_out=None, stream=None):
    """Prefill over a packed batch of variable-length sequences (fav_prefill_varlen).

    q [total_q, Hq, D], k / v [total_k, Hkv, D]: contiguous torch CUDA tensors; cu_seqlens_q /
    cu_seqlens_k: length-B+1 host sequences of ints (lists, numpy arrays or CPU tensors).
    Returns (o [total_q, Hq, D], lse [Hq, total_q] fp32 or None).
    """
    import numpy as np
    import torch
    for t in (q, k, v):
        if not t.is_cuda or not t.is_contiguous() or t.dim() != 3:
            raise ValueError("q, k, v must be contiguous 3-D CUDA tensors")
    if k.dtype != q.dtype or v.dtype != q.dtype:
        raise TypeError("q, k and v must share a dtype")
    cq = np.ascontiguousarray(np.asarray(cu_seqlens_q, dtype=np.int32))
    ck = np.ascontiguousarray(np.asarray(cu_seqlens_k, dtype=np.int32))
    if cq.ndim != 1 or cq.shape != ck.shape or cq.size < 2:
        raise ValueError("cu_seqlens_q and cu_seqlens_k must both have B + 1 entries")
    B = cq.size - 1
    total_q, Hq, D = q.shape
    total_k, Hkv, Dk = k.shape
    if tuple(v.shape) != tuple(k.shape) or Dk != D or cq[-1] != total_q or ck[-1] != total_k:
        raise ValueError("shape mismatch between q, k, v and the sequence offsets")
    if scale is None:
        scale = float(np.float32(1.0 / np.sqrt(D)))
    o = out if out is not None else torch.empty(q.shape, dtype=q.dtype, device=q.device)
    lse = None
    if return_lse:
        lse = lse_out if lse_out is not None else torch.empty((Hq, total_q), device=q.device,
                                                              dtype=torch.float32)
    s = stream if stream is not None else torch.cuda.current_stream(q.device)
    with torch.cuda.device(q.device):
        st = lib().fav_prefill_varlen(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                                      lse.data_ptr() if lse is not None else None,
                                      cq.ctypes.data, ck.ctypes.data, B, Hq, Hkv, D, float(scale),
                                      int(bool(causal)), _dtype_code(q), s.cuda_stream)
    _check(st)
    return o, lse


def forward_host(q, k, v, o, lse, B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype, stream=0):
    """End-to-end call on host buffers (numpy arrays or raw addresses); synchronises."""
    def addr(a):
        if a is None:
            return None
        if isinstance(a, int):
            return a
        if hasattr(a, "ctypes"):
            return a.ctypes.data
        return a.data_ptr()
    st = lib().fav_forward_host(addr(q), addr(k), addr(v), addr(o), addr(lse), B, Hq, Hkv, Nq,
                                Nkv, D, float(scale), int(bool(causal)), int(dtype), stream)
    _check(st)


def set_path(path):
    _check(lib().fav_set_path(int(path)))


def last_path():
    return lib().fav_last_path()


def set_decode_splits(n):
    _check(lib().fav_set_decode_splits(int(n)))


def last_decode_splits():
    return lib().fav_last_decode_splits()


def set_prefill_grid(n):
    """Cap on the persistent prefill kernel's thread blocks (0 = one per SM)."""
    _check(lib().fav_set_prefill_grid(int(n)))


def device_status():
    """Synchronises; returns and clears the kernels' bounded-wait status (0 = ok)."""
    return lib().fav_get_last_device_status()


def check_wait_timeout(limit_us=1000, stream=None):
    """Launches the bounded-wait self-test (fav_check_wait_timeout) on the current torch stream
    (or `stream`): one warp waits on an mbarrier that nothing arrives on and gives up after
    limit_us; the outcome is read with device_status()."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    _check(lib().fav_check_wait_timeout(int(limit_us), s.cuda_stream))


def release_workspace():
    lib().fav_release_workspace()
