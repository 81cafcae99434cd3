"""Python binding of libchronostitch, the C ABI in include/chronostitch.h.

ChronoStitch (arxiv 2607.19547) composes independently prefilled video-chunk
KV caches at query time.  The four calls of its hot path, each one CUDA
kernel launch in the library:

  cs_rebase_keys       Eq. 3  re-base stored post-rotary keys onto global 3-axis mRoPE coords
  cs_score_deviation   Eq. 5  squared deviation of fresh vs re-based layer-1 keys
  cs_select_topk       Sec. 2 top-rho later-chunk tokens, lower index wins ties
  cs_repair_attention  Eq. 1  causal GQA attention of the selected rows over the cache
plus cs_rebase_and_score (steps 1 and 2 in one launch where possible) and the
scatter-back of the repaired rows' fresh keys and values:
  cs_scatter_rows      Sec. 2 cache[l, idx[r]] = rows[l, r]

This module only marshals torch tensors (device memory and streams) into the
C calls and raises CsError on a non-OK status.  There is no CPU path: if the
library is not built, every call raises.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libchronostitch.so")

CS_OK, CS_ERR_INVALID_ARG, CS_ERR_UNSUPPORTED, CS_ERR_CUDA, CS_ERR_TIMEOUT, CS_ERR_DEVICE_ARG = range(6)
CS_DTYPE_F32, CS_DTYPE_BF16 = 0, 1


class CsError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        self.status = status
        super().__init__(f"{where}: status {status} ({cs_status_string(status)}): {detail}")


class _RopeCfg(ctypes.Structure):
    _fields_ = [("theta", ctypes.c_double), ("sections", ctypes.c_int32 * 3)]


_lib = None
_vp, _i32, _i64, _f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float

_SIGS = {
    "cs_abi_version": (ctypes.c_int, []),
    "cs_rebase_keys": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i64, _i32, _i32, _i32, _vp, _vp,
                                      ctypes.POINTER(_RopeCfg), _vp]),
    "cs_score_deviation": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _i32, _i64, _i64, _vp, _vp]),
    "cs_rebase_and_score": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i64, _i32, _i32, _i32, _vp, _vp,
                                           ctypes.POINTER(_RopeCfg), _i32, _i32, _i32, _vp, _i64,
                                           _vp, _vp]),
    "cs_select_topk": (ctypes.c_int, [_vp, _i32, _i32, ctypes.c_int32, _vp, _vp]),
    "cs_repair_attention": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _i32,
                                           _i32, _i32, _i64, _vp, _f32, _vp]),
    "cs_scatter_rows": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _i64, _i32, _i64, _i32, _vp,
                                       _vp]),
    "cs_sync_status": (ctypes.c_int, [_vp]),
    "cs_debug_wait_timeout": (ctypes.c_int, [ctypes.c_uint32, _vp]),
    "cs_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "cs_last_error_detail": (ctypes.c_char_p, []),
}


def lib():
    """The loaded libchronostitch (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        handle = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(handle, name)
            fn.restype = res
            fn.argtypes = args
        _lib = handle
    return _lib


def cs_status_string(status: int) -> str:
    return lib().cs_status_string(int(status)).decode()


def cs_last_error_detail() -> str:
    return lib().cs_last_error_detail().decode()


def cs_abi_version() -> int:
    return int(lib().cs_abi_version())


def _check(status: int, where: str):
    if status != CS_OK:
        raise CsError(status, where, cs_last_error_detail())


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _fresh(stream, make):
    """An output tensor allocated here for a call launched on `stream`.  torch's caching
    allocator tracks the current stream; when the call runs on another one, the tensor is
    recorded on it, so its memory is not handed out again before the kernel has written it."""
    t = make()
    if stream is not None:
        s = stream if isinstance(stream, torch.cuda.Stream) else torch.cuda.ExternalStream(int(stream))
        if s.cuda_stream != torch.cuda.current_stream(t.device).cuda_stream:
            t.record_stream(s)
    return t


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return CS_DTYPE_BF16
    if t.dtype == torch.float32:
        return CS_DTYPE_F32
    raise TypeError(f"unsupported dtype {t.dtype} (bf16 or fp32)")


def _need_cuda(*ts):
    """CUDA tensors, all on the current device (the library launches there)."""
    for t in ts:
        if not (isinstance(t, torch.Tensor) and t.is_cuda):
            raise ValueError("all tensors must be CUDA tensors")
    cur = torch.cuda.current_device()
    for t in ts:
        if t.device.index != cur:
            raise ValueError(f"tensor on {t.device}, but the current device is cuda:{cur}")


def _inner_contiguous(t: torch.Tensor, what: str):
    """Every dimension but the first must be densely packed (the first may be strided)."""
    expect = 1
    for d in range(t.dim() - 1, 0, -1):
        if t.size(d) > 1 and t.stride(d) != expect:
            raise ValueError(f"{what}: dimensions after the first must be contiguous")
        expect *= t.size(d)


def cs_rebase_keys(k: torch.Tensor, pos_local: torch.Tensor, pos_global: torch.Tensor, *,
                   k_out: torch.Tensor | None = None, theta: float = 1e6,
                   sections=(16, 24, 24), stream=None) -> torch.Tensor:
    """Eq. 3: re-base keys [L, T, Hkv, D] from pos_local to pos_global (int32 [T, 3]).

    In place unless k_out is given.  Returns the re-based tensor."""
    _need_cuda(k, pos_local, pos_global)
    if k.dim() != 4:
        raise ValueError("k must be [L, T, Hkv, D]")
    _inner_contiguous(k, "k")
    out = k if k_out is None else k_out
    if out is not k:
        _need_cuda(out)
        if out.shape != k.shape or out.dtype != k.dtype or out.stride() != k.stride():
            raise ValueError("k_out must match k in shape, dtype and strides")
    for p in (pos_local, pos_global):
        if p.dtype != torch.int32 or not p.is_contiguous() or p.shape != (k.shape[1], 3):
            raise ValueError("coordinates must be contiguous int32 [T, 3]")
    L, T, H, D = k.shape
    cfg = _RopeCfg(float(theta), (ctypes.c_int32 * 3)(*[int(s) for s in sections]))
    st = lib().cs_rebase_keys(k.data_ptr(), out.data_ptr(), _dtype_code(k), L, k.stride(0) if L > 1 else T * H * D,
                              T, H, D, pos_local.data_ptr(), pos_global.data_ptr(),
                              ctypes.byref(cfg), _stream(stream))
    _check(st, "cs_rebase_keys")
    return out


def cs_rebase_and_score(k: torch.Tensor, pos_local: torch.Tensor, pos_global: torch.Tensor,
                        k_fresh: torch.Tensor, score_layer: int, cand0: int, *,
                        score_out: torch.Tensor | None = None, k_out: torch.Tensor | None = None,
                        theta: float = 1e6, sections=(16, 24, 24), stream=None):
    """Eq. 3 then Eq. 5: re-base k [L, T, Hkv, D] (in place unless k_out) and score the
    n = k_fresh.shape[0] candidate tokens [cand0, cand0 + n) at layer score_layer against
    k_fresh [n, Hkv, D] (rows may be strided).  One launch where the library can fuse them.
    Returns (re-based keys, fp32 scores [n])."""
    _need_cuda(k, pos_local, pos_global, k_fresh)
    if k.dim() != 4:
        raise ValueError("k must be [L, T, Hkv, D]")
    _inner_contiguous(k, "k")
    out = k if k_out is None else k_out
    if out is not k:
        _need_cuda(out)
        if out.shape != k.shape or out.dtype != k.dtype or out.stride() != k.stride():
            raise ValueError("k_out must match k in shape, dtype and strides")
    for p in (pos_local, pos_global):
        if p.dtype != torch.int32 or not p.is_contiguous() or p.shape != (k.shape[1], 3):
            raise ValueError("coordinates must be contiguous int32 [T, 3]")
    L, T, H, D = k.shape
    if k_fresh.dim() != 3 or k_fresh.shape[1:] != (H, D) or k_fresh.dtype != k.dtype:
        raise ValueError("k_fresh must be [n, Hkv, D] of the keys' dtype")
    _inner_contiguous(k_fresh, "k_fresh")
    n = k_fresh.shape[0]
    if score_out is None:
        score_out = _fresh(stream, lambda: torch.empty(n, dtype=torch.float32, device=k.device))
    _need_cuda(score_out)
    if score_out.dtype != torch.float32 or score_out.numel() < n or not score_out.is_contiguous():
        raise ValueError("score_out must be contiguous fp32 with n elements")
    cfg = _RopeCfg(float(theta), (ctypes.c_int32 * 3)(*[int(s) for s in sections]))
    fs = k_fresh.stride(0) if n > 1 else H * D
    st = lib().cs_rebase_and_score(k.data_ptr(), out.data_ptr(), _dtype_code(k), L,
                                   k.stride(0) if L > 1 else T * H * D, T, H, D,
                                   pos_local.data_ptr(), pos_global.data_ptr(), ctypes.byref(cfg),
                                   int(score_layer), int(cand0), n, k_fresh.data_ptr(), fs,
                                   score_out.data_ptr(), _stream(stream))
    _check(st, "cs_rebase_and_score")
    return out, score_out


def cs_score_deviation(k_fresh: torch.Tensor, k_cached: torch.Tensor, *,
                       out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Eq. 5 (squared): fp32 [n] from rows k_fresh, k_cached [n, Hkv, D] (rows may be strided)."""
    _need_cuda(k_fresh, k_cached)
    if k_fresh.dim() != 3 or k_fresh.shape != k_cached.shape or k_fresh.dtype != k_cached.dtype:
        raise ValueError("k_fresh and k_cached must both be [n, Hkv, D] of one dtype")
    _inner_contiguous(k_fresh, "k_fresh")
    _inner_contiguous(k_cached, "k_cached")
    n, H, D = k_fresh.shape
    if out is None:
        out = _fresh(stream, lambda: torch.empty(n, dtype=torch.float32, device=k_fresh.device))
    _need_cuda(out)
    if out.dtype != torch.float32 or out.numel() < n or not out.is_contiguous():
        raise ValueError("out must be contiguous fp32 with n elements")
    fs = k_fresh.stride(0) if n > 1 else H * D
    cs = k_cached.stride(0) if n > 1 else H * D
    st = lib().cs_score_deviation(k_fresh.data_ptr(), k_cached.data_ptr(), _dtype_code(k_fresh),
                                  n, H, D, fs, cs, out.data_ptr(), _stream(stream))
    _check(st, "cs_score_deviation")
    return out


def cs_select_topk(score: torch.Tensor, k: int, idx_base: int = 0, *,
                   out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Sec. 2: ascending int32 indices idx_base + i of the k largest scores (lower i wins ties)."""
    _need_cuda(score)
    if score.dtype != torch.float32 or score.dim() != 1 or not score.is_contiguous():
        raise ValueError("score must be contiguous fp32 [n]")
    if out is None:
        out = _fresh(stream, lambda: torch.empty(int(k), dtype=torch.int32, device=score.device))
    _need_cuda(out)
    if out.dtype != torch.int32 or out.numel() < k or not out.is_contiguous():
        raise ValueError("out must be contiguous int32 with k elements")
    st = lib().cs_select_topk(score.data_ptr(), score.numel(), int(k), int(idx_base),
                              out.data_ptr(), _stream(stream))
    _check(st, "cs_select_topk")
    return out


def cs_repair_attention(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, qpos: torch.Tensor, *,
                        scale: float | None = None, out: torch.Tensor | None = None,
                        lse: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Eq. 1 over selected rows: q [L, M, Hq, D], k/v [L, T, Hkv, D], qpos int32 [M] ascending."""
    _need_cuda(q, k, v, qpos)
    if q.dim() != 4 or k.dim() != 4 or k.shape != v.shape or k.stride() != v.stride():
        raise ValueError("q must be [L, M, Hq, D]; k and v [L, T, Hkv, D] with equal strides")
    if not q.is_contiguous():
        raise ValueError("q must be contiguous")
    _inner_contiguous(k, "k")
    L, M, Hq, D = q.shape
    _, T, Hkv, Dk = k.shape
    if k.shape[0] != L or Dk != D or k.dtype != q.dtype or v.dtype != q.dtype:
        raise ValueError("q, k, v must share layers, head dim and dtype")
    if qpos.dtype != torch.int32 or qpos.numel() != M or not qpos.is_contiguous():
        raise ValueError("qpos must be contiguous int32 [M]")
    if out is None:
        out = _fresh(stream, lambda: torch.empty_like(q))
    _need_cuda(out)
    if out.shape != q.shape or out.dtype != q.dtype or not out.is_contiguous():
        raise ValueError("out must match q")
    if lse is not None:
        _need_cuda(lse)
        if lse.dtype != torch.float32 or lse.numel() != L * M * Hq or not lse.is_contiguous():
            raise ValueError("lse must be contiguous fp32 [L, M, Hq]")
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    st = lib().cs_repair_attention(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                   lse.data_ptr() if lse is not None else None, _dtype_code(q),
                                   L, M, T, Hq, Hkv, D, k.stride(0) if L > 1 else T * Hkv * D,
                                   qpos.data_ptr(), float(scale), _stream(stream))
    _check(st, "cs_repair_attention")
    return out


def cs_scatter_rows(cache: torch.Tensor, rows: torch.Tensor, idx: torch.Tensor, *,
                    stream=None) -> torch.Tensor:
    """Sec. 2 scatter-back: cache[l, idx[r]] = rows[l, r] for cache [L, T, ...], rows [L, n, ...].

    idx is int32 [n] of distinct tokens.  The cache is written in place and returned."""
    _need_cuda(cache, rows, idx)
    if cache.dim() < 2 or rows.dim() != cache.dim() or rows.shape[0] != cache.shape[0] or \
            rows.shape[2:] != cache.shape[2:] or rows.dtype != cache.dtype:
        raise ValueError("rows must be [L, n, ...] matching cache [L, T, ...] past the second dim")
    _inner_contiguous(cache, "cache")
    _inner_contiguous(rows, "rows")
    if idx.dtype != torch.int32 or idx.dim() != 1 or idx.numel() != rows.shape[1] or \
            not idx.is_contiguous():
        raise ValueError("idx must be contiguous int32 [n]")
    L, T = cache.shape[0], cache.shape[1]
    n = rows.shape[1]
    row_elems = 1
    for d in cache.shape[2:]:
        row_elems *= d
    cs_stride = cache.stride(0) if L > 1 else T * row_elems
    rs_stride = rows.stride(0) if L > 1 else n * row_elems
    st = lib().cs_scatter_rows(cache.data_ptr(), rows.data_ptr(), _dtype_code(cache), L, T, cs_stride,
                               n, rs_stride, row_elems, idx.data_ptr(), _stream(stream))
    _check(st, "cs_scatter_rows")
    return cache


def cs_sync_status(stream=None) -> None:
    """Waits for the stream and raises CsError if a kernel recorded a device-side error."""
    _check(lib().cs_sync_status(_stream(stream)), "cs_sync_status")


def cs_debug_wait_timeout(limit_us: int, stream=None) -> None:
    """Launches a bounded wait that nothing completes (diagnostics for failure detection)."""
    _check(lib().cs_debug_wait_timeout(int(limit_us), _stream(stream)), "cs_debug_wait_timeout")


__all__ = ["cs_rebase_keys", "cs_rebase_and_score", "cs_score_deviation", "cs_select_topk", "cs_repair_attention",
           "cs_scatter_rows", "cs_sync_status", "cs_debug_wait_timeout", "cs_status_string", "cs_last_error_detail",
           "cs_abi_version", "CsError", "lib", "LIB_PATH"]
