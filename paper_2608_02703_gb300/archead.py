"""Python binding of libarchead (ctypes).  Argument marshalling only: every
step of the forward runs in the library's CUDA kernels.  Functions carry the
C ABI's names (include/archead.h) and take torch tensors for device buffers;
torch is used for device memory and streams only.

The library must have been built (``paper_2608_02703_gb300.build.build()``);
loading fails loudly otherwise -- there is no fallback path.
"""

from __future__ import annotations

import ctypes
import os
from typing import Dict, List, Optional

import numpy as np

from .build import LIB

OK = 0
ERR_INVALID_ARG = 1
ERR_UNSUPPORTED = 2
ERR_OOM = 3
ERR_CUDA = 4
ERR_DEVICE_TIMEOUT = 5
ERR_TARGET_RANGE = 6

OUT_BF16 = 0
OUT_FP32 = 1

FORMAT_INT8 = 0
FORMAT_SC4 = 1

PATH_AUTO = 0
PATH_DECODE = 1
PATH_PREFILL = 2

COMPONENTS = {"residual": 0, "core_u": 1, "core_v": 2, "corr_a": 3, "corr_b": 4}

EXPORTED = (
    "archead_pack_create", "archead_destroy", "archead_forward", "archead_forward_path", "archead_forward_ce",
    "archead_forward_ce_path", "archead_forward_host", "archead_pack_bytes", "archead_device_bytes",
    "archead_debug_dequant", "archead_sync_status", "archead_set_wait_budget", "archead_debug_wait_timeout",
    "archead_profile_enable", "archead_profile_read", "archead_status_string", "archead_last_error",
    "archead_forward_decode_noalloc", "archead_forward_argmax", "archead_forward_argmax_path",
    "archead_forward_lse_partial", "archead_lse_combine", "archead_argmax_combine",
    "archead_quantize_symmetric", "archead_quantize_residual_sc4", "archead_pack_codes", "archead_dequant_symmetric",
    "archead_dequant_residual_sc4", "archead_pack_create_ex", "archead_abi_version",
)


class ArcheadError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = f"{where}: {_status_string(status)}"
        detail = _last_error()
        if status in (ERR_CUDA, ERR_UNSUPPORTED) and detail:
            msg += f" ({detail})"
        super().__init__(msg)


class archead_desc(ctypes.Structure):  # noqa: N801 - mirrors the C struct name
    _fields_ = [
        ("vocab", ctypes.c_int64), ("hidden", ctypes.c_int64),
        ("core_rank", ctypes.c_int32), ("corr_rank", ctypes.c_int32),
        ("group_size", ctypes.c_int32), ("format", ctypes.c_int32),
        ("res_codes", ctypes.c_void_p), ("res_scales", ctypes.c_void_p),
        ("core_u", ctypes.c_void_p), ("core_u_scale", ctypes.c_void_p),
        ("core_v", ctypes.c_void_p), ("core_v_scale", ctypes.c_void_p),
        ("corr_a", ctypes.c_void_p), ("corr_a_scale", ctypes.c_void_p),
        ("corr_b", ctypes.c_void_p), ("corr_b_scale", ctypes.c_void_p),
        ("res_row_scale", ctypes.c_void_p),
    ]


class archead_kernel_stat(ctypes.Structure):  # noqa: N801
    _fields_ = [("name", ctypes.c_char_p), ("launches", ctypes.c_int64), ("total_ms", ctypes.c_double)]


_lib: Optional[ctypes.CDLL] = None


def library_path() -> str:
    return LIB


def load() -> ctypes.CDLL:
    """Load libarchead.so; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB):
        raise RuntimeError(f"libarchead.so is not built ({LIB}); run paper_2608_02703_gb300.build.build()")
    lib = ctypes.CDLL(LIB)
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    sig = {
        "archead_pack_create": (i32, [ctypes.POINTER(archead_desc), vp, ctypes.POINTER(vp)]),
        "archead_pack_create_ex": (i32, [ctypes.POINTER(archead_desc), ctypes.c_size_t, vp, ctypes.POINTER(vp)]),
        "archead_abi_version": (i32, []),
        "archead_destroy": (None, [vp]),
        "archead_forward": (i32, [vp, vp, i64, vp, i32, vp]),
        "archead_forward_path": (i32, [vp, vp, i64, vp, i32, i32, vp]),
        "archead_forward_ce": (i32, [vp, vp, i64, vp, vp, vp]),
        "archead_forward_ce_path": (i32, [vp, vp, i64, vp, vp, i32, vp]),
        "archead_forward_host": (i32, [vp, vp, i64, vp, i32, vp]),
        "archead_forward_decode_noalloc": (i32, [vp, vp, i64, vp, i32, vp]),
        "archead_forward_argmax": (i32, [vp, vp, i64, vp, vp, vp]),
        "archead_forward_argmax_path": (i32, [vp, vp, i64, vp, vp, i32, vp]),
        "archead_forward_lse_partial": (i32, [vp, vp, i64, vp, i64, vp, i32, vp]),
        "archead_lse_combine": (i32, [vp, i32, i64, vp, vp]),
        "archead_argmax_combine": (i32, [vp, vp, vp, i32, i64, vp, vp, vp]),
        "archead_quantize_symmetric": (i32, [vp, i64, i64, i64, i64, i32, vp, vp, vp]),
        "archead_quantize_residual_sc4": (i32, [vp, i64, i64, i32, vp, vp, vp, vp]),
        "archead_pack_codes": (i32, [vp, i64, i64, i32, vp, vp]),
        "archead_dequant_symmetric": (i32, [vp, vp, i64, i64, i64, i64, vp, vp]),
        "archead_dequant_residual_sc4": (i32, [vp, vp, vp, i64, i64, i32, vp, vp]),
        "archead_pack_bytes": (i64, [vp]),
        "archead_device_bytes": (i64, [vp]),
        "archead_debug_dequant": (i32, [vp, i32, i64, i64, vp, vp]),
        "archead_sync_status": (i32, [vp, vp]),
        "archead_set_wait_budget": (i32, [vp, i64]),
        "archead_debug_wait_timeout": (i32, [vp, vp]),
        "archead_profile_enable": (i32, [vp, i32]),
        "archead_profile_read": (i32, [vp, ctypes.POINTER(archead_kernel_stat), i32]),
        "archead_status_string": (ctypes.c_char_p, [i32]),
        "archead_last_error": (ctypes.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _status_string(st: int) -> str:
    return load().archead_status_string(st).decode()


def _last_error() -> str:
    return load().archead_last_error().decode()


def _check(st: int, where: str) -> None:
    if st != OK:
        raise ArcheadError(st, where)


def _stream_ptr(stream) -> Optional[int]:
    import torch

    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


class Pack:
    """A packed head living on one CUDA device (wraps archead_pack*)."""

    def __init__(self, handle: int, shape):
        self.handle = handle
        self.shape = shape

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def close(self) -> None:
        if self.handle:
            load().archead_destroy(self.handle)
            self.handle = None


def archead_pack_create(head: Dict, shape, stream=None, desc_size=None) -> Pack:
    """Build a pack from canonical arrays (numpy host arrays or torch tensors).

    The INT8 format takes the arrays named as the struct fields; the paper's
    format (shape.fmt == "sc4") takes res_scale_codes, res_row_scale and
    core_u5 in place of res_scales and core_u.  With desc_size the call goes
    through archead_pack_create_ex with that struct size."""
    sc4 = getattr(shape, "fmt", "int8") == "sc4"
    d = archead_desc(vocab=shape.V, hidden=shape.d, core_rank=shape.core_rank, corr_rank=shape.corr_rank,
                     group_size=shape.group_size, format=FORMAT_SC4 if sc4 else FORMAT_INT8)
    source = {"res_scales": "res_scale_codes", "core_u": "core_u5"} if sc4 else {"res_row_scale": None}
    keep = []
    for name, _ in archead_desc._fields_[6:]:
        key = source.get(name, name)
        a = head.get(key) if key is not None else None
        if a is not None and hasattr(a, "flags") and not a.flags["C_CONTIGUOUS"]:
            a = np.ascontiguousarray(a)
        if a is not None and hasattr(a, "is_contiguous") and not a.is_contiguous():
            a = a.contiguous()
        keep.append(a)
        setattr(d, name, _ptr(a) if a is not None and getattr(a, "size", 1) != 0 else None)
    h = ctypes.c_void_p()
    if desc_size is None:
        _check(load().archead_pack_create(ctypes.byref(d), _stream_ptr(stream), ctypes.byref(h)), "archead_pack_create")
    else:
        _check(load().archead_pack_create_ex(ctypes.byref(d), desc_size, _stream_ptr(stream), ctypes.byref(h)),
               "archead_pack_create_ex")
    return Pack(h.value, shape)


def archead_abi_version() -> int:
    return int(load().archead_abi_version())


def archead_destroy(pack: Pack) -> None:
    pack.close()


def archead_forward(pack: Pack, x, M: int, logits, out_dtype: int = OUT_BF16, stream=None) -> None:
    _check(load().archead_forward(pack.handle, _ptr(x), M, _ptr(logits), out_dtype, _stream_ptr(stream)),
           "archead_forward")


def archead_forward_path(pack: Pack, x, M: int, logits, out_dtype: int, path: int, stream=None) -> None:
    _check(load().archead_forward_path(pack.handle, _ptr(x), M, _ptr(logits), out_dtype, path, _stream_ptr(stream)),
           "archead_forward_path")


def archead_forward_ce(pack: Pack, x, M: int, targets, ce, stream=None) -> None:
    _check(load().archead_forward_ce(pack.handle, _ptr(x), M, _ptr(targets), _ptr(ce), _stream_ptr(stream)),
           "archead_forward_ce")


def archead_forward_ce_path(pack: Pack, x, M: int, targets, ce, path: int, stream=None) -> None:
    _check(load().archead_forward_ce_path(pack.handle, _ptr(x), M, _ptr(targets), _ptr(ce), path,
                                          _stream_ptr(stream)), "archead_forward_ce_path")


def archead_forward_host(pack: Pack, x_host, M: int, logits_host, out_dtype: int = OUT_BF16, stream=None) -> None:
    _check(load().archead_forward_host(pack.handle, _ptr(x_host), M, _ptr(logits_host), out_dtype,
                                       _stream_ptr(stream)), "archead_forward_host")


def archead_forward_argmax(pack: Pack, x, M: int, index, value=None, stream=None) -> None:
    """Greedy next token per row of x: index (int32 [M]) and, optionally, its logit (fp32 [M])."""
    _check(load().archead_forward_argmax(pack.handle, _ptr(x), M, _ptr(index), _ptr(value), _stream_ptr(stream)),
           "archead_forward_argmax")


def archead_forward_argmax_path(pack: Pack, x, M: int, index, value, path: int, stream=None) -> None:
    _check(load().archead_forward_argmax_path(pack.handle, _ptr(x), M, _ptr(index), _ptr(value), path,
                                              _stream_ptr(stream)), "archead_forward_argmax_path")


def archead_forward_decode_noalloc(pack: Pack, x, M: int, logits, out_dtype: int = OUT_BF16, stream=None) -> None:
    """archead_forward for M <= 16 without any device allocation (fixed 512 KiB scratch array in the library)."""
    _check(load().archead_forward_decode_noalloc(pack.handle, _ptr(x), M, _ptr(logits), out_dtype,
                                                 _stream_ptr(stream)), "archead_forward_decode_noalloc")


def archead_forward_lse_partial(pack: Pack, x, M: int, targets, row0: int, parts, path: int = PATH_AUTO,
                                stream=None) -> None:
    """Per-token (max, sum of exp, target logit or -inf) over this shard's rows (fp32 [M][3])."""
    _check(load().archead_forward_lse_partial(pack.handle, _ptr(x), M, _ptr(targets), row0, _ptr(parts), path,
                                              _stream_ptr(stream)), "archead_forward_lse_partial")


def archead_lse_combine(parts, num_shards: int, M: int, ce, stream=None) -> None:
    """Cross entropy from the shards' partials (fp32 [num_shards][M][3], shard order)."""
    _check(load().archead_lse_combine(_ptr(parts), num_shards, M, _ptr(ce), _stream_ptr(stream)),
           "archead_lse_combine")


def archead_argmax_combine(values, indices, row0, num_shards: int, M: int, index, value=None, stream=None) -> None:
    """Greedy output from the shards' (value, local index) and their first global rows."""
    _check(load().archead_argmax_combine(_ptr(values), _ptr(indices), _ptr(row0), num_shards, M, _ptr(index),
                                         _ptr(value), _stream_ptr(stream)), "archead_argmax_combine")


def archead_quantize_symmetric(x, group_rows: int, group_cols: int, bits: int, codes, scales, stream=None) -> None:
    """Symmetric quantisation of the fp32 matrix x (rows x cols), one fp16 scale per group block."""
    rows, cols = x.shape
    _check(load().archead_quantize_symmetric(_ptr(x), rows, cols, group_rows, group_cols, bits, _ptr(codes),
                                             _ptr(scales), _stream_ptr(stream)), "archead_quantize_symmetric")


def archead_quantize_residual_sc4(r, group_size: int, codes, scale_codes, row_scale, stream=None) -> None:
    rows, cols = r.shape
    _check(load().archead_quantize_residual_sc4(_ptr(r), rows, cols, group_size, _ptr(codes), _ptr(scale_codes),
                                                _ptr(row_scale), _stream_ptr(stream)), "archead_quantize_residual_sc4")


def archead_pack_codes(codes, bits: int, packed, stream=None) -> None:
    rows, cols = codes.shape
    _check(load().archead_pack_codes(_ptr(codes), rows, cols, bits, _ptr(packed), _stream_ptr(stream)),
           "archead_pack_codes")


def archead_dequant_symmetric(codes, scales, group_rows: int, group_cols: int, out, stream=None) -> None:
    rows, cols = codes.shape
    _check(load().archead_dequant_symmetric(_ptr(codes), _ptr(scales), rows, cols, group_rows, group_cols, _ptr(out),
                                            _stream_ptr(stream)), "archead_dequant_symmetric")


def archead_dequant_residual_sc4(codes, scale_codes, row_scale, group_size: int, out, stream=None) -> None:
    rows, cols = codes.shape
    _check(load().archead_dequant_residual_sc4(_ptr(codes), _ptr(scale_codes), _ptr(row_scale), rows, cols,
                                               group_size, _ptr(out), _stream_ptr(stream)),
           "archead_dequant_residual_sc4")


def archead_pack_bytes(pack: Pack) -> int:
    return int(load().archead_pack_bytes(pack.handle))


def archead_device_bytes(pack: Pack) -> int:
    return int(load().archead_device_bytes(pack.handle))


def archead_debug_dequant(pack: Pack, component, row0: int, nrows: int, out, stream=None) -> None:
    c = COMPONENTS[component] if isinstance(component, str) else int(component)
    _check(load().archead_debug_dequant(pack.handle, c, row0, nrows, _ptr(out), _stream_ptr(stream)),
           "archead_debug_dequant")


def archead_sync_status(pack: Pack, stream=None) -> int:
    return int(load().archead_sync_status(pack.handle, _stream_ptr(stream)))


def archead_set_wait_budget(pack: Pack, cycles: int) -> None:
    _check(load().archead_set_wait_budget(pack.handle, cycles), "archead_set_wait_budget")


def archead_debug_wait_timeout(pack: Pack, stream=None) -> None:
    _check(load().archead_debug_wait_timeout(pack.handle, _stream_ptr(stream)), "archead_debug_wait_timeout")


def archead_profile_enable(pack: Pack, enable: bool = True) -> None:
    _check(load().archead_profile_enable(pack.handle, 1 if enable else 0), "archead_profile_enable")


def archead_profile_read(pack: Pack) -> List[dict]:
    buf = (archead_kernel_stat * 32)()
    n = load().archead_profile_read(pack.handle, buf, 32)
    return [{"name": buf[i].name.decode(), "launches": int(buf[i].launches), "total_ms": float(buf[i].total_ms)}
            for i in range(max(n, 0))]


def archead_status_string(status: int) -> str:
    return _status_string(status)


def archead_last_error() -> str:
    return _last_error()
