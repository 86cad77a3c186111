"""fp64 CPU oracle of the packed LM-head forward (ctypes wrapper of plain C).

TEST INFRASTRUCTURE.  Only the test suite, the package smoke check and the
benchmark's CPU-baseline leg may import this package.  It shares no code with
the CUDA path; the C source states what it computes and cites the paper.

Functions take the canonical packed head produced by ``synth.make_head``
(a dict of numpy arrays) and bf16 hidden states as uint16 bit patterns.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Dict, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "archead_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lib: Optional[ctypes.CDLL] = None

COMPONENTS = {"residual": 0, "core_u": 1, "core_v": 2, "corr_a": 3, "corr_b": 4}


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP over vocabulary rows)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Head(ctypes.Structure):
    _fields_ = [
        ("V", ctypes.c_int64), ("d", ctypes.c_int64),
        ("core_rank", ctypes.c_int32), ("corr_rank", ctypes.c_int32),
        ("group_size", ctypes.c_int32), ("format", ctypes.c_int32),
        ("res_codes", ctypes.c_void_p), ("res_scales", ctypes.c_void_p),
        ("core_u", ctypes.c_void_p), ("core_u_scale", ctypes.c_void_p),
        ("core_v", ctypes.c_void_p), ("core_v_scale", ctypes.c_void_p),
        ("corr_a", ctypes.c_void_p), ("corr_a_scale", ctypes.c_void_p),
        ("corr_b", ctypes.c_void_p), ("corr_b_scale", ctypes.c_void_p),
        ("res_scale_codes", ctypes.c_void_p), ("res_row_scale", ctypes.c_void_p),
        ("core_u5", ctypes.c_void_p),
    ]

FORMATS = {"int8": 0, "sc4": 1}


def use_library(path: Optional[str]) -> None:
    """Load the oracle from another build of the same source (None: default).

    The tests use this to check that the pins reject deliberately mutated
    copies of the oracle.
    """
    global _lib
    _lib = None if path is None else _configure(ctypes.CDLL(path))


def _load() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = _configure(ctypes.CDLL(build()))
    return _lib


def _configure(lib: ctypes.CDLL) -> ctypes.CDLL:
    i64, i32, vp, dp = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_double
    lib.oracle_fp16_value.restype = dp
    lib.oracle_fp16_value.argtypes = [ctypes.c_uint16]
    lib.oracle_bf16_value.restype = dp
    lib.oracle_bf16_value.argtypes = [ctypes.c_uint16]
    lib.oracle_fp16_values.argtypes = [vp, i64, vp]
    lib.oracle_bf16_values.argtypes = [vp, i64, vp]
    lib.oracle_unpack_int4.argtypes = [vp, i64, vp]
    lib.oracle_unpack_int5.argtypes = [vp, i64, i64, vp]
    lib.oracle_unpack_scale_codes.argtypes = [vp, i64, i64, vp]
    lib.oracle_dequant_rows.argtypes = [ctypes.POINTER(_Head), i64, i64, vp]
    lib.oracle_component.argtypes = [ctypes.POINTER(_Head), ctypes.c_int, i64, i64, vp]
    lib.oracle_logits.argtypes = [ctypes.POINTER(_Head), vp, i64, i64, i64, vp]
    lib.oracle_ce.argtypes = [ctypes.POINTER(_Head), vp, i64, vp, vp, vp, vp, vp]
    lib.oracle_packed_bytes.restype = i64
    lib.oracle_packed_bytes.argtypes = [i64, i64, i64, i64, i64]
    lib.oracle_packed_bytes_sc4.restype = i64
    lib.oracle_packed_bytes_sc4.argtypes = [i64, i64, i64, i64, i64]
    lib.oracle_dense_bf16_bytes.restype = i64
    lib.oracle_dense_bf16_bytes.argtypes = [i64, i64]
    lib.oracle_threads.restype = ctypes.c_int
    for name in ("oracle_dequant_rows", "oracle_component", "oracle_logits", "oracle_ce"):
        getattr(lib, name).restype = i32
    return lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _head_struct(head: Dict[str, np.ndarray], shape) -> _Head:
    fmt = getattr(shape, "fmt", "int8")
    G = shape.d // shape.group_size
    if fmt == "sc4":
        need = {
            "res_scale_codes": (np.uint8, (shape.V, (G + 1) // 2)),
            "res_row_scale": (np.uint16, (shape.V,)),
            "core_u5": (np.uint8, (shape.V, (5 * shape.core_rank + 7) // 8)),
        }
    else:
        need = {
            "res_scales": (np.uint16, (shape.V, G)),
            "core_u": (np.int8, (shape.V, shape.core_rank)),
        }
    need.update({
        "res_codes": (np.uint8, (shape.V, shape.d // 2)),
        "core_u_scale": (np.uint16, (shape.core_rank,)),
        "core_v": (np.int8, (shape.d, shape.core_rank)),
        "core_v_scale": (np.uint16, (shape.core_rank,)),
        "corr_a": (np.int8, (shape.V, shape.corr_rank)),
        "corr_a_scale": (np.uint16, (shape.V,)),
        "corr_b": (np.int8, (shape.d, shape.corr_rank)),
        "corr_b_scale": (np.uint16, (shape.d // shape.group_size, shape.corr_rank)),
    })
    h = _Head(V=shape.V, d=shape.d, core_rank=shape.core_rank, corr_rank=shape.corr_rank,
              group_size=shape.group_size, format=FORMATS[fmt])
    for name, (dt, shp) in need.items():
        a = head[name]
        if a.dtype != dt or tuple(a.shape) != shp or not a.flags["C_CONTIGUOUS"]:
            raise ValueError(f"{name}: expected {np.dtype(dt)} {shp} contiguous, got {a.dtype} {a.shape}")
        setattr(h, name, _ptr(a))
    return h


def fp16_values(bits: np.ndarray) -> np.ndarray:
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(bits.shape, dtype=np.float64)
    _load().oracle_fp16_values(_ptr(bits), bits.size, _ptr(out))
    return out


def bf16_values(bits: np.ndarray) -> np.ndarray:
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(bits.shape, dtype=np.float64)
    _load().oracle_bf16_values(_ptr(bits), bits.size, _ptr(out))
    return out


def unpack_int4(packed: np.ndarray) -> np.ndarray:
    """Signed codes of a packed byte array (two per byte, low nibble first)."""
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    out = np.empty(packed.size * 2, dtype=np.int8)
    _load().oracle_unpack_int4(_ptr(packed), packed.size * 2, _ptr(out))
    return out.reshape(packed.shape[:-1] + (packed.shape[-1] * 2,)) if packed.ndim else out


def unpack_int5(packed: np.ndarray, rank: int) -> np.ndarray:
    """Signed 5-bit codes [rows, rank] of rows of ceil(5 rank / 8) packed bytes."""
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    rows = packed.shape[0]
    out = np.empty((rows, rank), dtype=np.int8)
    _load().oracle_unpack_int5(_ptr(packed), rows, rank, _ptr(out))
    return out


def unpack_scale_codes(packed: np.ndarray, groups: int) -> np.ndarray:
    """4-bit unsigned group-scale codes [rows, groups] (two per byte, low nibble first)."""
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    rows = packed.shape[0]
    out = np.empty((rows, groups), dtype=np.int8)
    _load().oracle_unpack_scale_codes(_ptr(packed), rows, groups, _ptr(out))
    return out


def dequant_rows(head, shape, row0: int = 0, nrows: Optional[int] = None) -> np.ndarray:
    """Dense fp64 rows of W_hat = W_d + A_w B_w (never used by the CUDA path)."""
    nrows = shape.V - row0 if nrows is None else nrows
    h = _head_struct(head, shape)
    out = np.empty((nrows, shape.d), dtype=np.float64)
    if _load().oracle_dequant_rows(ctypes.byref(h), row0, nrows, _ptr(out)):
        raise ValueError("oracle_dequant_rows rejected its arguments")
    return out


def component(head, shape, comp, row0: int = 0, nrows: Optional[int] = None) -> np.ndarray:
    """One stored component dequantised element by element (code * scale)."""
    c = COMPONENTS[comp] if isinstance(comp, str) else int(comp)
    rows = shape.d if c in (2, 4) else shape.V
    cols = {0: shape.d, 1: shape.core_rank, 2: shape.core_rank, 3: shape.corr_rank, 4: shape.corr_rank}[c]
    nrows = rows - row0 if nrows is None else nrows
    h = _head_struct(head, shape)
    out = np.empty((nrows, cols), dtype=np.float64)
    if _load().oracle_component(ctypes.byref(h), c, row0, nrows, _ptr(out)):
        raise ValueError("oracle_component rejected its arguments")
    return out


def logits(head, shape, x_bits: np.ndarray, row0: int = 0, nrows: Optional[int] = None) -> np.ndarray:
    """fp64 logits [M, nrows] of vocabulary rows [row0, row0 + nrows)."""
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    M = x_bits.shape[0]
    nrows = shape.V - row0 if nrows is None else nrows
    h = _head_struct(head, shape)
    y = np.empty((M, nrows), dtype=np.float64)
    rc = _load().oracle_logits(ctypes.byref(h), _ptr(x_bits), M, row0, nrows, _ptr(y))
    if rc:
        raise ValueError(f"oracle_logits failed ({rc})")
    return y


def cross_entropy(head, shape, x_bits: np.ndarray, targets: np.ndarray, chunk: int = 32) -> Dict[str, np.ndarray]:
    """Per-token CE over the full vocabulary, with argmax and top-2 gap."""
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    targets = np.ascontiguousarray(targets, dtype=np.int32)
    M = x_bits.shape[0]
    h = _head_struct(head, shape)
    out = {
        "ce": np.empty(M, dtype=np.float64),
        "argmax": np.empty(M, dtype=np.int64),
        "top2_gap": np.empty(M, dtype=np.float64),
        "target_logit": np.empty(M, dtype=np.float64),
    }
    lib = _load()
    for m0 in range(0, M, chunk):
        m1 = min(M, m0 + chunk)
        xs = np.ascontiguousarray(x_bits[m0:m1])
        ts = np.ascontiguousarray(targets[m0:m1])
        parts = {k: np.empty(m1 - m0, dtype=v.dtype) for k, v in out.items()}
        rc = lib.oracle_ce(ctypes.byref(h), _ptr(xs), m1 - m0, _ptr(ts), _ptr(parts["ce"]),
                           _ptr(parts["argmax"]), _ptr(parts["top2_gap"]), _ptr(parts["target_logit"]))
        if rc < 0:
            raise ValueError(f"oracle_ce failed ({rc})")
        for k in out:
            out[k][m0:m1] = parts[k]
    return out


def packed_bytes(shape) -> int:
    """Eq. 10 of the paper over the stored components of this packed format."""
    fn = _load().oracle_packed_bytes_sc4 if getattr(shape, "fmt", "int8") == "sc4" else _load().oracle_packed_bytes
    return int(fn(shape.V, shape.d, shape.core_rank, shape.corr_rank, shape.group_size))


def dense_bf16_bytes(V: int, d: int) -> int:
    return int(_load().oracle_dense_bf16_bytes(V, d))


def threads() -> int:
    return int(_load().oracle_threads())


# ---------------------------------------------------------------------------
# Vocabulary shards (the forward is row-separable, paper Section 3.2, Eq. 7).
# ---------------------------------------------------------------------------
def lse_partial(head, shape, x_bits: np.ndarray, targets: np.ndarray, row0: int, nrows: int) -> np.ndarray:
    """fp64 (max, sum of exp(y - max), target logit or -inf) per token over
    global rows [row0, row0 + nrows) of the head: [M, 3]."""
    y = logits(head, shape, x_bits, row0=row0, nrows=nrows)
    mx = y.max(axis=1)
    s = np.exp(y - mx[:, None]).sum(axis=1)
    t = np.asarray(targets, dtype=np.int64) - row0
    mine = (t >= 0) & (t < nrows)
    tl = np.where(mine, y[np.arange(y.shape[0]), np.clip(t, 0, nrows - 1)], -np.inf)
    return np.stack([mx, s, tl], axis=1)


def lse_combine(parts: np.ndarray) -> np.ndarray:
    """CE per token from shard partials [P, M, 3] (shard order): the log-sum-
    exp of the union of the shards' rows minus the one reported target logit;
    NaN where the number of shards reporting the target is not one."""
    parts = np.asarray(parts, dtype=np.float64)
    mx = parts[:, :, 0].max(axis=0)
    s = (parts[:, :, 1] * np.exp(parts[:, :, 0] - mx[None, :])).sum(axis=0)
    owners = np.isfinite(parts[:, :, 2]).sum(axis=0)
    t = np.where(np.isfinite(parts[:, :, 2]), parts[:, :, 2], 0.0).sum(axis=0)
    return np.where(owners == 1, mx + np.log(s) - t, np.nan)


def argmax_combine(values: np.ndarray, indices: np.ndarray, row0: np.ndarray):
    """Greedy output over shards: the largest value, the lowest global row
    (local index + the shard's row0) on ties.  values, indices [P, M]."""
    values = np.asarray(values, dtype=np.float64)
    glob = np.asarray(indices, dtype=np.int64) + np.asarray(row0, dtype=np.int64).reshape(-1, 1)
    best = values.max(axis=0)
    cand = np.where(values == best[None, :], glob, np.iinfo(np.int64).max)
    return cand.min(axis=0), best
