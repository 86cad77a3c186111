"""Seeded generator of packed ARCHead heads, hidden states and targets.

The packed head follows the component list of the paper's packed state
dictionary (Appendix C, Table "Logical contents of the packed ARCHead state
dictionary") in the symmetric INT8/INT4 variant used by this library:

    res_codes     uint8  [V, d/2]    signed INT4 residual, two codes per byte:
                                     byte j of row n holds k=2j in the low
                                     nibble and k=2j+1 in the high nibble,
                                     two's complement (-8..7)
    res_scales    uint16 [V, d/g]    fp16 bit patterns, one per (row, group)
    core_u        int8   [V, r_c]    core left factor codes (A_c, Eq. 3)
    core_u_scale  uint16 [r_c]       fp16, one per column
    core_v        int8   [d, r_c]    core right factor codes (B_c transposed)
    core_v_scale  uint16 [r_c]       fp16, one per column
    corr_a        int8   [V, r_r]    correction left codes (A_w, Eq. 5)
    corr_a_scale  uint16 [V]         fp16, one per row (row-wise INT8)
    corr_b        int8   [d, r_r]    correction right codes (B_w transposed)
    corr_b_scale  uint16 [d/g, r_r]  fp16, one per (d-group, column)
                                     (group-wise INT8 along d)

The paper's own packed format (Section 3.2, Eq. 3: a 5-bit core left
factor and the SC4 residual with quantised group scales; Appendix C) is the
"sc4" variant.  It changes three arrays and keeps the rest:

    res_scale_codes uint8 [V, ceil(G/2)]  4-bit unsigned group-scale codes q,
                                          two per byte, low nibble = even
                                          group; the group scale is
                                          res_row_scale[n] * (q + 1)
    res_row_scale   uint16 [V]            fp16, one per row
    core_u5         uint8 [V, ceil(5 r_c / 8)]  5-bit two's complement core
                                          left codes (-16..15); code j of a
                                          row is bits 5j..5j+4 of the row's
                                          bytes read as one little-endian
                                          bit string; unused top bits zero

Hidden states follow the anisotropic recipe x = z diag(s) Q with s
log-spaced over [1e-2, 1e1], Q a Haar-random orthogonal matrix and a few
outlier channels scaled by 20, cast to bf16 (round to nearest even).  The
paper measures on real hidden states of its five heads (Section 4); those
are not available here, so these seeded inputs stand in for them.

Nothing in this module evaluates the head: it only draws codes, scales,
hidden states and targets.
"""

from __future__ import annotations

import dataclasses
from typing import Dict

import numpy as np


@dataclasses.dataclass(frozen=True)
class HeadShape:
    """Shape metadata of one packed head (vocab V, hidden d, ranks, group)."""

    V: int
    d: int
    core_rank: int
    corr_rank: int
    group_size: int
    n_outliers: int = 4
    fmt: str = "int8"  # "int8": INT8 core, fp16 group scales; "sc4": the paper's packed format

    @property
    def groups(self) -> int:
        return self.d // self.group_size

    @property
    def core_u5_bytes(self) -> int:
        """Bytes per row of the 5-bit core left factor (sc4)."""
        return (5 * self.core_rank + 7) // 8

    @property
    def scale_code_bytes(self) -> int:
        """Bytes per row of the 4-bit group-scale codes (sc4)."""
        return (self.groups + 1) // 2


# Head shapes of the paper's models (Section 4, "Models") in this library's
# packed variant, plus a tiny head that the CPU oracle finishes in seconds.
SHAPES: Dict[str, HeadShape] = {
    "tiny": HeadShape(V=4096, d=512, core_rank=64, corr_rank=16, group_size=64, n_outliers=4),
    "qwen3-8b": HeadShape(V=151936, d=4096, core_rank=128, corr_rank=32, group_size=128, n_outliers=4),
    "gemma-4-e4b": HeadShape(V=262144, d=2560, core_rank=128, corr_rank=32, group_size=128, n_outliers=8),
    # The paper's packed format with its Qwen hyper-parameters (Section 4,
    # "Baselines and implementation": r_c = 10, r_r = 6, groups of 64).
    "tiny-sc4": HeadShape(V=4096, d=512, core_rank=10, corr_rank=6, group_size=64, n_outliers=4, fmt="sc4"),
    "qwen3-8b-sc4": HeadShape(V=151936, d=4096, core_rank=10, corr_rank=6, group_size=64, n_outliers=4, fmt="sc4"),
}

# Element rms targets of the three parts of the head.  The paper prints no
# weight statistics; these give logits with rms near 2 on the Qwen shape.
_RMS_CORE = 0.008
_RMS_RESIDUAL = 0.004
_RMS_CORRECTION = 0.0012
# rms of a code drawn uniformly from [-8, 7] and from [-127, 127]
_RMS_INT4 = float(np.sqrt(np.mean(np.arange(-8, 8, dtype=np.float64) ** 2)))
_MS_INT8 = float(np.mean(np.arange(-127, 128, dtype=np.float64) ** 2))
_MS_INT5 = float(np.mean(np.arange(-16, 16, dtype=np.float64) ** 2))
# rms of the group-scale multiplier q + 1 for q uniform over [0, 15]
_RMS_SCALE_MULT = float(np.sqrt(np.mean(np.arange(1, 17, dtype=np.float64) ** 2)))

_HEAD_STREAMS = (
    "res_codes", "res_scales", "core_u", "core_u_scale", "core_v", "core_v_scale",
    "corr_a", "corr_a_scale", "corr_b", "corr_b_scale",
)


def _streams(seed: int, names) -> Dict[str, np.random.Generator]:
    children = np.random.SeedSequence(seed).spawn(len(names))
    return {n: np.random.default_rng(c) for n, c in zip(names, children)}


def _fp16_scales(rng: np.random.Generator, base: float, shape) -> np.ndarray:
    # base * 2^U(-1/2, 1/2): a full random mantissa, rounded to fp16.
    vals = base * np.exp2(rng.uniform(-0.5, 0.5, size=shape))
    return vals.astype(np.float16).view(np.uint16)


def _int8_codes(rng: np.random.Generator, shape) -> np.ndarray:
    return rng.integers(-127, 128, size=shape, dtype=np.int8)


def _uniform_bits(rng: np.random.Generator, rows: int, nbytes: int, used_bits: int) -> np.ndarray:
    """Uniform random bytes [rows, nbytes] with the bits past used_bits of
    each row zero: every field of the row is then uniform over its range."""
    b = rng.integers(0, 256, size=(rows, nbytes), dtype=np.uint8)
    spare = 8 * nbytes - used_bits
    if nbytes and spare:
        b[:, -1] &= np.uint8((1 << (8 - spare)) - 1)
    return b


def make_head(shape: HeadShape, seed: int = 0) -> Dict[str, np.ndarray]:
    """Draw one packed head in the canonical layout described above."""
    if shape.fmt == "sc4":
        return _make_head_sc4(shape, seed)
    if shape.fmt != "int8":
        raise ValueError(f"unknown packed format {shape.fmt!r}")
    V, d, rc, rr, g = shape.V, shape.d, shape.core_rank, shape.corr_rank, shape.group_size
    if d % 2 or d % g:
        raise ValueError("d must be even and a multiple of the group size")
    s = _streams(seed, _HEAD_STREAMS)
    base_r = _RMS_RESIDUAL / _RMS_INT4
    base_c = float(np.sqrt(_RMS_CORE / (np.sqrt(max(rc, 1)) * _MS_INT8)))
    base_w = float(np.sqrt(_RMS_CORRECTION / (np.sqrt(max(rr, 1)) * _MS_INT8)))
    head = {
        # Uniform bytes are two independent uniform nibbles, i.e. codes
        # uniform over [-8, 7] in two's complement.
        "res_codes": s["res_codes"].integers(0, 256, size=(V, d // 2), dtype=np.uint8),
        "res_scales": _fp16_scales(s["res_scales"], base_r, (V, d // g)),
        "core_u": _int8_codes(s["core_u"], (V, rc)),
        "core_u_scale": _fp16_scales(s["core_u_scale"], base_c, (rc,)),
        "core_v": _int8_codes(s["core_v"], (d, rc)),
        "core_v_scale": _fp16_scales(s["core_v_scale"], base_c, (rc,)),
        "corr_a": _int8_codes(s["corr_a"], (V, rr)),
        "corr_a_scale": _fp16_scales(s["corr_a_scale"], base_w, (V,)),
        "corr_b": _int8_codes(s["corr_b"], (d, rr)),
        "corr_b_scale": _fp16_scales(s["corr_b_scale"], base_w, (d // g, rr)),
    }
    return {k: np.ascontiguousarray(v) for k, v in head.items()}


_HEAD_STREAMS_SC4 = (
    "res_codes", "res_scale_codes", "res_row_scale", "core_u5", "core_u_scale", "core_v", "core_v_scale",
    "corr_a", "corr_a_scale", "corr_b", "corr_b_scale",
)


def _make_head_sc4(shape: HeadShape, seed: int) -> Dict[str, np.ndarray]:
    """The paper's packed format ("sc4" above), same element rms targets."""
    V, d, rc, rr, g = shape.V, shape.d, shape.core_rank, shape.corr_rank, shape.group_size
    if d % 2 or d % g:
        raise ValueError("d must be even and a multiple of the group size")
    s = _streams(seed, _HEAD_STREAMS_SC4)
    base_r = _RMS_RESIDUAL / _RMS_INT4 / _RMS_SCALE_MULT
    base_c = float(np.sqrt(_RMS_CORE / (np.sqrt(max(rc, 1)) * _MS_INT8)))
    base_w = float(np.sqrt(_RMS_CORRECTION / (np.sqrt(max(rr, 1)) * _MS_INT8)))
    G = d // g
    head = {
        "res_codes": s["res_codes"].integers(0, 256, size=(V, d // 2), dtype=np.uint8),
        "res_scale_codes": _uniform_bits(s["res_scale_codes"], V, shape.scale_code_bytes, 4 * G),
        "res_row_scale": _fp16_scales(s["res_row_scale"], base_r, (V,)),
        "core_u5": _uniform_bits(s["core_u5"], V, shape.core_u5_bytes, 5 * rc),
        "core_u_scale": _fp16_scales(s["core_u_scale"], base_c * np.sqrt(_MS_INT8 / _MS_INT5), (rc,)),
        "core_v": _int8_codes(s["core_v"], (d, rc)),
        "core_v_scale": _fp16_scales(s["core_v_scale"], base_c, (rc,)),
        "corr_a": _int8_codes(s["corr_a"], (V, rr)),
        "corr_a_scale": _fp16_scales(s["corr_a_scale"], base_w, (V,)),
        "corr_b": _int8_codes(s["corr_b"], (d, rr)),
        "corr_b_scale": _fp16_scales(s["corr_b_scale"], base_w, (d // g, rr)),
    }
    return {k: np.ascontiguousarray(v) for k, v in head.items()}


def with_extreme_codes(head: Dict[str, np.ndarray], shape: HeadShape, seed: int = 0,
                       frac: float = 0.125) -> Dict[str, np.ndarray]:
    """A copy of a packed head with the most negative code of each factor
    array planted: INT8 -128 in core_v, corr_a and corr_b (and core_u in the
    INT8 format), the 5-bit code -16 in core_u5 (the paper's format), and
    INT4 -8 in every residual code of row 0.  A seeded fraction `frac` of the
    entries, plus the whole first row and first column of each array, are
    overwritten; everything else is left as drawn.  The symmetric generators
    above draw INT8 codes in [-127, 127], so -128 only appears this way."""
    out = {k: v.copy() for k, v in head.items()}
    rng = _streams(seed + 3_000_017, ("mask",))["mask"]

    def plant(a: np.ndarray, value) -> None:
        if a.size == 0:
            return
        mask = rng.random(a.shape) < frac
        mask[0, :] = True
        mask[:, 0] = True
        a[mask] = value

    for name in ("core_v", "corr_a", "corr_b") + (("core_u",) if shape.fmt != "sc4" else ()):
        plant(out[name], np.int8(-128))
    if shape.fmt == "sc4" and shape.core_rank > 0:
        # code j of a row lives in bits 5j..5j+4 of the row's little-endian
        # bit string; -16 is 0b10000 in five-bit two's complement.
        bits = np.unpackbits(out["core_u5"], axis=1, bitorder="little")
        codes = np.zeros((shape.V, shape.core_rank), dtype=bool)
        plant_mask = rng.random(codes.shape) < frac
        plant_mask[0, :] = True
        plant_mask[:, 0] = True
        rows, cols = np.nonzero(plant_mask)
        for b in range(4):
            bits[rows, 5 * cols + b] = 0
        bits[rows, 5 * cols + 4] = 1
        out["core_u5"] = np.ascontiguousarray(np.packbits(bits, axis=1, bitorder="little")[:, :shape.core_u5_bytes])
    out["res_codes"][0, :] = 0x88  # both nibbles -8
    return {k: np.ascontiguousarray(v) for k, v in out.items()}


def head_nbytes_canonical(head: Dict[str, np.ndarray]) -> int:
    """Sum of numel * element size over the canonical arrays."""
    return int(sum(a.nbytes for a in head.values()))


def _haar_orthogonal(rng: np.random.Generator, d: int) -> np.ndarray:
    g = rng.standard_normal((d, d))
    q, r = np.linalg.qr(g)
    # Fold the signs of diag(R) into Q so that Q is Haar distributed.
    return q * np.sign(np.diag(r))[None, :]


def _f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    bits = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (bits + 0x7FFF + ((bits >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def make_hidden(d: int, M: int, seed: int = 0, n_outliers: int = 4) -> np.ndarray:
    """Anisotropic hidden states x = z diag(s) Q, as bf16 bits [M, d].

    Q and the outlier channels depend only on (seed, d); z depends on M too.
    The outlier channels are scaled by 20 after the rotation.  The result is
    rounded to fp32 and then to bf16, both to nearest even.
    """
    s = _streams(seed + 1_000_003, ("z", "q", "outlier"))
    scales = np.logspace(-2.0, 1.0, d)
    q = _haar_orthogonal(s["q"], d)
    idx = s["outlier"].choice(d, size=min(n_outliers, d), replace=False)
    z = s["z"].standard_normal((M, d))
    x = (z * scales[None, :]) @ q
    x[:, idx] *= 20.0
    return _f32_to_bf16_bits(x.astype(np.float32))


def make_dense_head(V: int, D: int, seed: int = 0, rank: int = 64, noise: float = 0.01) -> np.ndarray:
    """A dense fp32 output head [V, D] standing in for a real one: a
    rank-`rank` part with singular values log-spaced from 3 down to 0.05 (x
    0.5), plus i.i.d. Gaussian noise of standard deviation `noise` (the
    offline construction's input; the real heads are not available)."""
    s = _streams(seed + 4_000_037, ("u", "v", "noise"))
    k = min(rank, V, D)
    U, _ = np.linalg.qr(s["u"].standard_normal((V, k)))
    Vm, _ = np.linalg.qr(s["v"].standard_normal((D, k)))
    W = (U * (0.5 * np.geomspace(3.0, 0.05, k))[None, :]) @ Vm.T
    W += noise * s["noise"].standard_normal((V, D))
    return W.astype(np.float32)


def make_dense_head_device(V: int, D: int, seed: int = 0, rank: int = 64, noise: float = 0.01, device="cuda"):
    """make_dense_head's recipe drawn on a torch device (fp32), for sizes where
    a host draw would take long (the full Qwen3-8B-shaped head): the same
    spectrum and noise level from a seeded torch generator (not the same
    numbers as make_dense_head)."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(seed + 6_000_001)
    k = min(rank, V, D)
    U, _ = torch.linalg.qr(torch.randn((V, k), generator=gen, device=device))
    Vm, _ = torch.linalg.qr(torch.randn((D, k), generator=gen, device=device))
    s = 0.5 * torch.logspace(np.log10(3.0), np.log10(0.05), k, device=device)
    W = (U * s[None, :]) @ Vm.T
    W += noise * torch.randn((V, D), generator=gen, device=device)
    return W


def make_test_matrix(D: int, k: int, seed: int = 0) -> np.ndarray:
    """Gaussian random test matrix [D, k] for a randomized range finder."""
    return _streams(seed + 5_000_011, ("omega",))["omega"].standard_normal((D, k))


def make_targets(V: int, M: int, seed: int = 0) -> np.ndarray:
    """Next-token targets drawn uniformly over [0, V)."""
    rng = _streams(seed + 2_000_003, ("targets",))["targets"]
    return rng.integers(0, V, size=M, dtype=np.int64).astype(np.int32)
