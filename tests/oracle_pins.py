"""Pins of the fp64 oracle to facts fixed outside the oracle itself.

Each check raises AssertionError when the oracle disagrees with:
  - the definitions of two's complement INT4, IEEE binary16 and bfloat16
    (checked over every bit pattern against numpy's own conversions);
  - special cases that reduce to textbook products (core only = explicit
    U V^T; zero ranks = plain group-wise INT4 matmul);
  - closed forms of the cross entropy (uniform logits give log V);
  - a pure-Python brute force of Eqs. 3, 6 and 7 on tiny heads;
  - the paper's printed dense-head sizes and its packed Qwen head size
    (Section 3.3, Table 1);
  - for the paper's own format (5-bit core codes, quantised group scales):
    numpy's bit unpacking, a brute force, and the equal int8-format head;
  - invariants (linearity in x, vocabulary permutation, argmax tie rule).

The same checks run against deliberately mutated builds of the oracle in
test_oracle_mutants.py, to show that plausible mistakes are caught.
"""

from __future__ import annotations

import math
import os
import struct

import numpy as np

from synth import HeadShape, make_head, make_hidden, make_targets

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

# Small head with every dimension distinct so that a transposed index or a
# swapped rank cannot go unnoticed: V != d, r_c != r_r, several groups.
PIN_SHAPE = HeadShape(V=24, d=64, core_rank=5, corr_rank=3, group_size=16)


def _f16(bits: int) -> float:
    return float(np.array([bits], dtype=np.uint16).view(np.float16)[0])


def _bf16(bits: int) -> float:
    return struct.unpack("<f", struct.pack("<I", (int(bits) & 0xFFFF) << 16))[0]


def _int4_from_byte(b: int, high: bool) -> int:
    nib = (b >> 4) & 0xF if high else b & 0xF
    return nib - 16 if nib & 0x8 else nib


def check_int4_unpack(oracle):
    all_bytes = np.arange(256, dtype=np.uint8)
    codes = oracle.unpack_int4(all_bytes[None, :])[0]
    expect = np.array([[_int4_from_byte(b, False), _int4_from_byte(b, True)] for b in range(256)]).ravel()
    assert np.array_equal(codes, expect), "INT4 unpack disagrees with two's complement nibbles"
    # A few bytes written out by hand: low nibble is the even index.
    hand = {0x00: (0, 0), 0x0F: (-1, 0), 0xF0: (0, -1), 0x87: (7, -8), 0x78: (-8, 7), 0x19: (-7, 1)}
    for b, pair in hand.items():
        assert tuple(codes[2 * b:2 * b + 2]) == pair, f"byte {b:#x}"
    # Round trip: repacking the codes gives the bytes back.
    lo = codes[0::2].astype(np.int64) & 0xF
    hi = codes[1::2].astype(np.int64) & 0xF
    assert np.array_equal((lo | (hi << 4)).astype(np.uint8), all_bytes)
    # Random rows: repack(unpack) is the identity along d.
    rng = np.random.default_rng(7)
    c = rng.integers(-8, 8, size=(5, 46))
    packed = ((c[:, 0::2] & 0xF) | ((c[:, 1::2] & 0xF) << 4)).astype(np.uint8)
    assert np.array_equal(oracle.unpack_int4(packed), c)


def check_fp16_decode(oracle):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    got = oracle.fp16_values(bits)
    ref = bits.view(np.float16).astype(np.float64)
    finite = np.isfinite(ref)
    assert np.array_equal(got[finite], ref[finite]), "fp16 decode differs from IEEE binary16"
    assert np.all(np.isinf(got[np.isinf(ref)])) and np.all(np.isnan(got[np.isnan(ref)]))
    assert np.array_equal(np.signbit(got[finite]), np.signbit(ref[finite]))


def check_bf16_decode(oracle):
    bits = np.arange(65536, dtype=np.uint32)
    got = oracle.bf16_values(bits.astype(np.uint16))
    with np.errstate(invalid="ignore"):
        ref = (bits << 16).view(np.float32).astype(np.float64)
    finite = np.isfinite(ref)
    assert np.array_equal(got[finite], ref[finite]), "bf16 decode differs from the upper half of fp32"
    assert np.all(np.isinf(got[np.isinf(ref)])) and np.all(np.isnan(got[np.isnan(ref)]))


def _dq(head, shape):
    """Components decoded with numpy's conversions (not the oracle's)."""
    g = shape.group_size
    codes = np.empty((shape.V, shape.d), dtype=np.int64)
    b = head["res_codes"].astype(np.int64)
    codes[:, 0::2] = ((b & 0xF) ^ 0x8) - 0x8
    codes[:, 1::2] = (((b >> 4) & 0xF) ^ 0x8) - 0x8
    f16 = lambda a: a.view(np.float16).astype(np.float64)  # noqa: E731
    res = codes * np.repeat(f16(head["res_scales"]), g, axis=1)
    U = head["core_u"].astype(np.float64) * f16(head["core_u_scale"])[None, :]
    Vc = head["core_v"].astype(np.float64) * f16(head["core_v_scale"])[None, :]
    A = head["corr_a"].astype(np.float64) * f16(head["corr_a_scale"])[:, None]
    B = head["corr_b"].astype(np.float64) * np.repeat(f16(head["corr_b_scale"]), g, axis=0)
    return res, U, Vc, A, B


def _x64(x_bits):
    return (x_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def check_core_only(oracle, shape=PIN_SHAPE):
    """Zero residual and zero correction: logits are x (U V^T)^T."""
    head = make_head(shape, seed=11)
    head["res_codes"][:] = 0
    head["corr_a"][:] = 0
    x = make_hidden(shape.d, 3, seed=11)
    _, U, Vc, _, _ = _dq(head, shape)
    W = U @ Vc.T                                   # explicit dense product
    ref = _x64(x) @ W.T
    got = oracle.logits(head, shape, x)
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max()), "core-only logits"
    # The factored evaluation (x V) U^T gives the same numbers.
    fact = (_x64(x) @ Vc) @ U.T
    assert np.allclose(got, fact, rtol=1e-12, atol=1e-12 * np.abs(ref).max())


def check_group_int4(oracle):
    """r_c = r_r = 0: a plain group-wise INT4 matmul (the "Group INT4" head)."""
    shape = HeadShape(V=40, d=96, core_rank=0, corr_rank=0, group_size=32)
    head = make_head(shape, seed=12)
    x = make_hidden(shape.d, 4, seed=12)
    res, _, _, _, _ = _dq(head, shape)
    ref = _x64(x) @ res.T
    got = oracle.logits(head, shape, x)
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-13 * np.abs(ref).max()), "group INT4 logits"


def check_components(oracle, shape=PIN_SHAPE):
    head = make_head(shape, seed=13)
    res, U, Vc, A, B = _dq(head, shape)
    for name, ref in (("residual", res), ("core_u", U), ("core_v", Vc), ("corr_a", A), ("corr_b", B)):
        got = oracle.component(head, shape, name)
        assert np.array_equal(got, ref), f"component {name} is not exactly code * scale"
    W = oracle.dequant_rows(head, shape)
    assert np.allclose(W, res + U @ Vc.T + A @ B.T, rtol=1e-13, atol=1e-15)


def _brute_force_logits(head, shape, x_bits):
    """Pure-Python loops over Eqs. 3, 6, 7 with per-element decoding."""
    V, d, g, rc, rr = shape.V, shape.d, shape.group_size, shape.core_rank, shape.corr_rank
    y = [[0.0] * V for _ in range(x_bits.shape[0])]
    for n in range(V):
        w = []
        for k in range(d):
            c = _int4_from_byte(int(head["res_codes"][n, k // 2]), high=(k % 2 == 1))
            v = c * _f16(head["res_scales"][n, k // g])
            for j in range(rc):
                v += (int(head["core_u"][n, j]) * _f16(head["core_u_scale"][j])) * (
                    int(head["core_v"][k, j]) * _f16(head["core_v_scale"][j]))
            for j in range(rr):
                v += (int(head["corr_a"][n, j]) * _f16(head["corr_a_scale"][n])) * (
                    int(head["corr_b"][k, j]) * _f16(head["corr_b_scale"][k // g, j]))
            w.append(v)
        for m in range(x_bits.shape[0]):
            y[m][n] = math.fsum(_bf16(x_bits[m, k]) * w[k] for k in range(d))
    return np.array(y)


def check_brute_force(oracle, shape=PIN_SHAPE):
    head = make_head(shape, seed=14)
    x = make_hidden(shape.d, 3, seed=14)
    ref = _brute_force_logits(head, shape, x)
    got = oracle.logits(head, shape, x)
    scale = np.abs(ref).max()
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12 * scale), "oracle logits differ from brute force"
    # A sub-range of vocabulary rows is the same slice.
    part = oracle.logits(head, shape, x, row0=5, nrows=7)
    assert np.array_equal(part, got[:, 5:12])


def check_cross_entropy(oracle, shape=PIN_SHAPE):
    # Closed form: an all-zero head gives y = 0 and CE = log V for any target.
    head = make_head(shape, seed=15)
    for k in ("res_codes", "core_u", "corr_a"):
        head[k][:] = 0
    x = make_hidden(shape.d, 3, seed=15)
    t = make_targets(shape.V, 3, seed=15)
    out = oracle.cross_entropy(head, shape, x, t)
    assert np.allclose(out["ce"], math.log(shape.V), rtol=0, atol=1e-14)
    assert np.all(out["argmax"] == 0) and np.all(out["top2_gap"] == 0), "ties break to the lowest index"
    # Random head: CE equals logsumexp of the (pinned) logits minus the target logit.
    head = make_head(shape, seed=16)
    x = make_hidden(shape.d, 5, seed=16)
    t = make_targets(shape.V, 5, seed=16)
    y = _brute_force_logits(head, shape, x)
    out = oracle.cross_entropy(head, shape, x, t)
    lse = np.logaddexp.reduce(y, axis=1)
    assert np.allclose(out["ce"], lse - y[np.arange(5), t], rtol=0, atol=1e-12)
    assert np.array_equal(out["argmax"], np.argmax(y, axis=1))
    srt = np.sort(y, axis=1)
    assert np.allclose(out["top2_gap"], srt[:, -1] - srt[:, -2], rtol=0, atol=1e-12)
    assert np.allclose(out["target_logit"], y[np.arange(5), t], rtol=0, atol=1e-12)
    # One dominant logit: CE of that target is log(1 + (V-1) e^{-gap}) in closed form.
    head = make_head(shape, seed=17)
    for k in ("res_codes", "core_u", "corr_a"):
        head[k][:] = 0
    head["res_codes"][3, :] = 0x11                  # every code of row 3 is +1
    head["res_scales"][3, :] = 0x2C00               # fp16 scale 1/16
    xb = np.full((1, shape.d), 0x3F80, dtype=np.uint16)   # bf16 1.0, so y[3] = d/16
    out = oracle.cross_entropy(head, shape, xb, np.array([3], dtype=np.int32))
    gap = shape.d / 16.0
    assert math.isclose(out["ce"][0], math.log1p((shape.V - 1) * math.exp(-gap)), rel_tol=1e-12, abs_tol=1e-300)
    assert out["argmax"][0] == 3 and out["top2_gap"][0] == gap


def check_invariants(oracle, shape=PIN_SHAPE):
    head = make_head(shape, seed=18)
    x = make_hidden(shape.d, 2, seed=18)
    y = oracle.logits(head, shape, x)
    # Doubling x (exact in bf16: exponent + 1) doubles every logit exactly.
    x2 = x.copy()
    nz = (x2 & 0x7F80) != 0
    x2[nz] = x2[nz] + 0x0080
    assert np.array_equal(oracle.logits(head, shape, x2), 2 * y)
    # Permuting vocabulary rows permutes the logits.
    perm = np.random.default_rng(3).permutation(shape.V)
    hp = dict(head)
    for k in ("res_codes", "res_scales", "core_u", "corr_a", "corr_a_scale"):
        hp[k] = np.ascontiguousarray(head[k][perm])
    assert np.array_equal(oracle.logits(hp, shape, x), y[:, perm])
    # One-hot hidden state e_k reads out column k of W_hat.
    W = oracle.dequant_rows(head, shape)
    e = np.zeros((1, shape.d), dtype=np.uint16)
    e[0, 37] = 0x3F80
    assert np.array_equal(oracle.logits(head, shape, e)[0], W[:, 37])


def check_paper_dense_sizes(oracle):
    rows = []
    with open(os.path.join(GOLDEN, "paper_table1_dense_mib.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                name, V, D, mb = line.split()
                rows.append((name, int(V), int(D), float(mb)))
    assert len(rows) == 5
    for name, V, D, mb in rows:
        assert round(oracle.dense_bf16_bytes(V, D) / 2**20, 1) == mb, name


def check_packed_bytes(oracle):
    for shape in (PIN_SHAPE, HeadShape(V=40, d=96, core_rank=0, corr_rank=0, group_size=32),
                  HeadShape(V=4096, d=512, core_rank=64, corr_rank=16, group_size=64)):
        head = make_head(shape, seed=19)
        counted = sum(a.nbytes for k, a in head.items() if not (k == "corr_a_scale" and shape.corr_rank == 0))
        assert oracle.packed_bytes(shape) == counted, shape


# ---------------------------------------------------------------------------
# The paper's packed format ("sc4": 5-bit core left factor, 4-bit group-scale
# codes times an fp16 row scale).
# ---------------------------------------------------------------------------
PIN_SHAPE_SC4 = HeadShape(V=24, d=80, core_rank=5, corr_rank=3, group_size=16, fmt="sc4")  # 5 groups: odd


def _np_int5(packed: np.ndarray, rank: int) -> np.ndarray:
    """5-bit two's complement fields, LSB first, through numpy's unpackbits."""
    bits = np.unpackbits(packed, axis=1, bitorder="little")[:, :5 * rank].reshape(packed.shape[0], rank, 5)
    v = (bits.astype(np.int64) << np.arange(5)).sum(axis=2)
    return np.where(v >= 16, v - 32, v)


def _np_scale_codes(packed: np.ndarray, groups: int) -> np.ndarray:
    q = np.empty((packed.shape[0], 2 * packed.shape[1]), dtype=np.int64)
    q[:, 0::2] = packed & 0xF
    q[:, 1::2] = packed >> 4
    return q[:, :groups]


def check_int5_unpack(oracle):
    # Written out by hand: codes (1, -1, -16) are the bit string
    # 10000 11111 00001 (LSB first), i.e. bytes 0xE1, 0x43.
    assert oracle.unpack_int5(np.array([[0xE1, 0x43]], dtype=np.uint8), 3).tolist() == [[1, -1, -16]]
    # (15, 0, 7, -8): bits 0-3, 10-12, 18-19 set -> 0x0F, 0x1C, 0x0C (padding bits zero).
    assert oracle.unpack_int5(np.array([[0x0F, 0x1C, 0x0C]], dtype=np.uint8), 4).tolist() == [[15, 0, 7, -8]]
    # Every code value at every bit offset (j = 0..7 covers offsets 0, 5, 2, 7, 4, 1, 6, 3).
    codes = np.array([[(v + 7 * j) % 32 - 16 for j in range(8)] for v in range(32)], dtype=np.int64)
    bits = ((codes[:, :, None] & 31) >> np.arange(5)) & 1
    packed = np.packbits(bits.reshape(32, 40).astype(np.uint8), axis=1, bitorder="little")
    assert np.array_equal(oracle.unpack_int5(packed, 8), codes)
    # Random rows of several ranks against numpy's bit unpacking.
    rng = np.random.default_rng(21)
    for rank in (1, 3, 10, 13):
        nb = (5 * rank + 7) // 8
        raw = rng.integers(0, 256, size=(9, nb), dtype=np.uint8)
        assert np.array_equal(oracle.unpack_int5(raw, rank), _np_int5(raw, rank)), rank


def check_scale_code_unpack(oracle):
    assert oracle.unpack_scale_codes(np.array([[0x5A, 0xF0]], dtype=np.uint8), 4).tolist() == [[10, 5, 0, 15]]
    assert oracle.unpack_scale_codes(np.array([[0x31, 0x07]], dtype=np.uint8), 3).tolist() == [[1, 3, 7]]
    raw = np.random.default_rng(22).integers(0, 256, size=(7, 5), dtype=np.uint8)
    assert np.array_equal(oracle.unpack_scale_codes(raw, 9), _np_scale_codes(raw, 9))


def _dq_sc4(head, shape):
    """Components of an sc4 head decoded with numpy (not the oracle)."""
    g = shape.group_size
    codes = np.empty((shape.V, shape.d), dtype=np.int64)
    b = head["res_codes"].astype(np.int64)
    codes[:, 0::2] = ((b & 0xF) ^ 0x8) - 0x8
    codes[:, 1::2] = (((b >> 4) & 0xF) ^ 0x8) - 0x8
    f16 = lambda a: a.view(np.float16).astype(np.float64)  # noqa: E731
    s = f16(head["res_row_scale"])[:, None] * (_np_scale_codes(head["res_scale_codes"], shape.groups) + 1)
    res = codes * np.repeat(s, g, axis=1)
    U = _np_int5(head["core_u5"], shape.core_rank) * f16(head["core_u_scale"])[None, :]
    Vc = head["core_v"].astype(np.float64) * f16(head["core_v_scale"])[None, :]
    A = head["corr_a"].astype(np.float64) * f16(head["corr_a_scale"])[:, None]
    B = head["corr_b"].astype(np.float64) * np.repeat(f16(head["corr_b_scale"]), g, axis=0)
    return res, U, Vc, A, B


def check_sc4_components(oracle, shape=PIN_SHAPE_SC4):
    head = make_head(shape, seed=23)
    res, U, Vc, A, B = _dq_sc4(head, shape)
    for name, ref in (("residual", res), ("core_u", U), ("core_v", Vc), ("corr_a", A), ("corr_b", B)):
        got = oracle.component(head, shape, name)
        assert np.array_equal(got, ref), f"sc4 component {name} is not exactly code * scale"
    W = oracle.dequant_rows(head, shape)
    assert np.allclose(W, res + U @ Vc.T + A @ B.T, rtol=1e-13, atol=1e-15)


def _brute_force_logits_sc4(head, shape, x_bits):
    """Pure-Python loops with per-element bit decoding of the sc4 fields."""
    V, d, g, rc, rr = shape.V, shape.d, shape.group_size, shape.core_rank, shape.corr_rank
    nb_u = (5 * rc + 7) // 8

    def u5(n, j):
        row = [int(v) for v in head["core_u5"][n, :nb_u]]
        word = sum(v << (8 * i) for i, v in enumerate(row))
        c = (word >> (5 * j)) & 31
        return c - 32 if c >= 16 else c

    def scale(n, grp):
        byte = int(head["res_scale_codes"][n, grp // 2])
        q = (byte >> 4) if grp % 2 else (byte & 15)
        return _f16(head["res_row_scale"][n]) * (q + 1)

    y = [[0.0] * V for _ in range(x_bits.shape[0])]
    for n in range(V):
        w = []
        for k in range(d):
            v = _int4_from_byte(int(head["res_codes"][n, k // 2]), high=(k % 2 == 1)) * scale(n, k // g)
            for j in range(rc):
                v += (u5(n, j) * _f16(head["core_u_scale"][j])) * (
                    int(head["core_v"][k, j]) * _f16(head["core_v_scale"][j]))
            for j in range(rr):
                v += (int(head["corr_a"][n, j]) * _f16(head["corr_a_scale"][n])) * (
                    int(head["corr_b"][k, j]) * _f16(head["corr_b_scale"][k // g, j]))
            w.append(v)
        for m in range(x_bits.shape[0]):
            y[m][n] = math.fsum(_bf16(x_bits[m, k]) * w[k] for k in range(d))
    return np.array(y)


def check_sc4_brute_force(oracle, shape=PIN_SHAPE_SC4):
    head = make_head(shape, seed=24)
    x = make_hidden(shape.d, 2, seed=24)
    ref = _brute_force_logits_sc4(head, shape, x)
    got = oracle.logits(head, shape, x)
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max()), "sc4 logits differ from brute force"


def check_sc4_equals_int8_form(oracle):
    """An sc4 head whose group scales s_row (q + 1) are exact in fp16 is the
    same head as the int8-format head holding those scales and the widened
    5-bit codes: the two must give identical logits."""
    shape = HeadShape(V=33, d=128, core_rank=7, corr_rank=4, group_size=32, fmt="sc4")
    head = make_head(shape, seed=25)
    rng = np.random.default_rng(25)
    # Row scales 2^-12 (1 + k/64): 7 significant bits, so s_row * (q + 1) <= 16 s_row fits fp16 exactly.
    s_row = (2.0 ** -12) * (1 + rng.integers(0, 64, size=shape.V) / 64.0)
    head["res_row_scale"] = s_row.astype(np.float16).view(np.uint16)
    q = _np_scale_codes(head["res_scale_codes"], shape.groups)
    scales = (s_row[:, None] * (q + 1)).astype(np.float16)
    assert np.array_equal(scales.astype(np.float64), s_row[:, None] * (q + 1))
    i8shape = HeadShape(V=shape.V, d=shape.d, core_rank=shape.core_rank, corr_rank=shape.corr_rank,
                        group_size=shape.group_size)
    i8 = {k: v for k, v in head.items() if k not in ("res_scale_codes", "res_row_scale", "core_u5")}
    i8["res_scales"] = np.ascontiguousarray(scales.view(np.uint16))
    i8["core_u"] = np.ascontiguousarray(_np_int5(head["core_u5"], shape.core_rank).astype(np.int8))
    x = make_hidden(shape.d, 3, seed=25)
    assert np.array_equal(oracle.logits(head, shape, x), oracle.logits(i8, i8shape, x))


def check_paper_packed_storage(oracle):
    """Eq. 10 over the sc4 format reproduces the paper's packed size of the
    Qwen3-8B head (Table 1) within 0.1 MiB (0.03 %) and its compression."""
    rows = []
    with open(os.path.join(GOLDEN, "paper_table1_packed_qwen_mib.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                name, V, D, rc, rr, g, mb, ratio = line.split()
                rows.append((name, int(V), int(D), int(rc), int(rr), int(g), float(mb), float(ratio)))
    assert len(rows) == 1
    for name, V, D, rc, rr, g, mb, ratio in rows:
        shape = HeadShape(V=V, d=D, core_rank=rc, corr_rank=rr, group_size=g, fmt="sc4")
        got = oracle.packed_bytes(shape)
        assert abs(got / 2**20 - mb) < 0.1, (name, got / 2**20)
        assert abs(oracle.dense_bf16_bytes(V, D) / got - ratio) < 0.002, name
        # The format's own arrays count to the same bytes (small head, same rule).
    for shape in (PIN_SHAPE_SC4, HeadShape(V=50, d=192, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
                  HeadShape(V=7, d=96, core_rank=0, corr_rank=0, group_size=32, fmt="sc4")):
        head = make_head(shape, seed=26)
        counted = sum(a.nbytes for k, a in head.items() if not (k == "corr_a_scale" and shape.corr_rank == 0))
        assert oracle.packed_bytes(shape) == counted, shape


ALL_CHECKS = [
    check_int4_unpack, check_fp16_decode, check_bf16_decode, check_core_only, check_group_int4,
    check_components, check_brute_force, check_cross_entropy, check_invariants,
    check_paper_dense_sizes, check_packed_bytes,
    check_int5_unpack, check_scale_code_unpack, check_sc4_components, check_sc4_brute_force,
    check_sc4_equals_int8_form, check_paper_packed_storage,
]
