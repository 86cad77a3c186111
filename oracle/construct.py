"""fp64 CPU oracle of the offline construction of a packed head (paper,
Section 3.4, Algorithm 1, and its expanded form in Appendix B).

TEST INFRASTRUCTURE, like the rest of this package: only the test suite and
the benchmark's CPU-baseline leg may import it.  It shares no code with the
CUDA path.

Steps, in the paper's order and notation (W: V x D dense head, H: N x D
calibration hidden states):

  C_lambda = H^T H / N + lambda * cbar * I      (Section 3.1; cbar = mean diagonal of H^T H / N)
  Q, Lambda = eigh(C_lambda)
  T_p = Q Lambda^p Q^T,  T_p^-1 = Q Lambda^-p Q^T
  W_d = QuantizeCore(W, r_c, g):
        A_c B_c = rank-r_c approximation of W (truncated SVD, split as
                  U S^1/2 and S^1/2 V^T)
        core_u = Q(A_c) per column, core_v = Q(B_c^T) per column
        residual = Q_g(W - A_c B_c) group-wise along D (the unquantized core
                   is subtracted, Appendix B step 4)
        W_d = deq(core_u) deq(core_v)^T + deq(residual)   (the realized core)
  E = W - W_d
  U, S, V = TruncatedSVD(E T_p, r_r)   (exact, or randomized with a given
                                         test matrix Omega)
  A_w = U S,  B_w = V^T T_p^-1
  corr_a = Q(A_w) row-wise INT8, corr_b = Q(B_w^T) group-wise INT8 along D

Quantizers (symmetric, no zero points): scale = fp16(max|x| / qmax) over the
scale's group, code = clamp(rint(x / scale), -qmax, qmax) with x, the
division and the rounding in fp32 (round to nearest, ties to even), code 0
where the scale is 0.  The integer decisions are taken in fp32 because that
is the precision in which the GPU kernels take them.  qmax: 127 (INT8), 15
(5-bit), 7 (INT4).  The paper's format stores the residual's group scales as
4-bit codes q times one fp16 scale per row (s_group = s_row (q + 1));
quantize_residual_sc4 picks s_row = fp16(max over groups of max|x| / (7 * 16))
and q = clamp(ceil(max|x| / (7 s_row)) - 1, 0, 15).

The result is a head dict in the canonical layout of synth.make_head (INT8
format) or of its "sc4" variant, which oracle.logits and the library's
archead_pack_create both accept.
"""

from __future__ import annotations

from typing import Dict, Optional, Tuple

import numpy as np

QMAX = {8: 127, 5: 15, 4: 7}


# ---------------------------------------------------------------------------
# Metric transform (Section 3.1)
# ---------------------------------------------------------------------------
def damped_covariance(H: np.ndarray, lam: float) -> np.ndarray:
    """C_lambda = H^T H / N + lambda * cbar * I."""
    H = np.asarray(H, dtype=np.float64)
    C = H.T @ H / H.shape[0]
    cbar = float(np.mean(np.diag(C)))
    return C + lam * cbar * np.eye(C.shape[0])


def metric_transform(C_lambda: np.ndarray, p: float) -> Tuple[np.ndarray, np.ndarray]:
    """T_p = Q Lambda^p Q^T and its inverse, from the eigendecomposition of C_lambda."""
    lam, Q = np.linalg.eigh(C_lambda)
    T = (Q * lam ** p) @ Q.T
    Tinv = (Q * lam ** (-p)) @ Q.T
    return T, Tinv


# ---------------------------------------------------------------------------
# Truncated SVD: exact, or randomized (range finder with power iterations)
# ---------------------------------------------------------------------------
def truncated_svd(A: np.ndarray, r: int, omega: Optional[np.ndarray] = None, power_iters: int = 2):
    """Rank-r truncated SVD of A (fp64).  With omega (D x k, k >= r) the
    randomized range finder: Y = A omega, `power_iters` rounds of
    Y = A (A^T Y) with re-orthonormalisation, Q = orth(Y), then the SVD of the
    small matrix Q^T A.  Without omega, the exact SVD."""
    A = np.asarray(A, dtype=np.float64)
    if omega is None:
        U, S, Vt = np.linalg.svd(A, full_matrices=False)
        return _fix_signs(U[:, :r], S[:r], Vt[:r])
    Y = A @ np.asarray(omega, dtype=np.float64)
    Q, _ = np.linalg.qr(Y)
    for _ in range(power_iters):
        Z, _ = np.linalg.qr(A.T @ Q)
        Q, _ = np.linalg.qr(A @ Z)
    B = Q.T @ A
    Ub, S, Vt = np.linalg.svd(B, full_matrices=False)
    U = Q @ Ub
    return _fix_signs(U[:, :r], S[:r], Vt[:r])


def _fix_signs(U, S, Vt):
    """Singular vectors are defined up to sign; fix it so that the entry of
    largest magnitude of each left vector is positive (reading: the paper
    leaves it open, and the stored factors depend on it)."""
    idx = np.argmax(np.abs(U), axis=0)
    sgn = np.sign(U[idx, np.arange(U.shape[1])])
    sgn[sgn == 0] = 1.0
    return U * sgn[None, :], S, Vt * sgn[:, None]


# ---------------------------------------------------------------------------
# Quantizers (integer decisions in fp32)
# ---------------------------------------------------------------------------
def _fp16_bits(x32: np.ndarray) -> np.ndarray:
    return np.asarray(x32, dtype=np.float32).astype(np.float16).view(np.uint16)


def quantize_symmetric(x: np.ndarray, group_rows: int, group_cols: int, bits: int):
    """Symmetric quantisation of x [R, C] with one scale per (group_rows x
    group_cols) block: codes int8 [R, C], scales fp16 bits [R/gr, C/gc]."""
    qmax = QMAX[bits]
    x32 = np.asarray(x, dtype=np.float32)
    R, C = x32.shape
    assert R % group_rows == 0 and C % group_cols == 0
    blocks = np.abs(x32).reshape(R // group_rows, group_rows, C // group_cols, group_cols)
    mx = blocks.max(axis=(1, 3))                                     # exact in fp32
    s16 = _fp16_bits(mx / np.float32(qmax))                          # fp32 division, RNE to fp16
    s32 = s16.view(np.float16).astype(np.float32)
    s_full = np.repeat(np.repeat(s32, group_rows, axis=0), group_cols, axis=1)
    with np.errstate(divide="ignore", invalid="ignore"):
        q = np.rint(x32 / s_full)                                    # fp32 division, ties to even
    q = np.where(s_full > 0, np.clip(q, -qmax, qmax), 0.0)
    return q.astype(np.int8), s16


def quantize_residual_sc4(r: np.ndarray, g: int):
    """The paper's format: INT4 codes with a 4-bit scale code per group and one
    fp16 scale per row (reading: s_group = s_row (q + 1))."""
    r32 = np.asarray(r, dtype=np.float32)
    V, D = r32.shape
    G = D // g
    gmax = np.abs(r32).reshape(V, G, g).max(axis=2)                 # [V, G]
    s_row16 = _fp16_bits(gmax.max(axis=1) / np.float32(7 * 16))      # [V]
    s_row = s_row16.view(np.float16).astype(np.float32)
    with np.errstate(divide="ignore", invalid="ignore"):
        need = np.ceil(gmax / (np.float32(7) * s_row[:, None]))
    q = np.where(s_row[:, None] > 0, np.clip(need - 1, 0, 15), 0).astype(np.int64)
    s_grp = s_row[:, None] * (q + 1).astype(np.float32)             # exact: fp16 x small integer
    s_full = np.repeat(s_grp, g, axis=1)
    with np.errstate(divide="ignore", invalid="ignore"):
        c = np.rint(r32 / s_full)
    c = np.where(s_full > 0, np.clip(c, -7, 7), 0.0).astype(np.int8)
    return c, q.astype(np.uint8), s_row16


# ---------------------------------------------------------------------------
# Packing into the canonical layouts
# ---------------------------------------------------------------------------
def pack_int4(codes: np.ndarray) -> np.ndarray:
    """Two's complement nibbles, byte j of a row = columns 2j (low) and 2j+1."""
    c = np.asarray(codes, dtype=np.int64) & 15
    return (c[:, 0::2] | (c[:, 1::2] << 4)).astype(np.uint8)


def pack_scale_codes(q: np.ndarray) -> np.ndarray:
    """4-bit unsigned codes, two per byte, low nibble = even group."""
    q = np.asarray(q, dtype=np.int64)
    V, G = q.shape
    if G % 2:
        q = np.concatenate([q, np.zeros((V, 1), dtype=np.int64)], axis=1)
    return (q[:, 0::2] | (q[:, 1::2] << 4)).astype(np.uint8)


def pack_int5(codes: np.ndarray) -> np.ndarray:
    """5-bit two's complement codes, code j in bits 5j..5j+4 of the row's
    little-endian bit string, ceil(5 r / 8) bytes per row."""
    c = np.asarray(codes, dtype=np.int64) & 31
    V, r = c.shape
    bits = ((c[:, :, None] >> np.arange(5)[None, None, :]) & 1).reshape(V, 5 * r).astype(np.uint8)
    nbytes = (5 * r + 7) // 8
    pad = np.zeros((V, 8 * nbytes - 5 * r), dtype=np.uint8)
    return np.packbits(np.concatenate([bits, pad], axis=1), axis=1, bitorder="little")


# ---------------------------------------------------------------------------
# Dequantisation of what was stored (the realized core)
# ---------------------------------------------------------------------------
def _deq(codes, s16, group_rows, group_cols):
    s = s16.view(np.float16).astype(np.float64)
    s = np.repeat(np.repeat(s, group_rows, axis=0), group_cols, axis=1)
    return np.asarray(codes, dtype=np.float64) * s


# ---------------------------------------------------------------------------
# Algorithm 1
# ---------------------------------------------------------------------------
def construct(W: np.ndarray, H: np.ndarray, core_rank: int, corr_rank: int, group_size: int, p: float = 0.75,
              lam: float = 1e-3, fmt: str = "int8", omega_core: Optional[np.ndarray] = None,
              omega_corr: Optional[np.ndarray] = None, power_iters: int = 2) -> Dict[str, np.ndarray]:
    """Build a packed head from a dense head W and calibration states H.

    Returns the canonical arrays plus the intermediate fp64 quantities under
    keys starting with an underscore (T_p, the realized core, E, the
    unquantized correction) for the tests."""
    W = np.asarray(W, dtype=np.float64)
    V, D = W.shape
    g = group_size
    assert D % g == 0
    # C_lambda, its eigendecomposition and the metric transform.
    C = damped_covariance(H, lam)
    T, Tinv = metric_transform(C, p)
    # QuantizeCore: rank-r_c approximation, quantised factors, INT4 residual.
    if core_rank > 0:
        U, S, Vt = truncated_svd(W, core_rank, omega_core, power_iters)
        A_c = U * np.sqrt(S)[None, :]
        B_c = np.sqrt(S)[:, None] * Vt
    else:
        A_c = np.zeros((V, 0))
        B_c = np.zeros((0, D))
    head: Dict[str, np.ndarray] = {}
    cu_bits = 5 if fmt == "sc4" else 8
    cu_codes, cu_s = quantize_symmetric(A_c, V, 1, cu_bits) if core_rank else (
        np.zeros((V, 0), np.int8), np.zeros((1, 0), np.uint16))
    cv_codes, cv_s = quantize_symmetric(B_c.T, D, 1, 8) if core_rank else (
        np.zeros((D, 0), np.int8), np.zeros((1, 0), np.uint16))
    resid = W - A_c @ B_c
    if fmt == "sc4":
        rc, rq, rs = quantize_residual_sc4(resid, g)
        s_grp = rs.view(np.float16).astype(np.float64)[:, None] * (rq.astype(np.float64) + 1.0)
        res_deq = rc.astype(np.float64) * np.repeat(s_grp, g, axis=1)
        head["res_codes"] = pack_int4(rc)
        head["res_scale_codes"] = pack_scale_codes(rq)
        head["res_row_scale"] = np.ascontiguousarray(rs)
        head["core_u5"] = pack_int5(cu_codes) if core_rank else np.zeros((V, 0), np.uint8)
    else:
        rc, rs = quantize_symmetric(resid, 1, g, 4)
        res_deq = _deq(rc, rs, 1, g)
        head["res_codes"] = pack_int4(rc)
        head["res_scales"] = np.ascontiguousarray(rs)
        head["core_u"] = cu_codes
    head["core_u_scale"] = np.ascontiguousarray(cu_s.reshape(-1))
    head["core_v"] = cv_codes
    head["core_v_scale"] = np.ascontiguousarray(cv_s.reshape(-1))
    core_deq = _deq(cu_codes, cu_s, V, 1) @ _deq(cv_codes, cv_s, D, 1).T if core_rank else np.zeros((V, D))
    W_d = core_deq + res_deq
    # Realized core error, its truncated SVD in the metric, and the correction.
    E = W - W_d
    Et = E @ T
    if corr_rank > 0:
        U2, S2, V2t = truncated_svd(Et, corr_rank, omega_corr, power_iters)
        A_w = U2 * S2[None, :]
        B_w = V2t @ Tinv
        ca, sa = quantize_symmetric(A_w, 1, corr_rank, 8)
        cb, sb = quantize_symmetric(B_w.T, g, 1, 8)
    else:
        A_w = np.zeros((V, 0))
        B_w = np.zeros((0, D))
        ca, sa = np.zeros((V, 0), np.int8), np.zeros((V, 1), np.uint16)
        cb, sb = np.zeros((D, 0), np.int8), np.zeros((D // g, 0), np.uint16)
    head["corr_a"] = ca
    head["corr_a_scale"] = np.ascontiguousarray(sa.reshape(-1))
    head["corr_b"] = cb
    head["corr_b_scale"] = np.ascontiguousarray(sb)
    out = {k: np.ascontiguousarray(v) for k, v in head.items()}
    out.update({"_T": T, "_Tinv": Tinv, "_C": C, "_W_d": W_d, "_E": E, "_A_w": A_w, "_B_w": B_w,
                "_A_c": A_c, "_B_c": B_c})
    return out


def canonical(head: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    """The stored arrays only (drops the intermediate quantities)."""
    return {k: v for k, v in head.items() if not k.startswith("_")}


def metric_error(W: np.ndarray, W_hat: np.ndarray, T: np.ndarray) -> float:
    """||(W - W_hat) T_p||_F^2, the objective of the correction stage (Section 3.2)."""
    return float(np.sum(((np.asarray(W, np.float64) - W_hat) @ T) ** 2))
