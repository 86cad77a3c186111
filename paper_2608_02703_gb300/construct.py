"""Offline construction of a packed head on the GPU (paper, Section 3.4,
Algorithm 1; Appendix B): from a dense head W (V x D) and calibration hidden
states H (N x D) to the canonical packed arrays that archead_pack_create
takes.

Steps, in the paper's order:

  C_lambda = H^T H / N + lambda * cbar * I          (cbar = mean diagonal)
  Q, Lambda = eigh(C_lambda);  T_p = Q Lambda^p Q^T,  T_p^-1 = Q Lambda^-p Q^T
  QuantizeCore:  A_c B_c = rank-r_c truncated SVD of W (U S^1/2, S^1/2 V^T);
                 core_u = Q_8 (or Q_5) of A_c per column, core_v = Q_8 of
                 B_c^T per column; residual = INT4 of W - A_c B_c group-wise
                 along D (fp16 group scales, or the paper's 4-bit scale codes
                 times a row scale)
  E = W - W_d  (W_d dequantised from what was stored: the realized core)
  U, S, V = randomized SVD of E T_p (rank r_r);  A_w = U S,  B_w = V^T T_p^-1
  corr_a = row-wise INT8 of A_w,  corr_b = group-wise INT8 of B_w^T

The dense linear algebra (the covariance product, the eigendecomposition, the
GEMMs, QR factorisations and small SVDs of the randomized range finder) runs
on the GPU through torch (cuBLAS / cuSOLVER library routines).  Every
quantisation, packing and dequantisation step runs in the library's own
kernels (archead_quantize_symmetric, archead_quantize_residual_sc4,
archead_pack_codes, archead_dequant_*), which take the integer decisions in
fp32.  The random test matrices of the range finder are inputs (omega_core,
omega_corr), so that two implementations can be run on the same draws.
Singular vectors are returned with a fixed sign: the entry of largest
magnitude of each left vector is positive.
"""

from __future__ import annotations

from typing import Dict, Optional

from . import archead


def _torch():
    import torch

    return torch


def damped_covariance(H, lam: float, dtype=None):
    t = _torch()
    dtype = dtype or t.float64
    Hd = H.to(dtype)
    C = Hd.T @ Hd / Hd.shape[0]
    cbar = t.diagonal(C).mean()
    return C + lam * cbar * t.eye(C.shape[0], dtype=dtype, device=C.device)


def metric_transform(C_lambda, p: float):
    t = _torch()
    lam, Q = t.linalg.eigh(C_lambda)
    T = (Q * lam.pow(p)) @ Q.T
    Tinv = (Q * lam.pow(-p)) @ Q.T
    return T, Tinv


def _fix_signs(U, Vt):
    """Make the largest-magnitude entry of each left singular vector positive
    (flipping the matching right vector)."""
    t = _torch()
    idx = U.abs().argmax(dim=0)
    sgn = t.sign(U[idx, t.arange(U.shape[1], device=U.device)])
    sgn = t.where(sgn == 0, t.ones_like(sgn), sgn)
    return U * sgn[None, :], Vt * sgn[:, None]


def randomized_svd(A, r: int, omega, power_iters: int = 2):
    """Rank-r truncated SVD of A from the range of A omega, refined by
    `power_iters` rounds of A (A^T Q) with re-orthonormalisation."""
    t = _torch()
    Y = A @ omega.to(A.dtype)
    Q, _ = t.linalg.qr(Y)
    for _ in range(power_iters):
        Z, _ = t.linalg.qr(A.T @ Q)
        Q, _ = t.linalg.qr(A @ Z)
    B = Q.T @ A
    Ub, S, Vt = t.linalg.svd(B, full_matrices=False)
    U = Q @ Ub
    U, Vt = _fix_signs(U[:, :r], Vt[:r])
    return U, S[:r], Vt


def quantize(x, group_rows: int, group_cols: int, bits: int):
    """Library quantiser: int8 codes and fp16 scale bits (int16 tensor) of the fp32 matrix x."""
    t = _torch()
    x = x.to(t.float32).contiguous()
    R, C = x.shape
    codes = t.empty((R, C), dtype=t.int8, device=x.device)
    scales = t.empty((R // group_rows, C // group_cols), dtype=t.int16, device=x.device)
    archead.archead_quantize_symmetric(x, group_rows, group_cols, bits, codes, scales)
    return codes, scales


def dequantize(codes, scales, group_rows: int, group_cols: int):
    t = _torch()
    out = t.empty(codes.shape, dtype=t.float32, device=codes.device)
    archead.archead_dequant_symmetric(codes, scales, group_rows, group_cols, out)
    return out


def pack(codes, bits: int):
    t = _torch()
    R, C = codes.shape
    nb = (C + 1) // 2 if bits == 4 else (5 * C + 7) // 8
    out = t.empty((R, nb), dtype=t.uint8, device=codes.device)
    if R and C:
        archead.archead_pack_codes(codes.contiguous(), bits, out)
    return out


def construct(W, H, core_rank: int, corr_rank: int, group_size: int, p: float = 0.75, lam: float = 1e-3,
              fmt: str = "int8", omega_core=None, omega_corr=None, power_iters: int = 2, dtype=None,
              keep_intermediates: bool = False) -> Dict[str, object]:
    """Packed head of dense W [V, D] from calibration states H [N, D] (torch
    CUDA tensors).  dtype: precision of the dense linear algebra (float64 by
    default; the quantisers always decide in fp32).  Returns torch tensors in
    the canonical layout of the chosen format (numpy-compatible dtypes)."""
    t = _torch()
    dtype = dtype or t.float64
    dev = W.device
    V, D = W.shape
    g = group_size
    if D % g:
        raise ValueError("D must be a multiple of the group size")
    Wd = W.to(dtype)
    # Activation metric.
    C = damped_covariance(H, lam, dtype)
    T, Tinv = metric_transform(C, p)
    # QuantizeCore.
    head: Dict[str, object] = {}
    if core_rank > 0:
        if omega_core is None:
            raise ValueError("omega_core (D x k random test matrix) is required")
        U, S, Vt = randomized_svd(Wd, core_rank, omega_core.to(dev), power_iters)
        A_c = U * S.sqrt()[None, :]
        B_c = S.sqrt()[:, None] * Vt
        cu_codes, cu_s = quantize(A_c, V, 1, 5 if fmt == "sc4" else 8)
        cv_codes, cv_s = quantize(B_c.T, D, 1, 8)
        core = dequantize(cu_codes, cu_s, V, 1).to(dtype) @ dequantize(cv_codes, cv_s, D, 1).to(dtype).T
        resid = Wd - A_c @ B_c
    else:
        cu_codes = t.zeros((V, 0), dtype=t.int8, device=dev)
        cu_s = cv_s = t.zeros((1, 0), dtype=t.int16, device=dev)
        cv_codes = t.zeros((D, 0), dtype=t.int8, device=dev)
        core = t.zeros((V, D), dtype=dtype, device=dev)
        resid = Wd
    resid32 = resid.to(t.float32).contiguous()
    if fmt == "sc4":
        rc = t.empty((V, D), dtype=t.int8, device=dev)
        rq = t.empty((V, D // g), dtype=t.uint8, device=dev)
        rs = t.empty(V, dtype=t.int16, device=dev)
        archead.archead_quantize_residual_sc4(resid32, g, rc, rq, rs)
        res_deq = t.empty((V, D), dtype=t.float32, device=dev)
        archead.archead_dequant_residual_sc4(rc, rq, rs, g, res_deq)
        head["res_codes"] = pack(rc, 4)
        head["res_scale_codes"] = pack(rq.view(t.int8), 4)
        head["res_row_scale"] = rs
        head["core_u5"] = pack(cu_codes, 5) if core_rank else t.zeros((V, 0), dtype=t.uint8, device=dev)
    else:
        rc, rs = quantize(resid32, 1, g, 4)
        res_deq = dequantize(rc, rs, 1, g)
        head["res_codes"] = pack(rc, 4)
        head["res_scales"] = rs
        head["core_u"] = cu_codes
    head["core_u_scale"] = cu_s.reshape(-1)
    head["core_v"] = cv_codes
    head["core_v_scale"] = cv_s.reshape(-1)
    # Realized core error and its correction in the metric.
    W_core = core + res_deq.to(dtype)
    E = Wd - W_core
    if corr_rank > 0:
        if omega_corr is None:
            raise ValueError("omega_corr (D x k random test matrix) is required")
        U2, S2, V2t = randomized_svd(E @ T, corr_rank, omega_corr.to(dev), power_iters)
        A_w = U2 * S2[None, :]
        B_w = V2t @ Tinv
        ca, sa = quantize(A_w, 1, corr_rank, 8)
        cb, sb = quantize(B_w.T, g, 1, 8)
    else:
        A_w = t.zeros((V, 0), dtype=dtype, device=dev)
        B_w = t.zeros((0, D), dtype=dtype, device=dev)
        ca, sa = t.zeros((V, 0), dtype=t.int8, device=dev), t.zeros((V, 1), dtype=t.int16, device=dev)
        cb, sb = t.zeros((D, 0), dtype=t.int8, device=dev), t.zeros((D // g, 0), dtype=t.int16, device=dev)
    head["corr_a"] = ca
    head["corr_a_scale"] = sa.reshape(-1)
    head["corr_b"] = cb
    head["corr_b_scale"] = sb
    head = {k: v.contiguous() for k, v in head.items()}
    if keep_intermediates:
        head.update({"_T": T, "_Tinv": Tinv, "_W_d": W_core, "_E": E, "_A_w": A_w, "_B_w": B_w})
    return head


def to_numpy(head: Dict[str, object]) -> Dict[str, object]:
    """Canonical arrays as numpy (fp16 bits as uint16), ready for
    archead_pack_create or the oracle."""
    import numpy as np

    out = {}
    for k, v in head.items():
        if k.startswith("_"):
            continue
        a = v.cpu().numpy()
        if a.dtype == np.int16:
            a = a.view(np.uint16)
        out[k] = np.ascontiguousarray(a)
    return out
