"""Shared helpers of the GPU parity tests: upload synthetic inputs, call the
library through its C ABI, compare with the oracle under the stated bars."""

from __future__ import annotations

import numpy as np

from paper_2608_02703_gb300 import archead

# Acceptance bars (floating point): logits max|d| <= 1e-2 * rms(oracle logits),
# per-token CE |d| <= 1e-3 nats, argmax exact where the top-2 gap > 1e-2.
LOGIT_REL = 1e-2
CE_ABS = 1e-3
ARGMAX_GAP = 1e-2


def torch():
    import torch as _t

    return _t


def to_dev(a: np.ndarray):
    t = torch()
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return t.from_numpy(np.ascontiguousarray(a)).cuda()


def forward(pack, x_bits: np.ndarray, out_dtype=archead.OUT_FP32, path=archead.PATH_AUTO) -> np.ndarray:
    t = torch()
    M = x_bits.shape[0]
    V = pack.shape.V
    dt = t.float32 if out_dtype == archead.OUT_FP32 else t.bfloat16
    y = t.full((M, V), float("nan"), dtype=dt, device="cuda")
    archead.archead_forward_path(pack, to_dev(x_bits), M, y, out_dtype, path)
    assert archead.archead_sync_status(pack) == archead.OK
    return y.float().cpu().numpy().astype(np.float64)


def forward_ce(pack, x_bits: np.ndarray, targets: np.ndarray, path=archead.PATH_AUTO):
    t = torch()
    M = x_bits.shape[0]
    ce = t.full((M,), float("nan"), dtype=t.float32, device="cuda")
    archead.archead_forward_ce_path(pack, to_dev(x_bits), M, to_dev(targets.astype(np.int32)), ce, path)
    st = archead.archead_sync_status(pack)
    return ce.cpu().numpy().astype(np.float64), st


def bf16_half_ulp(y: np.ndarray) -> np.ndarray:
    a = np.abs(y)
    e = np.floor(np.log2(np.maximum(a, 1e-30)))
    return np.where(a > 0, 2.0 ** (e - 8), 0.0)  # half of 2^(e-7)


def check_logits(got: np.ndarray, ref: np.ndarray, bf16: bool = False, where: str = "") -> float:
    assert got.shape == ref.shape
    assert np.all(np.isfinite(got)), f"{where}: non-finite logits"
    rms = float(np.sqrt(np.mean(ref ** 2)))
    err = np.abs(got - ref)
    bound = LOGIT_REL * rms + (bf16_half_ulp(ref) if bf16 else 0.0)
    worst = float(np.max(err - bound))
    assert worst <= 0, f"{where}: max|d|={err.max():.4e} exceeds bound (rms={rms:.4e})"
    return float(err.max() / rms)


def check_argmax(got: np.ndarray, ref: np.ndarray, where: str = "") -> int:
    srt = np.sort(ref, axis=1)
    gap = srt[:, -1] - srt[:, -2] if ref.shape[1] > 1 else np.full(ref.shape[0], np.inf)
    sel = gap > ARGMAX_GAP
    a_got = np.argmax(got, axis=1)
    a_ref = np.argmax(ref, axis=1)
    bad = np.nonzero(sel & (a_got != a_ref))[0]
    assert bad.size == 0, f"{where}: argmax differs for tokens {bad[:8]}"
    return int(sel.sum())


def forward_argmax(pack, x_bits: np.ndarray, path=archead.PATH_AUTO):
    t = torch()
    M = x_bits.shape[0]
    idx = t.full((M,), -1, dtype=t.int32, device="cuda")
    val = t.full((M,), float("nan"), dtype=t.float32, device="cuda")
    archead.archead_forward_argmax_path(pack, to_dev(x_bits), M, idx, val, path)
    assert archead.archead_sync_status(pack) == archead.OK
    return idx.cpu().numpy().astype(np.int64), val.cpu().numpy().astype(np.float64)


def check_greedy(idx: np.ndarray, val: np.ndarray, ref: np.ndarray, where: str = "") -> None:
    """Greedy output against oracle logits: the index must be the oracle's
    argmax wherever the top-2 gap exceeds ARGMAX_GAP, and must always name a
    row whose oracle logit is within the logit bar of the maximum; the value
    must be the logit of that row within the logit bar."""
    rms = float(np.sqrt(np.mean(ref ** 2)))
    tol = LOGIT_REL * rms
    M = ref.shape[0]
    assert np.all((idx >= 0) & (idx < ref.shape[1])), f"{where}: index out of range"
    srt = np.sort(ref, axis=1)
    gap = srt[:, -1] - srt[:, -2] if ref.shape[1] > 1 else np.full(M, np.inf)
    a_ref = np.argmax(ref, axis=1)
    sel = gap > ARGMAX_GAP
    bad = np.nonzero(sel & (idx != a_ref))[0]
    assert bad.size == 0, f"{where}: greedy index differs for tokens {bad[:8]}"
    picked = ref[np.arange(M), idx]
    assert np.all(srt[:, -1] - picked <= 2 * tol), f"{where}: greedy index names a row far below the maximum"
    assert np.all(np.abs(val - picked) <= tol), f"{where}: greedy value max|d|={np.max(np.abs(val - picked)):.3e}"


def ce_bound(ref: dict) -> np.ndarray:
    """Per-token CE bar: CE_ABS, widened where the logits are so large that
    fp32 cannot resolve it.  The kernels carry each logit in fp32 and build
    it from sums whose terms reach CE_REL_LOGIT^-1 times the logit's own
    size (biased residual operands, the bf16 hi/lo split of t), so a logit
    of size L is resolved to about CE_REL_LOGIT * L; CE, a difference of two
    logits, gets twice that.  At logit rms ~2 the widening is below 1e-4."""
    big = np.maximum(np.abs(ref["target_logit"]), np.abs(ref["ce"] + ref["target_logit"]))
    return CE_ABS + 2.0 * CE_REL_LOGIT * big


# Relative resolution of a logit computed by the kernels (see ce_bound).
CE_REL_LOGIT = 2.0 ** -14
