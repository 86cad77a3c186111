"""Pins of the construction oracle (oracle/construct.py; paper Section 3.4,
Algorithm 1) against what the paper and the mathematics fix, CPU only:

- the metric transform: T_p T_p^-1 = I, T_1/2 squared = C_lambda, T_0 = I;
  Eq. 1's identity (1/N) ||H Delta^T||^2 = Tr(Delta C Delta^T);
- the conditional optimum of Section 3.2 (Eckart-Young-Mirsky): with the
  exact SVD the correction's error in the metric equals the tail of the
  squared singular values of E T_p, and random rank-r alternatives do worse;
  the randomized range finder recovers a known spectrum;
- the quantisers: code range, half-step rounding error, the maximum landing
  on +-qmax, zero groups, fp16 scales; the packers against the oracle's own
  (pinned) decoders;
- end to end: the stored head decodes (through oracle.dequant_rows, the
  forward oracle) to the realized core plus the quantised correction, and
  the correction lowers the metric error, in both packed formats.
"""

import numpy as np
import pytest

import oracle
from oracle import construct as oc
from synth import HeadShape, make_dense_head, make_hidden, make_test_matrix


def _H(D, N, seed=1):
    return oracle.bf16_values(make_hidden(D, N, seed=seed))


def test_metric_transform_identities():
    D, N = 64, 512
    C = oc.damped_covariance(_H(D, N), 1e-3)
    T, Tinv = oc.metric_transform(C, 0.75)
    assert np.allclose(T @ Tinv, np.eye(D), atol=1e-9)
    T2, _ = oc.metric_transform(C, 0.5)
    assert np.allclose(T2 @ T2, C, rtol=1e-9, atol=1e-12 * np.abs(C).max())
    T0, T0inv = oc.metric_transform(C, 0.0)
    assert np.allclose(T0, np.eye(D), atol=1e-12) and np.allclose(T0inv, np.eye(D), atol=1e-12)
    # lambda * cbar on the diagonal, cbar = mean diagonal of H^T H / N
    H = _H(D, N)
    raw = H.T @ H / N
    assert np.allclose(np.diag(C - raw), 1e-3 * np.mean(np.diag(raw)), rtol=1e-12)


def test_logit_error_identity_eq1():
    D, N, V = 48, 300, 40
    H = _H(D, N)
    rng = np.random.default_rng(2)
    Delta = rng.standard_normal((V, D))
    lhs = np.sum((H @ Delta.T) ** 2) / N
    C = H.T @ H / N
    assert np.isclose(lhs, np.trace(Delta @ C @ Delta.T), rtol=1e-10)
    # and with the damped metric at p = 1/2: Tr(Delta C_lambda Delta^T) = ||Delta T_1/2||^2
    Cl = oc.damped_covariance(H, 1e-3)
    T, _ = oc.metric_transform(Cl, 0.5)
    assert np.isclose(np.trace(Delta @ Cl @ Delta.T), np.sum((Delta @ T) ** 2), rtol=1e-10)


def test_conditional_optimum_eckart_young():
    V, D, N, r = 300, 64, 500, 6
    W = make_dense_head(V, D, seed=3).astype(np.float64)
    H = _H(D, N)
    h = oc.construct(W, H, core_rank=8, corr_rank=r, group_size=32, p=0.75)
    T, E = h["_T"], h["_E"]
    s = np.linalg.svd(E @ T, compute_uv=False)
    best = oc.metric_error(E, h["_A_w"] @ h["_B_w"], T)
    assert np.isclose(best, np.sum(s[r:] ** 2), rtol=1e-9)
    rng = np.random.default_rng(4)
    for _ in range(5):  # any other rank-r correction does worse
        A = h["_A_w"] + 0.05 * rng.standard_normal(h["_A_w"].shape) * np.abs(h["_A_w"]).mean()
        B = h["_B_w"] + 0.05 * rng.standard_normal(h["_B_w"].shape) * np.abs(h["_B_w"]).mean()
        assert oc.metric_error(E, A @ B, T) > best
    # the unquantised correction factors satisfy A_w = U S, B_w = V^T T^-1
    U, S, Vt = oc.truncated_svd(E @ T, r)
    assert np.allclose(h["_A_w"] @ h["_B_w"] @ T, (U * S) @ Vt, atol=1e-10 * np.abs(E).max())


def test_randomized_svd_recovers_a_known_spectrum():
    rng = np.random.default_rng(5)
    m, n, r = 400, 120, 8
    U, _ = np.linalg.qr(rng.standard_normal((m, n)))
    V, _ = np.linalg.qr(rng.standard_normal((n, n)))
    # a gap after the first r values: the range finder's error falls as
    # (s_{r+1} / s_r)^(2 q + 1) with q power iterations
    s = np.concatenate([np.geomspace(10, 5, r), np.geomspace(1e-2, 1e-4, n - r)])
    A = (U * s) @ V.T
    Ur, Sr, Vr = oc.truncated_svd(A, r, make_test_matrix(n, r + 10, seed=5), power_iters=2)
    assert np.allclose(Sr, s[:r], rtol=1e-8)
    Ue, Se, Ve = oc.truncated_svd(A, r)
    assert np.allclose(Ur, Ue, atol=1e-6) and np.allclose(Vr, Ve, atol=1e-6)  # same signs after the fix
    assert np.all(Ur[np.argmax(np.abs(Ur), axis=0), np.arange(r)] > 0)


@pytest.mark.parametrize("bits", [8, 5, 4])
@pytest.mark.parametrize("groups", [(1, 16), (24, 1), (4, 4)])
def test_symmetric_quantiser(bits, groups):
    gr, gc = groups
    rng = np.random.default_rng(bits)
    x = (rng.standard_normal((48, 32)) * np.exp2(rng.integers(-6, 6, (48, 32)))).astype(np.float32)
    x[:gr, :gc] = 0.0  # an all-zero group
    q, s16 = oc.quantize_symmetric(x, gr, gc, bits)
    qmax = oc.QMAX[bits]
    assert q.dtype == np.int8 and np.all(np.abs(q.astype(int)) <= qmax)
    s = s16.view(np.float16).astype(np.float64)
    assert s[0, 0] == 0 and np.all(q[:gr, :gc] == 0)
    sf = np.repeat(np.repeat(s, gr, 0), gc, 1)
    err = np.abs(x - q * sf)
    assert np.all(err <= 0.5 * sf * (1 + 1e-6) + (sf == 0) * 0)
    # the group maximum lands on +-qmax (the scale is its fp16-rounded 1/qmax)
    blocks = np.abs(q.astype(int)).reshape(48 // gr, gr, 32 // gc, gc).max(axis=(1, 3))
    nz = s > 0
    assert np.all(blocks[nz] >= qmax - 1)
    mx = np.abs(x).reshape(48 // gr, gr, 32 // gc, gc).max(axis=(1, 3))
    assert np.array_equal(s16, (mx / np.float32(qmax)).astype(np.float16).view(np.uint16))


def test_residual_quantiser_of_the_papers_format():
    rng = np.random.default_rng(7)
    r = (rng.standard_normal((40, 256)) * np.exp2(rng.integers(-4, 3, (40, 1)))).astype(np.float32)
    r[3] = 0.0
    c, q, s16 = oc.quantize_residual_sc4(r, 64)
    assert np.all(np.abs(c.astype(int)) <= 7) and np.all(q <= 15)
    s_row = s16.view(np.float16).astype(np.float64)
    sg = s_row[:, None] * (q.astype(np.float64) + 1)
    gmax = np.abs(r.astype(np.float64)).reshape(40, 4, 64).max(axis=2)
    ok = s_row > 0
    # every group's maximum is within rounding of a code: s_row may round
    # below max / 112 by 2^-11, so the largest group can sit at 7.003 steps
    assert np.all(7.5 * sg[ok] >= gmax[ok])
    assert np.all(np.abs(r - c * np.repeat(sg, 64, 1)) <= 0.5 * np.repeat(sg, 64, 1) * (1 + 1e-6))
    assert s_row[3] == 0 and np.all(c[3] == 0) and np.all(q[3] == 0)


def test_packers_against_the_oracle_decoders():
    rng = np.random.default_rng(8)
    c4 = rng.integers(-8, 8, (9, 34)).astype(np.int8)
    assert np.array_equal(oracle.unpack_int4(oc.pack_int4(c4)), c4)
    for r in (1, 3, 10, 13):
        c5 = rng.integers(-16, 16, (7, r)).astype(np.int8)
        assert np.array_equal(oracle.unpack_int5(oc.pack_int5(c5), r), c5)
    for G in (4, 5):
        q = rng.integers(0, 16, (6, G))
        assert np.array_equal(oracle.unpack_scale_codes(oc.pack_scale_codes(q), G), q)


@pytest.mark.parametrize("fmt,ranks,g", [("int8", (16, 8), 64), ("sc4", (10, 6), 64), ("int8", (0, 8), 32),
                                         ("int8", (8, 0), 64)])
def test_constructed_head_decodes_to_the_realized_core_plus_correction(fmt, ranks, g):
    V, D, N = 320, 128, 512
    rc, rr = ranks
    W = make_dense_head(V, D, seed=9).astype(np.float64)
    H = _H(D, N)
    h = oc.construct(W, H, rc, rr, g, fmt=fmt, omega_core=make_test_matrix(D, rc + 10, 1) if rc else None,
                     omega_corr=make_test_matrix(D, rr + 10, 2) if rr else None)
    shape = HeadShape(V=V, d=D, core_rank=rc, corr_rank=rr, group_size=g, fmt=fmt)
    Wq = oracle.dequant_rows(oc.canonical(h), shape)
    # the stored correction, dequantised
    if rr:
        ca = h["corr_a"].astype(np.float64) * h["corr_a_scale"].view(np.float16).astype(np.float64)[:, None]
        sb = np.repeat(h["corr_b_scale"].view(np.float16).astype(np.float64), g, axis=0)
        corr = ca @ (h["corr_b"].astype(np.float64) * sb).T
    else:
        corr = 0.0
    assert np.allclose(Wq, h["_W_d"] + corr, rtol=0, atol=1e-12 * np.abs(W).max())
    T = h["_T"]
    e_core = oc.metric_error(W, h["_W_d"], T)
    e_full = oc.metric_error(W, Wq, T)
    if rr:
        assert e_full < 0.5 * e_core, (e_full, e_core)
    assert np.all(np.isfinite(Wq))
