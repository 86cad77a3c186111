"""Pins of the construction oracle (paper, Section 3.4, Algorithm 1), written
as functions of the module under test so that the same checks run on the
oracle itself (test_construct_oracle.py) and on planted mistakes in copies
of it (test_construct_mutants.py).  Every check is fixed by the paper or by
the mathematics, never by the oracle's own output:

- the metric transform (Section 3.1): T_p T_p^-1 = I, T_1/2^2 = C_lambda,
  T_0 = I, lambda * cbar on the diagonal; Eq. 1's identity
  (1/N) ||H Delta^T||^2 = Tr(Delta C Delta^T);
- the conditional optimum (Section 3.2, Eckart-Young-Mirsky) and the
  randomized range finder on a known spectrum;
- QuantizeCore: balanced factors A_c = U S^1/2, B_c = S^1/2 V^T, the
  residual taken against the unquantised core (Appendix B);
- the quantisers (code range, half-step error, maximum on +-qmax, fp16
  scales) and the paper's SC4 scale codes (each group's code is the
  smallest that covers its maximum; the largest group uses the top codes);
- the packers against the forward oracle's (separately pinned) decoders;
- end to end: the stored head decodes, through the forward oracle, to the
  realized core plus the quantised correction, W - E is that realized core,
  and the correction lowers the metric error.
"""

import numpy as np

import oracle
from synth import HeadShape, make_dense_head, make_hidden, make_test_matrix


def _H(D, N, seed=1):
    return oracle.bf16_values(make_hidden(D, N, seed=seed))


def check_metric_transform_identities(oc):
    D, N = 64, 512
    H = _H(D, N)
    C = oc.damped_covariance(H, 1e-3)
    T, Tinv = oc.metric_transform(C, 0.75)
    assert np.allclose(T @ Tinv, np.eye(D), atol=1e-9)
    T2, _ = oc.metric_transform(C, 0.5)
    assert np.allclose(T2 @ T2, C, rtol=1e-9, atol=1e-12 * np.abs(C).max())
    T0, T0inv = oc.metric_transform(C, 0.0)
    assert np.allclose(T0, np.eye(D), atol=1e-12) and np.allclose(T0inv, np.eye(D), atol=1e-12)
    raw = H.T @ H / N  # lambda * cbar on the diagonal, cbar = mean diagonal of H^T H / N
    assert np.allclose(np.diag(C - raw), 1e-3 * np.mean(np.diag(raw)), rtol=1e-9)
    off = ~np.eye(D, dtype=bool)
    assert np.allclose((C - raw)[off], 0.0, atol=1e-12 * np.abs(raw).max())


def check_logit_error_identity_eq1(oc):
    D, N, V = 48, 300, 40
    H = _H(D, N)
    rng = np.random.default_rng(2)
    Delta = rng.standard_normal((V, D))
    Cl = oc.damped_covariance(H, 0.0)  # lambda = 0: the plain covariance
    assert np.isclose(np.sum((H @ Delta.T) ** 2) / N, np.trace(Delta @ Cl @ Delta.T), rtol=1e-10)
    Cl = oc.damped_covariance(H, 1e-3)
    T, _ = oc.metric_transform(Cl, 0.5)
    assert np.isclose(np.trace(Delta @ Cl @ Delta.T), np.sum((Delta @ T) ** 2), rtol=1e-10)


def check_conditional_optimum_eckart_young(oc):
    V, D, N, r = 300, 64, 500, 6
    W = make_dense_head(V, D, seed=3).astype(np.float64)
    h = oc.construct(W, _H(D, N), core_rank=8, corr_rank=r, group_size=32, p=0.75)
    T, E = h["_T"], h["_E"]
    s = np.linalg.svd(E @ T, compute_uv=False)
    best = np.sum(((E - h["_A_w"] @ h["_B_w"]) @ T) ** 2)
    assert np.isclose(best, np.sum(s[r:] ** 2), rtol=1e-9)
    rng = np.random.default_rng(4)
    for _ in range(5):  # any other rank-r correction does worse
        A = h["_A_w"] + 0.05 * rng.standard_normal(h["_A_w"].shape) * np.abs(h["_A_w"]).mean()
        B = h["_B_w"] + 0.05 * rng.standard_normal(h["_B_w"].shape) * np.abs(h["_B_w"]).mean()
        assert np.sum(((E - A @ B) @ T) ** 2) > best
    # A_w = U S, B_w = V^T T^-1 for the SVD of E T: (A_w B_w) T = U S V^T, and
    # A_w's columns are orthogonal with norms the singular values.
    U, S, Vt = np.linalg.svd(E @ T, full_matrices=False)
    assert np.allclose(h["_A_w"] @ h["_B_w"] @ T, (U[:, :r] * S[:r]) @ Vt[:r], atol=1e-10 * np.abs(E).max())
    assert np.allclose(np.linalg.norm(h["_A_w"], axis=0), S[:r], rtol=1e-9)


def check_randomized_svd_recovers_a_known_spectrum(oc):
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
    assert np.allclose((Ur * Sr) @ Vr, (U[:, :r] * s[:r]) @ V[:, :r].T, atol=1e-8)
    Ue, Se, Ve = oc.truncated_svd(A, r)
    assert np.allclose(Se, s[:r], rtol=1e-12)
    assert np.allclose(Ur, Ue, atol=1e-6) and np.allclose(Vr, Ve, atol=1e-6)  # same signs after the fix
    assert np.all(Ur[np.argmax(np.abs(Ur), axis=0), np.arange(r)] > 0)


def _check_symmetric_quantiser(oc, bits, gr, gc):
    rng = np.random.default_rng(bits)
    x = (rng.standard_normal((48, 32)) * np.exp2(rng.integers(-6, 6, (48, 32)))).astype(np.float32)
    x[:gr, :gc] = 0.0  # an all-zero group
    q, s16 = oc.quantize_symmetric(x, gr, gc, bits)
    qmax = {8: 127, 5: 15, 4: 7}[bits]  # the bit width's symmetric range
    assert q.dtype == np.int8 and np.all(np.abs(q.astype(int)) <= qmax)
    s = s16.view(np.float16).astype(np.float64)
    assert s[0, 0] == 0 and np.all(q[:gr, :gc] == 0)
    sf = np.repeat(np.repeat(s, gr, 0), gc, 1)
    assert np.all(np.abs(x - q * sf) <= 0.5 * sf * (1 + 1e-6))
    blocks = np.abs(q.astype(int)).reshape(48 // gr, gr, 32 // gc, gc).max(axis=(1, 3))
    assert np.all(blocks[s > 0] >= qmax - 1)  # the group maximum lands on +-qmax
    mx = np.abs(x).reshape(48 // gr, gr, 32 // gc, gc).max(axis=(1, 3))
    assert np.array_equal(s16, (mx / np.float32(qmax)).astype(np.float16).view(np.uint16))


def check_symmetric_quantisers(oc):
    for bits in (8, 5, 4):
        for gr, gc in ((1, 16), (24, 1), (4, 4)):
            _check_symmetric_quantiser(oc, bits, gr, gc)


def check_residual_quantiser_of_the_papers_format(oc):
    rng = np.random.default_rng(7)
    r = (rng.standard_normal((40, 256)) * np.exp2(rng.integers(-4, 3, (40, 1)))).astype(np.float32)
    r[3] = 0.0
    r[5, 64:128] = 0.0  # one empty group in a non-empty row
    c, q, s16 = oc.quantize_residual_sc4(r, 64)
    assert np.all(np.abs(c.astype(int)) <= 7) and np.all(q <= 15)
    s_row = s16.view(np.float16).astype(np.float64)
    sg = s_row[:, None] * (q.astype(np.float64) + 1)
    gmax = np.abs(r.astype(np.float64)).reshape(40, 4, 64).max(axis=2)
    ok = s_row > 0
    # every group's maximum is within rounding of a code (s_row may round
    # below max / 112 by 2^-11, so the largest group can sit at 7.003 steps)
    assert np.all(7.5 * sg[ok] >= gmax[ok])
    assert np.all(np.abs(r - c * np.repeat(sg, 64, 1)) <= 0.5 * np.repeat(sg, 64, 1) * (1 + 1e-6))
    assert s_row[3] == 0 and np.all(c[3] == 0) and np.all(q[3] == 0)
    # q is the smallest code whose scale reaches the group's maximum at 7
    # steps (up to fp32 rounding; the top code may be clipped), and s_row
    # puts the row's largest group on the top codes
    reach = 7.0 * s_row[:, None] * (q + 1.0)
    below = 7.0 * s_row[:, None] * q
    rows = ok.nonzero()[0]
    assert np.all(((q == 15) | (reach >= gmax * (1 - 1e-6)))[rows])
    assert np.all(((q == 0) | (below < gmax * (1 + 1e-6)))[rows])
    assert np.all(q.max(axis=1)[rows] >= 14)
    assert q[5, 1] == 0 and np.all(c[5, 64:128] == 0)


def check_packers_against_the_oracle_decoders(oc):
    rng = np.random.default_rng(8)
    c4 = rng.integers(-8, 8, (9, 34)).astype(np.int8)
    assert np.array_equal(oracle.unpack_int4(oc.pack_int4(c4)), c4)
    for r in (1, 3, 10, 13):
        c5 = rng.integers(-16, 16, (7, r)).astype(np.int8)
        assert np.array_equal(oracle.unpack_int5(oc.pack_int5(c5), r), c5)
    for G in (4, 5):
        q = rng.integers(0, 16, (6, G))
        assert np.array_equal(oracle.unpack_scale_codes(oc.pack_scale_codes(q), G), q)


def _constructed(oc, fmt, rc, rr, g, V=320, D=128, N=512):
    W = make_dense_head(V, D, seed=9).astype(np.float64)
    h = oc.construct(W, _H(D, N), rc, rr, g, fmt=fmt, omega_core=make_test_matrix(D, rc + 10, 1) if rc else None,
                     omega_corr=make_test_matrix(D, rr + 10, 2) if rr else None)
    return W, h, HeadShape(V=V, d=D, core_rank=rc, corr_rank=rr, group_size=g, fmt=fmt)


def check_core_factors_are_balanced(oc):
    """QuantizeCore splits the rank-r_c SVD as A_c = U S^1/2, B_c = S^1/2 V^T:
    column j of A_c and row j of B_c have the same norm sqrt(s_j)."""
    for fmt in ("int8", "sc4"):
        W, h, _ = _constructed(oc, fmt, 10, 6, 64)
        na, nb = np.linalg.norm(h["_A_c"], axis=0), np.linalg.norm(h["_B_c"], axis=1)
        assert np.allclose(na, nb, rtol=1e-9)
        # their product is the rank-10 approximation's singular values (from a
        # randomized range finder: close to, not equal to, the exact ones)
        s = np.linalg.svd(W, compute_uv=False)[:10]
        assert np.allclose(na * nb, s, rtol=5e-2)


def check_residual_is_taken_against_the_unquantised_core(oc):
    """Appendix B: the residual quantised to INT4 is W - A_c B_c (the core
    before its factors are quantised); each stored code is within half a
    step of it."""
    for fmt in ("int8", "sc4"):
        W, h, shape = _constructed(oc, fmt, 10, 0, 64)
        resid = W - h["_A_c"] @ h["_B_c"]
        codes = oracle.unpack_int4(h["res_codes"]).astype(np.float64)
        if fmt == "sc4":
            q = oracle.unpack_scale_codes(h["res_scale_codes"], W.shape[1] // 64).astype(np.float64)
            sg = h["res_row_scale"].view(np.float16).astype(np.float64)[:, None] * (q + 1)
        else:
            sg = h["res_scales"].view(np.float16).astype(np.float64)
        step = np.repeat(sg, 64, axis=1)
        assert np.all(np.abs(resid - codes * step) <= 0.5 * step * (1 + 1e-6) + 1e-12)


def check_constructed_head_decodes_to_the_realized_core_plus_correction(oc):
    for fmt, (rc, rr), g in (("int8", (16, 8), 64), ("sc4", (10, 6), 64), ("int8", (0, 8), 32), ("int8", (8, 0), 64)):
        W, h, shape = _constructed(oc, fmt, rc, rr, g, D=128)
        can = oc.canonical(h)
        Wq = oracle.dequant_rows(can, shape)
        if rr:
            ca = h["corr_a"].astype(np.float64) * h["corr_a_scale"].view(np.float16).astype(np.float64)[:, None]
            sb = np.repeat(h["corr_b_scale"].view(np.float16).astype(np.float64), g, axis=0)
            corr = ca @ (h["corr_b"].astype(np.float64) * sb).T
        else:
            corr = 0.0
        assert np.allclose(Wq, h["_W_d"] + corr, rtol=0, atol=1e-12 * np.abs(W).max())
        # E is measured against what was stored: W - E is the forward oracle's
        # dequantisation of the stored core and residual alone.
        core_only = dict(can)
        core_only["corr_a"] = np.zeros((shape.V, 0), np.int8)
        core_only["corr_a_scale"] = np.zeros(shape.V, np.uint16)
        core_only["corr_b"] = np.zeros((shape.d, 0), np.int8)
        core_only["corr_b_scale"] = np.zeros((shape.d // g, 0), np.uint16)
        shape0 = HeadShape(V=shape.V, d=shape.d, core_rank=rc, corr_rank=0, group_size=g, fmt=fmt)
        assert np.allclose(W - h["_E"], oracle.dequant_rows(core_only, shape0), rtol=0,
                           atol=1e-12 * np.abs(W).max())
        T = h["_T"]
        e_core = oc.metric_error(W, h["_W_d"], T)
        e_full = oc.metric_error(W, Wq, T)
        if rr:
            assert e_full < 0.5 * e_core, (e_full, e_core)
        assert np.all(np.isfinite(Wq))


ALL_CHECKS = [
    check_metric_transform_identities,
    check_logit_error_identity_eq1,
    check_conditional_optimum_eckart_young,
    check_randomized_svd_recovers_a_known_spectrum,
    check_symmetric_quantisers,
    check_residual_quantiser_of_the_papers_format,
    check_packers_against_the_oracle_decoders,
    check_core_factors_are_balanced,
    check_residual_is_taken_against_the_unquantised_core,
    check_constructed_head_decodes_to_the_realized_core_plus_correction,
]
