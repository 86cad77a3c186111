"""Plant plausible mistakes in copies of the construction oracle and check
that the pins (construct_pins.py) reject every one.

Each mutant is oracle/construct.py with one edit: a dropped or misplaced
factor, a wrong exponent sign, a transposed operand, a scale on the wrong
axis, an off-by-one in a code range, the core subtracted after instead of
before quantisation, and so on.  The unmodified oracle passes the same pins
(test_construct_oracle.py)."""

import importlib.util
import os

import pytest

import oracle
from tests import construct_pins

SRC = os.path.join(os.path.dirname(os.path.abspath(oracle.__file__)), "construct.py")

MUTANTS = {
    "covariance_not_averaged": ("C = H.T @ H / H.shape[0]", "C = H.T @ H"),
    "damping_not_scaled_by_cbar": ("return C + lam * cbar * np.eye(C.shape[0])", "return C + lam * np.eye(C.shape[0])"),
    "cbar_trace_not_mean": ("cbar = float(np.mean(np.diag(C)))", "cbar = float(np.sum(np.diag(C)))"),
    "metric_inverse_sign": ("Tinv = (Q * lam ** (-p)) @ Q.T", "Tinv = (Q * lam ** (p)) @ Q.T"),
    "metric_transposed": ("T = (Q * lam ** p) @ Q.T", "T = (Q.T * lam ** p) @ Q"),
    "no_power_iterations": ("for _ in range(power_iters):", "for _ in range(0):"),
    "right_vectors_misaligned": ("U = Q @ Ub\n    return _fix_signs(U[:, :r], S[:r], Vt[:r])",
                                 "U = Q @ Ub\n    return _fix_signs(U[:, :r], S[:r], Vt[1:r + 1])"),
    "signs_not_fixed": ("sgn[sgn == 0] = 1.0", "sgn[:] = 1.0"),
    "core_split_unbalanced": ("A_c = U * np.sqrt(S)[None, :]\n        B_c = np.sqrt(S)[:, None] * Vt",
                              "A_c = U * S[None, :]\n        B_c = Vt"),
    "residual_against_quantised_core": ("resid = W - A_c @ B_c",
                                        "resid = W - (_deq(cu_codes, cu_s, V, 1) @ _deq(cv_codes, cv_s, D, 1).T "
                                        "if core_rank else 0.0)"),
    "error_against_unquantised_core": ("E = W - W_d\n    Et = E @ T", "E = W - (A_c @ B_c + res_deq)\n    Et = E @ T"),
    "correction_singular_values_dropped": ("A_w = U2 * S2[None, :]", "A_w = U2"),
    "correction_metric_not_undone": ("B_w = V2t @ Tinv", "B_w = V2t @ T"),
    "correction_not_in_metric": ("Et = E @ T", "Et = E"),
    "rounding_floor": ("q = np.rint(x32 / s_full)", "q = np.floor(x32 / s_full)"),
    "int5_range": ("QMAX = {8: 127, 5: 15, 4: 7}", "QMAX = {8: 127, 5: 16, 4: 7}"),
    "scale_off_by_one": ("s16 = _fp16_bits(mx / np.float32(qmax))", "s16 = _fp16_bits(mx / np.float32(qmax + 1))"),
    "corr_b_scale_per_row": ("cb, sb = quantize_symmetric(B_w.T, g, 1, 8)", "cb, sb = quantize_symmetric(B_w.T, 1, 1, 8)"),
    "corr_a_scale_per_column": ("ca, sa = quantize_symmetric(A_w, 1, corr_rank, 8)",
                                "ca, sa = quantize_symmetric(A_w, V, 1, 8)"),
    "sc4_row_scale_range": ("gmax.max(axis=1) / np.float32(7 * 16)", "gmax.max(axis=1) / np.float32(7)"),
    "sc4_code_not_minimal": ("np.clip(need - 1, 0, 15)", "np.clip(need, 0, 15)"),
    "int4_nibble_order": ("(c[:, 0::2] | (c[:, 1::2] << 4)).astype(np.uint8)",
                          "(c[:, 1::2] | (c[:, 0::2] << 4)).astype(np.uint8)"),
    "int5_bit_order": ("(c[:, :, None] >> np.arange(5)[None, None, :])", "(c[:, :, None] >> np.arange(4, -1, -1)[None, None, :])"),
    "scale_codes_nibble_order": ("return (q[:, 0::2] | (q[:, 1::2] << 4)).astype(np.uint8)",
                                 "return (q[:, 1::2] | (q[:, 0::2] << 4)).astype(np.uint8)"),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(name, source, tmp_path):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name} not found exactly once"
    path = tmp_path / f"construct_{name}.py"
    path.write_text(source.replace(old, new))
    spec = importlib.util.spec_from_file_location(f"construct_{name}", str(path))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    failures = []
    for check in construct_pins.ALL_CHECKS:
        try:
            check(mod)
        except Exception:  # a failed assertion, or the mutant breaking a shape
            failures.append(check.__name__)
    assert failures, f"no pin rejects the mutant {name}"
