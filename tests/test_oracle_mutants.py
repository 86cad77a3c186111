"""Plant plausible mistakes in copies of the oracle and check the pins fail.

Each mutant is the oracle's C source with one edit (a dropped term, a wrong
sign, index, scale axis or exponent bias, a transposed operand).  Every edit
keeps all memory accesses in bounds.  The pins of oracle_pins.py must reject
every mutant; the unmodified source must pass them (test_oracle_pins.py).
"""

import os
import subprocess

import pytest

import oracle
from tests import oracle_pins

SRC = os.path.join(os.path.dirname(os.path.abspath(oracle.__file__)), "archead_oracle.c")

MUTANTS = {
    "int4_sign_extension": ("return nib >= 8 ? nib - 16 : nib;", "return nib >= 8 ? nib - 15 : nib;"),
    "int4_nibble_order": ("int nib = (k % 2 == 0) ? (byte & 0x0F)", "int nib = (k % 2 == 1) ? (byte & 0x0F)"),
    "fp16_exponent_bias": ("v = ldexp((double)(1024 + f), e - 25);", "v = ldexp((double)(1024 + f), e - 24);"),
    "bf16_exponent_bias": ("v = ldexp((double)(128 + f), e - 134);", "v = ldexp((double)(128 + f), e - 135);"),
    "residual_scale_group": ("double s_r = oracle_fp16_value(h->res_scales[n * G + k / g]);",
                             "double s_r = oracle_fp16_value(h->res_scales[n * G + (k / g + 1) % G]);"),
    "core_scale_swapped": ("c->su[j] = oracle_fp16_value(h->core_u_scale[j]);",
                           "c->su[j] = oracle_fp16_value(h->core_v_scale[j]);"),
    "core_right_transposed": ("c->vdq[k * rc + j] = (double)h->core_v[k * rc + j]",
                              "c->vdq[k * rc + j] = (double)h->core_v[j * d + k]"),
    "corr_scale_table_transposed": ("h->corr_b_scale[(k / g) * rr + j]);\n  }\n  return 0;",
                                    "h->corr_b_scale[j * (d / g) + (k / g)]);\n  }\n  return 0;"),
    "corr_left_scale_per_column": ("a[j] = (double)h->corr_a[n * rr + j] * s_a;",
                                   "a[j] = (double)h->corr_a[n * rr + j] * oracle_fp16_value(h->corr_a_scale[j]);"),
    "correction_dropped": ("w[k] = v + core + corr;", "w[k] = v + core;"),
    "core_sign": ("w[k] = v + core + corr;", "w[k] = v - core + corr;"),
    "hidden_reversed": ("acc += x[m * d + k] * w[k];", "acc += x[m * d + (d - 1 - k)] * w[k];"),
    "lse_not_shifted": ("s += exp(row[n] - mx);", "s += exp(row[n]);"),
    "ce_wrong_logit": ("ce[m] = lse - row[t];", "ce[m] = lse - row[arg];"),
    "argmax_tie_high": ("if (row[n] > mx) { mx = row[n]; arg = n; }", "if (row[n] >= mx) { mx = row[n]; arg = n; }"),
    "bytes_scale_dropped": ("bytes += G * rr * 2;", "bytes += 0;"),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(name, source, tmp_path):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name} not found exactly once"
    path_c = tmp_path / f"{name}.c"
    path_so = tmp_path / f"{name}.so"
    path_c.write_text(source.replace(old, new))
    subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", str(path_so), str(path_c), "-lm"],
                   check=True)
    failures = []
    try:
        oracle.use_library(str(path_so))
        for check in oracle_pins.ALL_CHECKS:
            try:
                check(oracle)
            except AssertionError:
                failures.append(check.__name__)
    finally:
        oracle.use_library(None)
    assert failures, f"no pin rejects the mutant {name}"
