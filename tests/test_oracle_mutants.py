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
    "residual_scale_group": ("double s_r = res_scale(h, n, k / g);",
                             "double s_r = res_scale(h, n, (k / g + 1) % (d / g));"),
    "int8_residual_scale_row": ("return oracle_fp16_value(h->res_scales[n * G + grp]);",
                                "return oracle_fp16_value(h->res_scales[((n + 1) % h->V) * G + grp]);"),
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
    "bytes_scale_dropped": ("bytes += G * rr * 2;     /* correction group scales */", "bytes += 0;"),
    # the paper's packed format (5-bit core codes, 4-bit group-scale codes)
    "int5_sign_extension": ("return v >= 16 ? v - 32 : v;", "return v >= 16 ? v - 31 : v;"),
    "int5_bit_order": ("v |= ((row[bit / 8] >> (bit % 8)) & 1) << b;", "v |= ((row[bit / 8] >> (bit % 8)) & 1) << (4 - b);"),
    "int5_row_stride": ("h->core_u5 + n * ((5 * (int64_t)h->core_rank + 7) / 8)",
                        "h->core_u5 + n * ((5 * (int64_t)h->core_rank) / 8)"),
    "scale_code_offset_dropped": ("scale_code(h->res_scale_codes + n * nb, grp) + 1);",
                                  "scale_code(h->res_scale_codes + n * nb, grp) + 0);"),
    "scale_code_nibble_order": ("return (grp % 2 == 0) ? (byte & 0x0F)", "return (grp % 2 == 1) ? (byte & 0x0F)"),
    "scale_code_row_stride": ("const int64_t nb = (G + 1) / 2;\n    return", "const int64_t nb = G / 2;\n    return"),
    "row_scale_index": ("oracle_fp16_value(h->res_row_scale[n])", "oracle_fp16_value(h->res_row_scale[(n + 1) % h->V])"),
    "sc4_bytes_row_scales_dropped": ("bytes += V * 2;                /* residual row scales", "bytes += 0;  /*"),
    "sc4_bytes_core_unpacked": ("bytes += V * ((5 * rc + 7) / 8);", "bytes += V * rc;"),
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
