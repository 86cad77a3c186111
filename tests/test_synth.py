"""The seeded generator: determinism, layout and value ranges."""

import numpy as np

from synth import SHAPES, HeadShape, make_head, make_hidden, make_targets


def test_head_layout_and_determinism():
    shape = HeadShape(V=300, d=256, core_rank=16, corr_rank=8, group_size=64)
    a = make_head(shape, seed=5)
    b = make_head(shape, seed=5)
    c = make_head(shape, seed=6)
    expect = {
        "res_codes": (np.uint8, (300, 128)), "res_scales": (np.uint16, (300, 4)),
        "core_u": (np.int8, (300, 16)), "core_u_scale": (np.uint16, (16,)),
        "core_v": (np.int8, (256, 16)), "core_v_scale": (np.uint16, (16,)),
        "corr_a": (np.int8, (300, 8)), "corr_a_scale": (np.uint16, (300,)),
        "corr_b": (np.int8, (256, 8)), "corr_b_scale": (np.uint16, (4, 8)),
    }
    for k, (dt, shp) in expect.items():
        assert a[k].dtype == dt and a[k].shape == shp, k
        assert np.array_equal(a[k], b[k]), k
        assert not np.array_equal(a[k], c[k]), k
    for k in ("core_u", "core_v", "corr_a", "corr_b"):
        assert a[k].min() >= -127 and a[k].max() <= 127
    for k in ("res_scales", "core_u_scale", "core_v_scale", "corr_a_scale", "corr_b_scale"):
        v = a[k].view(np.float16).astype(np.float64)
        assert np.all(np.isfinite(v)) and np.all(v > 0), k
    # Every nibble value occurs, both in the low and the high half of a byte.
    assert len(np.unique(a["res_codes"] & 0xF)) == 16 and len(np.unique(a["res_codes"] >> 4)) == 16


def test_hidden_states_anisotropic():
    x = make_hidden(256, 64, seed=0, n_outliers=4)
    assert x.dtype == np.uint16 and x.shape == (64, 256)
    assert np.array_equal(x, make_hidden(256, 64, seed=0, n_outliers=4))
    xf = (x.astype(np.uint32) << 16).view(np.float32)
    rms = np.sqrt((xf.astype(np.float64) ** 2).mean(axis=0))
    # Four outlier channels stand far above the rest.
    top = np.sort(rms)[::-1]
    assert top[3] > 5 * np.median(rms) and top[4] < 5 * np.median(rms)


def test_targets_range():
    t = make_targets(1000, 5000, seed=1)
    assert t.dtype == np.int32 and t.min() >= 0 and t.max() < 1000
    assert np.array_equal(t, make_targets(1000, 5000, seed=1))


def test_named_shapes():
    assert SHAPES["qwen3-8b"].V == 151936 and SHAPES["qwen3-8b"].d == 4096
    assert SHAPES["gemma-4-e4b"].V == 262144 and SHAPES["gemma-4-e4b"].d == 2560
    assert SHAPES["gemma-4-e4b"].n_outliers == 8


def test_sc4_head_layout_and_ranges():
    """The paper's packed format: 5-bit core codes and 4-bit scale codes with
    zero padding bits, every field value drawn."""
    shape = HeadShape(V=500, d=320, core_rank=10, corr_rank=6, group_size=64, fmt="sc4")
    a = make_head(shape, seed=5)
    assert np.array_equal(a["core_u5"], make_head(shape, seed=5)["core_u5"])
    expect = {
        "res_codes": (np.uint8, (500, 160)), "res_scale_codes": (np.uint8, (500, 3)),
        "res_row_scale": (np.uint16, (500,)), "core_u5": (np.uint8, (500, 7)),
        "core_u_scale": (np.uint16, (10,)), "core_v": (np.int8, (320, 10)),
        "corr_a": (np.int8, (500, 6)), "corr_b_scale": (np.uint16, (5, 6)),
    }
    for k, (dt, shp) in expect.items():
        assert a[k].dtype == dt and a[k].shape == shp, k
    assert "res_scales" not in a and "core_u" not in a
    # 50 bits of codes in 7 bytes: the top 6 bits of the last byte are zero.
    assert np.all(a["core_u5"][:, 6] >> 2 == 0) and len(np.unique(a["core_u5"][:, 6])) == 4
    # 5 groups in 3 bytes: the last high nibble is zero, the others take all 16 values.
    assert np.all(a["res_scale_codes"][:, 2] >> 4 == 0)
    assert len(np.unique(a["res_scale_codes"][:, :2] >> 4)) == 16
    v = a["res_row_scale"].view(np.float16).astype(np.float64)
    assert np.all(np.isfinite(v)) and np.all(v > 0)


def test_named_sc4_shapes():
    s = SHAPES["qwen3-8b-sc4"]
    assert (s.V, s.d, s.core_rank, s.corr_rank, s.group_size, s.fmt) == (151936, 4096, 10, 6, 64, "sc4")
