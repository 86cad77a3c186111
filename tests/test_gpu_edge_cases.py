"""Edge cases of the CUDA path against the fp64 oracle, through the C ABI:

- the most negative code of every factor array (INT8 -128, which the
  symmetric generator never draws; the 5-bit code -16 of the paper's format;
  INT4 -8), through the dequantiser and both streaming kernels;
- token counts that fill several 256-token prefill tiles and end in a ragged
  one (M = 257, 300, 700), on every path;
- ties: a head whose rows are all the same gives bitwise-equal logits on
  every path, and the lowest vocabulary row wins; an all-zero head gives
  CE = log V and near-zero logits;
- cross entropy far from logit rms 2: one dominant row (CE from ~0 to far
  above log V) and hidden states scaled by 2^3, 2^6 and 2^10;
- zero group, row and correction scales (+0 and -0).
"""

import math
import zlib

import numpy as np
import pytest

import oracle
from paper_2608_02703_gb300 import archead
from synth import HeadShape, make_head, make_hidden, make_targets, with_extreme_codes
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

PATHS = (archead.PATH_AUTO, archead.PATH_DECODE, archead.PATH_PREFILL)

SHAPES = {
    "tiny": HeadShape(V=4096, d=512, core_rank=64, corr_rank=16, group_size=64),
    "ragged": HeadShape(V=1000, d=256, core_rank=16, corr_rank=8, group_size=64),
    "g32": HeadShape(V=700, d=512, core_rank=24, corr_rank=40, group_size=32),
    "g128": HeadShape(V=513, d=512, core_rank=128, corr_rank=32, group_size=128),
    "max_rank": HeadShape(V=384, d=256, core_rank=256, corr_rank=256, group_size=64),
    "sc4": HeadShape(V=4096, d=512, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
    "sc4_g32": HeadShape(V=700, d=512, core_rank=24, corr_rank=40, group_size=32, fmt="sc4"),
    "sc4_ragged": HeadShape(V=1000, d=320, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
}

_packs = {}


@pytest.fixture(scope="module", autouse=True)
def _build():
    from paper_2608_02703_gb300.build import build

    build()
    yield
    for p, _ in _packs.values():
        p.close()
    _packs.clear()


def _seed(key: str) -> int:
    return zlib.crc32(key.encode()) % 1000


def get(name, variant="plain"):
    key = (name, variant)
    if key not in _packs:
        shape = SHAPES[name]
        head = make_head(shape, seed=_seed(name))
        if variant == "extreme":
            head = with_extreme_codes(head, shape, seed=_seed(name))
        _packs[key] = (archead.archead_pack_create(head, shape), head)
    return _packs[key]


# ---------------------------------------------------------------------------
# Most negative codes
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["tiny", "g32", "g128", "max_rank", "sc4", "sc4_g32"])
def test_extreme_codes_dequant_bit_exact(name):
    import torch

    pack, head = get(name, "extreme")
    shape = SHAPES[name]
    comps = [("residual", shape.V, shape.d)]
    if shape.core_rank:
        comps += [("core_u", shape.V, shape.core_rank), ("core_v", shape.d, shape.core_rank)]
    if shape.corr_rank:
        comps += [("corr_a", shape.V, shape.corr_rank), ("corr_b", shape.d, shape.corr_rank)]
    for comp, rows, cols in comps:
        out = torch.full((rows, cols), float("nan"), dtype=torch.float32, device="cuda")
        archead.archead_debug_dequant(pack, comp, 0, rows, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        ref = oracle.component(head, shape, comp)
        assert np.array_equal(got.view(np.uint32), ref.astype(np.float32).view(np.uint32)), f"{name}/{comp}"


@pytest.mark.parametrize("name", ["tiny", "g32", "g128", "max_rank", "sc4", "sc4_g32"])
@pytest.mark.parametrize("M,path", [(1, archead.PATH_DECODE), (9, archead.PATH_DECODE), (16, archead.PATH_DECODE),
                                    (40, archead.PATH_PREFILL), (300, archead.PATH_PREFILL)])
def test_extreme_codes_logits(name, M, path):
    pack, head = get(name, "extreme")
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=700 + M)
    ref = oracle.logits(head, shape, x)
    got = gu.forward(pack, x, archead.OUT_FP32, path)
    gu.check_logits(got, ref, where=f"{name} extreme codes M={M} path={path}")
    gu.check_argmax(got, ref, where=f"{name} extreme codes M={M} path={path}")


@pytest.mark.parametrize("name", ["tiny", "max_rank", "sc4"])
@pytest.mark.parametrize("M,path", [(16, archead.PATH_DECODE), (300, archead.PATH_PREFILL)])
def test_extreme_codes_cross_entropy(name, M, path):
    pack, head = get(name, "extreme")
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=750 + M)
    t = make_targets(shape.V, M, seed=750 + M)
    ref = oracle.cross_entropy(head, shape, x, t)["ce"]
    got, st = gu.forward_ce(pack, x, t, path)
    assert st == archead.OK
    assert np.max(np.abs(got - ref)) <= gu.CE_ABS


# ---------------------------------------------------------------------------
# Several prefill tiles with a ragged last one
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["tiny", "ragged", "g32", "max_rank", "sc4", "sc4_ragged"])
@pytest.mark.parametrize("M", [257, 300, 700])
def test_ragged_token_tiles_every_path(name, M):
    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=800 + M)
    ref = oracle.logits(head, shape, x)
    for path in PATHS:
        got = gu.forward(pack, x, archead.OUT_FP32, path)
        gu.check_logits(got, ref, where=f"{name} M={M} path={path}")
        gu.check_argmax(got, ref, where=f"{name} M={M} path={path}")
    got16 = gu.forward(pack, x, archead.OUT_BF16, archead.PATH_PREFILL)
    gu.check_logits(got16, ref, bf16=True, where=f"{name} M={M} prefill bf16")


@pytest.mark.parametrize("name", ["tiny", "g32", "sc4", "sc4_ragged"])
@pytest.mark.parametrize("M", [257, 700])
def test_ragged_token_tiles_ce_and_greedy(name, M):
    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=900 + M)
    t = make_targets(shape.V, M, seed=900 + M)
    ref = oracle.cross_entropy(head, shape, x, t)["ce"]
    ref_y = oracle.logits(head, shape, x)
    for path in PATHS:
        got, st = gu.forward_ce(pack, x, t, path)
        assert st == archead.OK
        err = np.abs(got - ref)
        assert np.all(err <= gu.CE_ABS), f"{name} M={M} path={path}: max|dCE|={err.max():.3e}"
        idx, val = gu.forward_argmax(pack, x, path)
        gu.check_greedy(idx, val, ref_y, where=f"{name} M={M} path={path}")


# ---------------------------------------------------------------------------
# Zero scales
# ---------------------------------------------------------------------------
def _zero_scale_head(shape, seed):
    """About one in eight residual group scales (INT8 format) or row scales
    (SC4) set to +0 or -0, one whole row of them, and as many correction row
    scales.  Their weights are zero whatever the codes; the pack stores zero
    codes there, and the 64-token decode instance runs such groups at scale 1."""
    head = make_head(shape, seed=seed)
    rng = np.random.default_rng(seed)
    key = "res_row_scale" if shape.fmt == "sc4" else "res_scales"
    s = head[key]
    mask = rng.random(s.shape) < 0.125
    s[mask] = np.where(rng.random(int(mask.sum())) < 0.5, 0x0000, 0x8000).astype(np.uint16)
    s[3] = 0
    if shape.corr_rank:
        a = head["corr_a_scale"]
        a[rng.random(a.shape) < 0.125] = 0
        a[5] = 0x8000
    return head


@pytest.mark.parametrize("name", ["tiny", "g32", "g128", "max_rank", "sc4", "sc4_g32"])
def test_zero_scales(name):
    """Zero group, row and correction scales against the oracle: logits on
    every path at the token counts of every decode instance, and the
    dequantised components (equal as numbers: a zero weight may come back
    as +0 where the oracle's product is -0)."""
    import torch

    shape = SHAPES[name]
    head = _zero_scale_head(shape, seed=_seed(name) + 1)
    pack = archead.archead_pack_create(head, shape)
    try:
        comps = [("residual", shape.V, shape.d)] + ([("corr_a", shape.V, shape.corr_rank)] if shape.corr_rank else [])
        for comp, rows, cols in comps:
            out = torch.full((rows, cols), float("nan"), dtype=torch.float32, device="cuda")
            archead.archead_debug_dequant(pack, comp, 0, rows, out)
            torch.cuda.synchronize()
            assert np.array_equal(out.cpu().numpy().astype(np.float64), oracle.component(head, shape, comp)), comp
        x = make_hidden(shape.d, 64, seed=31)
        ref = oracle.logits(head, shape, x)
        for M in (1, 9, 16, 27, 40, 64):
            for path in PATHS:
                got = gu.forward(pack, x[:M], archead.OUT_FP32, path)
                gu.check_logits(got, ref[:M], where=f"{name} zero scales M={M} path={path}")
    finally:
        pack.close()


# ---------------------------------------------------------------------------
# Exact ties
# ---------------------------------------------------------------------------
def _zero_head(shape, seed):
    head = make_head(shape, seed=seed)
    zero = ("res_codes", "core_u5", "corr_a") if shape.fmt == "sc4" else ("res_codes", "core_u", "corr_a")
    for k in zero:
        head[k][:] = 0
    return head


def _residual_scale_bound(head, shape, x_bits):
    """Per token, max over rows of sum_g s[n, g] * sum_{k in g} |x[k]|: the
    largest logit a residual of unit codes could reach (decoded by the
    oracle's pinned fp16/bf16/scale-code decoders)."""
    g = shape.group_size
    if shape.fmt == "sc4":
        q = oracle.unpack_scale_codes(head["res_scale_codes"], shape.groups).astype(np.float64)
        s = oracle.fp16_values(head["res_row_scale"])[:, None] * (q + 1.0)
    else:
        s = oracle.fp16_values(head["res_scales"])
    ax = np.abs(oracle.bf16_values(x_bits)).reshape(x_bits.shape[0], shape.groups, g).sum(axis=2)
    return (ax @ s.T).max(axis=1)


@pytest.mark.parametrize("name", ["tiny", "ragged", "sc4"])
@pytest.mark.parametrize("M", [1, 9, 16, 40, 300])
def test_all_zero_head(name, M):
    """Zero codes everywhere: the oracle's logits are exactly zero (CE = log V,
    argmax 0).  The kernels multiply offset operands (code + 1032 and the
    like) and start each group from minus the offset times the sum of x, so
    a zero code leaves only the fp32 rounding of that cancellation: logits
    within 2^-12 of a unit-code residual's size, CE = log V within the bar,
    and the greedy output the first maximum of the same path's own fp32
    logits."""
    shape = SHAPES[name]
    head = _zero_head(shape, seed=11)
    ref = oracle.cross_entropy(head, shape, make_hidden(shape.d, 1, seed=11), np.zeros(1, np.int32))
    assert ref["argmax"][0] == 0 and ref["top2_gap"][0] == 0.0  # the oracle's own tie rule
    pack = archead.archead_pack_create(head, shape)
    try:
        x = make_hidden(shape.d, M, seed=12 + M)
        t = make_targets(shape.V, M, seed=12 + M)
        bound = 2.0 ** -12 * _residual_scale_bound(head, shape, x)
        for path in PATHS:
            y = gu.forward(pack, x, archead.OUT_FP32, path)
            assert np.all(np.abs(y) <= bound[:, None]), f"{name} M={M} path={path}: |y| up to {np.abs(y).max():.3e}"
            idx, val = gu.forward_argmax(pack, x, path)
            first = np.argmax(y, axis=1)
            assert np.array_equal(idx, first), f"{name} M={M} path={path}: not the first maximum"
            assert np.array_equal(val, y[np.arange(M), first])
            ce, st = gu.forward_ce(pack, x, t, path)
            assert st == archead.OK
            assert np.max(np.abs(ce - math.log(shape.V))) <= gu.CE_ABS
    finally:
        pack.close()


def _repeated_rows_head(shape, seed):
    """Every vocabulary row a copy of row 0: all logits of a token are equal
    in exact arithmetic."""
    head = make_head(shape, seed=seed)
    for k, a in head.items():
        if a.ndim >= 1 and a.shape[0] == shape.V and k != "core_v" and k != "corr_b":
            a[:] = a[0]
    return head


@pytest.mark.parametrize("name", ["tiny", "ragged", "sc4", "sc4_ragged"])
@pytest.mark.parametrize("M", [1, 9, 16, 40, 300])
def test_repeated_rows_exact_ties(name, M):
    """All rows equal: the oracle's logits tie exactly (argmax 0, CE = log V).
    The prefill kernel computes every row by the same operations, so its fp32
    logits of a token are bitwise equal across the whole vocabulary; the
    decode kernel encodes rows 16i + 0..7 and 16i + 8..15 of each 16-row
    fragment differently (code + 1032 and 16 code + 1152), so there the two
    classes tie bitwise among themselves.  On every path the largest logit is
    shared by at least a third of the rows (ties across tiles, warps and
    vocabulary slices), greedy returns the lowest of them with that value,
    and CE is log V."""
    shape = SHAPES[name]
    head = _repeated_rows_head(shape, seed=13)
    pack = archead.archead_pack_create(head, shape)
    try:
        x = make_hidden(shape.d, M, seed=14 + M)
        t = make_targets(shape.V, M, seed=14 + M)
        ref = oracle.cross_entropy(head, shape, x, t)
        assert np.all(ref["argmax"] == 0) and np.all(ref["top2_gap"] == 0.0)
        for path in PATHS:
            y = gu.forward(pack, x, archead.OUT_FP32, path)
            gu.check_logits(y, oracle.logits(head, shape, x), where=f"{name} M={M} path={path}")
            mx = y.max(axis=1)
            ties = (y == mx[:, None]).sum(axis=1)
            assert np.all(ties >= shape.V // 3), f"{name} M={M} path={path}: only {ties.min()} rows hold the max"
            assert np.all(np.unique(y, axis=None).size <= 2 * M), f"{name} M={M} path={path}: rows differ"
            idx, val = gu.forward_argmax(pack, x, path)
            first = np.argmax(y, axis=1)  # numpy: the first index of the maximum
            assert np.array_equal(idx, first), f"{name} M={M} path={path}: not the lowest row of the maximum"
            assert np.array_equal(val, mx)
            ce, st = gu.forward_ce(pack, x, t, path)
            assert st == archead.OK
            assert np.max(np.abs(ce - math.log(shape.V))) <= gu.CE_ABS
    finally:
        pack.close()


# ---------------------------------------------------------------------------
# Cross entropy far from logit rms 2
# ---------------------------------------------------------------------------
def _scaled(x_bits: np.ndarray, e: int) -> np.ndarray:
    """x * 2^e, exactly (bf16 exponent shift; zeros stay zero)."""
    x = x_bits.astype(np.uint32)
    exp = ((x >> 7) & 0xFF).astype(np.int64)
    nz = exp > 0
    new = np.where(nz, exp + e, 0)
    assert new.max() < 255 and (not nz.any() or new[nz].min() > 0)
    return ((x & 0x807F) | (new.astype(np.uint32) << 7)).astype(np.uint16)


def _dominant_row_head(shape, x_ref_bits, row, target_logit, seed):
    """A head whose row `row` holds the sign pattern of x_ref (every residual
    code +-1, every group scale s): that row's logit for x_ref is
    s * sum|x_ref| + its rank-r terms, set near target_logit by the choice of
    s, far above every other row."""
    head = make_head(shape, seed=seed)
    xr = oracle.bf16_values(x_ref_bits)[0]
    codes = np.where(xr > 0, 1, -1).astype(np.int64) & 15
    head["res_codes"][row, :] = (codes[0::2] | (codes[1::2] << 4)).astype(np.uint8)
    s = np.float16(target_logit / np.sum(np.abs(xr)))
    if shape.fmt == "sc4":
        head["res_scale_codes"][row, :] = 0  # q = 0: group scale = s_row
        head["res_row_scale"][row] = s.view(np.uint16)
    else:
        head["res_scales"][row, :] = s.view(np.uint16)
    return head


@pytest.mark.parametrize("name", ["tiny", "sc4"])
def test_cross_entropy_dominant_row(name):
    """One row ~40 above the rest for every token (scaled by 1, 2, 4 and 8):
    CE ~ 0 when it is the target, ~40..320 otherwise, on every path."""
    shape = SHAPES[name]
    base = make_hidden(shape.d, 1, seed=21)
    row = 1234
    head = _dominant_row_head(shape, base, row, 40.0, seed=21)
    pack = archead.archead_pack_create(head, shape)
    try:
        M = 24
        x = np.concatenate([_scaled(base, m % 4) for m in range(M)])
        t = make_targets(shape.V, M, seed=21)
        t[::2] = row
        ref = oracle.cross_entropy(head, shape, x, t)
        assert np.all(ref["argmax"] == row)
        assert ref["ce"][::2].max() < 1e-6 and ref["ce"][1::2].min() > 20.0
        for path in PATHS:
            got, st = gu.forward_ce(pack, x, t, path)
            assert st == archead.OK
            err = np.abs(got - ref["ce"])
            assert np.all(err <= gu.ce_bound(ref)), f"{name} path={path}: max|dCE|={err.max():.3e}"
            idx, _ = gu.forward_argmax(pack, x, path)
            assert np.all(idx == row)
    finally:
        pack.close()


@pytest.mark.parametrize("name", ["tiny", "g128", "sc4"])
@pytest.mark.parametrize("e", [3, 6, 10])
@pytest.mark.parametrize("M,path", [(16, archead.PATH_DECODE), (300, archead.PATH_PREFILL)])
def test_cross_entropy_large_logit_scale(name, e, M, path):
    """Hidden states scaled by 2^e (logit rms ~2^(e+1)): CE from near zero to
    thousands of nats against the oracle, under the CE bar widened by the
    fp32 resolution of the logits (gpu_util.ce_bound)."""
    pack, head = get(name)
    shape = SHAPES[name]
    x = _scaled(make_hidden(shape.d, M, seed=1000 + M), e)
    t = make_targets(shape.V, M, seed=1000 + M)
    ref = oracle.cross_entropy(head, shape, x, t)
    got, st = gu.forward_ce(pack, x, t, path)
    assert st == archead.OK
    err = np.abs(got - ref["ce"])
    bound = gu.ce_bound(ref)
    assert np.all(err <= bound), (f"{name} 2^{e} M={M} path={path}: max|dCE|={err.max():.3e} "
                                  f"(bound {bound.min():.3e}..{bound.max():.3e})")
