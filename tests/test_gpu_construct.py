"""Offline construction on the GPU (paper Section 3.4, Algorithm 1) against
the construction oracle (oracle/construct.py):

- the library's quantisers, packers and dequantisers bit for bit on the same
  fp32 inputs (both take every integer decision in fp32);
- the whole construction (fp64 linear algebra on the GPU, the same random
  test matrices) giving the same stored arrays as the oracle, in both packed
  formats;
- the constructed head through archead_pack_create and the forward kernels
  against the forward oracle, and its error in the activation metric.
"""

import numpy as np
import pytest

import oracle
from oracle import construct as oc
from paper_2608_02703_gb300 import archead
from synth import HeadShape, make_dense_head, make_hidden, make_test_matrix
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _build():
    from paper_2608_02703_gb300.build import build

    build()


def _dev(a):
    import torch

    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _inputs(seed, shape=(96, 64)):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal(shape) * np.exp2(rng.integers(-20, 8, shape))).astype(np.float32)
    x[:4, :8] = 0.0
    x[5, 3] = 1e-30  # far below the smallest fp16 scale step
    return x


@pytest.mark.parametrize("bits", [8, 5, 4])
@pytest.mark.parametrize("groups", [(1, 64), (1, 8), (96, 1), (8, 1), (4, 4)])
def test_quantiser_bit_exact(bits, groups):
    import torch
    from paper_2608_02703_gb300 import construct as gc

    x = _inputs(bits * 7 + groups[0])
    codes, scales = gc.quantize(_dev(x), groups[0], groups[1], bits)
    rq, rs = oc.quantize_symmetric(x, groups[0], groups[1], bits)
    assert np.array_equal(codes.cpu().numpy(), rq)
    assert np.array_equal(scales.cpu().numpy().view(np.uint16), rs)
    back = gc.dequantize(codes, scales, groups[0], groups[1])
    torch.cuda.synchronize()
    ref = rq.astype(np.float64) * np.repeat(np.repeat(rs.view(np.float16).astype(np.float64), groups[0], 0),
                                            groups[1], 1)
    assert np.array_equal(back.cpu().numpy().astype(np.float64), ref)


@pytest.mark.parametrize("g", [32, 64, 128])
def test_residual_quantiser_of_the_papers_format_bit_exact(g):
    import torch

    x = _inputs(g, (80, 512))
    rc = torch.empty((80, 512), dtype=torch.int8, device="cuda")
    rq = torch.empty((80, 512 // g), dtype=torch.uint8, device="cuda")
    rs = torch.empty(80, dtype=torch.int16, device="cuda")
    archead.archead_quantize_residual_sc4(_dev(x), g, rc, rq, rs)
    c, q, s = oc.quantize_residual_sc4(x, g)
    assert np.array_equal(rc.cpu().numpy(), c)
    assert np.array_equal(rq.cpu().numpy(), q)
    assert np.array_equal(rs.cpu().numpy().view(np.uint16), s)
    out = torch.empty((80, 512), dtype=torch.float32, device="cuda")
    archead.archead_dequant_residual_sc4(rc, rq, rs, g, out)
    sg = s.view(np.float16).astype(np.float64)[:, None] * (q.astype(np.float64) + 1)
    assert np.array_equal(out.cpu().numpy().astype(np.float64), c * np.repeat(sg, g, axis=1))


def test_packers_bit_exact():
    from paper_2608_02703_gb300 import construct as gc

    rng = np.random.default_rng(3)
    c4 = rng.integers(-8, 8, (33, 70)).astype(np.int8)
    assert np.array_equal(gc.pack(_dev(c4), 4).cpu().numpy(), oc.pack_int4(c4))
    q = rng.integers(0, 16, (33, 5)).astype(np.int8)
    assert np.array_equal(gc.pack(_dev(q), 4).cpu().numpy(), oc.pack_scale_codes(q))
    for r in (1, 3, 10, 13, 64):
        c5 = rng.integers(-16, 16, (33, r)).astype(np.int8)
        assert np.array_equal(gc.pack(_dev(c5), 5).cpu().numpy(), oc.pack_int5(c5))


CASES = [
    ("int8", 1000, 256, 16, 8, 64),
    ("sc4", 700, 320, 10, 6, 64),
    ("int8", 513, 256, 0, 8, 32),
]


@pytest.mark.parametrize("fmt,V,D,rc,rr,g", CASES, ids=[f"{c[0]}-V{c[1]}-d{c[2]}-r{c[3]}-{c[4]}" for c in CASES])
def test_construction_matches_the_oracle(fmt, V, D, rc, rr, g):
    import torch
    from paper_2608_02703_gb300 import construct as gc

    N = 1024
    W = make_dense_head(V, D, seed=11)
    Hb = make_hidden(D, N, seed=11)
    H = oracle.bf16_values(Hb)
    om_c = make_test_matrix(D, rc + 10, seed=12) if rc else None
    om_r = make_test_matrix(D, rr + 10, seed=13)
    ref = oc.construct(W.astype(np.float64), H, rc, rr, g, fmt=fmt, omega_core=om_c, omega_corr=om_r)
    Hd = torch.from_numpy(Hb.view(np.int16)).cuda().view(torch.bfloat16).float()
    got = gc.construct(_dev(W), Hd, rc, rr, g, fmt=fmt, omega_core=_dev(om_c) if rc else None, omega_corr=_dev(om_r))
    got = gc.to_numpy(got)
    can = oc.canonical(ref)
    assert set(got) == set(can)
    for k in can:
        assert got[k].shape == can[k].shape and got[k].dtype == can[k].dtype, k
        mism = int(np.sum(got[k] != can[k]))
        assert mism == 0, f"{k}: {mism} of {can[k].size} entries differ"
    # the constructed head runs through the library like any other
    shape = HeadShape(V=V, d=D, core_rank=rc, corr_rank=rr, group_size=g, fmt=fmt)
    pack = archead.archead_pack_create(got, shape)
    try:
        x = make_hidden(D, 16, seed=14)
        yref = oracle.logits(can, shape, x)
        for M, path in ((16, archead.PATH_DECODE), (16, archead.PATH_PREFILL)):
            gu.check_logits(gu.forward(pack, x[:M], archead.OUT_FP32, path), yref[:M], where=f"{fmt} constructed")
    finally:
        pack.close()
    # the correction lowers the error in the activation metric
    Wq = oracle.dequant_rows(can, shape)
    T = ref["_T"]
    assert oc.metric_error(W, Wq, T) < 0.5 * oc.metric_error(W, ref["_W_d"], T)
