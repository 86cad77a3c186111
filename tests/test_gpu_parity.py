"""CUDA path vs the fp64 oracle on small heads (several tiles, ragged tails,
every supported group size, rank 0 branches), through the C ABI."""

import zlib

import numpy as np
import pytest

import oracle
from paper_2608_02703_gb300 import archead
from synth import HeadShape, make_head, make_hidden, make_targets
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

SHAPES = {
    "ragged": HeadShape(V=1000, d=256, core_rank=16, corr_rank=8, group_size=64),
    "tiny": HeadShape(V=4096, d=512, core_rank=64, corr_rank=16, group_size=64),
    "g32": HeadShape(V=700, d=512, core_rank=24, corr_rank=40, group_size=32),
    "g128": HeadShape(V=513, d=512, core_rank=128, corr_rank=32, group_size=128),
    "g256": HeadShape(V=300, d=768, core_rank=8, corr_rank=8, group_size=256),
    "d320": HeadShape(V=333, d=320, core_rank=5, corr_rank=3, group_size=64),
    "group_int4": HeadShape(V=640, d=256, core_rank=0, corr_rank=0, group_size=64),
    "core_only": HeadShape(V=640, d=256, core_rank=32, corr_rank=0, group_size=64),
    "corr_only": HeadShape(V=640, d=256, core_rank=0, corr_rank=32, group_size=64),
    "max_rank": HeadShape(V=384, d=256, core_rank=256, corr_rank=256, group_size=64),
    "one_row": HeadShape(V=1, d=64, core_rank=4, corr_rank=4, group_size=32),
    # The paper's packed format (5-bit core left codes, 4-bit group-scale
    # codes times a row scale), with its Qwen ranks and group size first.
    "sc4": HeadShape(V=4096, d=512, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
    "sc4_ragged": HeadShape(V=1000, d=320, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),  # 5 groups
    "sc4_g32": HeadShape(V=700, d=512, core_rank=24, corr_rank=40, group_size=32, fmt="sc4"),
    "sc4_g128": HeadShape(V=513, d=512, core_rank=3, corr_rank=0, group_size=128, fmt="sc4"),
    "sc4_g256": HeadShape(V=300, d=768, core_rank=13, corr_rank=5, group_size=256, fmt="sc4"),
    "sc4_int4": HeadShape(V=640, d=256, core_rank=0, corr_rank=0, group_size=64, fmt="sc4"),
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


def get(name):
    if name not in _packs:
        shape = SHAPES[name]
        head = make_head(shape, seed=zlib.crc32(name.encode()) % 1000)
        _packs[name] = (archead.archead_pack_create(head, shape), head)
    return _packs[name]


def test_pack_create_ex_version1_struct():
    """An INT8 head described by a version-1 struct (no res_row_scale)
    through archead_pack_create_ex gives the same logits as the full struct."""
    import ctypes

    pack, head = get("tiny")
    shape = SHAPES["tiny"]
    v1 = archead.archead_desc.res_row_scale.offset
    old = archead.archead_pack_create(head, shape, desc_size=v1)
    try:
        x = make_hidden(shape.d, 9, seed=21)
        a = gu.forward(pack, x, archead.OUT_FP32, archead.PATH_AUTO)
        b = gu.forward(old, x, archead.OUT_FP32, archead.PATH_AUTO)
        assert np.array_equal(a, b)
        assert ctypes.sizeof(archead.archead_desc) > v1
    finally:
        old.close()


@pytest.mark.parametrize("name", sorted(SHAPES))
def test_dequant_bit_exact(name):
    import torch

    pack, head = get(name)
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
        assert np.array_equal(got.astype(np.float64), ref), f"{name}/{comp} not bit-exact"
        assert np.array_equal(got.view(np.uint32), ref.astype(np.float32).view(np.uint32))


@pytest.mark.parametrize("name", sorted(SHAPES))
@pytest.mark.parametrize("M", [1, 3, 8, 9, 16, 32, 64])
def test_decode_logits(name, M):
    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=M, n_outliers=shape.n_outliers)
    ref = oracle.logits(head, shape, x)
    got = gu.forward(pack, x, archead.OUT_FP32, archead.PATH_DECODE)
    gu.check_logits(got, ref, where=f"{name} M={M} fp32")
    gu.check_argmax(got, ref, where=f"{name} M={M}")
    got16 = gu.forward(pack, x, archead.OUT_BF16, archead.PATH_DECODE)
    gu.check_logits(got16, ref, bf16=True, where=f"{name} M={M} bf16")


@pytest.mark.parametrize("M", [1, 2, 12])
def test_decode_hidden_state_range(M):
    """Hidden states far outside fp16 range, or tiny, one scale per token: the
    decode path stages them in fp16 under a per-token power-of-two scale."""
    pack, head = get("tiny")
    shape = SHAPES["tiny"]
    x = make_hidden(shape.d, M, seed=50 + M).view(np.uint16).astype(np.uint32)
    # Shift bf16 exponents by +14 or -40 (powers of two: exact), alternating per token.
    shift = np.where(np.arange(M) % 2 == 0, 14, -40)[:, None].astype(np.int64)
    exp = ((x >> 7) & 0xFF).astype(np.int64)
    nz = exp > 0
    new_exp = np.where(nz, exp + shift, 0)
    assert new_exp.max() < 255 and new_exp[nz].min() > 0
    xs = ((x & 0x807F) | (new_exp.astype(np.uint32) << 7)).astype(np.uint16)
    ref = oracle.logits(head, shape, xs)
    got = gu.forward(pack, xs, archead.OUT_FP32, archead.PATH_DECODE)
    for m in range(M):  # each token against its own scale
        gu.check_logits(got[m:m + 1], ref[m:m + 1], where=f"M={M} token {m}")


@pytest.mark.parametrize("name", ["ragged", "tiny", "g32", "max_rank", "sc4", "sc4_ragged", "sc4_g256", "sc4_int4"])
@pytest.mark.parametrize("M", [17, 40, 133])
def test_logits_many_tokens(name, M):
    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=M)
    ref = oracle.logits(head, shape, x)
    for path in (archead.PATH_AUTO, archead.PATH_DECODE, archead.PATH_PREFILL):
        got = gu.forward(pack, x, archead.OUT_FP32, path)
        gu.check_logits(got, ref, where=f"{name} M={M} path={path}")
        gu.check_argmax(got, ref, where=f"{name} M={M} path={path}")


@pytest.mark.parametrize("name", ["ragged", "tiny", "g32", "g256", "corr_only", "one_row", "max_rank", "sc4",
                                  "sc4_g32"])
@pytest.mark.parametrize("M", [1, 7, 16, 40])
def test_greedy(name, M):
    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=300 + M)
    ref = oracle.logits(head, shape, x)
    for path in (archead.PATH_AUTO, archead.PATH_DECODE, archead.PATH_PREFILL):
        idx, val = gu.forward_argmax(pack, x, path)
        gu.check_greedy(idx, val, ref, where=f"{name} M={M} path={path}")


@pytest.mark.parametrize("name", ["ragged", "tiny", "g32", "g256", "corr_only", "one_row", "sc4", "sc4_ragged",
                                  "sc4_g128"])
@pytest.mark.parametrize("M", [1, 5, 16, 33])
def test_cross_entropy(name, M):
    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=100 + M)
    t = make_targets(shape.V, M, seed=M)
    ref = oracle.cross_entropy(head, shape, x, t)["ce"]
    for path in (archead.PATH_AUTO, archead.PATH_DECODE, archead.PATH_PREFILL):
        got, st = gu.forward_ce(pack, x, t, path)
        assert st == archead.OK
        err = np.abs(got - ref)
        assert np.all(err <= gu.CE_ABS), f"{name} M={M} path={path}: max|dCE|={err.max():.3e}"


@pytest.mark.parametrize("shape", [
    HeadShape(V=520, d=8192, core_rank=16, corr_rank=8, group_size=128),
    HeadShape(V=300, d=6144, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
], ids=["d8192", "d6144_sc4"])
def test_wide_head(shape):
    """Heads so wide that eight tokens of x do not fit in shared memory next to
    a deep enough ring: the decode path switches to its streamed-x instance
    (at d = 8192 for M = 8); every path against the oracle.  One set of hidden
    states (and its prefixes) keeps the Haar rotation of x to one draw."""
    head = make_head(shape, seed=5)
    pack = archead.archead_pack_create(head, shape)
    try:
        x = make_hidden(shape.d, 64, seed=5)
        ref = oracle.logits(head, shape, x)
        for M in (1, 5, 8, 16, 27, 64):
            got = gu.forward(pack, x[:M], archead.OUT_FP32, archead.PATH_DECODE)
            gu.check_logits(got, ref[:M], where=f"d={shape.d} decode M={M}")
        got = gu.forward(pack, x, archead.OUT_FP32, archead.PATH_PREFILL)
        gu.check_logits(got, ref, where=f"d={shape.d} prefill M=64")
        t = make_targets(shape.V, 16, seed=5)
        ce, st = gu.forward_ce(pack, x[:16], t)
        assert st == archead.OK
        ref_ce = oracle.cross_entropy(head, shape, x[:16], t)["ce"]
        assert np.max(np.abs(ce - ref_ce)) <= gu.CE_ABS
    finally:
        pack.close()


def test_very_wide_head_takes_prefill_under_auto():
    """d = 65536 at g = 32: the decode kernel's per-group sums of x do not fit
    its shared memory, so an explicit decode request is refused as
    unsupported and AUTO runs the prefill kernel, for any M."""
    import torch

    shape = HeadShape(V=300, d=65536, core_rank=8, corr_rank=8, group_size=32)
    head = make_head(shape, seed=6)
    pack = archead.archead_pack_create(head, shape)
    try:
        rng = np.random.default_rng(6)
        M = 3
        # bf16 values of both signs with exponents 2^-7 .. 2^3 (no rotation: the
        # Haar draw of make_hidden is a 65536 x 65536 QR).
        x = ((rng.integers(0, 2, (M, shape.d)) << 15) | (rng.integers(120, 131, (M, shape.d)) << 7)
             | rng.integers(0, 128, (M, shape.d))).astype(np.uint16)
        ref = oracle.logits(head, shape, x)
        got = gu.forward(pack, x, archead.OUT_FP32, archead.PATH_AUTO)
        gu.check_logits(got, ref, where="d=65536 auto")
        y = torch.empty((M, shape.V), dtype=torch.float32, device="cuda")
        with pytest.raises(archead.ArcheadError) as ei:
            archead.archead_forward_path(pack, gu.to_dev(x), M, y, archead.OUT_FP32, archead.PATH_DECODE)
        assert ei.value.status == archead.ERR_UNSUPPORTED
    finally:
        pack.close()


def test_ce_target_out_of_range():
    pack, head = get("ragged")
    shape = SHAPES["ragged"]
    x = make_hidden(shape.d, 4, seed=3)
    t = np.array([5, shape.V, -1, 7], dtype=np.int32)
    got, st = gu.forward_ce(pack, x, t)
    assert st == archead.ERR_TARGET_RANGE
    assert np.isnan(got[1]) and np.isnan(got[2])
    ref = oracle.cross_entropy(head, shape, x[[0, 3]], t[[0, 3]])["ce"]
    assert np.all(np.abs(got[[0, 3]] - ref) <= gu.CE_ABS)
    assert archead.archead_sync_status(pack) == archead.OK  # the error word was cleared


def test_zero_tokens_is_a_no_op():
    import torch

    pack, _ = get("ragged")
    y = torch.zeros((1, 1), dtype=torch.float32, device="cuda")
    archead.archead_forward(pack, y, 0, y, archead.OUT_FP32)
    assert archead.archead_sync_status(pack) == archead.OK


@pytest.mark.parametrize("M", [4, 300])
def test_forward_host_matches_device(M):
    """Host buffers: pinned (the kernels write the output in place) and
    pageable (staged through the pack's device buffer), bit for bit the
    device-buffer forward, on the decode and the prefill kernel."""
    import torch

    pack, head = get("tiny")
    shape = SHAPES["tiny"]
    x = make_hidden(shape.d, M, seed=9)
    for dt, out in ((torch.bfloat16, archead.OUT_BF16), (torch.float32, archead.OUT_FP32)):
        dev = gu.forward(pack, x, out)
        xh = torch.from_numpy(x.view(np.int16)).pin_memory()
        yh = torch.full((M, shape.V), float("nan"), dtype=dt).pin_memory()
        archead.archead_forward_host(pack, xh, M, yh, out)
        assert np.array_equal(yh.float().numpy().astype(np.float64), dev)
        yp = torch.full((M, shape.V), float("nan"), dtype=dt)  # pageable
        archead.archead_forward_host(pack, torch.from_numpy(x.view(np.int16).copy()), M, yp, out)
        assert np.array_equal(yp.float().numpy().astype(np.float64), dev)


def test_forward_host_repeated_calls_with_new_inputs():
    """Repeated host calls on the same pinned buffers: every call must read
    the buffers' current contents and match the device-buffer forward bit
    for bit, also after M changes and after the pack's workspace is
    reallocated by a larger forward in between."""
    import torch

    pack, head = get("ragged")
    shape = SHAPES["ragged"]
    for M in (3, 16, 3):
        xh = torch.empty((M, shape.d), dtype=torch.int16).pin_memory()
        yh = torch.empty((M, shape.V), dtype=torch.bfloat16).pin_memory()
        for call in range(5):
            x = make_hidden(shape.d, M, seed=40 + 7 * M + call)
            xh.copy_(torch.from_numpy(x.view(np.int16)))
            yh.fill_(float("nan"))
            archead.archead_forward_host(pack, xh, M, yh, archead.OUT_BF16)
            dev = gu.forward(pack, x, archead.OUT_BF16)
            assert np.array_equal(yh.float().numpy().astype(np.float64), dev), f"M={M} call {call}"
            if call == 2:  # a larger forward grows the workspace between two replays
                big = make_hidden(shape.d, 600, seed=5)
                gu.forward(pack, big, archead.OUT_BF16)
    assert archead.archead_sync_status(pack) == archead.OK


def test_wait_timeout_is_reported_and_recoverable():
    pack, head = get("ragged")
    archead.archead_set_wait_budget(pack, 20_000)  # cycles: a few microseconds
    archead.archead_debug_wait_timeout(pack)
    assert archead.archead_sync_status(pack) == archead.ERR_DEVICE_TIMEOUT
    archead.archead_set_wait_budget(pack, 2_000_000_000)
    shape = SHAPES["ragged"]
    x = make_hidden(shape.d, 2, seed=1)
    gu.check_logits(gu.forward(pack, x), oracle.logits(head, shape, x), where="after timeout")


def test_pack_bytes_follow_eq10():
    for name in ("tiny", "group_int4", "core_only", "max_rank", "sc4", "sc4_ragged", "sc4_int4"):
        pack, head = get(name)
        assert archead.archead_pack_bytes(pack) == oracle.packed_bytes(SHAPES[name])
        assert archead.archead_device_bytes(pack) >= archead.archead_pack_bytes(pack)


def test_deterministic():
    pack, _ = get("tiny")
    shape = SHAPES["tiny"]
    x = make_hidden(shape.d, 16, seed=4)
    a = gu.forward(pack, x)
    b = gu.forward(pack, x)
    assert np.array_equal(a, b)
