"""archead_forward_decode_noalloc: the decode forward for callers that must
not allocate device memory while they run the head (memory reserved up front,
graph capture under a pool that forbids new allocations, latency-critical
loops).  Its scratch is a fixed 512 KiB array inside the library instead of the
pack's cudaMalloc-grown workspace.

The tests call it through the C ABI and check its logits against the fp64
oracle under the same bars as every other parity test, on two calls in a row
(the second call finds the first call's data in the shared array; both must
give the same bits).  This file is collected last on purpose.
"""

import zlib

import numpy as np
import pytest

import oracle
from paper_2608_02703_gb300 import archead
from synth import HeadShape, make_head, make_hidden
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

SHAPES = [
    HeadShape(V=1000, d=256, core_rank=16, corr_rank=8, group_size=64),
    HeadShape(V=4096, d=512, core_rank=64, corr_rank=16, group_size=64),
    HeadShape(V=700, d=320, core_rank=24, corr_rank=40, group_size=32),
    # the paper's packed format (5-bit core codes, 4-bit group-scale codes)
    HeadShape(V=1500, d=384, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
]


@pytest.fixture(scope="module", autouse=True)
def _build():
    from paper_2608_02703_gb300.build import build

    build()


def _run_noalloc(pack, x_bits, out_dtype):
    import torch

    M = x_bits.shape[0]
    dt = torch.float32 if out_dtype == archead.OUT_FP32 else torch.bfloat16
    y = torch.full((M, pack.shape.V), float("nan"), dtype=dt, device="cuda")
    archead.archead_forward_decode_noalloc(pack, gu.to_dev(x_bits), M, y, out_dtype)
    assert archead.archead_sync_status(pack) == archead.OK
    return y.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"V{s.V}_d{s.d}_g{s.group_size}_{s.fmt}")
@pytest.mark.parametrize("out_dtype", [archead.OUT_FP32, archead.OUT_BF16])
def test_noalloc_matches_oracle_on_two_calls_in_a_row(shape, out_dtype):
    head = make_head(shape, seed=zlib.crc32(repr(shape).encode()) % 1000)
    pack = archead.archead_pack_create(head, shape)
    try:
        for M, seed in ((7, 1), (16, 2), (1, 3)):
            x = make_hidden(shape.d, M, seed=seed)
            ref = oracle.logits(head, shape, x)
            first = _run_noalloc(pack, x, out_dtype)
            second = _run_noalloc(pack, x, out_dtype)
            bf16 = out_dtype == archead.OUT_BF16
            for got in (first, second):
                gu.check_logits(got, ref, bf16=bf16, where=f"noalloc M={M}")
            assert np.array_equal(first, second)
            # and the same bits as the allocating entry point
            assert np.array_equal(first, gu.forward(pack, x, out_dtype, archead.PATH_DECODE))
    finally:
        pack.close()


def test_noalloc_rejects_more_than_16_tokens():
    import torch

    shape = SHAPES[0]
    pack = archead.archead_pack_create(make_head(shape, seed=5), shape)
    try:
        x = gu.to_dev(make_hidden(shape.d, 17, seed=5))
        y = torch.empty((17, shape.V), dtype=torch.float32, device="cuda")
        with pytest.raises(archead.ArcheadError) as exc:
            archead.archead_forward_decode_noalloc(pack, x, 17, y, archead.OUT_FP32)
        assert exc.value.status == archead.ERR_UNSUPPORTED
        assert "at most 16" in str(exc.value)
    finally:
        pack.close()


def test_noalloc_rejects_heads_needing_more_scratch():
    import torch

    # Ranks 256 + 256 at d = 4096: the pre-pass partial sums alone take
    # 16 column blocks x 16 splits x 2 KB = 512 KiB, beyond the fixed array.
    shape = HeadShape(V=128, d=4096, core_rank=256, corr_rank=256, group_size=128)
    pack = archead.archead_pack_create(make_head(shape, seed=6), shape)
    try:
        x = gu.to_dev(make_hidden(shape.d, 1, seed=6))
        y = torch.empty((1, shape.V), dtype=torch.float32, device="cuda")
        with pytest.raises(archead.ArcheadError) as exc:
            archead.archead_forward_decode_noalloc(pack, x, 1, y, archead.OUT_FP32)
        assert exc.value.status == archead.ERR_UNSUPPORTED
        assert "512 KiB" in str(exc.value)
    finally:
        pack.close()


def test_noalloc_forward_replays_as_a_cuda_graph():
    """The allocation-free decode captured once into a CUDA graph (pre-pass and
    decode grids with their programmatic dependency) and replayed on new
    hidden states written into the captured input buffer."""
    import torch

    shape = SHAPES[1]
    head = make_head(shape, seed=7)
    pack = archead.archead_pack_create(head, shape)
    try:
        M = 5
        xd = torch.zeros((M, shape.d), dtype=torch.int16, device="cuda")
        y = torch.zeros((M, shape.V), dtype=torch.float32, device="cuda")
        # First call outside the capture: it looks up the scratch array's
        # device address and opts the kernels into their shared memory.
        archead.archead_forward_decode_noalloc(pack, xd, M, y, archead.OUT_FP32)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            archead.archead_forward_decode_noalloc(pack, xd, M, y, archead.OUT_FP32)
        for seed in (8, 9):
            x = make_hidden(shape.d, M, seed=seed)
            xd.copy_(torch.from_numpy(x.view(np.int16)))
            g.replay()
            torch.cuda.synchronize()
            assert archead.archead_sync_status(pack) == archead.OK
            got = y.cpu().numpy().astype(np.float64)
            gu.check_logits(got, oracle.logits(head, shape, x), where=f"graph replay seed={seed}")
    finally:
        pack.close()


def test_noalloc_capture_after_warm_up_at_another_token_count():
    """A warm-up call at M = 1 prepares every decode instance the pack can
    use (one and two 8-token tiles), so a capture at M = 16 does no first-time
    set-up inside the capture; the replay is checked against the oracle."""
    import torch

    shape = SHAPES[3]
    head = make_head(shape, seed=17)
    pack = archead.archead_pack_create(head, shape)
    try:
        x1 = gu.to_dev(make_hidden(shape.d, 1, seed=17))
        y1 = torch.zeros((1, shape.V), dtype=torch.float32, device="cuda")
        archead.archead_forward_decode_noalloc(pack, x1, 1, y1, archead.OUT_FP32)
        torch.cuda.synchronize()
        M = 16
        xd = torch.zeros((M, shape.d), dtype=torch.int16, device="cuda")
        y = torch.zeros((M, shape.V), dtype=torch.bfloat16, device="cuda")
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            archead.archead_forward_decode_noalloc(pack, xd, M, y, archead.OUT_BF16)
        x = make_hidden(shape.d, M, seed=18)
        xd.copy_(torch.from_numpy(x.view(np.int16)))
        g.replay()
        torch.cuda.synchronize()
        assert archead.archead_sync_status(pack) == archead.OK
        gu.check_logits(y.float().cpu().numpy().astype(np.float64), oracle.logits(head, shape, x), bf16=True,
                        where="capture at M=16 after warm-up at M=1")
    finally:
        pack.close()


def test_noalloc_capture_of_the_resident_instance_after_warm_up_at_m8():
    """d = 8192: eight tokens of x do not stay resident next to a full ring,
    so M = 8 runs the streamed-x instance and M = 1 the resident one.  A
    warm-up at M = 8 still prepares the resident instance, and a capture at
    M = 1 replays against the oracle."""
    import torch

    shape = HeadShape(V=520, d=8192, core_rank=16, corr_rank=8, group_size=128)
    head = make_head(shape, seed=19)
    pack = archead.archead_pack_create(head, shape)
    try:
        x8 = gu.to_dev(make_hidden(shape.d, 8, seed=19))
        y8 = torch.zeros((8, shape.V), dtype=torch.float32, device="cuda")
        archead.archead_forward_decode_noalloc(pack, x8, 8, y8, archead.OUT_FP32)
        torch.cuda.synchronize()
        xd = torch.zeros((1, shape.d), dtype=torch.int16, device="cuda")
        y = torch.zeros((1, shape.V), dtype=torch.float32, device="cuda")
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            archead.archead_forward_decode_noalloc(pack, xd, 1, y, archead.OUT_FP32)
        x = make_hidden(shape.d, 1, seed=20)
        xd.copy_(torch.from_numpy(x.view(np.int16)))
        g.replay()
        torch.cuda.synchronize()
        assert archead.archead_sync_status(pack) == archead.OK
        gu.check_logits(y.cpu().numpy().astype(np.float64), oracle.logits(head, shape, x),
                        where="capture at M=1 after warm-up at M=8, d=8192")
    finally:
        pack.close()
