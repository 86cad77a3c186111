"""Vocabulary-parallel evaluation through the C ABI on one GPU: a head cut
into P row blocks, one pack each (what P ranks would hold), against the
oracle and against the unsharded pack.  The exchange itself is a host-side
all-gather (tests/test_sharded.py covers it on gloo ranks); here the blocks'
outputs are stacked on the device in shard order and fed to the combines."""

import numpy as np
import pytest

import oracle
from paper_2608_02703_gb300 import archead, sharded
from synth import HeadShape, make_head, make_hidden, make_targets
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

SHAPES = {
    "tiny": HeadShape(V=4096, d=512, core_rank=64, corr_rank=16, group_size=64),
    "ragged": HeadShape(V=1000, d=256, core_rank=16, corr_rank=8, group_size=64),
    "sc4": HeadShape(V=4096, d=512, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
}


@pytest.fixture(scope="module", autouse=True)
def _build():
    from paper_2608_02703_gb300.build import build

    build()


def _cuts(V, how):
    if how == "tiles2":
        return [sharded.shard_rows(V, 2, r)[0] for r in range(2)] + [V]
    if how == "tiles3":
        return [sharded.shard_rows(V, 3, r)[0] for r in range(3)] + [V]
    return [0, 333, 700, V]  # blocks that start inside a 128-row tile


def _packs(head, shape, cuts):
    out = []
    for a, b in zip(cuts[:-1], cuts[1:]):
        sub, sub_shape = sharded.shard_head(head, shape, a, b - a)
        out.append((a, archead.archead_pack_create(sub, sub_shape)))
    return out


@pytest.mark.parametrize("name", sorted(SHAPES))
@pytest.mark.parametrize("how", ["tiles2", "tiles3", "ragged"])
@pytest.mark.parametrize("M,path", [(1, archead.PATH_DECODE), (16, archead.PATH_DECODE), (40, archead.PATH_AUTO),
                                    (300, archead.PATH_PREFILL)])
def test_shards_match_the_whole_head(name, how, M, path):
    import torch

    shape = SHAPES[name]
    head = make_head(shape, seed=31)
    cuts = _cuts(shape.V, how)
    whole = archead.archead_pack_create(head, shape)
    packs = _packs(head, shape, cuts)
    try:
        x = make_hidden(shape.d, M, seed=32 + M)
        t = make_targets(shape.V, M, seed=32 + M)
        xd = gu.to_dev(x)
        td = gu.to_dev(t)
        ref = oracle.cross_entropy(head, shape, x, t)
        ref_y = oracle.logits(head, shape, x)
        # Logits: each block is its own columns.  Blocks cut at multiples of
        # 16 rows keep every row's place in its 16-row MMA fragment, and the
        # kernels then give the unsharded pack's logits bit for bit (the
        # decode kernel encodes the two 8-row halves of a fragment
        # differently, so other cuts round differently, within the bar).
        full = gu.forward(whole, x, archead.OUT_FP32, path)
        blocks = np.concatenate([gu.forward(p, x, archead.OUT_FP32, path) for _, p in packs], axis=1)
        aligned = all(c % 16 == 0 for c in cuts)
        if aligned:
            assert np.array_equal(blocks, full)
        gu.check_logits(blocks, ref_y, where=f"{name} {how} M={M} shards")
        # Cross entropy: partials in shard order, then the combine.
        # (each shard's output in its own buffer, as on its own rank; stacked
        # in shard order like the all-gather does)
        own = [torch.full((M, 3), float("nan"), dtype=torch.float32, device="cuda") for _ in packs]
        for (a, p), buf in zip(packs, own):
            archead.archead_forward_lse_partial(p, xd, M, td, a, buf, path)
        parts = torch.stack(own)
        ce = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
        archead.archead_lse_combine(parts, len(packs), M, ce)
        torch.cuda.synchronize()
        got = ce.cpu().numpy().astype(np.float64)
        assert np.max(np.abs(got - ref["ce"])) <= gu.CE_ABS
        whole_ce, st = gu.forward_ce(whole, x, t, path)
        assert st == archead.OK
        # same rows, same arithmetic up to the merge order (cuts inside a
        # fragment also change the rows' rounding, within the CE bar above)
        if aligned:
            assert np.max(np.abs(got - whole_ce)) <= 1e-5
        # Partials against the oracle's: max and target logit within the logit bar.
        pn = parts.cpu().numpy().astype(np.float64)
        rms = float(np.sqrt(np.mean(ref_y ** 2)))
        for i, (a, b) in enumerate(zip(cuts[:-1], cuts[1:])):
            op = oracle.lse_partial(head, shape, x, t, a, b - a)
            assert np.all(np.abs(pn[i, :, 0] - op[:, 0]) <= gu.LOGIT_REL * rms)
            assert np.array_equal(np.isinf(pn[i, :, 2]), np.isinf(op[:, 2]))
        # Greedy: per-shard (value, local row), then the combine.
        own_v = [torch.empty(M, dtype=torch.float32, device="cuda") for _ in packs]
        own_i = [torch.empty(M, dtype=torch.int32, device="cuda") for _ in packs]
        for (_, p), v, i in zip(packs, own_v, own_i):
            archead.archead_forward_argmax_path(p, xd, M, i, v, path)
        vals, idxs = torch.stack(own_v), torch.stack(own_i)
        row0 = torch.tensor(cuts[:-1], dtype=torch.int32, device="cuda")
        gi = torch.empty(M, dtype=torch.int32, device="cuda")
        gv = torch.empty(M, dtype=torch.float32, device="cuda")
        archead.archead_argmax_combine(vals, idxs, row0, len(packs), M, gi, gv)
        gi_n, gv_n = gi.cpu().numpy().astype(np.int64), gv.cpu().numpy().astype(np.float64)
        gu.check_greedy(gi_n, gv_n, ref_y, where=f"{name} {how} M={M} greedy")
        # the combine picks the first maximum of the shards' own logits
        assert np.array_equal(gi_n, np.argmax(blocks, axis=1)) and np.array_equal(gv_n, blocks.max(axis=1))
        if aligned:
            wi, wv = gu.forward_argmax(whole, x, path)
            assert np.array_equal(gi_n, wi) and np.array_equal(gv_n, wv)
    finally:
        whole.close()
        for _, p in packs:
            p.close()


def test_target_outside_every_shard_gives_nan():
    import torch

    shape = SHAPES["ragged"]
    head = make_head(shape, seed=33)
    cuts = _cuts(shape.V, "ragged")
    packs = _packs(head, shape, cuts)
    try:
        M = 4
        x = gu.to_dev(make_hidden(shape.d, M, seed=33))
        t = gu.to_dev(np.array([0, shape.V, 999, -1], dtype=np.int32))
        own = [torch.empty((M, 3), dtype=torch.float32, device="cuda") for _ in packs]
        for (a, p), buf in zip(packs, own):
            archead.archead_forward_lse_partial(p, x, M, t, a, buf)
        parts = torch.stack(own)
        ce = torch.empty(M, dtype=torch.float32, device="cuda")
        archead.archead_lse_combine(parts, len(packs), M, ce)
        got = ce.cpu().numpy()
        assert np.isfinite(got[0]) and np.isfinite(got[2]) and np.isnan(got[1]) and np.isnan(got[3])
    finally:
        for _, p in packs:
            p.close()


def test_sharded_head_class_on_a_one_rank_group():
    """ShardedHead end to end on a single-rank NCCL group (the exchange is the
    all-gather a multi-GPU run makes, with one participant)."""
    import os
    import socket

    import torch
    import torch.distributed as dist

    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("nccl", rank=0, world_size=1, device_id=torch.device("cuda", 0))
    try:
        shape = SHAPES["tiny"]
        head = make_head(shape, seed=34)
        sh = sharded.ShardedHead(head, shape)
        M = 16
        x = make_hidden(shape.d, M, seed=34)
        t = make_targets(shape.V, M, seed=34)
        ce = torch.empty(M, dtype=torch.float32, device="cuda")
        sh.cross_entropy(gu.to_dev(x), M, gu.to_dev(t), ce)
        gi = torch.empty(M, dtype=torch.int32, device="cuda")
        gv = torch.empty(M, dtype=torch.float32, device="cuda")
        sh.greedy(gu.to_dev(x), M, gi, gv)
        y = torch.empty((M, sh.rows), dtype=torch.float32, device="cuda")
        sh.logits(gu.to_dev(x), M, y, archead.OUT_FP32)
        torch.cuda.synchronize()
        ref = oracle.cross_entropy(head, shape, x, t)
        ref_y = oracle.logits(head, shape, x)
        assert np.max(np.abs(ce.cpu().numpy() - ref["ce"])) <= gu.CE_ABS
        gu.check_greedy(gi.cpu().numpy().astype(np.int64), gv.cpu().numpy().astype(np.float64), ref_y)
        gu.check_logits(y.cpu().numpy().astype(np.float64), ref_y)
        sh.close()
    finally:
        dist.destroy_process_group()
