"""Vocabulary-parallel evaluation, host side (CPU): the split of the rows
over ranks, the sliced heads, the oracle's shard partials and combines
against its whole-head results, and the exchange on gloo ranks (world size 2)
feeding the combines.  The CUDA partials and combines are tested against the
oracle in test_gpu_sharded.py."""

import os
import socket

import numpy as np
import pytest

import oracle
from paper_2608_02703_gb300 import sharded
from synth import HeadShape, make_head, make_hidden, make_targets

SHAPES = {
    "int8": HeadShape(V=1000, d=256, core_rank=16, corr_rank=8, group_size=64),
    "sc4": HeadShape(V=700, d=320, core_rank=10, corr_rank=6, group_size=64, fmt="sc4"),
}


@pytest.mark.parametrize("V", [2, 5, 127, 128, 129, 1000, 4096, 151936, 262144])
@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
def test_shard_rows_cover_the_vocabulary_once(V, world):
    if V < world:
        with pytest.raises(ValueError):
            sharded.shard_rows(V, world, 0)
        return
    blocks = [sharded.shard_rows(V, world, r) for r in range(world)]
    pos = 0
    for r0, n in blocks:
        assert r0 == pos and n >= 1
        pos += n
    assert pos == V
    if -(-V // 128) >= world:  # whole tiles per rank
        assert all(r0 % 128 == 0 for r0, _ in blocks)
        sizes = [-(-n // 128) for _, n in blocks]
        assert max(sizes) - min(sizes) <= 1


@pytest.mark.parametrize("fmt", sorted(SHAPES))
def test_shard_heads_give_the_column_blocks(fmt):
    shape = SHAPES[fmt]
    head = make_head(shape, seed=3)
    x = make_hidden(shape.d, 3, seed=3)
    full = oracle.logits(head, shape, x)
    for world in (2, 3):
        for r in range(world):
            r0, n = sharded.shard_rows(shape.V, world, r, align=64)
            sub, sub_shape = sharded.shard_head(head, shape, r0, n)
            assert sub_shape.V == n and oracle.packed_bytes(sub_shape) < oracle.packed_bytes(shape)
            assert np.array_equal(oracle.logits(sub, sub_shape, x), full[:, r0:r0 + n])


@pytest.mark.parametrize("fmt", sorted(SHAPES))
def test_oracle_shard_combine_equals_the_whole_head(fmt):
    shape = SHAPES[fmt]
    head = make_head(shape, seed=4)
    M = 6
    x = make_hidden(shape.d, M, seed=4)
    t = make_targets(shape.V, M, seed=4)
    ref = oracle.cross_entropy(head, shape, x, t)
    y = oracle.logits(head, shape, x)
    for cuts in ([0, shape.V], [0, 300, shape.V], [0, 1, 2, 333, shape.V]):
        parts = np.stack([oracle.lse_partial(head, shape, x, t, a, b - a) for a, b in zip(cuts[:-1], cuts[1:])])
        ce = oracle.lse_combine(parts)
        assert np.allclose(ce, ref["ce"], rtol=0, atol=1e-12)
        assert np.allclose(ce, np.logaddexp.reduce(y, axis=1) - y[np.arange(M), t], rtol=0, atol=1e-12)
        vals = np.stack([y[:, a:b].max(axis=1) for a, b in zip(cuts[:-1], cuts[1:])])
        idxs = np.stack([y[:, a:b].argmax(axis=1) for a, b in zip(cuts[:-1], cuts[1:])])
        gi, gv = oracle.argmax_combine(vals, idxs, np.array(cuts[:-1]))
        assert np.array_equal(gi, np.argmax(y, axis=1)) and np.array_equal(gv, y.max(axis=1))
    # A target that no shard holds gives NaN.
    parts = np.stack([oracle.lse_partial(head, shape, x, np.full(M, shape.V + 5), 0, shape.V)])
    assert np.all(np.isnan(oracle.lse_combine(parts)))


def test_oracle_argmax_combine_ties_go_to_the_lowest_global_row():
    vals = np.array([[1.0, 2.0], [1.0, 2.0], [0.5, 2.0]])
    idxs = np.array([[7, 0], [3, 5], [0, 1]])
    row0 = np.array([0, 100, 200])
    gi, gv = oracle.argmax_combine(vals, idxs, row0)
    assert gi.tolist() == [7, 0] and gv.tolist() == [1.0, 2.0]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch
    import torch.distributed as dist

    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        for fmt, shape in sorted(SHAPES.items()):
            head = make_head(shape, seed=5)
            M = 5
            x = make_hidden(shape.d, M, seed=5)
            t = make_targets(shape.V, M, seed=5)
            r0, n = sharded.shard_rows(shape.V, world, rank)
            sub, sub_shape = sharded.shard_head(head, shape, r0, n)
            # This rank's partials, from its own slice of the head.
            mine = oracle.lse_partial(sub, sub_shape, x, t - r0, 0, n)
            assert np.array_equal(mine, oracle.lse_partial(head, shape, x, t, r0, n))
            gathered = sharded.exchange(torch.from_numpy(mine), None).numpy()
            y = oracle.logits(sub, sub_shape, x)
            vals = sharded.exchange(torch.from_numpy(y.max(axis=1)), None).numpy()
            idxs = sharded.exchange(torch.from_numpy(y.argmax(axis=1).astype(np.int32)), None).numpy()
            row0s = sharded.exchange(torch.tensor([r0], dtype=torch.int32), None).numpy().reshape(-1)
            gi, gv = oracle.argmax_combine(vals, idxs, row0s)
            out[(rank, fmt)] = (oracle.lse_combine(gathered).tolist(), gi.tolist(), gv.tolist(), row0s.tolist())
    finally:
        dist.destroy_process_group()


def test_exchange_and_combine_on_gloo_ranks():
    import torch.multiprocessing as mp

    world = 2
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, start_method="spawn", join=True)
    for fmt, shape in sorted(SHAPES.items()):
        head = make_head(shape, seed=5)
        M = 5
        x = make_hidden(shape.d, M, seed=5)
        t = make_targets(shape.V, M, seed=5)
        ref = oracle.cross_entropy(head, shape, x, t)
        for rank in range(world):
            ce, gi, gv, row0s = out[(rank, fmt)]
            assert row0s == [sharded.shard_rows(shape.V, world, r)[0] for r in range(world)]
            assert np.allclose(ce, ref["ce"], rtol=0, atol=1e-12), fmt
            assert gi == ref["argmax"].tolist(), fmt
        assert out[(0, fmt)] == out[(1, fmt)]  # every rank ends with the same result
