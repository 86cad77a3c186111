"""Full-size heads (the Qwen3-8B and Gemma-shaped configurations and the
Qwen3-8B head in the paper's own packed format, the same seeded heads
bench.py times) through the C ABI against the fp64 oracle:
the whole vocabulary for decode token counts (all tokens up to 16, sampled
tokens of the 32- and 64-token launches), sampled tokens for prefill
(a token's logits depend on that token's hidden state only, so the oracle
checks sampled rows exactly)."""

import numpy as np
import pytest

import oracle
from paper_2608_02703_gb300 import archead
from synth import SHAPES, make_head, make_hidden, make_targets
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

FULL = ("qwen3-8b", "gemma-4-e4b", "qwen3-8b-sc4")
PREFILL_M = {"qwen3-8b": 4096, "gemma-4-e4b": 2048, "qwen3-8b-sc4": 4096}

_state = {}


@pytest.fixture(scope="module", autouse=True)
def _build():
    from paper_2608_02703_gb300.build import build

    build()
    yield
    for pack, _ in _state.values():
        pack.close()
    _state.clear()


def get(name):
    if name not in _state:
        shape = SHAPES[name]
        head = make_head(shape, seed=0)
        _state[name] = (archead.archead_pack_create(head, shape), head)
    return _state[name]


def _rows(y, idx):
    return y[idx].float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("name", FULL)
@pytest.mark.parametrize("M", [1, 16])
def test_decode_full_vocabulary(name, M):
    import torch

    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=1, n_outliers=shape.n_outliers)
    ref = oracle.logits(head, shape, x)
    y = torch.full((M, shape.V), float("nan"), dtype=torch.float32, device="cuda")
    archead.archead_forward(pack, gu.to_dev(x), M, y, archead.OUT_FP32)
    assert archead.archead_sync_status(pack) == archead.OK
    got = _rows(y, slice(None))
    gu.check_logits(got, ref, where=f"{name} decode M={M}")
    gu.check_argmax(got, ref, where=f"{name} decode M={M}")


@pytest.mark.parametrize("name", FULL)
def test_decode_cross_entropy_full_vocabulary(name):
    pack, head = get(name)
    shape = SHAPES[name]
    M = 16
    x = make_hidden(shape.d, M, seed=2, n_outliers=shape.n_outliers)
    t = make_targets(shape.V, M, seed=2)
    ref = oracle.cross_entropy(head, shape, x, t)
    ce, st = gu.forward_ce(pack, x, t)
    assert st == archead.OK
    assert np.max(np.abs(ce - ref["ce"])) <= gu.CE_ABS, f"{name}: CE max|d|={np.max(np.abs(ce - ref['ce'])):.3e}"


@pytest.mark.parametrize("name", FULL)
def test_greedy_full_vocabulary(name):
    pack, head = get(name)
    shape = SHAPES[name]
    M = 16
    x = make_hidden(shape.d, M, seed=3, n_outliers=shape.n_outliers)
    ref = oracle.logits(head, shape, x)
    idx, val = gu.forward_argmax(pack, x)
    gu.check_greedy(idx, val, ref, where=f"{name} greedy M={M}")


@pytest.mark.parametrize("name", FULL)
@pytest.mark.parametrize("M", [27, 64])
def test_decode_wide_sampled_tokens(name, M):
    """One launch of the 32- resp. 64-token decode instance (every n-tile of
    the launch, the ragged one included) over the whole vocabulary: logits,
    greedy output and fused CE on one token of each 8-token n-tile."""
    import torch

    pack, head = get(name)
    shape = SHAPES[name]
    x = make_hidden(shape.d, M, seed=4, n_outliers=shape.n_outliers)
    t = make_targets(shape.V, M, seed=4)
    idx = np.unique(np.minimum(np.arange(0, M + 7, 8) + (np.arange(0, M + 7, 8) // 8) % 8, M - 1))
    ref = oracle.logits(head, shape, x[idx])
    y = torch.full((M, shape.V), float("nan"), dtype=torch.float32, device="cuda")
    archead.archead_forward(pack, gu.to_dev(x), M, y, archead.OUT_FP32)
    assert archead.archead_sync_status(pack) == archead.OK
    got = _rows(y, torch.from_numpy(idx).cuda())
    gu.check_logits(got, ref, where=f"{name} decode M={M} sampled")
    gu.check_argmax(got, ref, where=f"{name} decode M={M} sampled")
    del y
    gi, gv = gu.forward_argmax(pack, x)
    gu.check_greedy(gi[idx], gv[idx], ref, where=f"{name} decode greedy M={M} sampled")
    ce, st = gu.forward_ce(pack, x, t)
    assert st == archead.OK
    ref_ce = oracle.cross_entropy(head, shape, x[idx], t[idx])
    d = np.abs(ce[idx] - ref_ce["ce"])
    assert np.max(d) <= gu.CE_ABS, f"{name}: decode CE M={M} max|d|={np.max(d):.3e}"


@pytest.mark.parametrize("name", FULL)
def test_prefill_sampled_tokens(name):
    """The bench's prefill launch (M = 4096 / 2048 tokens: logits, greedy
    output and fused CE), checked on sampled tokens: first and last of the 256-token tiles,
    the ragged end and a few random ones."""
    import torch

    pack, head = get(name)
    shape = SHAPES[name]
    M = PREFILL_M[name]
    x = make_hidden(shape.d, M, seed=1, n_outliers=shape.n_outliers)
    t = make_targets(shape.V, M, seed=1)
    rng = np.random.default_rng(7)
    idx = np.unique(np.concatenate([[0, 1, 255, 256, 511, M // 2, M - 2, M - 1], rng.integers(0, M, 4)]))
    ref = oracle.logits(head, shape, x[idx])
    y = torch.empty((M, shape.V), dtype=torch.bfloat16, device="cuda")
    archead.archead_forward(pack, gu.to_dev(x), M, y, archead.OUT_BF16)
    assert archead.archead_sync_status(pack) == archead.OK
    got = _rows(y, torch.from_numpy(idx).cuda())
    gu.check_logits(got, ref, bf16=True, where=f"{name} prefill M={M} sampled")
    gu.check_argmax(got, ref, where=f"{name} prefill M={M} sampled")
    del y
    gi, gv = gu.forward_argmax(pack, x)
    gu.check_greedy(gi[idx], gv[idx], ref, where=f"{name} prefill greedy M={M} sampled")
    ce, st = gu.forward_ce(pack, x, t)
    assert st == archead.OK
    ref_ce = oracle.cross_entropy(head, shape, x[idx], t[idx])
    d = np.abs(ce[idx] - ref_ce["ce"])
    assert np.max(d) <= gu.CE_ABS, f"{name}: prefill CE max|d|={np.max(d):.3e}"
    assert np.all(np.isfinite(ce))
