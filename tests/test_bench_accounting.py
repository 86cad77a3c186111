"""bench.py's algorithmic byte and flop accounting and its use of the
committed traffic captures (host logic, CPU only)."""

import json

import bench
import oracle
from synth import SHAPES, HeadShape


def test_packed_bytes_match_the_oracle_eq10():
    for name in ("tiny", "qwen3-8b", "gemma-4-e4b", "tiny-sc4", "qwen3-8b-sc4"):
        assert bench.packed_bytes(SHAPES[name]) == oracle.packed_bytes(SHAPES[name]), name
    odd = HeadShape(V=333, d=320, core_rank=13, corr_rank=0, group_size=64, fmt="sc4")
    assert bench.packed_bytes(odd) == oracle.packed_bytes(odd)


def test_streamed_bytes_are_the_vocabulary_side_of_the_pack():
    s = SHAPES["qwen3-8b"]
    d_side = s.d * s.core_rank + 2 * 2 * s.core_rank + s.d * s.corr_rank + (s.d // s.group_size) * s.corr_rank * 2
    assert bench.packed_vocab_bytes(s) + d_side == bench.packed_bytes(s)
    assert bench.kernel_bytes(s, 1, "logits") == bench.packed_vocab_bytes(s) + 2 * s.d + 2 * s.V
    assert bench.call_flops(s, 4096) == 2 * 4096 * s.V * s.d + 2 * 4096 * (s.V + s.d) * (s.core_rank + s.corr_rank)


def test_traffic_is_used_only_for_the_sources_it_was_captured_with(tmp_path, monkeypatch):
    """A capture counts only for its kernel, workload and M, and only while the
    kernel's sources hash to the ones it was taken with (else null)."""
    table = {"decode/qwen3-8b-decode/M=1": {"dram_bytes_per_launch": 123, "sources_sha256": bench.kernel_source_hash("decode")},
             "prefill/qwen3-8b-prefill/M=1024": {"dram_bytes_per_launch": 456, "sources_sha256": "0" * 64}}
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(table))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_source_hash", lambda k: table["decode/qwen3-8b-decode/M=1"]["sources_sha256"]
                        if k == "decode" else "1" * 64)
    assert bench.captured_traffic("decode", "qwen3-8b-decode", 1) == 123
    assert bench.captured_traffic("decode", "qwen3-8b-decode", 16) is None      # no capture at this M
    assert bench.captured_traffic("prefill", "qwen3-8b-prefill", 1024) is None  # sources changed since



def test_flat_keys_repeat_the_nested_headline_figures():
    res = {
        "prefill": {"M": 4096, "logits": {"ms_per_call": 4.2, "frac_bf16_peak": 0.66},
                    "ce": {"ms_per_call": 4.8, "frac_bf16_peak": 0.58}},
        "decode_sweep": [{"M": 1, "us_per_call": 68.5, "frac_hbm": 0.77}, {"M": 16, "us_per_call": 80.0, "frac_hbm": 0.7}],
        "sc4": {"decode_sweep": [{"M": 1, "us_per_call": 66.0, "frac_hbm": 0.72}],
                "prefill": {"M": 4096, "logits": {"ms_per_call": 3.9, "frac_bf16_peak": 0.69}}},
        "gemma": {"decode_sweep": [], "prefill": {"M": 2048, "ce": {"ms_per_call": 3.0, "frac_bf16_peak": 0.51}}},
        "tiny": {"us_per_call": 9.5, "oracle": {"us_per_call": 12000.0}},
        "crossover": {"rows": [{"M": 16, "auto_us": 89.0, "dense_bf16_us": 204.0},
                               {"M": 64, "auto_us": 245.4, "dense_bf16_us": 210.7}]},
    }
    flat = bench.flat_keys(res)
    assert flat["qwen_crossover_m64_auto_us"] == 245.4 and flat["qwen_crossover_m64_dense_bf16_us"] == 210.7
    assert "qwen_crossover_m16_auto_us" not in flat  # only the rows the headline table quotes
    assert flat["qwen_prefill_m4096_logits_ms"] == 4.2 and flat["qwen_prefill_m4096_ce_frac_bf16_peak"] == 0.58
    assert flat["qwen_decode_m16_us"] == 80.0 and flat["qwen_decode_m1_kernel_frac_hbm"] == 0.77
    assert flat["qwen_sc4_decode_m1_us"] == 66.0 and flat["qwen_sc4_prefill_m4096_logits_ms"] == 3.9
    assert flat["gemma_prefill_m2048_ce_ms"] == 3.0
    assert flat["tiny_m4_us"] == 9.5 and flat["tiny_m4_oracle_us"] == 12000.0
    assert all(not isinstance(v, (dict, list)) for v in flat.values())
