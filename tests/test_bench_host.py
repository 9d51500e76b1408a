"""Host-side pieces of bench.py on the CPU: the traffic record read from a profile
summary is used only while the profiled sources are unchanged, the algorithmic
byte counts follow the per-unit figures of the measurement section, and the
reference arm's line carries the keys of the benchmark's contract."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
import workloads as wl  # noqa: E402


def test_profiled_traffic_needs_matching_sources(tmp_path, monkeypatch):
    src = tmp_path / "k.cu"
    src.write_text("__global__ void k() {}\n")
    prof = tmp_path / "profiles"
    prof.mkdir()
    sha = bench.source_sha256([str(src)])
    (prof / "k.md").write_text(f"# k\n\ntraffic_bytes_per_launch: 1234\nsource_sha256: {sha}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic([str(src)], "k.md") == 1234.0
    src.write_text("__global__ void k() { }\n")                 # the kernel changed: no record
    assert bench.profiled_traffic([str(src)], "k.md") is None
    assert bench.profiled_traffic([str(src)], "missing.md") is None


def test_step_bytes_follow_the_per_unit_figures():
    w = wl.CONFIGS["decode_loop_b128_ctx32k"]
    L, cand = 33716.6, 1.15
    by = bench.step_bytes(w, L, cand)
    B = w.B
    assert by["verify_greedy"] == 2 * B * (w.K + 1) * w.V                  # the logits, bf16
    assert by["find_candidates"] == pytest.approx(4 * B * L)                # ids scanned
    assert by["rank_hidden"] == pytest.approx(2 * B * (cand + 1) * w.d)     # H_{j-1} rows and H_{t-1}
    assert by["rank_attention"] == pytest.approx(2 * B * cand * w.R)
    assert by["draft_step"] == pytest.approx(by["find_candidates"] + by["rank_hidden"] + by["rank_attention"]
                                             + by["extract_draft"])
    # the indexed drafting reads no context: an index entry and the appended ids instead
    assert by["draft_index"] < by["draft_step"] - by["find_candidates"] + B * 64 * 2
    assert by["verify_greedy_draft"] == pytest.approx(by["verify_greedy"] + by["draft_index"])
    assert 426e6 < by["verify_greedy"] < 427e6


def test_reference_arm_line_has_the_contract_keys(monkeypatch):
    """bench.py --impl reference on a shrunken decode loop (the oracle on the host):
    one JSON-ready dict with the reference arm's keys, its own timing as value, and a
    cpu_baseline and an e2e that describe this run (no host-device copies)."""
    small = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=4, prompt_len=192, out_len=64, V=300, d=32,
                                                          layers=1, heads=4, planted_heads=1)
    monkeypatch.setattr(bench, "workload", lambda args: small)
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--steps", "3", "--warmup", "3"])
    out = bench.run_reference(bench.parse(), 1, 0)
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in out, k
    assert out["impl"] == "reference" and out["unit"] == "steps/s" and out["value"] > 0
    assert out["steps"] == 3 and out["warmup"] == 3 and out["metric"] == bench.METRIC
    assert out["config"]["workload"] == bench.workload_name(small)
    assert out["config"] == bench.bench_config(small, bench.parse(), 1)       # the same dict as our arm's
    cb = out["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] == 1 and cb["value"] == out["value"] and "sample" in cb
    e = out["e2e"]
    assert e["value"] == out["value"] and e["unit"] == out["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_oracle_single_step_on_sparse_rows_matches_dense():
    """The configs' oracle timing runs the oracle on host arrays holding only the rows
    its ranking reads; its rankings there equal those on the whole tensors."""
    import numpy as np
    import torch
    import oracle
    w = wl.CONFIGS["attention_b32_ctx8k"].replace(B=3, prompt_len=300, out_len=100, V=50, d=64)
    inp = wl.single_step(w, device="cpu")
    ids, L = inp["ids"].numpy(), inp["seq_len"].numpy()
    cand, cnt, _, _ = oracle.find_candidates(ids, L, w.ngram_min, w.ngram_max, w.C_cap)
    Hs, As = bench.sparse_rows(inp["H"], inp["A"], L, cand, cnt)
    dense_h = inp["H"].contiguous().view(torch.int16).numpy().view(np.uint16)
    dense_a = inp["A"].contiguous().view(torch.int16).numpy().view(np.uint16)
    for rank, full, sparse in ((oracle.rank_hidden, dense_h, Hs), (oracle.rank_attention, dense_a, As)):
        s_f, b_f, _ = rank(full, L, cand, cnt)
        s_s, b_s, _ = rank(sparse, L, cand, cnt)
        assert np.array_equal(s_f, s_s, equal_nan=True) and np.array_equal(b_f, b_s)
    assert bench.oracle_single_step(oracle, inp, w) > 0
