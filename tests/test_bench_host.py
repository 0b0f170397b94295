"""Host logic of the benchmark (no GPU): the byte and flop counts behind the
roofline objects, the traffic figures' tie to the kernel sources, the clock
record's parsing and the peaks file.  Each count is checked against a route
other than its own formula: a per-row tally, a closed form of the paper's
shapes (Eq. 6-8: c = W_c [m; u] is d x 2d, [v; g] = [W_v; W_g] r is 2d x d),
or an invariant."""

import json
import os

import numpy as np
import pytest

import bench
from paper_2608_29748_gb300.workloads import CONFIGS, PROFILE_CONFIG

CFG5 = CONFIGS[5]


def per_row_tally(cfg, accept, windows):
    """Rows a windowed schedule reads, one (sequence, row) at a time: row i of
    sequence b is read when its window starts at or before A_b (every draft
    before the window matched)."""
    rows = 0
    for b in range(len(accept)):
        for k in range(len(windows) - 1):
            if accept[b] >= windows[k]:
                rows += windows[k + 1] - windows[k]
    return rows * cfg.V * cfg.elem_bytes


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_read_logits_bytes_matches_a_per_row_tally(seed):
    rng = np.random.default_rng(seed)
    K = CFG5.K
    accept = rng.integers(0, K + 1, size=37)
    for windows in ([0, K + 1], [0, 4, 10, K + 1], [0, 1, 2, 3, K + 1], list(range(K + 2))):
        got = bench.read_logits_bytes(CFG5, accept, windows)
        assert got == per_row_tally(CFG5, accept, windows)
        # between what the outputs need and what one pass reads
        assert bench.needed_logits_bytes(CFG5, accept) <= got <= len(accept) * (K + 1) * CFG5.V * 2
    # one window is one pass over every row; a window per row reads exactly the needed rows
    assert bench.read_logits_bytes(CFG5, accept, [0, K + 1]) == len(accept) * (K + 1) * CFG5.V * 2
    assert bench.read_logits_bytes(CFG5, accept, list(range(K + 2))) == bench.needed_logits_bytes(CFG5, accept)


def test_needed_logits_bytes_special_cases():
    K, V = CFG5.K, CFG5.V
    assert bench.needed_logits_bytes(CFG5, np.zeros(5, dtype=np.int32)) == 5 * V * 2       # row 0 only
    assert bench.needed_logits_bytes(CFG5, np.full(5, K, dtype=np.int32)) == 5 * (K + 1) * V * 2  # every row


def test_conditioning_flops_closed_forms():
    d, R = CFG5.d, 2876
    # broadcast e: 4 R d^2 (correction) + 4 R d^2 (v and the r half of the gate) + 2 d^2 (W_g,e e once)
    assert bench.conditioning_flops(CFG5, R, dense_e=False) == 8 * R * d * d + 2 * d * d
    # the bench line of config 5 quotes 386.04 GFLOP
    assert bench.conditioning_flops(CFG5, R, dense_e=False) == 386043740160
    # per-position e: W_g,e e for every row
    assert bench.conditioning_flops(CFG5, R, dense_e=True) == 10 * R * d * d
    # raw (r = m): no correction GEMM; overwrite / none: no projections
    assert bench.conditioning_flops(CFG5, R, dense_e=False, variant="raw") == 4 * R * d * d + 2 * d * d
    assert bench.conditioning_flops(CFG5, R, False, "overwrite") == bench.conditioning_flops(CFG5, R, False, "none") == 0
    assert bench.conditioning_flops(CFG5, 0, dense_e=False) == 2 * d * d


def test_verify_bytes_accounting():
    """Rows carried plus rows copied are all B K positions; packing reads and
    writes the [m; u] rows (2d each) and writes the row map."""
    cfg = PROFILE_CONFIG
    B, K, d, V = cfg.B, cfg.K, cfg.d, cfg.V
    rng = np.random.default_rng(3)
    accept = rng.integers(0, K + 1, size=B)
    n = np.maximum(0, K - 1 - accept)
    R = int(n.sum())
    base = bench.needed_logits_bytes(cfg, accept) + B * K * 4 + B * (K + 1) * 4 + 3 * B * 4
    copies = (B * K - R) * d * 2
    assert bench.verify_bytes(cfg, n, False, accept=accept) == base + copies
    assert bench.verify_bytes(cfg, n, True, accept=accept) - bench.verify_bytes(cfg, n, False, accept=accept) \
        == 2 * R * 2 * d * 2 + R * 4
    # overwrite writes every e~ row and reads the m rows of the carried ones
    assert bench.verify_bytes(cfg, n, False, "overwrite", accept) == base + B * K * d * 2 + R * d * 2
    # without accepted lengths the whole logits tensor counts
    assert bench.verify_bytes(cfg, n, False) - bench.verify_bytes(cfg, n, False, accept=accept) \
        == (B * (K + 1) - int(np.sum(accept + 1))) * V * 2


def test_measured_traffic_follows_the_kernel_sources(monkeypatch):
    w = CFG5.name
    for phase in ("verify", "conditioning"):
        entry = bench.TRAFFIC[(phase, w)]
        if entry["sources"] == bench.kernel_sources_hash():
            assert bench.measured_traffic(phase, w, "corrected") == entry["bytes"]
        # any other variant, or another workload, has no measured figure
        assert bench.measured_traffic(phase, w, "raw") is None
        assert bench.measured_traffic(phase, "no-such-workload", "corrected") is None
        # a figure taken on other sources is not reported
        monkeypatch.setitem(bench.TRAFFIC, (phase, w), dict(entry, sources="0" * 16))
        assert bench.measured_traffic(phase, w, "corrected") is None


def test_kernel_sources_hash_changes_with_any_source(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2608_29748_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "a.cu").write_text("kernel A\n")
    (csrc / "b.cuh").write_text("header\n")
    (csrc / "notes.txt").write_text("not a source\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_sources_hash()
    (csrc / "notes.txt").write_text("edited, still not a source\n")
    assert bench.kernel_sources_hash() == h0
    (csrc / "b.cuh").write_text("header // a comment\n")
    h1 = bench.kernel_sources_hash()
    assert h1 != h0 and len(h1) == 16
    (csrc / "c.h").write_text("")
    assert bench.kernel_sources_hash() != h1


def test_clock_summary_parses_nvidia_smi_rows(tmp_path):
    path = tmp_path / "clocks.csv"
    rows = [
        "0, 2070, 2070, 1200.5, 0x0, Not Active, Not Active, Not Active, Not Active",
        "0, 2055, 2070, 1350.0, 0x4, Not Active, Not Active, Not Active, Active",
        "0, 2070, 2070, 1390.2, 0x0, Not Active, Not Active, Not Active, Not Active",
        "garbled line",
        "0, [N/A], 2070, 0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    path.write_text("\n".join(rows) + "\n")
    s = bench.ClockSampler(0)
    s.path = str(path)
    out = s.summary()
    assert out == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    assert not path.exists()  # the record is removed once read
    empty = tmp_path / "empty.csv"
    empty.write_text("")
    s.path = str(empty)
    assert s.summary() is None


def test_load_peaks_reads_the_measured_file():
    p = bench.load_peaks()
    path = os.path.join(bench.ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            raw = json.load(f)
        assert p["source"] == "measured"
        assert p["hbm_gbs"] == raw["hbm_gbs"] and p["bf16_tflops"] == raw["bf16_tflops"]
        assert p["bf16_tflops_sustained"] == raw["bf16_tflops_sustained"]
    else:
        assert p == {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                     "source": "fallback"}


def test_round_hbm_bytes_is_at_least_the_logits_and_weights():
    R = 2876
    b = bench.round_hbm_bytes(CFG5, R)
    d = CFG5.d
    assert b >= CFG5.logits_bytes() + 5 * d * d * 2 + 2 * R * d * 2
    assert bench.round_hbm_bytes(CFG5, R + 1) - b == 2 * d * 2  # one more carried row: its m and u
