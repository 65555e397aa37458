"""Host-side checks of bench.py's measurement helpers (no GPU).

The bench reports a kernel's ncu DRAM traffic only while the kernel sources
still hash to the value the counters were taken on, divides whole-job tokens
by the slowest replica's time, and takes its roofline denominator from the
measured peaks file, else the recipe's fallback.
"""
import json
import os

import pytest

import bench


def test_traffic_reported_only_for_the_captured_sources(monkeypatch):
    digest = bench.kernel_sources_sha256(bench.NCU_TRAFFIC["sources"])
    # figures recorded for exactly these sources are reported
    same = dict(bench.NCU_TRAFFIC, sha256=digest)
    monkeypatch.setattr(bench, "NCU_TRAFFIC", same)
    assert bench.ncu_traffic("bf16") == bench.NCU_TRAFFIC["bytes"]["bf16"]
    assert bench.ncu_traffic("int4") == bench.NCU_TRAFFIC["bytes"]["int4"]
    # any change to the sources (here: a different recorded hash) withdraws them
    changed = dict(bench.NCU_TRAFFIC, sha256="0" * 64)
    monkeypatch.setattr(bench, "NCU_TRAFFIC", changed)
    assert bench.ncu_traffic("bf16") is None
    assert bench.ncu_traffic("int4") is None


def test_traffic_figures_are_close_to_the_algorithmic_bytes():
    # one full-size batch-1 layer: W_gate + gate-active W_up rows + both-active
    # W_down rows, 161.5 MB (bf16) / 45.4 MB (INT4); DRAM traffic well above
    # that would mean re-reads
    assert 161.5e6 <= bench.NCU_TRAFFIC["bytes"]["bf16"] <= 1.05 * 161.5e6
    assert 45.4e6 <= bench.NCU_TRAFFIC["bytes"]["int4"] <= 1.05 * 45.4e6


@pytest.mark.parametrize("batch,steps,world,t,expect", [(1, 50, 1, 0.5, 100.0), (8, 10, 4, 2.0, 160.0)])
def test_whole_job_value(batch, steps, world, t, expect):
    assert bench.whole_job_value(batch, steps, world, t) == pytest.approx(expect)


def test_peaks_measured_or_fallback(tmp_path, monkeypatch):
    peaks_file = os.path.join(bench.ROOT, "MEASURED_PEAKS.json")
    got = bench.load_peaks()
    if os.path.exists(peaks_file):
        with open(peaks_file) as f:
            assert got == {"hbm_gbs": float(json.load(f)["hbm_gbs"]), "source": "measured"}
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_peaks() == {"hbm_gbs": 6800.0, "source": "fallback"}
