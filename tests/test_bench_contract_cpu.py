"""The benchmark's contract on the CPU: the reference arm's JSON line, and the
algorithmic work the metric divides by, counted independently.

The attention FLOPs are 4 d Hq per (query, key) pair the mask allows (2 d for
q.k, 2 d for p.v); the decode bytes are each request's assembled K and V read
once.  Both are checked here against a brute-force count of the visible pairs
(the oracle's own mask rule, query i of S sees T_art + (S_kv - S) + i + 1 keys)
and against the figure worked out for the tiny configuration (3 artifacts of
37, 64, 100 tokens, 16 suffix tokens, d = 64, 4 query heads: 3.43 MFLOP).
"""
from __future__ import annotations

import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from gen import Geometry, make_custom, make_workload  # noqa: E402


def _visible_pairs(wl):
    n = 0
    for r in range(wl.n_req):
        t_art = wl.t_art(r)
        for i in range(wl.S):
            n += t_art + (wl.S_kv - wl.S) + i + 1
    return n


def test_tiny_attention_flops():
    wl = make_workload("tiny")
    assert _visible_pairs(wl) == 16 * 201 + 16 * 17 // 2
    assert bench.attention_flops(wl) == 4 * 64 * 4 * (16 * 201 + 136) == 3_432_448


def test_work_of_multi_request_decode_and_prefill_shapes():
    g = Geometry(hidden=128, n_q_heads=8, n_kv_heads=2, head_dim=64, rank=8)
    lengths = [70, 5, 130, 64]
    reqs = [[0, 2], [], [3, 1, 3], [2]]
    for S, S_kv in ((1, 9), (5, 5), (3, 40)):
        wl = make_custom("c", g, 7, lengths, reqs, S, S_kv)
        assert bench.attention_flops(wl) == 4 * 64 * 8 * _visible_pairs(wl)
        # K and V, Hkv heads of d bf16 values, for every assembled and suffix token
        toks = sum(sum(lengths[a] for a in r) + S_kv for r in reqs)
        assert bench.kv_bytes(wl) == toks * 2 * 2 * 64 * 2
        assert bench.is_decode(wl) == (S * g.group <= 16)
        # distinct K/V: artifacts 0, 1, 2, 3 once each (2 and 3 are used twice), and the suffixes
        assert bench.kv_distinct_bytes(wl) == (70 + 5 + 130 + 64 + 4 * S_kv) * 2 * 2 * 64 * 2


def test_qproj_flops_counts_base_and_low_rank_products():
    wl = make_workload("tiny")
    g = wl.geom
    M = wl.S
    assert bench.qproj_flops(wl) == 2 * M * 256 * 256 + 2 * M * 256 * 8 + 2 * M * 8 * 256
    assert g.d_q == 256 and g.rank == 8


def test_reference_arm_line_keeps_the_contract():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "3"], capture_output=True, text=True, timeout=300, cwd=ROOT,
                       env=dict(os.environ, RANK="0", WORLD_SIZE="1"))
    assert r.returncode == 0, r.stderr
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "impl", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["unit"] == "TFLOP/s" and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["config"]["workload"] == "tiny" and d["dtype"] == "f64"
    assert d["value"] > 0 and d["cpu_baseline"]["value"] == d["value"] and d["e2e"]["value"] == d["value"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1 and d["cpu_baseline"]["sample"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["vs_baseline"] is None


def test_warmup_below_three_is_raised_to_three():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=300, cwd=ROOT,
                       env=dict(os.environ, RANK="0", WORLD_SIZE="1"))
    assert r.returncode == 0, r.stderr
    assert json.loads(r.stdout)["warmup"] == 3


def test_clock_record_parsing():
    # nvidia-smi --format=csv,noheader,nounits lines of ClockSampler.FIELDS:
    # index, sm, max sm, power, active mask, hw_slowdown, hw_thermal, sw_thermal, sw_power_cap
    idle = "0, 345, 2070, 180.1, 0x0000000000000001, Not Active, Not Active, Not Active, Not Active"
    busy = "0, 2070, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active"
    capped = "0, 1965, 2070, 1399.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active"
    hot = "0, 1800, 2070, 1200.0, 0x0000000000000040, Not Active, Active, Not Active, Not Active"
    r = bench.parse_clocks("\n".join([idle, busy, busy, busy]))
    assert r == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 4}   # idle sample left out
    r = bench.parse_clocks("\n".join([busy, capped, capped]))
    assert r["reasons"] == ["sw_power_cap"] and r["sm_mhz"] == 1965.0
    r = bench.parse_clocks("\n".join([busy, hot, "garbage", "0, N/A, 2070, x, y, a, b, c, d"]))
    assert r["reasons"] == ["hw_thermal_slowdown"] and r["samples"] == 2
    assert bench.parse_clocks("") is None and bench.parse_clocks("no samples here") is None


def test_clock_sampler_without_nvidia_smi(monkeypatch):
    # a host without the tool records no clocks instead of failing the run
    monkeypatch.setenv("PATH", "")
    s = bench.ClockSampler(0)
    assert s.stop() is None


def test_decode_read_fractions():
    # the decode roofline in the bytes a launch must move: distinct K/V per
    # second against the peak, and the measured DRAM bytes when a current
    # traffic record exists
    g = Geometry(hidden=128, n_q_heads=8, n_kv_heads=2, head_dim=64, rank=8)
    wl = make_custom("d", g, 7, [70, 5, 130, 64], [[0, 2], [2, 1], [3, 1, 3], [2]], 1, 9)
    per_token = 2 * 2 * 64 * 2
    distinct = (70 + 5 + 130 + 64 + 4 * 9) * per_token
    f = bench.decode_read_fracs(wl, 0.5, 100.0, None)
    assert f["distinct_bytes"] == distinct and "dram_frac" not in f
    assert abs(f["distinct_frac"] - round(distinct / 0.5e-3 / 1e9 / 100.0, 4)) < 1e-12
    f = bench.decode_read_fracs(wl, 0.5, 100.0, 10_000_000)
    assert abs(f["dram_frac"] - round(1e7 / 0.5e-3 / 1e9 / 100.0, 4)) < 1e-12
