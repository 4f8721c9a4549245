"""bench.py contract checks that need no GPU: the reference arm (the float64 oracle timed on
the host on a bounded row sample) prints one JSON line with the agreed keys."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_contract_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                          "tiny_fp32", "--steps", "2", "--warmup", "3", "--ref-rows", "4"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = [l for l in out.stdout.splitlines() if l.startswith("{")][-1]
    d = json.loads(line)
    assert d["impl"] == "reference"
    assert d["unit"] == "response tokens/s" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert d["config"]["workload"] == "tiny_fp32"


def _bench():
    sys.path.insert(0, ROOT)
    import bench
    return bench


def test_peak_follows_the_clock_record():
    b = _bench()
    peaks = {"hbm_gbs": 7000.0, "bf16_tflops": 1926.0, "bf16_tflops_sustained": 1749.0}
    capped = {"sm_mhz": 1545.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}
    low_clock = {"sm_mhz": 1700.0, "sm_max_mhz": 2070.0, "reasons": []}
    full = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}
    assert b.choose_peak(capped, peaks, "measured")[0] == 1749.0
    assert b.choose_peak(low_clock, peaks, "measured")[0] == 1749.0
    assert b.choose_peak(full, peaks, "measured")[0] == 1926.0
    assert b.choose_peak(None, peaks, "measured")[0] == 1926.0
    # with the clock of the sustained measurement known: a capped kernel running well above
    # that clock is held to the burst figure, one at about that clock to the sustained one
    timed = dict(peaks, sustained_mhz=1507.0)
    assert b.choose_peak(capped, timed, "measured")[0] == 1749.0  # 1545 <= 1.05 * 1507
    assert b.choose_peak({"sm_mhz": 1811.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}, timed,
                         "measured")[0] == 1926.0
    p, src = b.load_peaks()
    assert src in ("measured", "fallback") and p["bf16_tflops"] > 0


def test_whole_job_rate_counts_every_rank_over_the_slowest_time():
    b = _bench()
    assert b.whole_job_rate(1000, 10, 4, 2000.0) == 1000 * 10 * 4 / 2.0


def test_recorded_traffic_only_while_the_source_hash_matches(tmp_path, monkeypatch):
    b = _bench()
    for rel in b.KERNEL_SOURCES["gemm_dH"]:
        p = tmp_path / rel
        p.parent.mkdir(parents=True, exist_ok=True)
        p.write_text("// kernel source " + rel)
    (tmp_path / "profiles").mkdir()
    monkeypatch.setattr(b, "ROOT", str(tmp_path))
    good = b.source_hash("gemm_dH")
    prof = tmp_path / "profiles" / "gemm_dH_qwen3_1p7b.txt"
    prof.write_text(f"# header\nsource_sha256: {good}\ndram_bytes_per_launch: 8400000000\n")
    assert b.recorded_traffic("gemm_dH", "qwen3_1p7b") == 8.4e9
    assert b.recorded_traffic("gemm_dH", "qwen3_1p7b", "kl_seqmean") == 8.4e9  # same kernels and shapes
    assert b.recorded_traffic("gemm_dH", "qwen3_1p7b", "surrogate") is None    # no record for that path
    (tmp_path / b.KERNEL_SOURCES["gemm_dH"][0]).write_text("// changed")
    assert b.recorded_traffic("gemm_dH", "qwen3_1p7b") is None


def test_sampled_parity_applies_the_bounds():
    import types

    import numpy as np
    import torch
    b = _bench()
    rng = np.random.default_rng(0)
    T, d, rows = 32, 16, [1, 5, 9, 30]
    kl = rng.random(T)
    dH = rng.standard_normal((T, d))
    ref = types.SimpleNamespace(kl=kl[rows].copy(), dH_s=dH[rows].copy())
    out = {"kl": torch.from_numpy(kl).float(), "dH": torch.from_numpy(dH).float()}
    ok = b.sampled_parity("kl", rows, ref, out)
    assert ok["rows"] == 4 and ok["kl_within_bound"] and ok["dH_within_bound"]
    bad_kl = kl.copy()
    bad_kl[5] += 1e-3 + 2e-3 * kl[5]
    r = b.sampled_parity("kl", rows, ref, {"kl": torch.from_numpy(bad_kl), "dH": out["dH"]})
    assert not r["kl_within_bound"] and r["dH_within_bound"]
    bad_dH = dH.copy()
    bad_dH[9] *= 1.5
    r = b.sampled_parity("kl", rows, ref, {"kl": out["kl"], "dH": torch.from_numpy(bad_dH)})
    assert r["kl_within_bound"] and not r["dH_within_bound"]
    bad_row = dH.copy()
    bad_row[2] = 0.0  # not a sampled row: not compared
    assert b.sampled_parity("kl", rows, ref, {"kl": out["kl"], "dH": torch.from_numpy(bad_row)})["dH_within_bound"]
    assert b.sampled_parity("kl", rows, ref, None) is None
