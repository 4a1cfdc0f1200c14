"""Host arithmetic of the benchmark's JSON line, checked by hand on CPU: the
visible-pair count, the roofline work models, the scaling of the captured DRAM
traffic to the workload, and the CUDA-core peak from unit counts."""
import os
import sys
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_03228_gb300 import synth  # noqa: E402

PK = dict(hbm_gbs=6000.0, bf16_tflops=2000.0, fp32_tflops=80.0, source="test")


def test_visible_pairs_by_hand():
    # causal prefill: query t sees keys 0..t, so a head has 1 + 2 + ... + 4096 pairs
    assert bench.visible_pairs(synth.WORKLOADS["llama31_8b_t4096_r32"]) == 1024 * 4096 * 4097 // 2
    # decode: 8 queries per head, each sees the whole 2^20-key cache
    assert bench.visible_pairs(synth.WORKLOADS["decode_n1m_b8_r32"]) == 32 * 8 * 2 ** 20


def test_selection_models():
    w = synth.WORKLOADS["llama31_8b_t4096_r32"]
    bound, work, unit, peak, _, _ = bench.selection_model(w, PK, 4096, 4096, "select")
    assert (bound, unit, peak) == ("tensor", "TFLOP/s", 2000.0)
    assert work == 2 * 32 * 8_592_031_744 == 549_890_031_616
    assert bench.selection_model(w, PK, 4096, 4096, "exact")[1] == 2 * 128 * 8_592_031_744
    d = synth.WORKLOADS["decode_n1m_b8_r32"]
    bound, work, unit, peak, _, _ = bench.selection_model(d, PK, 2 ** 20, 8, "select")
    assert (bound, unit, peak) == ("hbm", "GB/s", 6000.0)
    # bf16 codes of 32 heads x 2^20 keys x r = 32, plus the queries read and the
    # int32 top-64 lists written
    assert work == 32 * 2 ** 20 * 32 * 2 + 32 * 8 * 128 * 2 + 32 * 8 * 64 * 4 == 2_147_614_720
    # the exact decode reads the 8 KV heads' bf16 keys once
    assert bench.selection_model(d, PK, 2 ** 20, 8, "exact")[1] == 8 * 2 ** 20 * 128 * 2 + 32 * 8 * 128 * 2 + 32 * 8 * 64 * 4


def test_rooflines_rate_fraction_and_traffic_scaling():
    w = synth.WORKLOADS["llama31_8b_t4096_r32"]
    g = types.SimpleNamespace(N=4096, T=4096)
    ktime = {"select": (22.0, 2), "exact": (32.0, 2), "fit": (10.0, 2), "_steps": 2}
    out = bench.rooflines(w, PK, ktime, g)
    sel = out["select"]
    assert sel["ms_per_launch"] == 11.0 and sel["launches_per_step"] == 1.0
    assert sel["achieved"] == pytest.approx(549_890_031_616 / 11e-3 / 1e12)
    assert sel["frac"] == pytest.approx(sel["achieved"] / 2000.0)
    # the capture was taken at 256 of the 1024 query heads: four times its bytes
    assert sel["traffic"] == pytest.approx(4 * (566644480 + 224940800))
    assert out["exact"]["traffic"] == pytest.approx(4 * (970252544 + 235156992))
    assert out["exact"]["model"].endswith("(evaluation only: the exact top-k of the recall protocol)")
    # the fit changed after its capture: no traffic; kernels not timed: no entry
    assert out["fit"]["traffic"] is None and out["fit"]["bound"] == "alu"
    assert out["fit"]["work_per_launch"] == 1024 * (4 + 48) * 128 ** 3
    assert "moments" not in out and "build" not in out
    # the captured figures hold for the Llama-3.1-8B shapes only
    q = synth.WORKLOADS["qwen25_7b_t4096_r32"]
    assert bench.rooflines(q, PK, ktime, g)["select"]["traffic"] is None


def test_cuda_core_peak_from_unit_counts():
    pk = bench.peaks()
    assert pk["alu_tops"] == pytest.approx(152 * 128 * pk["sm_max_mhz"] * 1e6 / 1e12)
    assert pk["fp32_tflops"] == pytest.approx(2 * pk["alu_tops"])
    assert pk["source"] in ("measured", "fallback")


def test_clock_sampler_parses_the_query_lines(monkeypatch):
    """The sampler reads nvidia-smi's CSV lines (fields: SM clock, max SM clock,
    power, active reasons mask, then the four reason flags); a stand-in process
    prints canned lines, one of them malformed."""
    import subprocess
    import time
    lines = ["2070, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
             "2055, 2070, 1350.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
             "[N/A], 2070, 1000.0, 0x0, Not Active, Not Active, Not Active, Not Active",
             "2070, 2070, 1000.0, 0x0, Not Active, Not Active, Not Active, Not Active"]
    script = "import time\nfor l in %r: print(l, flush=True)\ntime.sleep(60)" % (lines,)
    real = subprocess.Popen
    monkeypatch.setattr(bench.subprocess, "Popen", lambda cmd, **kw: real([sys.executable, "-c", script], **kw))
    c = bench.ClockSampler(0)
    c.start()
    for _ in range(100):
        if len(c.lines) >= 4:
            break
        time.sleep(0.05)
    out = c.stop()
    assert out == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}


def test_clock_sampler_without_nvidia_smi(monkeypatch):
    def missing(*a, **kw):
        raise OSError("no nvidia-smi")
    monkeypatch.setattr(bench.subprocess, "Popen", missing)
    c = bench.ClockSampler(0)
    c.start()
    assert c.stop() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
