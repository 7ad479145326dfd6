"""Host-side logic of bench.py, on the CPU: the clock record, the roofline
fractions and the per-block token counts of a workload."""
import numpy as np
import pytest

import bench as B
import dora_synth as S


def _line(sm, mx=2070, reasons=("Not Active",) * 4, active="0x0"):
    return ", ".join(["2026/12/02 12:00:00.000", str(sm), str(mx), "900.00 W", active, *reasons])


def test_clock_summary_window_median_and_reasons():
    lines = [
        (0.0, _line(1000)),                                   # before the window
        (1.0, _line(1900)),
        (1.1, _line(1950, reasons=("Not Active", "Not Active", "Not Active", "Active"))),
        (1.2, _line(2000)),
        (1.3, "not, a, sample"),                              # skipped: too few fields
        (1.4, _line("[N/A]")),                                # skipped: no number
        (9.0, _line(500, reasons=("Active",) * 4)),           # after the window
    ]
    c = B.clock_summary(lines, 1.0, 1.25)
    assert c["samples"] == 3
    assert c["sm_mhz"] == 1950.0
    assert c["sm_max_mhz"] == 2070.0
    assert c["reasons"] == ["sw_power_cap"]


def test_clock_summary_throttle_reasons_named():
    c = B.clock_summary([(5.0, _line(1500, reasons=("Active", "Not Active", "Active",
                                                      "Not Active")))], 5.0, 5.0)
    assert c["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    assert B.clock_summary([], 0.0, 1.0) == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [],
                                             "samples": 0}


def _kern():
    # two steps' worth of work divided out already: per-step figures
    return {
        "gemm": dict(ms=4.0, launches=48, flops=5.4e12 * 1.0, bytes=48 * 2.0e8, rows=0.0,
                     share=0.78),
        "gemm_qkv": dict(ms=1.0, launches=12, flops=1.5e12, bytes=1.0, rows=400000.0, share=0.2),
        "gemm_proj": dict(ms=0.5, launches=12, flops=0.5e12, bytes=1.0, rows=400000.0, share=0.1),
        "gemm_fc1": dict(ms=1.3, launches=12, flops=1.7e12, bytes=1.0, rows=370000.0, share=0.26),
        "gemm_fc2": dict(ms=1.2, launches=12, flops=1.7e12, bytes=1.0, rows=370000.0, share=0.24),
        "attention": dict(ms=0.8, launches=12, flops=0.19e12, bytes=2.5e9, rows=0.0, share=0.16),
        "select_compact": dict(ms=0.06, launches=3, flops=0.0, bytes=2.3e8, rows=0.0,
                               share=0.012),
    }


PEAKS = {"hbm_gbs": 6757.2, "bf16_tflops": 1905.9, "bf16_tflops_sustained": 1705.0}


def test_roofline_fractions_follow_the_timed_work(monkeypatch):
    monkeypatch.setattr(B, "sha256_of", lambda path: "no capture for this source")
    out = B.roofline_report(_kern(), PEAKS, "measured", "cfg3")
    g = out["roofline"]
    assert g["achieved"] == pytest.approx(5.4e12 / 4.0e-3 / 1e12, abs=0.05)
    assert g["frac"] == pytest.approx(g["achieved"] / 1905.9, abs=1e-4)
    assert g["frac_of_sustained"] == pytest.approx(g["achieved"] / 1705.0, abs=1e-4)
    assert g["traffic"] is None and g["traffic_case"] is None     # source not captured
    a = out["roofline_attention"]
    ai = 0.19e12 / 2.5e9
    assert a["arith_intensity"] == pytest.approx(ai, abs=0.05)
    attain = min(1905.9, ai * 6757.2 / 1e3)
    assert a["attainable_from_hbm"] == pytest.approx(attain, abs=0.05)
    assert a["frac_of_attainable"] == pytest.approx(a["achieved"] / attain, abs=1e-3)
    c = out["roofline_compact"]
    assert c["achieved"] == pytest.approx(2.3e8 / 0.06e-3 / 1e9, abs=0.05)
    assert c["frac"] == pytest.approx(c["achieved"] / 6757.2, abs=1e-4)
    assert c["us_per_launch"] == pytest.approx(20.0, abs=0.01)


def test_roofline_traffic_only_for_the_captured_source_and_workload(monkeypatch):
    key_g, per_row = next(iter(B.NCU_GEMM_BYTES_PER_ROW.items()))
    key_c, cap = next(iter(B.NCU_TRAFFIC_SELECT_COMPACT.items()))
    monkeypatch.setattr(B, "sha256_of",
                        lambda path: key_g if path.endswith("gemm_tcgen05.cu") else key_c)
    k = _kern()
    out = B.roofline_report(k, PEAKS, "measured", "cfg3")
    want = round(sum(per_row[n] * k[n]["rows"] for n in per_row) / k["gemm"]["launches"])
    assert out["roofline"]["traffic"] == want
    assert out["roofline_compact"]["traffic"] == cap["traffic"]
    other = B.roofline_report(k, PEAKS, "measured", "cfg6")
    assert other["roofline"]["traffic"] is None
    assert other["roofline_compact"]["traffic"] is None


@pytest.mark.parametrize("name", ["cfg3", "cfg6"])
def test_lengths_per_block_follow_the_schedule(name):
    cfg = S.get_config(name, batch=16)
    hw = B.HostWorkload(cfg, 0, 1, host_tensors=False)
    keeps = hw.sets[0]["keeps"]
    lens = hw.lengths_per_block(0)
    assert len(lens) == cfg.depth
    n = np.full(cfg.batch, cfg.n_tokens)
    for l, (n_in, n_out) in enumerate(lens):
        assert np.array_equal(n_in, n)
        if l in cfg.prune_blocks:
            assert np.array_equal(n_out, keeps[list(cfg.prune_blocks).index(l)])
            assert np.all(n_out <= n_in) and np.all(n_out >= 1)
        else:
            assert np.array_equal(n_out, n_in)
        n = n_out


def test_workload_config_names_the_shape():
    cfg = S.get_config("cfg3")
    c = B.workload_config(cfg, world=2, nsets=3, graph=True, streams=1)
    assert c["global_batch"] == 2 * cfg.batch
    assert c["seq_len"] == cfg.n_tokens
    assert "prune at 3/6/9" in c["workload"] and "D=768" in c["workload"]
    assert c["cuda_graph"] is True and c["parallelism"].startswith("dp2")
