"""Host-side arithmetic of bench.py's JSON line, on the CPU.

Checks the connection and flop counts against the paper's own figures
(Section 6.3: 13,826 connections for 203-60-26, the true unit's included;
Section 7.2: about 4.23 flops per connection), the value, roofline and e2e
fields that the float32 and bf16 config entries derive from their timings, and
the rule that a workload with no DRAM capture of its current kernels reports
null traffic."""
import importlib.util
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_connection_and_flop_counts_match_the_paper():
    b = _bench()
    assert b.connections((203, 60, 26)) == 13_826
    f60 = b.algorithmic_flops_per_pattern((203, 60, 26))
    assert f60 == 58_476
    assert round(f60 / 13_826, 2) == 4.23
    assert b.connections((203, 120, 26)) == 27_626
    assert b.algorithmic_flops_per_pattern((203, 120, 26)) == 116_796


def test_alu_peak_is_lanes_times_two_times_clock():
    b = _bench()
    peak, mhz = b.alu_peak_tflops(152)
    assert peak == pytest.approx(152 * 128 * 2 * mhz * 1e6 / 1e12)


def test_f32_entry_fields_follow_from_the_timings():
    b = _bench()
    sizes, n, launches = (203, 120, 26), 65_536, 5
    e = b.f32_entry("nettalk120", sizes, n, 512, launches, [7.4, 7.6], [1.5, 1.5], (2.0, 100, 10, 3),
                    152, None, "203-120-26")
    W = 27_626
    assert e["value"] == pytest.approx(W * n * launches / 7.5e-3)
    assert e["ms_per_step"] == pytest.approx(7.5)
    r = e["roofline"]
    assert r["bound"] == "alu" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(116_796 * n / 1.5e-3 / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    tr = b.TRAFFIC_PER_PATTERN.get("nettalk120")
    assert r["traffic"] == (pytest.approx(tr * n) if tr else None)
    assert e["e2e"] == {"value": pytest.approx(W * n * launches * 3 / 2.0), "unit": b.UNIT,
                        "h2d_bytes_per_step": 100, "d2h_bytes_per_step": 10}
    assert "cpu_baseline" not in e


@pytest.mark.parametrize("name,sizes,B", [("wide3", (1024, 2048, 2048, 512), 8192),
                                          ("wide4096", (4096,) * 5, 16384),
                                          ("not_captured", (16, 8, 4), 64)])
def test_bf16_entry_fields_and_the_traffic_rule(name, sizes, B):
    b = _bench()
    cpu = {"value": 1.0, "unit": b.UNIT, "cores": 1, "kind": "oracle", "sample": "s"}
    e = b.bf16_entry(name, sizes, B, [0.39, 0.41], (1.0, 5, 4, 2), cpu, name)
    W = b.connections(sizes)
    assert e["value"] == pytest.approx(W * B / 0.4e-3)
    r = e["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(b.algorithmic_flops_per_pattern(sizes) * B / 0.4e-3 / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    tr = b.TRAFFIC_PER_PATTERN.get(name)
    assert r["traffic"] == (pytest.approx(tr * B) if tr else None)
    assert e["e2e"]["value"] == pytest.approx(W * B * 2 / 1.0)
    assert e["cpu_baseline"] is cpu
