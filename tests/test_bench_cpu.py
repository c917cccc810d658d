"""bench.py's host-side arithmetic, without a GPU: the algorithmic work of a
step, the roofline fractions and bound, the reading of the committed traffic
records, the clock sampler's parsing of nvidia-smi samples, and the config
object both bench arms print."""

import os

import pytest

import bench
from workloads import B256X8X64_E4M3, B8X2X32_BF16, TINY_F32, generate


def test_algorithmic_work_of_the_largest_window():
    cfg = B256X8X64_E4M3
    n = 52424
    flops, nbytes = bench.algorithmic(cfg, n)
    assert flops == 2.0 * n * 5120 * 157184
    # the E4M3 codes and their row scales once, the masked bf16 rows once,
    # 12 bytes of outputs and 1 byte of mask per window position
    assert nbytes == 157184 * 5120 + 4 * 157184 + n * 5120 * 2 + cfg.P * 13
    assert abs(nbytes - 1.344e9) < 1e6


def test_roofline_fractions_and_bound():
    hbm, tc, _, _ = bench.peaks()
    cfg, n = B8X2X32_BF16, 294
    flops, nbytes = bench.algorithmic(cfg, n)
    r = bench.roofline_of(cfg, n, [0.130] * 24, traffic=627e6, lm_launches=1)
    assert r["tensor_view"]["frac"] == pytest.approx(flops / 130e-6 / 1e12 / tc)
    assert r["hbm_view"]["frac"] == pytest.approx(nbytes / 130e-6 / 1e9 / hbm)
    # the bound is the roof with the longer floor; the headline fraction is its own
    expect = "tensor" if flops / (tc * 1e12) >= nbytes / (hbm * 1e9) else "hbm"
    assert r["bound"] == expect
    assert r["frac"] == pytest.approx(r["tensor_view" if expect == "tensor" else "hbm_view"]["frac"])
    assert r["traffic_over_algorithmic"] == pytest.approx(627e6 / nbytes)
    assert r["lmhead_launches_timed"] == 24 and r["lmhead_launches_per_step"] == 1
    # the largest window is far on the tensor side of the ridge
    big = bench.roofline_of(B256X8X64_E4M3, 52424, [47.0], lm_launches=2)
    assert big["bound"] == "tensor" and big["traffic"] is None and big["lmhead_launches_per_step"] == 2


def test_traffic_records_are_read_for_the_current_sources_only(tmp_path, monkeypatch):
    f = tmp_path / "traffic.txt"
    f.write_text("# header: the command\n\nworkload: w1\nkernel_sha256_16: aaaa\ndram_bytes_per_launch: 123\n\n"
                 "workload: w1\nkernel_sha256_16: bbbb\ndram_bytes_per_launch: 456\n\n"
                 "workload: w2\nkernel_sha256_16: aaaa\ndram_bytes_per_launch: 789\n")
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(f))
    monkeypatch.setattr(bench, "kernel_hash", lambda: "aaaa")
    assert bench.recorded_traffic("w1") == 123.0
    assert bench.recorded_traffic("w2") == 789.0
    assert bench.recorded_traffic("w3") is None
    monkeypatch.setattr(bench, "kernel_hash", lambda: "cccc")  # sources changed since: no record
    assert bench.recorded_traffic("w1") is None


def test_kernel_hash_covers_the_lm_head_sources():
    assert len(bench.KERNEL_SOURCES) == 3
    for f in bench.KERNEL_SOURCES:
        assert os.path.exists(os.path.join(bench.ROOT, f)), f
    h = bench.kernel_hash()
    assert len(h) == 16 and int(h, 16) >= 0


class _Proc:
    def terminate(self):
        pass

    def wait(self):
        return 0


def _sampler_with(tmp_path, rows):
    p = tmp_path / "clocks.csv"
    p.write_text("\n".join(rows) + "\n")
    s = bench.ClockSampler(0)
    s.proc, s.path = _Proc(), str(p)
    return s


def test_clock_sampler_reports_the_loaded_median_and_the_reasons(tmp_path):
    na = "Not Active"
    rows = [f"0, 345, 2070, 120.5, 0x0, {na}, {na}, {na}, {na}",          # idle sample: excluded
            f"0, 1500, 2070, 1300.0, 0x4, {na}, {na}, {na}, Active",
            f"0, 1550, 2070, 1350.5, 0x4, {na}, {na}, {na}, Active",
            f"0, 1600, 2070, 1380.0, 0x0, {na}, {na}, {na}, {na}"]
    out = _sampler_with(tmp_path, rows).stop()
    assert out["sm_mhz"] == 1550.0 and out["sm_max_mhz"] == 2070.0
    assert out["reasons"] == ["sw_power_cap"] and out["samples"] == 4
    assert out["power_w_max"] == 1380.0


def test_clock_sampler_flags_thermal_slowdown(tmp_path):
    na = "Not Active"
    out = _sampler_with(tmp_path, [f"0, 1200, 2070, 900.0, 0x40, {na}, Active, {na}, {na}"]).stop()
    assert out["reasons"] == ["hw_thermal_slowdown"]


def test_both_arms_print_the_same_config_object():
    wl = generate(TINY_F32)
    n = bench.masked_count(wl)
    a = bench.config_object(TINY_F32, wl, n, 1)
    b = bench.config_object(TINY_F32, generate(TINY_F32), n, 1)
    assert a == b
    assert a["workload"] == TINY_F32.name and a["masked_positions_per_rank"] == n
    assert set(a["inputs_sha256"]) >= {"hidden", "weight", "pos_masked", "block_flags"}
