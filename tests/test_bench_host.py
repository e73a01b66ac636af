"""bench.py's host-side arithmetic, on CPU: the algorithmic bytes of every workload, the kernel each
workload's call launches, the add count behind the ALU floor, the committed-traffic lookup (and its
turning null when the kernel it was measured on changes), the whole-job value and the clock summary.
Expected values are worked out by hand from the shapes, independently of the bench's own formulas."""
import json
import os

import pytest

import bench
from paper_2607_25234_gb300 import inputs

W = inputs.WORKLOADS


@pytest.mark.parametrize("name,ideal", [
    # read X + read G (fp32) + write Y
    ("tiny_1x256x64_f32", 2 * 256 * 64 * 4 + 256 * 64 * 4),                    # 196,608
    ("epipolar_128x512x128_bf16", 2 * 128 * 512 * 128 * 2 + 512 * 128 * 4),    # 33,816,576
    ("longseq_32x4096x64_f32", 2 * 32 * 4096 * 64 * 4 + 4096 * 64 * 4),        # 68,157,440
    ("fullimage_1x65536x128_bf16", 2 * 65536 * 128 * 2 + 65536 * 128 * 4),    # 67,108,864
    # forward (X, G, Y) + backward (X, dY, G read; dX, dG written)
    ("train_16x8192x256_bf16", 5 * 16 * 8192 * 256 * 2 + 3 * 8192 * 256 * 4),  # 360,710,144
])
def test_algorithmic_bytes_of_the_workloads(name, ideal):
    assert W[name].ideal_bytes() == ideal
    assert W["fullimage_1x65536x128_bf16"].ideal_bytes() == 67_108_864
    assert W["train_16x8192x256_bf16"].ideal_bytes(backward=False) == 142_606_336


def test_kernel_each_workload_launches():
    assert bench.kernel_name(W["fullimage_1x65536x128_bf16"]) == "k_forward_fast<bf16, R=13, Q=10>"
    assert bench.kernel_name(W["longseq_32x4096x64_f32"]) == "k_forward_fast<f32, R=13, Q=5>"
    assert bench.kernel_name(W["epipolar_128x512x128_bf16"]).startswith("k_forward_plane<bf16, column bits 2>")
    assert bench.kernel_name(W["tiny_1x256x64_f32"]).startswith("k_forward_plane<f32, column bits 0>")
    assert bench.kernel_name(W["train_16x8192x256_bf16"]) == "k_forward_fast<bf16, R=14, Q=7>"
    assert bench.backward_kernel_name(W["train_16x8192x256_bf16"]) == "k_backward_fast<bf16, R=14, Q=7>"
    assert bench.backward_kernel_name(W["fullimage_train_1x65536x128_bf16"]) == "k_backward_fast<bf16, R=14, Q=9>"
    # 2^16-element planes go one per CTA only from a batch of 80
    small = inputs.Workload("x", 79, 512, 128, "bf16")
    assert bench.kernel_name(small).startswith("k_forward_fast<bf16, R=13, Q=3>")


def test_alu_floor_counts_the_butterfly_adds():
    f = bench.alu_floor(W["fullimage_1x65536x128_bf16"], 152, 2070.0)
    assert f["adds"] == 2 * (1 << 23) * 23 and f["muls"] == 1 << 23
    assert f["floor_us"] == pytest.approx(2 * (1 << 23) * 23 / (152 * 128 * 2070e6) * 1e6)
    t = bench.alu_floor(W["train_16x8192x256_bf16"], 152, None)
    L = 8192 * 256
    assert t["adds"] == 16 * 5 * L * 21 and t["muls"] == 16 * 3 * L and t["floor_us"] is None


def test_whole_job_value_counts_every_rank():
    one = bench.whole_job_tokens_per_s(1, 65536, 100, 5.0)
    assert one == pytest.approx(65536 * 100 / 5e-3)
    assert bench.whole_job_tokens_per_s(4, 65536, 100, 5.0) == pytest.approx(4 * one)


def test_committed_traffic_is_used_only_for_the_unchanged_kernel(monkeypatch, tmp_path):
    committed = json.load(open(os.path.join(bench.ROOT, "profiles", "roofline_traffic.json")))
    for name, e in committed.items():
        assert name in W, name
        fresh = e["kernel_source_hash"] == bench.kernel_source_hash(e["kernel"])
        # a capture of the kernel as it stands is used; one taken before its sources changed is not
        assert bench.traffic_from_profile(name) == (e["dram_bytes_per_launch"] if fresh else None)
        assert e["dram_bytes_per_launch"] == e["dram_read_bytes"] + e["dram_write_bytes"]
    # another hash (the kernel's sources changed since the capture): no traffic figure; the same
    # hash: the committed figure
    monkeypatch.setattr(bench, "kernel_source_hash", lambda kernel: "0000000000000000")
    assert bench.traffic_from_profile("fullimage_1x65536x128_bf16") is None
    e0 = committed["fullimage_1x65536x128_bf16"]
    monkeypatch.setattr(bench, "kernel_source_hash", lambda kernel: e0["kernel_source_hash"])
    assert bench.traffic_from_profile("fullimage_1x65536x128_bf16") == e0["dram_bytes_per_launch"]
    monkeypatch.undo()
    # an entry that names a kernel the workload does not launch: no traffic figure
    fake_root = tmp_path
    os.makedirs(fake_root / "profiles")
    e = dict(committed["fullimage_1x65536x128_bf16"], kernel="k_forward_plane<bf16, column bits 2>")
    e["kernel_source_hash"] = bench.kernel_source_hash(e["kernel"])
    (fake_root / "profiles" / "roofline_traffic.json").write_text(json.dumps({"fullimage_1x65536x128_bf16": e}))
    monkeypatch.setattr(bench, "ROOT", str(fake_root))
    assert bench.traffic_from_profile("fullimage_1x65536x128_bf16") is None
    assert bench.traffic_from_profile("no_such_workload") is None


def test_clock_summary_uses_the_timed_window_and_decodes_reasons():
    s = bench.ClockSampler("0")
    s.samples = [(0.5, 1000.0, 2070.0, 0x1), (1.0, 2070.0, 2070.0, 0x0), (1.5, 2040.0, 2070.0, 0x4),
                 (2.0, 2070.0, 2070.0, 0x0), (3.0, 800.0, 2070.0, 0x8)]
    got = s.summary(1.0, 2.0)
    assert got["window"] == "timed_region" and got["samples"] == 3
    assert got["sm_mhz"] == 2070.0 and got["sm_max_mhz"] == 2070.0
    assert got["reasons"] == ["sw_power_cap"]
    late = s.summary(2.5, 3.5)
    assert late["reasons"] == ["hw_slowdown"] and late["sm_mhz"] == 800.0
    assert s.summary(10.0, 11.0)["window"] == "whole_run"   # nothing inside: every sample, marked so
    empty = bench.ClockSampler("0").summary(0.0, 1.0)
    assert empty["samples"] == 0 and empty["sm_mhz"] is None


def test_reference_arm_line_matches_ours_in_config_and_metric(monkeypatch, capsys):
    """The driver compares the two arms' lines: the reference arm (the CPU oracle) reports the same
    config (built by the same function as the GPU arm's) and, for a training step, the same
    forward + backward metric."""
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)

    class Args:
        steps, warmup, gpus = 1, 1, 1
    for name, metric in (("tiny_1x256x64_f32", "WHTMix fwd tokens/s"),
                         ("train_16x8192x256_bf16", "WHTMix fwd+bwd tokens/s")):
        w = W[name]
        small = w if w.B * w.N * w.C <= 1 << 16 else \
            bench.inputs.Workload(w.name, 1, 256, w.C, w.dtype, backward=w.backward)
        bench.reference_arm(Args(), small)
        line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
        assert line["impl"] == "reference" and line["metric"] == metric
        assert line["config"] == bench.workload_config(small, 1, bench.device_l2_bytes())
        assert line["cpu_baseline"]["cores"] >= 1 and line["value"] > 0


def test_bf16_exchange_workload():
    # the same shape, bytes and kernel as the full-image workload, with the exchange marked
    w, ref = W["fullimage_x16_1x65536x128_bf16"], W["fullimage_1x65536x128_bf16"]
    assert w.ideal_bytes() == ref.ideal_bytes() == 67_108_864
    assert bench.kernel_name(w) == "k_forward_fast<bf16, R=13, Q=10, bf16 exchange>"
    cfg, cfg_ref = bench.workload_config(w, 1, 126 << 20), bench.workload_config(ref, 1, 126 << 20)
    assert cfg["exchange"] == "bf16" and cfg_ref["exchange"] == "f32"
    assert {k: v for k, v in cfg.items() if k not in ("workload", "exchange")} == \
        {k: v for k, v in cfg_ref.items() if k not in ("workload", "exchange")}
