"""The benchmark's work accounting against closed forms of the workload definitions (CPU only).

The metric counts surviving work only: per output pixel, 2 FLOP for each of the 4 pattern taps of every
kept kernel (dense end layers: all 9 taps of every kernel).  Kept-kernel counts follow from each
workload's keep ratio (exactly round(keep * Co * Ci) kept), so the per-frame totals have closed forms
that do not depend on the generated weights.  The totals below are written out from the workload
definitions, not from the code under test.
"""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2004_11250_gb300 import synth  # noqa: E402


def surviving(N, H, W, Co, Ci, keep):
    return 2 * N * H * W * 4 * round(keep * Co * Ci)


def test_vgg16_frame_flops():
    chans = [64, 64, "P", 128, 128, "P", 256, 256, 256, "P", 512, 512, 512, "P", 512, 512, 512]
    expect, ci, h, first = [], 3, 224, True
    for c in chans:
        if c == "P":
            h //= 2
            continue
        expect.append(surviving(1, h, h, c, ci, 1.0 if first else 0.3))
        ci, first = c, False
    shapes = bench.op_shapes(synth.cfg1_vgg16())
    assert [s["flops"] for s in shapes] == expect
    assert [s["H"] for s in shapes] == [224, 224, 112, 112, 56, 56, 56, 28, 28, 28, 14, 14, 14]
    assert sum(expect) / 1e9 == pytest.approx(4.1465, abs=5e-4)
    assert shapes[0]["flops"] / 1e9 == pytest.approx(0.0771, abs=1e-4)  # conv1 keeps all 3 x 64 kernels


def test_style_vdsr_single_and_sweep_flops():
    style = bench.op_shapes(synth.cfg2_style())
    assert len(style) == 10 and all(s["flops"] == surviving(1, 128, 128, 128, 128, 0.25) for s in style)
    assert style[0]["flops"] / 1e9 == pytest.approx(0.5369, abs=1e-4)
    # the style blocks' second convs add the block input: their compulsory bytes include it
    assert style[1]["bytes"] - style[0]["bytes"] == 4 * 128 * 128 * 128

    vdsr = bench.op_shapes(synth.cfg3_vdsr())
    px = 720 * 1280
    assert len(vdsr) == 20
    assert vdsr[0]["flops"] == 2 * px * 9 * 64 and vdsr[-1]["flops"] == 2 * px * 9 * 64  # dense 1->64, 64->1
    assert all(s["flops"] == surviving(1, 720, 1280, 64, 64, 0.4) for s in vdsr[1:-1])
    assert vdsr[1]["flops"] / 1e9 == pytest.approx(12.08, abs=5e-3)
    assert sum(s["flops"] for s in vdsr) / 1e9 == pytest.approx(219.6, abs=0.1)

    single = bench.op_shapes(synth.cfg0_single())
    assert single[0]["flops"] == surviving(1, 32, 32, 16, 16, 0.5) == 2 * 1024 * 4 * 128

    for C, keep, gflop in ((64, 0.2, 0.164), (512, 1.0, 52.6)):
        s = bench.op_shapes(synth.cfg4_point(C, 8, keep))[0]
        assert s["flops"] == surviving(8, 56, 56, C, C, keep)
        assert s["flops"] / 1e9 == pytest.approx(gflop, abs=1e-3 if gflop < 1 else 0.05)


def test_roofline_time_is_the_slower_bound():
    # FP32 peak: 152 SMs x 128 FMA lanes x 2 FLOP x 2.07 GHz; the roofline time is the slower of
    # F / peak and B / HBM bandwidth
    peak = 152 * 128 * 2 * 2.07e9
    assert bench.FP32_PEAK_TFLOPS * 1e12 == pytest.approx(peak)
    assert bench.roof_time_s(peak, 0, 6756.2) == pytest.approx(1.0)
    assert bench.roof_time_s(0, 6756.2e9, 6756.2) == pytest.approx(1.0)
    assert bench.roof_time_s(peak, 2 * 6756.2e9, 6756.2) == pytest.approx(2.0)


def test_source_hash_ignores_comments_only():
    """The hash that ties profiles/ traffic figures to the kernel code skips // comments and blank lines,
    and changes with any code edit."""
    src = "int a = 1;  // one\n\n// a whole comment line\nint b = a + 2;\n"
    assert bench.code_lines(src) == "int a = 1;\nint b = a + 2;"
    assert bench.code_lines(src.replace("// one", "// another note")) == bench.code_lines(src)
    assert bench.code_lines(src.replace("a + 2", "a + 3")) != bench.code_lines(src)


def test_traffic_read_only_for_matching_code(tmp_path, monkeypatch):
    """roofline.traffic comes from a committed summary only while that summary's recorded source hash is
    the current one; otherwise the bench reports null."""
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "ppconv_vgg16_dram_traffic.txt").write_text(
        "# summary\nkernel_source_sha256: abc\ndram_bytes_per_launch_avg: 1000\n"
        "dram_bytes_per_launch_avg[ppconv_tcf_kernel]: 1234\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_from_profile("abc", "ppconv_tcf_kernel") == 1234.0
    assert bench.traffic_from_profile("abc") == 1000.0
    assert bench.traffic_from_profile("def", "ppconv_tcf_kernel") is None
    assert bench.traffic_from_profile("abc", "ppconv_tcf_kernel", precision="f16x3") is None  # no such file


def test_profile_commands_leave_clocks_alone():
    """Every ncu command quoted in profiles/ runs with --clock-control none (ncu would otherwise lock
    the GPU's clocks), and the summaries are short text."""
    pdir = os.path.join(ROOT, "profiles")
    names = sorted(os.listdir(pdir))
    assert names
    for name in names:
        assert name.endswith((".md", ".txt")), name
        text = open(os.path.join(pdir, name), encoding="utf-8").read()
        assert len(text) < 16384, name
        for line in text.splitlines():
            if "ncu " in line and ("--metrics" in line or "--set" in line or "--section" in line):
                assert "--clock-control none" in line, (name, line)
