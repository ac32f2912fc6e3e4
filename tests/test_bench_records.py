"""Host logic of bench.py: the check that a recorded ncu traffic capture still describes the
kernel's code (the hash covers the code of the listed sources and ignores their comments), and
the clock record of the timed region from nvidia-smi's samples."""

import bench


def test_code_text_drops_comments_and_keeps_code():
    src = ('// header\n#include "a.cuh"  // trailing\n\n/* block\n   comment */ int x = 1; /* mid */ int y;\n'
           'const char* s = "not // a comment /* either */";\nchar c = \'"\';  // quote char\n')
    assert bench.code_text(src) == ('#include "a.cuh"\n int x = 1;  int y;\n'
                                    'const char* s = "not // a comment /* either */";\nchar c = \'"\';')


def test_code_text_keeps_escaped_quotes_inside_literals():
    src = 'asm("mov %0, \\"x\\"; // kept");  // dropped\n'
    assert bench.code_text(src) == 'asm("mov %0, \\"x\\"; // kept");'


def test_sources_sha_ignores_comment_edits_only(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2609_24150_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (csrc / "k.cu").write_text("// v1\n__global__ void k() {}\n")
    a = bench.sources_sha(["k.cu"])
    (csrc / "k.cu").write_text("// v2: reworded\n\n__global__ void k() {}  // same code\n")
    assert bench.sources_sha(["k.cu"]) == a
    (csrc / "k.cu").write_text("__global__ void k() { int z; }\n")
    assert bench.sources_sha(["k.cu"]) != a
    assert bench.sources_sha(["missing.cu"]) is None


def test_clock_summary_takes_the_median_and_every_active_reason():
    text = "\n".join([
        "0, 2070, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, 1965, 2070, 1400.1, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 2070, 2070, 1200.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, [N/A], 2070, 1200.0, 0x0, Not Active, Not Active, Not Active, Not Active",   # skipped
        "0, 2070, 2070",                                                                 # partial
        "",
    ])
    c = bench.summarize_clocks(text)
    assert c == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "samples": 3, "reasons": ["sw_power_cap"]}


def test_clock_summary_reports_thermal_and_hardware_slowdowns():
    text = ("0, 1500, 2070, 800, 0x48, Active, Not Active, Active, Not Active\n"
            "0, 1400, 2070, 800, 0x48, Not Active, Active, Not Active, Not Active\n")
    c = bench.summarize_clocks(text)
    assert c["sm_mhz"] == 1450.0 and c["samples"] == 2
    assert c["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]
    assert bench.summarize_clocks("") is None
