"""bench.py's check that a recorded ncu traffic capture still describes the kernel's code:
the hash covers the code of the listed sources and ignores their comments."""

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
