"""bench.py's ncu traffic records: keyed by the kernel code (comments
stripped), read back only while that code is unchanged."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_strip_comments_keeps_code_and_literals():
    src = ('int a = 1; // line comment\n'
           '/* block\n   comment */ const char* s = "x//y /* not */";\n'
           "char c = '/'; const char* e = \"q\\\"//r\";  \n\n  int   b;")
    out = bench.strip_comments(src)
    assert "comment" not in out
    assert '"x//y /* not */"' in out and "'/'" in out and '"q\\"//r"' in out
    assert out.endswith("int b;") and "  " not in out


def test_comment_edits_do_not_change_the_hash(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2605_06675_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "include").mkdir()
    (tmp_path / "include" / "rq.h").write_text("/* abi */ int rq_x(void);\n")
    (csrc / "k.cuh").write_text("// helper\n__device__ int f(int x) { return x + 1; }\n")
    (csrc / "k.cu").write_text('#include "k.cuh"\n__global__ void g(int* p) { *p = f(*p); }\n')
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_source_hash("k.cu")
    (csrc / "k.cuh").write_text("// helper, reworded\n\n__device__ int f(int x) {  return x + 1; }\n")
    assert bench.kernel_source_hash("k.cu") == h0
    (csrc / "k.cuh").write_text("__device__ int f(int x) { return x + 2; }\n")
    assert bench.kernel_source_hash("k.cu") != h0


def test_records_parse_and_go_stale(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2605_06675_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "include").mkdir()
    (tmp_path / "profiles").mkdir()
    (tmp_path / "include" / "rq.h").write_text("int rq_x(void);\n")
    (csrc / "k.cu").write_text("__global__ void g() {}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h = bench.kernel_source_hash("k.cu")
    (tmp_path / "profiles" / "traffic.txt").write_text(
        f"# comment\nkern wl 1234 k.cu:{h}\nkern other 99 k.cu:0000000000000000\n")
    assert bench.recorded_traffic("kern", "wl") == 1234.0
    assert bench.recorded_traffic("kern", "other") is None
    assert bench.recorded_traffic("kern", "missing") is None
    (csrc / "k.cu").write_text("__global__ void g() { }\n__global__ void h() {}\n")
    assert bench.recorded_traffic("kern", "wl") is None


def test_only_included_headers_enter_the_hash(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2605_06675_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "include").mkdir()
    (tmp_path / "include" / "rq.h").write_text("int rq_x(void);\n")
    (csrc / "a.cuh").write_text('#include "rq.h"\n__device__ int f(int x) { return x; }\n')
    (csrc / "b.cuh").write_text("__device__ int g(int x) { return -x; }\n")
    (csrc / "k.cu").write_text('#include "a.cuh"\n__global__ void k(int* p) { *p = f(*p); }\n')
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_source_hash("k.cu")
    (csrc / "b.cuh").write_text("__device__ int g(int x) { return x * 3; }\n")   # not included
    assert bench.kernel_source_hash("k.cu") == h0
    (tmp_path / "include" / "rq.h").write_text("int rq_x(void); int rq_y(void);\n")  # included via a.cuh
    assert bench.kernel_source_hash("k.cu") != h0


def test_a_body_included_inside_a_function_enters_the_hash(tmp_path, monkeypatch):
    # the decode split kernel's body is a file included inside two kernels
    csrc = tmp_path / "paper_2605_06675_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "include").mkdir()
    (tmp_path / "include" / "rq.h").write_text("int rq_x(void);\n")
    (csrc / "body.inc").write_text("  *p += 1;\n")
    (csrc / "k.cu").write_text('__global__ void k(int* p) {\n#include "body.inc"\n}\n'
                               '__global__ void k2(int* p) {\n  #include "body.inc"\n}\n')
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_source_hash("k.cu")
    (csrc / "body.inc").write_text("  *p += 2;\n")
    assert bench.kernel_source_hash("k.cu") != h0
