"""Host helpers of the benchmark: the device-code hash that keys the recorded
DRAM traffic ignores comments but not code, and the recorded traffic is only
read back for the hash it was taken on."""
from __future__ import annotations

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_code_only_drops_comments_keeps_literals():
    src = ('int a = 1; // tail comment\n'
           '/* block\n comment */ const char* s = "// not a comment /* nor this */";\n'
           '\n'
           "char c = '/'; int b = a / 2;  \n")
    out = bench.code_only(src)
    assert "comment" not in out.replace("not a comment", "")
    assert '"// not a comment /* nor this */"' in out
    assert "char c = '/'; int b = a / 2;" in out
    assert "\n\n" not in out


def test_comment_edits_keep_the_hash_code_edits_change_it():
    a = 'asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(p));  // load\nint x = 3;\n'
    b = '// a new comment line\nasm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(p));  /* load */\nint x = 3;\n'
    c = 'asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(p));  // load\nint x = 4;\n'
    assert bench.code_only(a) == bench.code_only(b)
    assert bench.code_only(a) != bench.code_only(c)


def test_recorded_traffic_is_keyed_by_the_hash():
    h = bench.device_source_hash()
    assert len(h) == 64
    t = bench.traffic_from_profile(h)
    assert t is None or t > 0
    assert bench.traffic_from_profile("0" * 64) is None
