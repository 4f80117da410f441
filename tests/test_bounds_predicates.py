"""The debug-bounds predicates (csrc/echo_bounds.h) compiled for the host with g++.

The composition and validator kernels check every index they gather through with
these functions when echo_compose_opts.debug_bounds is set (a failed check skips
the access and reports ECHO_E_BOUNDS).  The header has no CUDA dependency, so the
same code is exercised here on the edge cases: empty buffers, negative indices, the
last element, one past the end, and 64-bit extremes.
"""
import os
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2412_12487_gb300", "csrc")

PROGRAM = r"""
#include <cstdio>
#include <cstdlib>
#include "echo_bounds.h"
using namespace echo;
static int fails = 0;
#define CHECK(x) do { if (!(x)) { std::printf("FAIL %s\n", #x); ++fails; } } while (0)
int main() {
  CHECK(!in_range(0, 0));
  CHECK(in_range(0, 1));
  CHECK(!in_range(1, 1));
  CHECK(!in_range(-1, 5));
  CHECK(in_range(4, 5));
  CHECK(!in_range(5, 5));
  CHECK(!in_range(INT64_MIN, INT64_MAX));
  CHECK(in_range(INT64_MAX - 1, INT64_MAX));
  CHECK(range_ok(0, 0, 0));
  CHECK(range_ok(3, 3, 3));
  CHECK(!range_ok(3, 4, 3));
  CHECK(!range_ok(-1, 2, 5));
  CHECK(!range_ok(4, 2, 5));
  CHECK(range_ok(0, 5, 5));
  CHECK(!range_ok(0, 6, 5));
  CHECK(masked_row_ok(7, 0, 0));              // no masked position: nothing to read
  CHECK(masked_row_ok(0, 0x1ull, 1));
  CHECK(!masked_row_ok(0, 0x3ull, 1));        // two rows from 0 need n >= 2
  CHECK(masked_row_ok(5, 0x8000000000000001ull, 7));
  CHECK(!masked_row_ok(5, 0x8000000000000001ull, 6));
  CHECK(!masked_row_ok(-1, 0x1ull, 10));
  CHECK(masked_row_ok(0, ~0ull, 64));
  CHECK(!masked_row_ok(1, ~0ull, 64));
  if (fails) return 1;
  std::printf("ok\n");
  return 0;
}
"""


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")
def test_bounds_predicates_on_the_host():
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "t.cpp")
        exe = os.path.join(d, "t")
        with open(src, "w") as f:
            f.write(PROGRAM)
        subprocess.check_call(["g++", "-std=c++17", "-O1", "-I", CSRC, src, "-o", exe])
        out = subprocess.run([exe], capture_output=True, text=True)
        assert out.returncode == 0, out.stdout
        assert out.stdout.strip() == "ok"
