"""The multiply-and-shift divider of the saliency kernel's bookkeeping (csrc/fastdiv.h) against the C `/`
operator: every divisor up to 4096 on every dividend up to 2^16, the dividends next to 2^31 - 1, and
random pairs.  The header is host-compilable, so the check runs on the CPU with g++."""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
HEADER = os.path.join(HERE, "..", "paper_2609_22158_gb300", "csrc", "fastdiv.h")

PROGRAM = r"""
#include "%s"
#include <cstdio>
#include <cstdint>
int main() {
  using namespace stepkv;
  long bad = 0;
  uint64_t x = 88172645463325252ull;
  for (int d = 1; d <= 4096; ++d) {
    const FastDiv f = make_fastdiv(d);
    for (int n = 0; n < 65536; ++n) bad += fdiv(n, f) != n / d;
    for (int n = 2147483647; n > 2147483647 - 4096; --n) {
      int r;
      const int q = fdivmod(n, f, r);
      bad += q != n / d || r != n %% d || fmodulo(n, f) != n %% d;
    }
  }
  for (int i = 0; i < 2000000; ++i) {
    x ^= x << 13; x ^= x >> 7; x ^= x << 17;
    const int d = (int)(x %% 2147483647u) + 1;
    const int n = (int)((x >> 32) & 0x7fffffffu);
    bad += fdiv(n, make_fastdiv(d)) != n / d;
  }
  std::printf("mismatches %%ld\n", bad);
  return bad != 0;
}
"""


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")
def test_fastdiv_matches_integer_division(tmp_path):
    src = tmp_path / "fd.cpp"
    exe = tmp_path / "fd"
    src.write_text(PROGRAM % os.path.abspath(HEADER))
    subprocess.run(["g++", "-O2", "-std=c++17", "-o", str(exe), str(src)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "mismatches 0" in r.stdout
