"""Host check of the fused kernel's work-item order (csrc/schedule.h): every
(GEMM1 / GEMM2, tile, column) item is issued exactly once, and every GEMM2
item comes after all GEMM1 items of its tile."""
import os
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_28979_gb300", "csrc")

DRIVER = r'''
#include <cstdio>
#include <cstdlib>
#include <vector>
#include "schedule.h"
using namespace mot;
int main(int argc, char** argv) {
  int bad = 0, cases = 0;
  for (int F = 1; F <= 70; ++F)
    for (int n1 : {1, 2, 3, 24, 32})
      for (int n2 : {1, 2, 3})
        for (int MB : {1, 2, 5, 8, 16}) {
          Schedule s{F, n1, n2, MB};
          std::vector<int> seen1(F * n1, 0), seen2(F * n2, 0), done1(F, 0);
          ++cases;
          for (int i = 0; i < s.total(); ++i) {
            Item it = schedule_item(s, i);
            if (it.f < 0 || it.f >= F) { ++bad; break; }
            if (it.type == 1) {
              if (it.n < 0 || it.n >= n1) { ++bad; break; }
              seen1[it.f * n1 + it.n]++;
              done1[it.f]++;
            } else if (it.type == 2) {
              if (it.n < 0 || it.n >= n2) { ++bad; break; }
              seen2[it.f * n2 + it.n]++;
              if (done1[it.f] != n1) { ++bad; break; }   // dependency issued earlier
            } else { ++bad; break; }
          }
          for (int v : seen1) if (v != 1) { ++bad; break; }
          for (int v : seen2) if (v != 1) { ++bad; break; }
        }
  printf("%d %d\n", cases, bad);
  return bad != 0;
}
'''


def test_schedule_is_a_dependency_respecting_permutation(tmp_path):
    src = tmp_path / "drv.cpp"
    src.write_text(DRIVER)
    exe = tmp_path / "drv"
    subprocess.check_call(["g++", "-O2", "-std=c++17", "-I", CSRC, str(src), "-o", str(exe)])
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    cases, bad = map(int, r.stdout.split())
    assert cases > 5000 and bad == 0, r.stdout
