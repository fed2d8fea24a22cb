"""Host check of the tensor-core read's launch order (no GPU needed).

The read kernel maps its CTA rank to a (head, query tile) pair with
tc_tile_of_rank (csrc/fem_order.h, compiled here for the host as it is for the
device).  Every output tile must be computed exactly once, and when causal the
ranks of each group of heads must visit the query tiles heaviest first.  The
checker program runs the map over ragged head counts and tile counts.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2602_07160_gb300", "csrc")

CHECKER = r"""
#include <cstdio>
#include <vector>
#include "fem_order.h"
int main() {
  int bad = 0, cases = 0;
  const int bhs[] = {1, 2, 3, 7, 8, 9, 15, 16, 17, 24, 64, 65, 96};
  const int qts[] = {1, 2, 3, 16, 64, 65, 256};
  for (int BH : bhs)
    for (int n_qt : qts)
      for (int causal = 0; causal < 2; ++causal) {
        ++cases;
        std::vector<int> seen(static_cast<size_t>(BH) * n_qt, 0);
        std::vector<int> last_qt(BH, -1);
        for (int rank = 0; rank < BH * n_qt; ++rank) {
          int bh = -1, qt = -1;
          fem::tc_tile_of_rank(rank, BH, n_qt, causal, bh, qt);
          if (bh < 0 || bh >= BH || qt < 0 || qt >= n_qt) { ++bad; continue; }
          ++seen[static_cast<size_t>(bh) * n_qt + qt];
          // per head, causal ranks take its tiles from the last (heaviest) down, else up
          if (last_qt[bh] >= 0 && (causal ? qt >= last_qt[bh] : qt <= last_qt[bh])) ++bad;
          last_qt[bh] = qt;
        }
        for (int c : seen) bad += c != 1;
      }
  std::printf("cases %d bad %d\n", cases, bad);
  return bad != 0;
}
"""


def test_launch_order_is_a_bijection(tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    src = tmp_path / "order_check.cu"
    src.write_text(CHECKER)
    exe = tmp_path / "order_check"
    subprocess.run([nvcc, "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True, capture_output=True,
                   timeout=300)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "bad 0" in r.stdout
