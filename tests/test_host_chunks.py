"""Host check of the host-buffer read's chunk schedule (no GPU needed).

fem_fwd_host copies, reads and copies back its work chunk by chunk
(csrc/fem_chunks.h, compiled here for the host as it is for the library).  The
chunks must cover every (batch element, head) exactly once, in the order of the
[B, H, T, d] arrays, each a run of heads of one batch element no longer than
host_chunk_heads(B, H); the very first and the very last chunk are a quarter of
the chunk length (at least one head) whenever the chunk they came from was
longer than that.
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
#include "fem_chunks.h"
int main() {
  int bad = 0, cases = 0;
  for (int B = 1; B <= 12; ++B)
    for (int H = 1; H <= 40; ++H) {
      ++cases;
      const int hc = fem::host_chunk_heads(B, H), edge = hc / 4 > 1 ? hc / 4 : 1;
      const std::vector<fem::HostChunk> ch = fem::host_chunks(B, H);
      int next = 0;  // the next (b, h) in the arrays' order, as b * H + h
      for (const fem::HostChunk &c : ch) {
        if (c.b < 0 || c.b >= B || c.h0 < 0 || c.nh < 1 || c.h0 + c.nh > H || c.nh > hc) ++bad;
        if (c.b * H + c.h0 != next) ++bad;
        next = c.b * H + c.h0 + c.nh;
      }
      if (next != B * H) ++bad;
      // the end chunks: the first and last runs of the unsplit schedule, cut to `edge` heads
      const int first_full = hc < H ? hc : H, last_full = H - (H - 1) / hc * hc;
      if (first_full > edge && ch.front().nh != edge) ++bad;
      if (last_full > edge && ch.back().nh != edge) ++bad;
      const int unsplit = B * ((H + hc - 1) / hc);
      if (static_cast<int>(ch.size()) != unsplit + (first_full > edge) + (last_full > edge)) ++bad;
      if (bad) { std::printf("B %d H %d bad\n", B, H); return 1; }
    }
  std::printf("cases %d bad %d\n", cases, bad);
  return 0;
}
"""


def test_host_chunks_cover_every_head_once(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no C++ compiler")
    src = tmp_path / "chunks_check.cpp"
    src.write_text(CHECKER)
    exe = tmp_path / "chunks_check"
    subprocess.run([cxx, "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True, capture_output=True,
                   timeout=300)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "bad 0" in r.stdout
