// Chunk schedule of the host-buffer read (fem_fwd_host; host code only).
//
// The read on host buffers copies its inputs in, reads and copies the results
// out chunk by chunk, so that the copies in of one chunk, the read of the one
// before and the copies out of the one before that overlap.  A chunk is a run
// of consecutive heads of one batch element (contiguous in every [B, H, T, d]
// array), at most host_chunk_heads(B, H) heads: about eight chunks in all.  The
// very first and the very last chunk are split into a quarter (at least one
// head) and the rest: only the first chunk's copies in run before any read and
// only the last chunk's read and copies out after the last copy in, so small
// end chunks shorten the pipeline's fill and drain.  The chunks cover every
// (b, h) once, in the arrays' order.
#pragma once

#include <algorithm>
#include <vector>

namespace fem {

struct HostChunk {
  int b, h0, nh;  // heads h0 .. h0 + nh - 1 of batch element b
};

inline int host_chunk_heads(int B, int H) {
  const int per_b = std::max(1, std::min(H, 8 / B));  // chunks per batch element
  return (H + per_b - 1) / per_b;
}

inline std::vector<HostChunk> host_chunks(int B, int H) {
  const int hc = host_chunk_heads(B, H);
  std::vector<HostChunk> chunks;
  for (int b = 0; b < B; ++b)
    for (int h0 = 0; h0 < H; h0 += hc) chunks.push_back({b, h0, std::min(hc, H - h0)});
  const int edge = std::max(1, hc / 4);
  if (chunks.front().nh > edge) {
    const HostChunk f = chunks.front();
    chunks.front() = {f.b, f.h0 + edge, f.nh - edge};
    chunks.insert(chunks.begin(), HostChunk{f.b, f.h0, edge});
  }
  if (chunks.back().nh > edge) {
    const HostChunk l = chunks.back();
    chunks.back() = {l.b, l.h0, l.nh - edge};
    chunks.push_back({l.b, l.h0 + l.nh - edge, edge});
  }
  return chunks;
}

}  // namespace fem
