// Launch order of the tensor-core read's CTAs (host and device): CTA `rank`
// of a grid of n_qt query tiles x BH heads reads query tile qt of head bh.
//
// The heads go in groups of kHeadGroup; within a group the query tiles go
// heaviest first across its heads when causal (the last diagonal tiles read
// the most key tiles), so the launch ends on the lightest tiles and the SMs
// finish together, while the CTAs in flight share the K and bank tiles of at
// most two groups in L2.  The map is a bijection of [0, n_qt BH) onto the
// (bh, qt) pairs; the last group may hold fewer than kHeadGroup heads.
#pragma once

namespace fem {

constexpr int kHeadGroup = 8;  // heads whose query tiles the launch order interleaves

__host__ __device__ inline void tc_tile_of_rank(int rank, int BH, int n_qt, int causal, int &bh, int &qt) {
  const int g0 = rank / (kHeadGroup * n_qt) * kHeadGroup, gsz = BH - g0 < kHeadGroup ? BH - g0 : kHeadGroup;
  const int idx = rank - g0 * n_qt;
  bh = g0 + idx % gsz;
  qt = causal ? n_qt - 1 - idx / gsz : idx / gsz;
}

}  // namespace fem
