// tile_order.cuh -- the order in which the persistent GEMMs visit their
// output tiles (internal).
//
// A GEMM's output is a grid of tt token tiles x nf feature blocks, visited by
// the CTA pairs in rounds of consecutive tile indices.  While the activations
// fit in L2 with room to spare, token tiles go fastest: the activations stay
// resident and each weight block is read once.  Beyond that, groups of G
// feature blocks whose weights fit in L2 (~40 MB) go in turn, feature block
// fastest within a group: the group's weights stay resident while the
// activations stream past once per group, instead of once per round.
#pragma once

namespace w8a8 {

// Token tile ti and feature block fi of tile `local` (G = 1: the plain order,
// token tile fastest).  A bijection of [0, tt * nf).
__device__ __forceinline__ void grouped_tile(int local, int tt, int nf, int G, int &ti, int &fi) {
    if (G == 1) {                      // the plain order, with one division
        fi = local / tt;
        ti = local - fi * tt;
        return;
    }
    const int g = local / (G * tt);
    const int i = local - g * G * tt;
    const int Gg = min(G, nf - g * G);
    ti = i / Gg;
    fi = g * G + (i - ti * Gg);
}

constexpr long long kTileL2Resident = 48ll << 20;

// Feature blocks per group for activations of act_bytes (one branch) and
// weight blocks of block_bytes.
inline int tile_group(long long act_bytes, long long block_bytes, int nf) {
    if (act_bytes <= kTileL2Resident) return 1;
    long long g = kTileL2Resident * 5 / 6 / block_bytes;
    if (g < 1) g = 1;
    if (g > nf) g = nf;
    return static_cast<int>(g);
}

}  // namespace w8a8
