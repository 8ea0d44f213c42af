// af1_layout.h — the device tile layout of a packed sign matrix, shared by the
// pack kernels, the forward kernels and the host planner.
//
// The forward pass evaluates two sign-matrix products (AF1 Eq. binary_paths,
// right to left): t = B z with B = V^T (r x n) and u = U s' (m x r). Each is a
// product of an R x C matrix of signs with a vector per token. The kernels
// feed the signs to FP8 (e4m3) tensor-core MMAs of shape m16n8k32, so the
// signs are stored in an order that lets every lane expand its own A-fragment
// registers with one LOP3 per 4 signs:
//
//   * The matrix is cut into tiles of 16 rows x 128 columns (256 bytes).
//   * In a tile, lane L = 4g + c (g = L / 4, c = L % 4) owns two 32-bit words:
//     word 0 for row g, word 1 for row g + 8.
//   * Bit (8e + p) of a lane's word (e = 0..3, p = 0..7) is the sign of column
//     16p + 4c + e of that row: 1 for +1, 0 for -1. Rows >= R and columns >= C
//     are 0 bits.
//   * "Slot" p of a word is the A-fragment register of MMA p/2 (a0/a1 for even
//     p, a2/a3 for odd p); its 4 bytes are columns 16p + 4c + {0,1,2,3}.
//   * Tiles are grouped in blocks of RTC row-tiles x KTC column-tiles; block
//     (rg, ks) is one CTA's work and is contiguous, ordered column-tile major
//     ([kt][rt]) so that each column tile of a block is one bulk copy.
#pragma once

#include <stdint.h>

#ifdef __CUDACC__
#define AF1_HD __host__ __device__ __forceinline__
#else
#define AF1_HD inline
#endif

namespace af1 {

constexpr int kTileRows = 16;
constexpr int kTileCols = 128;
constexpr int kTileBytes = 256;
constexpr int kTerms = 4;             // e4m3 terms per activation value
constexpr int kTokensPerGroup = 2;    // MMA n = 8 columns = 2 tokens x 4 terms
constexpr int kMaxPassTokens = 16;    // tokens per kernel pass
constexpr int kMaxKTC = 16;           // column tiles per CTA block (one mbarrier each)
constexpr int kMaxCols = kMaxKTC * 16 * 128;  // longest contraction: 16 CTAs x 16 tiles

struct TileMatrix {
  int64_t R = 0, C = 0;  // valid rows / columns
  int RT = 0, KT = 0;    // row tiles, column tiles
  int RTC = 0, KTC = 0;  // tiles per block along rows / columns
  int RG = 0, KS = 0;    // blocks along rows / columns (the grid)
};

AF1_HD int blk_rows(const TileMatrix& t, int rg) {
  int left = t.RT - rg * t.RTC;
  return left < t.RTC ? left : t.RTC;
}
AF1_HD int blk_cols(const TileMatrix& t, int ks) {
  int left = t.KT - ks * t.KTC;
  return left < t.KTC ? left : t.KTC;
}
// Index of the first tile of block (rg, ks).
AF1_HD int64_t blk_base(const TileMatrix& t, int rg, int ks) {
  return (int64_t)rg * t.RTC * t.KT + (int64_t)blk_rows(t, rg) * ks * t.KTC;
}
// Index of tile (rt, kt) in the layout.
AF1_HD int64_t tile_index(const TileMatrix& t, int rt, int kt) {
  int rg = rt / t.RTC, ks = kt / t.KTC;
  return blk_base(t, rg, ks) + (int64_t)(kt - ks * t.KTC) * blk_rows(t, rg) + (rt - rg * t.RTC);
}
// Column (within the tile) of bit b of the word of lane-column c.
AF1_HD int bit_col(int b, int c) { return 16 * (b & 7) + 4 * c + (b >> 3); }

}  // namespace af1
