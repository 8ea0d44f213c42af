// af1_layout.h — the device layout of a packed sign matrix, shared by the
// pack kernels, the decode and prefill kernels and the host planner.
//
// The forward pass evaluates two sign-matrix products (AF1 Eq. binary_paths,
// right to left): t = B z with B = V^T (r x n) and u = U s' (m x r). Each is
// an R x C matrix of signs times one vector per token. Both kernels expand
// the signs row by row into the A operand of a tcgen05 MMA with M = 128, one
// matrix row per tensor-memory lane (decode) or shared-memory row (prefill),
// so the layout groups rows in blocks of 128 and puts the words of 128
// consecutive rows next to each other:
//
//   * Row block rb holds rows 128 rb .. 128 rb + 127; rows >= R are 0 bits.
//   * Columns are cut into chunks of 128 (4 words of 32 per row); columns
//     >= C are 0 bits. A matrix has NCH = ceil(C / 128) chunks, so a row has
//     4 NCH words, the same count as a canonical row (16-byte padded).
//   * Word kw of row i is at index (rb * 4 NCH + kw) * 128 + (i mod 128):
//     chunk c of row block rb is 2 KB of contiguous memory ([word][row]).
//   * Bit (8e + p) of word kw (e = 0..3, p = 0..7) is the sign of column
//     32 kw + 4p + e: 1 for +1, 0 for -1. Masking bit p of every byte with
//     one LOP3 gives the four 8-bit A values of columns 32 kw + 4p .. + 3,
//     i.e. one 32-bit tensor-memory column (4 consecutive K elements).
#pragma once

#include <stdint.h>

#ifdef __CUDACC__
#define AF1_HD __host__ __device__ __forceinline__
#else
#define AF1_HD inline
#endif

namespace af1 {

constexpr int kBlockRows = 128;   // rows per block = MMA M = tensor-memory lanes
constexpr int kChunkCols = 128;   // columns per chunk
constexpr int kChunkWords = 4;    // 32-bit words per row and chunk
constexpr int kChunkBytes = kBlockRows * kChunkWords * 4;  // 2048
constexpr int kTerms = 4;           // e4m3 terms per activation value (decode)
constexpr int kMaxPassTokens = 16;  // tokens per decode pass
constexpr int kMaxCols = 32768;     // longest contraction (n and r)

struct SignMatrix {
  int64_t R = 0, C = 0;  // valid rows / columns
  int RB = 0;            // row blocks of 128
  int NCH = 0;           // column chunks of 128
};

AF1_HD SignMatrix make_sign_matrix(int64_t R, int64_t C) {
  SignMatrix s;
  s.R = R;
  s.C = C;
  s.RB = (int)((R + kBlockRows - 1) / kBlockRows);
  s.NCH = (int)((C + kChunkCols - 1) / kChunkCols);
  return s;
}
// Bytes of the packed matrix in this layout.
AF1_HD int64_t sign_matrix_bytes(const SignMatrix& s) { return (int64_t)s.RB * s.NCH * kChunkBytes; }
// Index (in 32-bit words) of word kw of row `row`.
AF1_HD int64_t word_index(const SignMatrix& s, int64_t row, int64_t kw) {
  return ((row / kBlockRows) * s.NCH * kChunkWords + kw) * kBlockRows + (row % kBlockRows);
}
// Column, within the 32 columns of a word, of bit b.
AF1_HD int bit_col(int b) { return 4 * (b & 7) + (b >> 3); }

}  // namespace af1
