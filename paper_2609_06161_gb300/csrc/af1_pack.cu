// af1_pack.cu — sign packing kernels.
//
// (1) pack_signs: an int8 matrix of +-1 (the sign factors of AF1 Sec. 3.1,
//     A_pm1 and B_pm1) -> the canonical words of the packed format declared in
//     include/af1.h (bit = 1 for +1, LSB first, rows padded to 16 bytes).
// (2) words_to_blocks: canonical words -> the internal row-block layout
//     described in af1_layout.h. The bit count is unchanged (1 bit per sign);
//     only the order differs, plus the zero rows of a partial row block.
// (3) blocks_to_words: the inverse, for exporting a layer.
// (4) bf16_to_f16: BF16 scale bit patterns -> FP16 bit patterns, flagging
//     any value FP16 does not represent exactly.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1_internal.h"
#include "af1_layout.h"

namespace af1 {
namespace {

__global__ void pack_signs_kernel(const int8_t* __restrict__ src, int64_t rows, int64_t cols,
                                  int64_t row_stride, int64_t col_stride, uint32_t* __restrict__ words,
                                  int64_t wpr, uint32_t* bad_flag) {
  int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= rows * wpr) return;
  // Consecutive threads take consecutive rows of one word column, so that a
  // column-strided source (V read as V^T) is read coalesced.
  int64_t row = t % rows;
  int64_t w = t / rows;
  uint32_t word = 0;
  bool bad = false;
#pragma unroll 4
  for (int b = 0; b < 32; ++b) {
    int64_t col = w * 32 + b;
    if (col < cols) {
      int8_t v = src[row * row_stride + col * col_stride];
      if (v == 1) {
        word |= 1u << b;
      } else if (v != -1) {
        bad = true;
      }
    }
  }
  words[row * wpr + w] = word;
  if (bad) atomicOr(bad_flag, 1u);
}

// One thread per device word: gather the 32 bits of word kw of row `row`
// from the canonical word of the same row and word index (same 32 columns,
// bit b of the device word = canonical bit bit_col(b)).
__global__ void words_to_blocks_kernel(const uint32_t* __restrict__ words, int64_t wpr, SignMatrix sm,
                                       uint32_t* __restrict__ out) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)sm.RB * sm.NCH * kChunkWords * kBlockRows;
  if (t >= total) return;
  const int64_t i = t % kBlockRows;               // row within the block
  const int64_t kw = (t / kBlockRows) % ((int64_t)sm.NCH * kChunkWords);
  const int64_t rb = t / ((int64_t)kBlockRows * sm.NCH * kChunkWords);
  const int64_t row = rb * kBlockRows + i;
  uint32_t v = 0;
  if (row < sm.R) {
    const uint32_t src = words[row * wpr + kw];
#pragma unroll
    for (int b = 0; b < 32; ++b) {
      const int col = bit_col(b);
      if (32 * kw + col < sm.C) v |= ((src >> col) & 1u) << b;  // padding columns stay 0
    }
  }
  out[t] = v;
}

// One thread per canonical word: the inverse gather of words_to_blocks
// (padding columns and rows beyond R are absent from, or zero in, the
// canonical words).
__global__ void blocks_to_words_kernel(const uint32_t* __restrict__ blocks, SignMatrix sm, int64_t wpr,
                                       uint32_t* __restrict__ words) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= sm.R * wpr) return;
  const int64_t row = t / wpr, kw = t - row * wpr;
  uint32_t v = 0;
  if (kw < (int64_t)sm.NCH * kChunkWords) {
    const uint32_t src = blocks[word_index(sm, row, kw)];
#pragma unroll
    for (int b = 0; b < 32; ++b) v |= ((src >> b) & 1u) << bit_col(b);
  }
  words[t] = v;
}

// BF16 value -> FP16 bits when FP16 holds the same value exactly (finite,
// inside the FP16 range, no mantissa bit below its resolution); else *bad.
__global__ void bf16_to_f16_kernel(const uint16_t* __restrict__ src, uint16_t* __restrict__ dst, int64_t count,
                                   uint32_t* bad) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= count) return;
  const float f = __uint_as_float((uint32_t)src[t] << 16);
  const __half h = __float2half_rn(f);
  if (!(__half2float(h) == f)) atomicOr(bad, 1u);  // also catches NaN
  dst[t] = __half_as_ushort(h);
}

// h = FP16(SiLU(g) u) elementwise (SiLU(g) = g / (1 + e^-g) in FP32): the
// SwiGLU input of a down projection, for the kernels that read their
// activations from memory. Thread i handles 8 columns of one row.
__global__ void swiglu_kernel(const __half* __restrict__ g, const __half* __restrict__ u, int64_t ldx,
                              int64_t tokens, int64_t n, __half* __restrict__ h, int64_t ldh) {
  const int64_t g8 = (n + 7) / 8;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= tokens * g8) return;
  const int64_t t = i / g8, j = (i - t * g8) * 8;
  const __half* gr = g + t * ldx + j;
  const __half* ur = u + t * ldx + j;
  __half* hr = h + t * ldh + j;
  if (j + 8 <= n) {
    const uint4 gv = *reinterpret_cast<const uint4*>(gr);
    const uint4 uv = *reinterpret_cast<const uint4*>(ur);
    const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w}, uw[4] = {uv.x, uv.y, uv.z, uv.w};
    uint32_t hw[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 gf = __half22float2(*reinterpret_cast<const __half2*>(&gw[k]));
      const float2 uf = __half22float2(*reinterpret_cast<const __half2*>(&uw[k]));
      const __half2 hv = __floats2half2_rn(gf.x / (1.f + expf(-gf.x)) * uf.x, gf.y / (1.f + expf(-gf.y)) * uf.y);
      hw[k] = *reinterpret_cast<const uint32_t*>(&hv);
    }
    *reinterpret_cast<uint4*>(hr) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
  } else {
    for (int64_t k = 0; j + k < n; ++k) {
      const float gf = __half2float(gr[k]), uf = __half2float(ur[k]);
      hr[k] = __float2half_rn(gf / (1.f + expf(-gf)) * uf);
    }
  }
}

}  // namespace

cudaError_t launch_blocks_to_words(const uint8_t* blocks, const SignMatrix& sm, int64_t wpr, uint32_t* words,
                                   cudaStream_t st) {
  const int64_t total = sm.R * wpr;
  if (total == 0) return cudaSuccess;
  const int threads = 256;
  blocks_to_words_kernel<<<(unsigned)((total + threads - 1) / threads), threads, 0, st>>>(
      reinterpret_cast<const uint32_t*>(blocks), sm, wpr, words);
  return cudaGetLastError();
}

cudaError_t launch_swiglu(const __half* g, const __half* u, int64_t ldx, int64_t tokens, int64_t n, __half* h,
                          int64_t ldh, cudaStream_t st) {
  const int64_t total = tokens * ((n + 7) / 8);
  if (total == 0) return cudaSuccess;
  const int threads = 256;
  swiglu_kernel<<<(unsigned)((total + threads - 1) / threads), threads, 0, st>>>(g, u, ldx, tokens, n, h, ldh);
  return cudaGetLastError();
}

cudaError_t launch_bf16_to_f16(const uint16_t* src, uint16_t* dst, int64_t count, uint32_t* bad, cudaStream_t st) {
  if (count == 0) return cudaSuccess;
  const int threads = 256;
  bf16_to_f16_kernel<<<(unsigned)((count + threads - 1) / threads), threads, 0, st>>>(src, dst, count, bad);
  return cudaGetLastError();
}

cudaError_t launch_pack_signs(const int8_t* src, int64_t rows, int64_t cols, int64_t row_stride,
                              int64_t col_stride, uint32_t* words, int64_t wpr, uint32_t* bad_flag,
                              cudaStream_t st) {
  int64_t total = rows * wpr;
  if (total == 0) return cudaSuccess;
  int threads = 256;
  int64_t blocks = (total + threads - 1) / threads;
  pack_signs_kernel<<<(unsigned)blocks, threads, 0, st>>>(src, rows, cols, row_stride, col_stride, words,
                                                          wpr, bad_flag);
  return cudaGetLastError();
}

cudaError_t launch_words_to_blocks(const uint32_t* words, int64_t wpr, const SignMatrix& sm, uint8_t* out,
                                   cudaStream_t st) {
  const int64_t total = (int64_t)sm.RB * sm.NCH * kChunkWords * kBlockRows;
  if (total == 0) return cudaSuccess;
  const int threads = 256;
  const int64_t blocks = (total + threads - 1) / threads;
  words_to_blocks_kernel<<<(unsigned)blocks, threads, 0, st>>>(words, wpr, sm, reinterpret_cast<uint32_t*>(out));
  return cudaGetLastError();
}

}  // namespace af1
