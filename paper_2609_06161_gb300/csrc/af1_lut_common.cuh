// af1_lut_common.cuh — pieces shared by the two CUDA-core decode kernels
// (af1_lut.cu: clustered split-K tiles; af1_stream.cu: balanced streaming
// ranges): the layout of the lookup tables of signed sums, the
// staging of activations, the table build and the lookups of one chunk.
//
// Tables. For every group of 4 columns {k_0..k_3} and every token, the 16 sums
//     T[i] = sum_q (bit q of i ? +z_{k_q} : -z_{k_q}),   i = 0..15,
// live in shared memory (FP32); a matrix row then needs one table read and
// one FP32 add per 4 signs (the 4 sign bits of the group are the index). In
// the row-block layout (af1_layout.h) bit 8e + p of word kw is column
// 32 kw + 4p + e, so nibble j = 2e + h of a word holds the signs of columns
// 32 kw + 16h + 4q + e, q = 0..3: the group of nibble j. The tables of one
// 128-column chunk take 2 KB per token (one token) or 4 KB per token pair
// (float2 entries {token 2p, 2p + 1}); group g = 4j + w (word w, nibble j)
// sits at g * 64 (one token) or p * 4096 + g * 128 (pairs). The byte offset
// of an entry inside its 256-byte window is built from the sign word with
// one shift and one LOP3 for four nibbles at a time, and PRMT splices it
// under the window's upper address bytes: a lookup is PRMT + LDS + FADD.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1_internal.h"
#include "af1_layout.h"
#include "af1_ptx.cuh"

namespace af1 {
namespace {

// v -> `local` in the shared memory of cluster CTA `rank`, completing 4
// bytes of the transaction count of that CTA's mbarrier `bar`.
__device__ __forceinline__ void st_async_f32(float* local, uint64_t* bar, uint32_t rank, float v) {
  uint32_t raddr, rbar;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(raddr) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rbar) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.f32 [%0], %1, [%2];" ::"r"(raddr), "f"(v),
               "r"(rbar)
               : "memory");
}
__device__ __forceinline__ float lds_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}
template <int OFF>
__device__ __forceinline__ float2 lds_f32x2(uint32_t addr) {
  float2 v;
  asm volatile("ld.shared.v2.f32 {%0,%1}, [%2+%3];" : "=f"(v.x), "=f"(v.y) : "r"(addr), "n"(OFF));
  return v;
}

// ---------------------------------------------------------------------------
// Table layout
// ---------------------------------------------------------------------------

// Token pairs of a pass: 0 stands for a single token (FP32 entries).
__host__ __device__ constexpr int pairs_for(int T) { return T == 1 ? 0 : (T + 1) / 2; }
// Table bytes of one chunk.
__host__ __device__ constexpr int table_chunk_bytes(int np) { return np == 0 ? 2048 : 4096 * np; }
// Staged activations: column k of the CTA at k + k / 32 (the skew keeps the
// table builders' stride-32 reads on distinct banks).
__host__ __device__ constexpr int zrow_floats(int CPC) { return CPC * kChunkCols + CPC * (kChunkCols / 32); }
// ---------------------------------------------------------------------------
// Activations, tables, lookups
// ---------------------------------------------------------------------------

// SwiGLU input h = FP16(SiLU(g) u), SiLU(g) = g / (1 + e^-g) in FP32.
__device__ __forceinline__ float swiglu_h(float g, float u) {
  return __half2float(__float2half_rn(g / (1.f + expf(-g)) * u));
}

// Activations of `nch` chunks from column k0 on -> zs[t][k + k / 32]
// (FP32), k the column within the staged chunks. Phase 1 stages z = b * x
// (an FP16 x FP16 product, exact in FP32; SWIGLU: x = swiglu_h(xg, x2g)),
// phase 2 its FP32 input; columns >= C stage 0. Written by the previous
// kernel, the inputs are read through L2 (ld.global.cg), 8 columns per load,
// a batch of loads per thread in flight at once.
template <int PHASE, int THREADS, bool SWIGLU = false>
__device__ __forceinline__ void stage_activations(const LutProblem& pb, const __half* xg, const __half* x2g,
                                                  const float* zg, int T, int nch, int64_t k0, float* zs, int zrow,
                                                  int tid) {
  const int g8 = nch * (kChunkCols / 8);  // 8-column groups per token
  const int ng = T * g8;
  constexpr int kBatch = 2;
  for (int i0 = tid; i0 < ng; i0 += kBatch * THREADS) {
    float v[kBatch][8];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int i = i0 + u * THREADS;
      const int t = i / g8, k = (i - t * g8) * 8;
      const int64_t col = k0 + k;
      if (i < ng && col + 7 < pb.sm.C) {
        if (PHASE == 1) {
          const uint4 xr = __ldcg(reinterpret_cast<const uint4*>(xg + (int64_t)t * pb.ldx + col));
          const uint4 br = __ldg(reinterpret_cast<const uint4*>(pb.colscale + col));
          const uint32_t xw[4] = {xr.x, xr.y, xr.z, xr.w}, bw[4] = {br.x, br.y, br.z, br.w};
          uint32_t uw[4] = {0u, 0u, 0u, 0u};
          if constexpr (SWIGLU) {
            const uint4 ur = __ldcg(reinterpret_cast<const uint4*>(x2g + (int64_t)t * pb.ldx + col));
            uw[0] = ur.x;
            uw[1] = ur.y;
            uw[2] = ur.z;
            uw[3] = ur.w;
          }
#pragma unroll
          for (int h2 = 0; h2 < 4; ++h2) {
            float2 xf = __half22float2(*reinterpret_cast<const __half2*>(&xw[h2]));
            const float2 bf = __half22float2(*reinterpret_cast<const __half2*>(&bw[h2]));
            if constexpr (SWIGLU) {
              const float2 uf = __half22float2(*reinterpret_cast<const __half2*>(&uw[h2]));
              xf.x = swiglu_h(xf.x, uf.x);
              xf.y = swiglu_h(xf.y, uf.y);
            }
            v[u][2 * h2] = xf.x * bf.x;
            v[u][2 * h2 + 1] = xf.y * bf.y;
          }
        } else {
          const float4 z0 = __ldcg(reinterpret_cast<const float4*>(zg + (int64_t)t * pb.ldz + col));
          const float4 z1 = __ldcg(reinterpret_cast<const float4*>(zg + (int64_t)t * pb.ldz + col + 4));
          v[u][0] = z0.x;
          v[u][1] = z0.y;
          v[u][2] = z0.z;
          v[u][3] = z0.w;
          v[u][4] = z1.x;
          v[u][5] = z1.y;
          v[u][6] = z1.z;
          v[u][7] = z1.w;
        }
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float z = 0.f;
          if (i < ng && col + q < pb.sm.C) {
            if (PHASE == 1) {
              float xv = __half2float(__ldcg(xg + (int64_t)t * pb.ldx + col + q));
              if constexpr (SWIGLU) xv = swiglu_h(xv, __half2float(__ldcg(x2g + (int64_t)t * pb.ldx + col + q)));
              z = xv * __half2float(pb.colscale[col + q]);
            } else
              z = __ldcg(zg + (int64_t)t * pb.ldz + col + q);
          }
          v[u][q] = z;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int i = i0 + u * THREADS;
      if (i < ng) {
        const int t = i / g8, k = (i - t * g8) * 8;
        float* dst = zs + t * zrow + k + (k >> 5);  // 8 columns within one 32-column block
#pragma unroll
        for (int q = 0; q < 8; ++q) dst[q] = v[u][q];
      }
    }
  }
}

// Tables of `nch` staged chunks at `tbl` from the staged activations: task
// (c, j, w, q) writes entries 4q .. 4q + 3 of group 4j + w of chunk c (a
// warp's 32 tasks write 512 contiguous bytes). Tokens >= T get zero tables.
template <int NP, int THREADS>
__device__ __forceinline__ void build_tables(uint8_t* tbl, const float* zs, int zrow, int T, int nch, int tid) {
  constexpr int TCB = table_chunk_bytes(NP);
  const int npair = NP == 0 ? 1 : NP;
  const int ntask = nch * 128 * npair;
  for (int task = tid; task < ntask; task += THREADS) {
    const int q = task & 3, w = (task >> 2) & 3, j = (task >> 4) & 7;
    const int rest = task >> 7;
    const int p = rest % npair, c = rest / npair;
    const int e = j >> 1, hh = j & 1;
    // columns of index bits 0..3 (chunk-local): c 128 + 32 w + 16 hh + 4 qq + e
    const int kb = c * kChunkCols + 32 * w + 16 * hh + e;
    const int zb = kb + (kb >> 5);  // same 32-column block for all four
    uint8_t* dst = tbl + c * TCB + (NP == 0 ? (4 * j + w) * 64 + q * 16 : p * 4096 + (4 * j + w) * 128 + q * 32);
    float ent[2][4];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int t = NP == 0 ? 0 : 2 * p + u;
      if (NP == 0 && u == 1) break;
      float z0 = 0.f, z1 = 0.f, z2 = 0.f, z3 = 0.f;
      if (t < T) {
        const float* zr = zs + t * zrow + zb;
        z0 = zr[0];
        z1 = zr[4];
        z2 = zr[8];
        z3 = zr[12];
      }
      const float c23 = ((q & 1) ? z2 : -z2) + ((q & 2) ? z3 : -z3);
      const float d = z0 + z1, f = z0 - z1;
      ent[u][0] = c23 - d;  // -z0 - z1
      ent[u][1] = c23 + f;  // +z0 - z1
      ent[u][2] = c23 - f;  // -z0 + z1
      ent[u][3] = c23 + d;  // +z0 + z1
    }
    if (NP == 0) {
      *reinterpret_cast<float4*>(dst) = make_float4(ent[0][0], ent[0][1], ent[0][2], ent[0][3]);
    } else {
      *reinterpret_cast<float4*>(dst) = make_float4(ent[0][0], ent[1][0], ent[0][1], ent[1][1]);
      *reinterpret_cast<float4*>(dst + 16) = make_float4(ent[0][2], ent[1][2], ent[0][3], ent[1][3]);
    }
  }
}

// Lookups of one word w (word wi of chunk, thread-constant) for one token:
// tables of the chunk at tb (one token, 64 bytes per group).
__device__ __forceinline__ void lookup_word1(uint32_t w, uint32_t pat, const uint32_t (&base)[8], float& acc) {
  const uint32_t lo = ((w << 2) & 0x3C3C3C3Cu) | pat;  // nibbles 0, 2, 4, 6 -> entry offsets
  const uint32_t hi = ((w >> 2) & 0x3C3C3C3Cu) | pat;  // nibbles 1, 3, 5, 7
#pragma unroll
  for (int j = 0; j < 8; ++j) acc += lds_f32(__byte_perm((j & 1) ? hi : lo, base[j], 0x7650 | (j >> 1)));
}

template <int NP>
__device__ __forceinline__ void lookup_word2(uint32_t w, uint32_t pat, const uint32_t (&base)[8], float (&acc)[2 * NP]) {
  const uint32_t lo = ((w << 3) & 0x78787878u) | pat;
  const uint32_t hi = ((w >> 1) & 0x78787878u) | pat;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t addr = __byte_perm((j & 1) ? hi : lo, base[j], 0x7650 | (j >> 1));
    const float2 v0 = lds_f32x2<0>(addr);
    acc[0] += v0.x;
    acc[1] += v0.y;
    if (NP > 1) {
      const float2 v1 = lds_f32x2<4096>(addr);
      acc[2] += v1.x;
      acc[3] += v1.y;
    }
  }
}

// Lookups of one chunk for thread (r, g): words 2g and 2g + 1 of row r
// (wc = the chunk's words + r) against the chunk's tables at tb.
template <int NP>
__device__ __forceinline__ void lookup_chunk(uint32_t tb, const uint32_t* wc, int g, float (&acc)[NP == 0 ? 1 : 2 * NP]) {
  // Entry-offset byte patterns of words 2g and 2g + 1 (their groups'
  // offsets below the 256-byte window).
  const uint32_t pat0 = NP == 0 ? (uint32_t)(2 * g * 64) * 0x01010101u : 0u;
  const uint32_t pat1 = NP == 0 ? (uint32_t)((2 * g + 1) * 64) * 0x01010101u : 0x80808080u;
  uint32_t base[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) base[j] = tb + (uint32_t)(NP == 0 ? j * 256 : j * 512 + g * 256);
  const uint32_t w0 = wc[(2 * g) * kBlockRows], w1 = wc[(2 * g + 1) * kBlockRows];
  if constexpr (NP == 0) {
    lookup_word1(w0, pat0, base, acc[0]);
    lookup_word1(w1, pat1, base, acc[0]);
  } else {
    lookup_word2<NP>(w0, pat0, base, acc);
    lookup_word2<NP>(w1, pat1, base, acc);
  }
}

}  // namespace
}  // namespace af1
