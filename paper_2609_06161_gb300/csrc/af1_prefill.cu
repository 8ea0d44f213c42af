// af1_prefill.cu — prefill path (more than 16 tokens): the two sign-matrix
// products of AF1 Eq. final_reconstruction as dense GEMMs on the sm_103a
// tensor cores (tcgen05), with the 1-bit factors expanded on the fly.
//
//   GEMM1: H[t][k] = s_k * sum_j B[k][j] * (b_j x[t][j])    (B = V^T, r x n)
//   GEMM2: y[t][i] = a_i * sum_k U[i][k] * H[t][k]          (U, m x r)
//
// Output tiles are 128 features x BN tokens (BN = 16, 32, 64, 128 or 256),
// with K cut into stages of 128 (BN = 256) or 64. The kernel is persistent
// and stream-K: the grid (at most one CTA per SM, chosen on the host by a
// cost model) splits the (tile, K-stage) iterations into equal contiguous
// ranges, so a CTA runs some whole tiles plus, at either end of its range,
// part of a tile shared with its neighbours. A shared tile's contributors
// take tickets when their part is final; all but the last store FP32
// partial tiles in the workspace, and the last sums the parts in a fixed
// contributor order (results do not depend on timing), applies the feature
// scale and stores the output (see sum_tile). No CTA waits for another that
// may not be running. Without room for the partials (the built-in-scratch
// entry) the grid is one CTA per tile.
//
// Roles of the 18 warps of a CTA, over the CTA's stages in order:
//   * warp 0, one thread: copies each stage's packed signs (the row block's
//     words of the stage, 1-2 KB contiguous in the row-block layout) and,
//     for GEMM1, its column scales into a ring of small slots
//     (cp.async.bulk), 6-14 stages ahead and independent of the MMA (with
//     the signs loaded by the expanders one stage ahead, each stage waited
//     about 1,500 cycles on the load); then the stage's FP16 activation
//     tile(s) (B, BN x 64 per box) by TMA (cp.async.bulk.tensor, 128-byte
//     swizzle, zero fill past the tokens / columns) into a ring of 3 stages
//     of 64 KB (BN = 256) or 8;
//   * warps 4-11 expand the signs into FP16 (+-b_j for GEMM1, +-1 for GEMM2:
//     exact) and store them into a ring of A buffers (one per stage) in
//     tensor memory (tcgen05.st; warp w writes rows 32 (w % 4) .. +31, one
//     row per thread = tensor-memory lane, and half (w - 4) / 4 of the
//     stage's columns); A in tensor memory leaves shared-memory bandwidth to
//     B;
//   * warp 1, one thread: the stage's tcgen05.mma.kind::f16 (K = 16 each,
//     N = BN, A from tensor memory, B from shared memory) into an
//     accumulator (D, FP32, BN columns), after one wait on the stage's
//     barrier (completed by the activation copy and the 8 expander warps),
//     then one commit. Measured: this thread needs 134 cycles per MMA, N =
//     128 or 256 alike, plus 77 per commit and 67 per barrier check, and the
//     tensor pipe idles meanwhile; hence stages of 128 and tiles of 256.
//     Tiles of up to 128 tokens alternate between two accumulators, so the
//     epilogue of one tile overlaps the MMAs of the next; tiles of 256 have
//     one (two would leave no tensor memory for A), and the MMAs of the next
//     tile wait for its read-back;
//   * two groups of four warps (12-15; 16, 17, 2, 3) read an accumulator
//     back (tcgen05.ld) in alternate chunks (32 tokens for FP16 outputs, 16
//     for FP32 ones and partial tiles), apply the feature scale and stage
//     each chunk in shared memory, which one thread of the group writes out
//     with a TMA store (or a bulk copy for a partial tile) (stores from the
//     warps themselves were latency-bound in the store queue).
// All waits are bounded; a wait that gives up sets the status word.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cstring>

#include "af1_internal.h"
#include "af1_layout.h"
#include "af1_ptx.cuh"

namespace af1 {
namespace {

constexpr int BM = 128;      // features per tile (MMA M, tensor-memory lanes)
constexpr int BOX = 64;      // K per activation box: one 128-byte swizzle row of FP16
constexpr int kThreads = 576;
constexpr int kTmemCols = 512;  // accumulators (2 x BN, or 1 x 256) + one A buffer per stage
constexpr int kExpandWarps = 8;  // warps 4..11
constexpr int kEpiWarp0 = 12;    // epilogue group 0: warps 12..15; group 1: warps 16, 17, 2, 3
constexpr int kEpiWarps = 8;
__device__ __forceinline__ bool is_epi_warp(int w) { return w == 2 || w == 3 || w >= kEpiWarp0; }
constexpr int kMaxStages = 8;
constexpr int kMaxWSlots = 14;

// K per stage: 128 for tiles of 256 tokens, 64 otherwise. One thread issues
// the MMAs and every operation of its loop besides them leaves the tensor
// pipe idle (measured: 134 cycles per MMA back to back, N = 128 or 256; a
// commit adds 77 and a completed mbarrier check 67), so long stages and one
// barrier per stage keep it busy.
template <int BN>
__host__ __device__ constexpr int bk() {
  return BN == 256 ? 128 : 64;
}
__host__ __device__ constexpr int bk_of(int bn) { return bn == 256 ? 128 : 64; }
template <int BN>
__host__ __device__ constexpr int tile_b_bytes() {
  return BN * bk<BN>() * 2;
}
// Stages of the activation ring (shared memory) and of the A ring (tensor
// memory, bk / 2 columns each), and accumulators.
template <int BN>
__host__ __device__ constexpr int stages() {
  return BN == 256 ? 3 : 8;
}
template <int BN>
__host__ __device__ constexpr int accumulators() {
  return BN == 256 ? 1 : 2;
}
static_assert(accumulators<256>() * 256 + stages<256>() * bk<256>() / 2 <= kTmemCols, "tensor memory");
static_assert(accumulators<128>() * 128 + stages<128>() * bk<128>() / 2 <= kTmemCols, "tensor memory");
// Sign ring: slots of one stage's packed words (bk / 32 words x 128 rows)
// followed by its bk FP16 column scales (GEMM1).
template <int BN>
__host__ __device__ constexpr int wsign_bytes() {
  return bk<BN>() / 32 * kBlockRows * 4;
}
template <int BN>
__host__ __device__ constexpr int wslot_bytes() {
  return wsign_bytes<BN>() + bk<BN>() * 2;
}
template <int BN>
__host__ __device__ constexpr int wslots() {
  return BN == 256 ? 6 : 14;
}
// Epilogue staging: two buffers of one 16-token x 128-row chunk (FP32 at
// most), [token][row].
constexpr int kEpiStageBytes = 16 * 128 * 4;
constexpr int kSmemCap = 227 * 1024;  // opt-in shared memory of a CTA
template <int BN>
__host__ __device__ constexpr int smem_base() {
  return stages<BN>() * tile_b_bytes<BN>() + wslots<BN>() * wslot_bytes<BN>() + 2 * kEpiStageBytes +
         1024 /* barriers */ + 1024 /* base alignment */;
}
// Extra landing space right after the activation ring, for the parts of a
// shared tile that a CTA sums (the ring alone holds 16 tokens of at most 2-4
// parts for tiles of 16-32 tokens, and pieces of 16 tokens each paid a
// round trip): what the CTA's shared memory has left, for tiles of up to
// 128 tokens. The whole CTA takes the SM anyway (it allocates all of its
// tensor memory).
template <int BN>
__host__ __device__ constexpr int land_bytes() {
  return BN == 256 ? 0 : (kSmemCap - smem_base<BN>()) / 1024 * 1024;
}
// Bytes a summing CTA can copy parts into: the activation ring and the land.
template <int BN>
__host__ __device__ constexpr int landing_bytes() {
  return stages<BN>() * tile_b_bytes<BN>() + land_bytes<BN>();
}
template <int BN>
__host__ __device__ constexpr int smem_bytes() {
  return smem_base<BN>() + land_bytes<BN>();
}
static_assert(smem_bytes<256>() <= kSmemCap, "shared memory");
static_assert(smem_bytes<16>() <= kSmemCap && smem_bytes<128>() <= kSmemCap, "shared memory");
// Host side: landing bytes for a tile width of bn tokens.
inline int64_t landing_bytes_of(int bn) {
  switch (bn) {
    case 16: return landing_bytes<16>();
    case 32: return landing_bytes<32>();
    case 64: return landing_bytes<64>();
    case 128: return landing_bytes<128>();
    default: return landing_bytes<256>();
  }
}

struct PrefillArgs {
  const uint32_t* signs;  // packed signs, af1_layout.h row-block layout
  SignMatrix sm;          // R = features, C = K
  int tokens;
  const __half* colscale;  // GEMM1: b (length C, zero-padded to 128-column stages); GEMM2: nullptr (+-1)
  const __half* rowscale;  // GEMM1: s (length R); GEMM2: a
  void* out;               // GEMM1: H [tokens][ld_out] FP16; GEMM2: y
  int64_t ld_out;
  int out_f32;
  int out_vec;             // out and ld_out allow 16-byte stores
  float* part;             // partial tiles: 2 slots per CTA of 128 rows x BN FP32 (nullptr: one tile per CTA)
  unsigned* count;         // per tile: tickets taken, partials stored (zero between calls)
  unsigned* status;
  long long wait_cycles;  // budget of every bounded wait (clock64 cycles)
};

struct __align__(8) PrefillBarriers {
  uint64_t full[kMaxStages];     // the stage's activation tile has landed and its A is stored
  uint64_t empty[kMaxStages];    // the stage's MMAs are done
  uint64_t full_w[kMaxWSlots];   // a stage's signs (and column scales) have landed
  uint64_t empty_w[kMaxWSlots];  // the expander warps have read them
  uint64_t dfull[2];           // accumulator d holds a finished tile (or segment)
  uint64_t dempty[2];          // the epilogue has read accumulator d
  uint32_t issued_b, issued_w; // copies issued (drained when a wait gave up)
  uint64_t red;                // partial tiles copied in for a reduction
  uint32_t tmem_addr;
  uint32_t err;
  uint32_t last;               // epilogue: this CTA holds the last ticket of the shared tile
  uint32_t npend;              // epilogue: a shared tile this CTA sums at the end of its range
  uint32_t pend[2];
};

__device__ __forceinline__ void tmem_ld16(uint32_t addr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(addr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 2-D TMA load of the box at (x = column, y = token) into shared memory,
// completing on `bar` with the box's byte count.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);  // start address
  d |= (uint64_t)1u << 16;                 // leading byte offset (unused for this layout)
  d |= (uint64_t)(1024u >> 4) << 32;       // stride byte offset
  d |= (uint64_t)1u << 46;                 // version
  d |= (uint64_t)2u << 61;                 // 128-byte swizzle
  return d;
}

// kind::f16: D F32, A and B F16, both K-major, M = 128, N = BN.
template <int BN>
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, bool accumulate) {
  constexpr uint32_t idesc = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate ? 1u : 0u)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// Sign bit (bit `p` of bytes b0 and b1 of the selected pair) -> the sign
// positions 15 and 31 of an FP16 pair, then value = +-v (bit 1 keeps v).
__device__ __forceinline__ uint32_t signed_pair(uint32_t pair_bytes, int p, uint32_t v) {
  const uint32_t sh = pair_bytes << (7 - p);
  return v ^ (~sh & 0x80008000u);
}

// TMA store of the [16 tokens][128 rows] box at (x = row, y = token) from
// shared memory, and a plain bulk store; both in the thread's bulk group.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(smem_u32(src))
               : "memory");
}
__device__ __forceinline__ void bulk_s2g(void* dst, const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_u32(src)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// No group still reading its shared-memory source.
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// Every group complete (its writes performed).
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void tmem_ld16_nowait(uint32_t addr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(addr));
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// A warp's 32-row x 16-token chunk, held one row per lane (v[q] = token
// q), to dst[token][row] (leading dimension ld): through a 16 x 32 staging
// tile in shared memory, so that each lane stores 16 contiguous bytes (one
// 2-byte store per lane and token was latency-bound in the store queue:
// about 70 cycles per store instruction). Rows row0 .. +31 (those below
// nrow), tokens tok0 .. +15 (those below ntok).
template <typename T>
__device__ __forceinline__ void store_chunk(const float (&v)[16], T* stage, T* dst, int64_t ld, int64_t row0,
                                            int64_t nrow, int64_t tok0, int64_t ntok, bool vec, int lane) {
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    if constexpr (sizeof(T) == 2)
      stage[q * 32 + lane] = __float2half_rn(v[q]);
    else
      stage[q * 32 + lane] = v[q];
  }
  __syncwarp();
  constexpr int VE = 16 / (int)sizeof(T);  // elements per 16-byte vector
  constexpr int VPR = 32 / VE;              // vectors per token
#pragma unroll
  for (int vi = lane; vi < 16 * VPR; vi += 32) {
    const int tk = vi / VPR, cg = vi % VPR;
    const int64_t tok = tok0 + tk, row = row0 + cg * VE;
    if (tok < ntok) {
      const T* src = stage + tk * 32 + cg * VE;
      T* p = dst + tok * ld + row;
      if (vec && row + VE <= nrow) {
        *reinterpret_cast<uint4*>(p) = *reinterpret_cast<const uint4*>(src);
      } else {
        for (int e = 0; e < VE; ++e)
          if (row + e < nrow) p[e] = src[e];
      }
    }
  }
  __syncwarp();
}

// The CTA that runs iteration i of I split over G CTAs: CTA c runs
// [floor(c I / G), floor((c + 1) I / G)).
__device__ __forceinline__ int cta_of(int64_t i, int64_t I, int G) { return (int)(((i + 1) * G - 1) / I); }
__device__ __forceinline__ int64_t range_start(int c, int64_t I, int G) { return (int64_t)c * I / G; }

template <bool GEMM1, int BN>
__global__ void __launch_bounds__(kThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap act_map, const __grid_constant__ CUtensorMap out_map,
                   const __grid_constant__ CUtensorMap out_map32, const PrefillArgs a) {
  constexpr int BK = bk<BN>();
  constexpr int kTileB = tile_b_bytes<BN>();
  constexpr int kBoxBytes = BN * BOX * 2;
  constexpr int kStages = stages<BN>();
  constexpr int ND = accumulators<BN>();
  constexpr int kWSlots = wslots<BN>();
  constexpr int kWSignBytes = wsign_bytes<BN>();
  constexpr int kWSlotBytes = wslot_bytes<BN>();
  constexpr int kACols = BK / 2;       // tensor-memory columns of one stage's A
  constexpr int kWPS = BK / 32;        // sign words per row and stage
  constexpr int kWPW = kWPS / 2;       // ... per expander warp (two warps per row)
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the swizzled operand tiles.
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tileB = smem;  // activation ring, then the landing space of sum_tile
  uint8_t* wring = smem + kStages * kTileB + land_bytes<BN>();
  uint8_t* estage = wring + kWSlots * kWSlotBytes;
  PrefillBarriers& bar = *reinterpret_cast<PrefillBarriers*>(estage + 2 * kEpiStageBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const SignMatrix& tm = a.sm;
  const int RB = tm.RB;
  const int nk = (int)((tm.C + BK - 1) / BK);        // K stages per tile
  const int NT = (a.tokens + BN - 1) / BN;           // token tiles
  const int64_t I = (int64_t)RB * NT * nk;           // iterations: tile t = tt * RB + rb, stage k
  const int G = (int)gridDim.x;
  const int c = (int)blockIdx.x;
  const int64_t i0 = range_start(c, I, G);
  const int n = (int)(range_start(c + 1, I, G) - i0);  // this CTA's stages

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bar.full[s], 1 + kExpandWarps);  // the producer's expect_tx arrival + one per expander warp
      mbar_init(&bar.empty[s], 1);
    }
    for (int s = 0; s < kWSlots; ++s) {
      mbar_init(&bar.full_w[s], 1);
      mbar_init(&bar.empty_w[s], kExpandWarps);
    }
    for (int d = 0; d < ND; ++d) {
      mbar_init(&bar.dfull[d], 1);
      mbar_init(&bar.dempty[d], kEpiWarps);
    }
    mbar_init(&bar.red, 1);
    bar.err = 0;
    bar.issued_b = 0;
    bar.issued_w = 0;
    bar.npend = 0;
    bar.last = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&act_map)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&bar.tmem_addr)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = bar.tmem_addr;  // accumulators at columns 0 (and BN), A buffers from ND BN

  if (warp == 0) {
    // ---- producer -----------------------------------------------------------
    // Stage j of this CTA is iteration i0 + j: tile t = (i0 + j) / nk, K stage
    // k = (i0 + j) % nk. Its signs are words 2k and 2k + 1 of the 128 rows of
    // row block t % RB (256 consecutive words); its column scales lie inside
    // the layer's 256-byte-padded, zero-filled scale array.
    // Two cursors over the stages (signs run ahead of the activation tiles),
    // each kept as (row block, token tile, K stage): no division per stage
    // in this single thread's loop (three 64-bit divisions per stage made
    // it the bottleneck).
    struct Cursor {
      int rb, tt, k;
    };
    const int t_first = (int)(i0 / nk);
    const Cursor c0 = {t_first % RB, t_first / RB, (int)(i0 - (int64_t)t_first * nk)};
    auto advance = [&](Cursor& cu) {
      if (++cu.k == nk) {
        cu.k = 0;
        if (++cu.rb == RB) {
          cu.rb = 0;
          ++cu.tt;
        }
      }
    };
    Cursor cw = c0, cb = c0;
    int wi = 0;  // next stage whose signs are copied (at cursor cw)
    auto issue_w = [&](int j) {
      const int ws = j % kWSlots;
      if (j >= kWSlots) mbar_wait(&bar.empty_w[ws], ((j / kWSlots) & 1) ^ 1, &bar.err, a.wait_cycles);
      uint8_t* dst = wring + ws * kWSlotBytes;
      mbar_expect_tx(&bar.full_w[ws], (uint32_t)(GEMM1 ? kWSlotBytes : kWSignBytes));
      bulk_g2s(dst, a.signs + ((int64_t)cw.rb * tm.NCH * kChunkWords + (int64_t)kWPS * cw.k) * kBlockRows,
               (uint32_t)kWSignBytes, &bar.full_w[ws]);
      if (GEMM1) bulk_g2s(dst + kWSignBytes, a.colscale + (int64_t)cw.k * BK, (uint32_t)(BK * 2), &bar.full_w[ws]);
      advance(cw);
    };
    if (lane == 0) {
      // The signs are constants: copy the first ones before the dependency wait.
      for (; wi < n && wi < kWSlots; ++wi) issue_w(wi);
    }
    griddep_wait();  // the activations are written by the previous kernel
    if (lane == 0) {
      for (int j = 0; j < n; ++j) {
        for (; wi < n && wi < j + kWSlots; ++wi) issue_w(wi);
        const int s = j % kStages;
        if (j >= kStages) mbar_wait(&bar.empty[s], ((j / kStages) & 1) ^ 1, &bar.err, a.wait_cycles);
        mbar_expect_tx(&bar.full[s], (uint32_t)kTileB);
#pragma unroll
        for (int bx = 0; bx < BK / BOX; ++bx)
          tma_load_2d(tileB + s * kTileB + bx * kBoxBytes, &act_map, cb.k * BK + bx * BOX, cb.tt * BN, &bar.full[s]);
        advance(cb);
      }
      bar.issued_b = (uint32_t)n;
      bar.issued_w = (uint32_t)wi;
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA issuer -----------------------------------------------------------
    if (lane == 0) {
      // The barriers of stage j + 1 are checked before the last MMA of
      // stage j is issued, while three MMAs are queued (checked after it,
      // the pipe drained during the two checks: about 200 cycles per stage).
      const uint32_t b0 = smem_u32(tileB);
      int u = 0;  // segment (tile or part of one) of this CTA
      uint32_t d_tmem = tmem;
      bool first = true;
      int k = (int)(i0 % nk);  // K stage of stage j, kept incrementally
      auto wait_stage = [&](int j) { mbar_wait(&bar.full[j % kStages], (j / kStages) & 1, &bar.err, a.wait_cycles); };
      if (n > 0) wait_stage(0);
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      for (int j = 0; j < n; ++j) {
        const int s = j % kStages;
        const bool seg_end = j == n - 1 || k == nk - 1;
        // MMA kk: K 16 kk .. + 15 of the stage = tensor-memory columns 8 kk ..
        // of its A buffer and, of its activation tile, box kk / 4, 32-byte
        // step kk % 4 of the swizzled rows. The stage's operand addresses are
        // all formed before its first MMA (the empty asm pins them there):
        // this thread's issue sets the tensor pipe's pace, and address
        // arithmetic between two MMAs is a gap in it.
        constexpr int kMma = BK / 16;
        uint64_t bdesc[kMma];
        uint32_t aaddr[kMma];
#pragma unroll
        for (int kk = 0; kk < kMma; ++kk) {
          bdesc[kk] = smem_desc(b0 + s * kTileB + (kk / 4) * kBoxBytes + (kk % 4) * 32);
          aaddr[kk] = tmem + (uint32_t)(ND * BN + s * kACols + kk * 8);
          asm volatile("" : "+l"(bdesc[kk]), "+r"(aaddr[kk]));
        }
#pragma unroll
        for (int kk = 0; kk < kMma - 1; ++kk) mma_f16_ts<BN>(d_tmem, aaddr[kk], bdesc[kk], !(first && kk == 0));
        // Stage j + 1: its accumulator must be free (with one accumulator
        // that needs this segment's epilogue, so it waits after the commit).
        const bool ahead = j + 1 < n && !(seg_end && ND == 1);
        if (ahead) {
          if (seg_end && u + 1 >= ND)
            mbar_wait(&bar.dempty[(u + 1) % ND], (((u + 1) / ND) & 1) ^ 1, &bar.err, a.wait_cycles);
          wait_stage(j + 1);
        }
        mma_f16_ts<BN>(d_tmem, aaddr[kMma - 1], bdesc[kMma - 1], true);
        mma_commit(&bar.empty[s]);
        if (seg_end) mma_commit(&bar.dfull[u % ND]);
        if (j + 1 < n) {
          if (seg_end) {
            ++u;
            d_tmem = tmem + (uint32_t)((u % ND) * BN);
            first = true;
            if (!ahead) {
              if (u >= ND) mbar_wait(&bar.dempty[u % ND], ((u / ND) & 1) ^ 1, &bar.err, a.wait_cycles);
              wait_stage(j + 1);
            }
          } else {
            first = false;
          }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        }
        if (++k == nk) k = 0;
      }
    }
    __syncwarp();
  } else if (warp >= 4 && warp < kEpiWarp0) {
    // ---- weight expansion: warp w, rows 32 (w % 4) + lane, half h = (w - 4)
    //      / 4 of the stage: its words h kWPW .. + kWPW - 1 (32 K each) ------
    const int q = warp & 3, h = (warp - 4) >> 2;
    const int R = q * 32 + lane;  // TMEM lane = row of the block
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    for (int j = 0; j < n; ++j) {
      const int s = j % kStages;
      const int ws = j % kWSlots;
      mbar_wait(&bar.full_w[ws], (j / kWSlots) & 1, &bar.err, a.wait_cycles);
      const uint32_t* wslot = reinterpret_cast<const uint32_t*>(wring + ws * kWSlotBytes);
      uint32_t av[16 * kWPW];
#pragma unroll
      for (int ww = 0; ww < kWPW; ++ww) {
        const int word = h * kWPW + ww;  // word of the stage: K 32 word .. + 31
        const uint32_t wd = wslot[word * kBlockRows + R];
        uint4 cs[4];
        if (GEMM1) {
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) cs[jj] = reinterpret_cast<const uint4*>(wslot + kWPS * kBlockRows)[4 * word + jj];
        }
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          // K 32 word + 8 jj .. + 7 (tensor-memory columns 16 word + 4 jj ..
          // + 3, two FP16 values each) = columns 4p + e of the word with
          // p = 2 jj (first 4) and p + 1 (last 4).
          const int p = 2 * jj;
          const uint32_t b01 = __byte_perm(wd, 0u, 0x1404);  // bytes 0,1 -> bytes 1,3 (e = 0, 1)
          const uint32_t b23 = __byte_perm(wd, 0u, 0x3424);  // bytes 2,3 -> bytes 1,3 (e = 2, 3)
          uint4 sv = make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);  // +-1 for GEMM2
          if (GEMM1) sv = cs[jj];
          av[16 * ww + 4 * jj + 0] = signed_pair(b01, p, sv.x);
          av[16 * ww + 4 * jj + 1] = signed_pair(b23, p, sv.y);
          av[16 * ww + 4 * jj + 2] = signed_pair(b01, p + 1, sv.z);
          av[16 * ww + 4 * jj + 3] = signed_pair(b23, p + 1, sv.w);
        }
      }
      // The words and scales are in registers: hand the slot back.
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar.empty_w[ws]);
      // The previous stage's store was left in flight while this stage was
      // expanded: complete it and count this warp on that stage.
      if (j > 0) {
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar.full[(j - 1) % kStages]);
      }
      if (j >= kStages) {
        if (lane == 0) mbar_wait(&bar.empty[s], ((j / kStages) & 1) ^ 1, &bar.err, a.wait_cycles);
        __syncwarp();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      }
      const uint32_t addr = tmem + lane_base + (uint32_t)(ND * BN + s * kACols + 16 * kWPW * h);
      if constexpr (kWPW == 2) {
        asm volatile(
            "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
            "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(addr),
            "r"(av[0]), "r"(av[1]), "r"(av[2]), "r"(av[3]), "r"(av[4]), "r"(av[5]), "r"(av[6]), "r"(av[7]),
            "r"(av[8]), "r"(av[9]), "r"(av[10]), "r"(av[11]), "r"(av[12]), "r"(av[13]), "r"(av[14]), "r"(av[15]),
            "r"(av[16]), "r"(av[17]), "r"(av[18]), "r"(av[19]), "r"(av[20]), "r"(av[21]), "r"(av[22]), "r"(av[23]),
            "r"(av[24]), "r"(av[25]), "r"(av[26]), "r"(av[27]), "r"(av[28]), "r"(av[29]), "r"(av[30]), "r"(av[31])
            : "memory");
      } else {
        asm volatile(
            "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
                addr),
            "r"(av[0]), "r"(av[1]), "r"(av[2]), "r"(av[3]), "r"(av[4]), "r"(av[5]), "r"(av[6]), "r"(av[7]),
            "r"(av[8]), "r"(av[9]), "r"(av[10]), "r"(av[11]), "r"(av[12]), "r"(av[13]), "r"(av[14]), "r"(av[15])
            : "memory");
      }
    }
    if (n > 0) {
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar.full[(n - 1) % kStages]);
    }
    // The next kernel may launch once this CTA has expanded its weights: its
    // own expansion needs no input and would otherwise compete with this
    // one's for the SMs.
    griddep_launch_dependents();
  } else if (is_epi_warp(warp)) {
    // ---- epilogue: accumulator -> registers -> output or partial tile --------
    // Two groups of four warps (one warp per tensor-memory lane quadrant
    // each) take alternate 16-token chunks, so two read-back chains run at
    // once (the MMA waits for this read-back when a tile has one
    // accumulator). Group g stages its chunk in buffer g; its first thread
    // writes it out.
    const int q = warp & 3;
    const int g = (warp >= kEpiWarp0 && warp < kEpiWarp0 + 4) ? 0 : 1;
    const int R = q * 32 + lane;
    const bool issuer = R == 0;                // the group's thread that writes chunks out
    const bool leader = issuer && g == 0;      // counts partials and copies parts in
    const int gbar = 1 + g;                    // named barrier of the group (128 threads)
    constexpr int kBothBar = 3;                // named barrier of both groups (256 threads)
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const bool tma_out = a.out_vec != 0;  // else each warp stores its own rows
    uint8_t* buf = estage + g * kEpiStageBytes;
    griddep_wait();  // the outputs (and partial tiles) may still be read by the previous kernel
    uint32_t red_phase = 0;  // completions of bar.red seen
    // One 16-token chunk of the tile (this thread's row R, v[q] = token
    // c0 + q), staged [token][row] and written by the group's first thread:
    // into the output (TMA store; rows and tokens past the matrix are not
    // written) or, with part != nullptr, into a partial slot (bulk copy).
    auto emit = [&](const float (&v)[16], float* part, int c0, int64_t row_base, int64_t tok) {
      if (issuer) bulk_wait_read0();  // the group's previous store has read the buffer
      named_sync(gbar, 128);
      if (part != nullptr || a.out_f32) {
        float* b = reinterpret_cast<float*>(buf);
#pragma unroll
        for (int qq = 0; qq < 16; ++qq) b[qq * BM + R] = v[qq];
      } else {
        __half* b = reinterpret_cast<__half*>(buf);
#pragma unroll
        for (int qq = 0; qq < 16; ++qq) b[qq * BM + R] = __float2half_rn(v[qq]);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      named_sync(gbar, 128);
      if (issuer) {
        if (part != nullptr)
          bulk_s2g(part + (size_t)c0 * BM, buf, 16 * BM * 4);
        else
          tma_store_2d(&out_map, buf, (int)row_base, (int)tok);
        bulk_commit();
      }
    };
    auto emit_out = [&](const float (&v)[16], int64_t row0, int64_t row_base, int64_t tok) {
      if (tma_out) {
        emit(v, nullptr, 0, row_base, tok);
      } else if (a.out_f32) {
        store_chunk<float>(v, reinterpret_cast<float*>(estage) + (g * 4 + q) * 512, reinterpret_cast<float*>(a.out),
                           a.ld_out, row0, tm.R, tok, a.tokens, false, lane);
      } else {
        store_chunk<__half>(v, reinterpret_cast<__half*>(estage) + (g * 4 + q) * 1024,
                            reinterpret_cast<__half*>(a.out), a.ld_out, row0, tm.R, tok, a.tokens, false, lane);
      }
    };
    // Sum shared tile t: wait (bounded) for the stored parts, copy them into
    // the activation ring PT tokens at a time, and add in contributor order;
    // this CTA's own part comes from accumulator columns own_dcol, or from
    // its slot when own_dcol is all ones.
    auto sum_tile = [&](int t, uint32_t own_dcol) {
      const int64_t it0 = (int64_t)t * nk;
      const int cf = cta_of(it0, I, G), cl = cta_of(it0 + nk - 1, I, G);
      const bool own_tmem = own_dcol != 0xFFFFFFFFu;
      const int parts = cl - cf + 1;
      const int copied = own_tmem ? parts - 1 : parts;  // parts read from the slots
      unsigned* tickets = a.count + 2 * (size_t)t;
      if (leader) {
        const long long w0 = clock64();
        while (ld_acquire_gpu(tickets + 1) < (unsigned)copied) {
          if (clock64() - w0 > a.wait_cycles) {
            atomicOr(&bar.err, 1u);
            break;
          }
        }
      }
      named_sync(kBothBar, 256);
      const int rb = t % RB, tok0 = (t / RB) * BN;
      const int64_t frow = (int64_t)rb * BM + R;
      const float rsc = frow < tm.R ? __half2float(a.rowscale[frow]) : 0.f;
      const int64_t row_base = (int64_t)rb * BM;
      const int64_t row0 = row_base + q * 32;
      int PT = (int)((int64_t)landing_bytes<BN>() / ((int64_t)copied * BM * 4)) / 16 * 16;
      if (PT > BN) PT = BN;
      if (PT < 16) {  // the host's grid keeps the parts within the ring; never taken
        if (leader) atomicOr(&bar.err, 1u);
        return;
      }
      const float* ringf = reinterpret_cast<const float*>(tileB);
#pragma unroll 1
      for (int p0 = 0; p0 < BN; p0 += PT) {
        const int pt = BN - p0 < PT ? BN - p0 : PT;
        if (leader) {
          // The parts were written by other CTAs (and perhaps this one).
          asm volatile("fence.proxy.async.global;" ::: "memory");
          mbar_expect_tx(&bar.red, (uint32_t)(copied * pt * BM * 4));
          int idx = 0;
          for (int cc = cf; cc <= cl; ++cc) {
            if (own_tmem && cc == c) continue;
            const int sl = 2 * cc + (range_start(cc, I, G) >= it0 ? 0 : 1);
            bulk_g2s(tileB + (size_t)idx * pt * BM * 4, a.part + (size_t)sl * BN * BM + (size_t)p0 * BM,
                     (uint32_t)(pt * BM * 4), &bar.red);
            ++idx;
          }
        }
        mbar_wait(&bar.red, red_phase & 1, &bar.err, a.wait_cycles);
        ++red_phase;
#pragma unroll 1
        for (int c0 = p0 + 16 * g; c0 < p0 + pt; c0 += 32) {
          uint32_t r[16];
          if (own_tmem) tmem_ld16(own_dcol + (uint32_t)c0, r);
          float acc[16];
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) acc[qq] = 0.f;
          int idx = 0;
          for (int cc = cf; cc <= cl; ++cc) {
            if (own_tmem && cc == c) {
#pragma unroll
              for (int qq = 0; qq < 16; ++qq) acc[qq] += __uint_as_float(r[qq]);
              continue;
            }
            const float* src = ringf + ((size_t)idx * pt + (c0 - p0)) * BM + R;
#pragma unroll
            for (int qq = 0; qq < 16; ++qq) acc[qq] += src[qq * BM];
            ++idx;
          }
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) acc[qq] *= rsc;
          emit_out(acc, row0, row_base, tok0 + c0);
        }
        named_sync(kBothBar, 256);  // the piece is read before the next copy overwrites it
      }
      if (leader) {
        tickets[0] = 0u;  // ready for the next call
        tickets[1] = 0u;
      }
    };
    int64_t i = i0;
    const int64_t iend = i0 + n;
    for (int u = 0; i < iend; ++u) {
      const int t = (int)(i / nk);
      const int ka = (int)(i - (int64_t)t * nk);
      const int kb = (int)min((int64_t)nk, (int64_t)ka + (iend - i));
      i += kb - ka;
      const int d = u % ND;
      if (lane == 0) mbar_wait(&bar.dfull[d], (u / ND) & 1, &bar.err, a.wait_cycles);
      __syncwarp();
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t dcol = tmem + lane_base + (uint32_t)(d * BN);
      const int rb = t % RB, tok0 = (t / RB) * BN;
      const int64_t frow = (int64_t)rb * BM + R;
      const float rsc = frow < tm.R ? __half2float(a.rowscale[frow]) : 0.f;
      const int64_t row_base = (int64_t)rb * BM;
      const int64_t row0 = row_base + q * 32;  // first row of this warp's quadrant
      if (ka == 0 && kb == nk && tma_out && !a.out_f32 && BN >= 32) {
        // A whole tile with FP16 output: 32-token chunks (alternating between
        // the groups), staged as two 16-token halves and written by one TMA
        // store (half the barriers, waits and store issues per token of
        // 16-token chunks). Both halves of the next chunk are read back from
        // tensor memory while this one is staged and stored: a read-back
        // takes about as long as staging a chunk (one 16-column read in
        // flight at a time left a 256-token tile's drain at ~2.9 us even
        // without any store).
        __half* hb = reinterpret_cast<__half*>(buf);
        uint32_t ra[16], rb[16];
        if (32 * g < BN) {
          tmem_ld16_nowait(dcol + (uint32_t)(32 * g), ra);
          tmem_ld16_nowait(dcol + (uint32_t)(32 * g + 16), rb);
        }
#pragma unroll 1
        for (int c0 = 32 * g; c0 < BN; c0 += 64) {
          if (issuer) bulk_wait_read0();  // the group's previous store has read the buffer
          named_sync(gbar, 128);
          tmem_wait_ld();  // this chunk's read-back
          const bool more = c0 + 64 < BN;
          float v[16];
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) v[qq] = __uint_as_float(ra[qq]) * rsc;
          if (more) tmem_ld16_nowait(dcol + (uint32_t)(c0 + 64), ra);
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) hb[qq * BM + R] = __float2half_rn(v[qq]);
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) v[qq] = __uint_as_float(rb[qq]) * rsc;
          if (more) tmem_ld16_nowait(dcol + (uint32_t)(c0 + 80), rb);
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) hb[(16 + qq) * BM + R] = __float2half_rn(v[qq]);
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          named_sync(gbar, 128);
          if (issuer) {
            tma_store_2d(&out_map32, buf, (int)row_base, (int)(tok0 + c0));
            bulk_commit();
          }
        }
        tmem_wait_ld();
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar.dempty[d]);
      } else if (ka == 0 && kb == nk) {
        // A whole tile: scale and store this group's chunks; the next
        // chunk's read-back is in flight while this one is staged.
        uint32_t r[16];
        if (16 * g < BN) tmem_ld16(dcol + (uint32_t)(16 * g), r);
#pragma unroll 1
        for (int c0 = 16 * g; c0 < BN; c0 += 32) {
          float v[16];
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) v[qq] = __uint_as_float(r[qq]) * rsc;
          if (c0 + 32 < BN) tmem_ld16_nowait(dcol + (uint32_t)(c0 + 32), r);
          emit_out(v, row0, row_base, tok0 + c0);
          tmem_wait_ld();
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar.dempty[d]);
      } else {
        // Part of a shared tile (CTAs cf .. cl contribute). Each takes a
        // ticket when its accumulator is final (acquire-release add). The
        // last ticket sums the tile: at once when this is the CTA's last
        // segment (its activation ring is then idle; its own part stays in
        // tensor memory), else at the end of its range. Every other part is
        // stored into its CTA's slot (0 for the segment the CTA's range starts
        // with, 1 for the one it ends with; [token][row] over the tile's 128
        // rows) and counted as stored (release add). The summing CTA waits
        // (bounded) only for parts of CTAs that hold a ticket, i.e. that are
        // resident and only storing.
        const int64_t it0 = (int64_t)t * nk;
        const int cf = cta_of(it0, I, G), cl = cta_of(it0 + nk - 1, I, G);
        unsigned* tickets = a.count + 2 * (size_t)t;
        if (leader) bar.last = atom_add_acq_rel_gpu(tickets, 1u) == (unsigned)(cl - cf) ? 1u : 0u;
        named_sync(kBothBar, 256);
        const bool last = bar.last != 0;
        named_sync(kBothBar, 256);  // bar.last is reused by the next shared tile
        if (last && i == iend) {
          sum_tile(t, dcol);
          asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar.dempty[d]);
        } else {
          const int slot = 2 * c + (i0 >= it0 ? 0 : 1);
          float* Pp = a.part + (size_t)slot * BN * BM;
          uint32_t r[16];
          if (16 * g < BN) tmem_ld16(dcol + (uint32_t)(16 * g), r);
#pragma unroll 1
          for (int c0 = 16 * g; c0 < BN; c0 += 32) {
            float v[16];
#pragma unroll
            for (int qq = 0; qq < 16; ++qq) v[qq] = __uint_as_float(r[qq]);
            if (c0 + 32 < BN) tmem_ld16_nowait(dcol + (uint32_t)(c0 + 32), r);
            emit(v, Pp, c0, 0, 0);
            tmem_wait_ld();
          }
          asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar.dempty[d]);
          // Both groups' copies complete (their writes performed), then one
          // release add.
          if (issuer) {
            bulk_wait_all();
            asm volatile("fence.proxy.async.global;" ::: "memory");
          }
          named_sync(kBothBar, 256);
          if (leader) {
            red_release_gpu(tickets + 1, 1u);
            if (last) bar.pend[bar.npend++] = (uint32_t)t;
          }
        }
      }
    }
    // A shared tile whose last ticket this CTA took before its last segment:
    // every part (its own too) is in the slots now that the ring is idle.
    named_sync(kBothBar, 256);
    const int npend = (int)bar.npend;
    for (int pi = 0; pi < npend; ++pi) sum_tile((int)bar.pend[pi], 0xFFFFFFFFu);
    if (issuer) bulk_wait_all();  // every store has been performed before the CTA exits
  }

  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncwarp();  // every lane of the warp arrives at the barrier (lanes of a role warp finish at different times)
  __syncthreads();
  if (bar.err != 0 && threadIdx.x == 0) {
    // A wait gave up: let the copies that may still be in flight land
    // (bounded: the last copy issued into each slot) before the CTA exits,
    // and report it.
    const int nb = (int)bar.issued_b, nw = (int)bar.issued_w;
    for (int j = nb - kStages < 0 ? 0 : nb - kStages; j < nb; ++j)
      mbar_wait(&bar.full[j % kStages], (j / kStages) & 1, &bar.err, a.wait_cycles);
    for (int j = nw - kWSlots < 0 ? 0 : nw - kWSlots; j < nw; ++j)
      mbar_wait(&bar.full_w[j % kWSlots], (j / kWSlots) & 1, &bar.err, a.wait_cycles);
    atomicOr(a.status, kStatusTimeout);
  }
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

// cuTensorMapEncodeTiled, looked up once through the runtime (no link
// dependency on the driver library).
// (A function-local static: initialised once, safe under concurrent callers.)
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
  return fn;
}

// Tensor map of an FP16 [rows][ld] activation matrix with `cols` valid
// columns: boxes of 64 columns x bn rows, 128-byte swizzle, zero fill
// outside the matrix.
cudaError_t make_act_map(CUtensorMap* map, const __half* base, int64_t rows, int64_t cols, int64_t ld, int bn) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return cudaErrorNotSupported;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * 2)};
  cuuint32_t box[2] = {(cuuint32_t)BOX, (cuuint32_t)bn};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Token tile of a pass of T tokens.
int prefill_bn(int64_t T) { return T <= 16 ? 16 : T <= 32 ? 32 : T <= 64 ? 64 : T <= 128 ? 128 : 256; }

// Grid of one GEMM. Without room for partial tiles: one CTA per tile.
// Otherwise the grid (at most one CTA per SM) that minimises a CTA's modelled
// time: its stages, a fixed cost (pipeline fill, epilogue) and, when tiles
// are shared, the summing CTA's read of the other parts (its slowest step:
// about 20 bytes per cycle measured). Filling every SM regardless spread
// the 8 row-block tiles of a 1024 x 8192 layer over 8 CTAs each and the
// sums took longer than the stages (64 tokens: 26 -> 37 us).
int prefill_grid(const SignMatrix& sm, int64_t T, int num_sms, bool split) {
  const int64_t bn = prefill_bn(T);
  const int64_t tiles = (int64_t)sm.RB * ((T + bn - 1) / bn);
  if (!split) return (int)tiles;
  const int64_t bkk = bk_of((int)bn);
  const int64_t nk = (sm.C + bkk - 1) / bkk;
  const int64_t iters = tiles * nk;
  const double t_stage = (double)(bkk / 16) * 134.0 + 150.0;  // cycles: MMAs, barrier check, commit
  const double t_fixed = 4000.0 + 45.0 * (double)bn;           // fill, epilogue of a tile
  const double part_cycles = (double)bn * BM * 4 / 20.0;       // reading one partial tile
  // The summing CTA copies 16 tokens of every part into its activation ring.
  const int64_t ring = landing_bytes_of((int)bn);
  const int64_t max_parts = ring / (16 * BM * 4);
  int64_t best_g = 1;
  double best = 1e300;
  for (int64_t g = 1; g <= num_sms && g <= iters; ++g) {
    const int64_t per = (iters + g - 1) / g;  // stages of the busiest CTA
    int64_t parts = 1;                        // CTAs sharing one tile (at most)
    if (per % nk != 0 || (iters % g) != 0) parts = per >= nk ? 2 : (nk + per - 1) / per + 1;
    if (parts > max_parts) continue;
    const double cost =
        (double)per * t_stage + t_fixed + (parts > 1 ? 3000.0 + (double)(parts - 1) * part_cycles : 0.0);
    if (cost < best * 0.995) {  // prefer fewer CTAs on ties
      best = cost;
      best_g = g;
    }
  }
  return (int)best_g;
}

// Tensor map of the output [tokens][ld] (FP16 or FP32) with `rows` valid
// columns: boxes of 128 columns x box_tokens tokens, no swizzle; stores past the
// matrix are dropped.
cudaError_t make_out_map(CUtensorMap* map, void* base, int64_t tokens, int64_t rows, int64_t ld, bool f32,
                         int box_tokens) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return cudaErrorNotSupported;
  const int64_t es = f32 ? 4 : 2;
  cuuint64_t dims[2] = {(cuuint64_t)rows, (cuuint64_t)tokens};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * es)};
  cuuint32_t box[2] = {(cuuint32_t)BM, (cuuint32_t)box_tokens};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, base, dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <bool GEMM1, int BN>
cudaError_t launch_gemm_bn(const PrefillArgs& a, const __half* act, int64_t ld_act, int grid, cudaStream_t st) {
  CUtensorMap map, omap, omap32;
  cudaError_t e = make_act_map(&map, act, a.tokens, a.sm.C, ld_act, BN);
  if (e != cudaSuccess) return e;
  std::memset(&omap, 0, sizeof(omap));
  std::memset(&omap32, 0, sizeof(omap32));
  if (a.out_vec) {
    e = make_out_map(&omap, a.out, a.tokens, a.sm.R, a.ld_out, a.out_f32 != 0, 16);
    if (e == cudaSuccess && !a.out_f32) e = make_out_map(&omap32, a.out, a.tokens, a.sm.R, a.ld_out, false, 32);
    if (e != cudaSuccess) return e;
  }
  auto kern = prefill_kernel<GEMM1, BN>;
  constexpr int smem = smem_bytes<BN>();
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, map, omap, omap32, a);
}

template <bool GEMM1>
cudaError_t launch_gemm(const PrefillArgs& a, const __half* act, int64_t ld_act, int num_sms, cudaStream_t st) {
  const int grid = prefill_grid(a.sm, a.tokens, num_sms, a.part != nullptr);
  switch (prefill_bn(a.tokens)) {
    case 16: return launch_gemm_bn<GEMM1, 16>(a, act, ld_act, grid, st);
    case 32: return launch_gemm_bn<GEMM1, 32>(a, act, ld_act, grid, st);
    case 64: return launch_gemm_bn<GEMM1, 64>(a, act, ld_act, grid, st);
    case 128: return launch_gemm_bn<GEMM1, 128>(a, act, ld_act, grid, st);
    default: return launch_gemm_bn<GEMM1, 256>(a, act, ld_act, grid, st);
  }
}

}  // namespace

int64_t prefill_h_ld(const af1_layer& L) { return (L.r + 7) / 8 * 8; }

int64_t prefill_part_bytes(const af1_layer& L, int64_t tokens) {
  const int64_t T = tokens < kPrefillPassTokens ? tokens : kPrefillPassTokens;
  return (int64_t)2 * L.num_sms * prefill_bn(T) * BM * 4;
}

int64_t prefill_count_bytes(const af1_layer& L, int64_t tokens) {
  const int64_t T = tokens < kPrefillPassTokens ? tokens : kPrefillPassTokens;
  const int64_t nt = (T + prefill_bn(T) - 1) / prefill_bn(T);
  const int64_t rb = L.p1.RB > L.p2.RB ? L.p1.RB : L.p2.RB;
  return rb * nt * 8;
}

cudaError_t launch_prefill(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y, int64_t ldy,
                           int y_dtype, uint8_t* h_buf, float* part, unsigned* count, unsigned* status,
                           cudaStream_t st) {
  const int64_t ldh = prefill_h_ld(L);
  const int ysize = y_dtype == 0 ? 2 : 4;
  for (int64_t t0 = 0; t0 < tokens; t0 += kPrefillPassTokens) {
    const int T = (int)((tokens - t0) < kPrefillPassTokens ? (tokens - t0) : kPrefillPassTokens);
    PrefillArgs g1 = {};
    g1.signs = reinterpret_cast<const uint32_t*>(L.signs1);
    g1.sm = L.p1;
    g1.tokens = T;
    g1.colscale = reinterpret_cast<const __half*>(L.b);
    g1.rowscale = reinterpret_cast<const __half*>(L.s);
    g1.out = h_buf;
    g1.ld_out = ldh;
    g1.out_f32 = 0;
    g1.out_vec = ((uintptr_t)h_buf % 16 == 0 && (ldh * 2) % 16 == 0) ? 1 : 0;
    g1.part = part;
    g1.count = count;
    g1.status = status;
    g1.wait_cycles = wait_budget();
    cudaError_t e = launch_gemm<true>(g1, static_cast<const __half*>(x) + t0 * ldx, ldx, L.num_sms, st);
    if (e != cudaSuccess) return e;
    PrefillArgs g2 = g1;
    g2.signs = reinterpret_cast<const uint32_t*>(L.signs2);
    g2.sm = L.p2;
    g2.colscale = nullptr;
    g2.rowscale = reinterpret_cast<const __half*>(L.a);
    g2.out = static_cast<uint8_t*>(y) + t0 * ldy * ysize;
    g2.ld_out = ldy;
    g2.out_f32 = y_dtype == 0 ? 0 : 1;
    g2.out_vec = ((uintptr_t)g2.out % 16 == 0 && (ldy * ysize) % 16 == 0) ? 1 : 0;
    e = launch_gemm<false>(g2, reinterpret_cast<const __half*>(h_buf), ldh, L.num_sms, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace af1
