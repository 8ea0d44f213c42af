// af1_prefill.cu — prefill path (more than 16 tokens): the two sign-matrix
// products of AF1 Eq. final_reconstruction as dense GEMMs on the sm_103a
// tensor cores (tcgen05), with the 1-bit factors expanded on the fly.
//
//   GEMM1: H[t][k] = s_k * sum_j B[k][j] * (b_j x[t][j])    (B = V^T, r x n)
//   GEMM2: y[t][i] = a_i * sum_k U[i][k] * H[t][k]          (U, m x r)
//
// A CTA computes D = A . B^T for 128 features x BN tokens (BN = 64, 128 or
// 256), D in tensor memory (128 lanes x BN FP32 columns). Per K-stage of 64:
//   * one thread of warp 0 loads the BN x 64 FP16 activation tile (B) with
//     one TMA copy (cp.async.bulk.tensor, 128-byte swizzle, zero fill past
//     the tokens / columns): the K-major layout the MMA descriptor describes;
//   * warps 4-7 (one feature row per thread = tensor-memory lane) expand the
//     packed signs of the 128 x 64 weight tile into FP16 (+-b_j for GEMM1,
//     +-1 for GEMM2: exact) and store them into a ring of A buffers in
//     tensor memory (tcgen05.st, 32 columns per stage); each thread loads
//     the next stage's sign words (and column scales) while it expands the
//     current one. A in tensor memory leaves shared-memory bandwidth to B
//     (measured: 848 vs 735 TFLOP/s with A in shared memory);
//   * one thread of warp 1 issues four tcgen05.mma.kind::f16 (K = 16 each,
//     N = BN, A from tensor memory, B from shared memory) and commits them to
//     the stage's "empty" mbarrier.
// Warps 4-7 then read D back with tcgen05.ld (warp w owns TMEM lanes
// 32 (w % 4) .. +31), apply the per-feature scale and store FP16 / FP32.
// All mbarrier waits are bounded; a wait that gives up sets the status word.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1_internal.h"
#include "af1_layout.h"
#include "af1_ptx.cuh"

namespace af1 {
namespace {

constexpr int BM = 128;  // features per CTA (MMA M, TMEM lanes)
constexpr int BK = 64;   // K per stage: one 128-byte swizzle row of FP16
constexpr int kMaxStages = 6;
constexpr int kThreads = 256;

template <int BN>
__host__ __device__ constexpr int tile_b_bytes() {
  return BN * BK * 2;
}
// Pipeline depth: 6 stages for tiles of 256 tokens (192 KB of activation
// tiles; tensor memory holds D in 256 columns plus an A ring of 6 x 32), 4
// for the smaller tiles.
template <int BN>
__host__ __device__ constexpr int stages() {
  return BN == 256 ? 6 : 4;
}
template <int BN>
__host__ __device__ constexpr int smem_bytes() {
  return stages<BN>() * tile_b_bytes<BN>() + 1024 /* barriers */ + 1024 /* base alignment */;
}

struct PrefillArgs {
  const uint32_t* signs;  // packed signs, af1_layout.h row-block layout
  SignMatrix sm;          // R = features, C = K
  int tokens;
  const __half* colscale;  // GEMM1: b (length C); GEMM2: nullptr (+-1)
  const __half* rowscale;  // GEMM1: s (length R); GEMM2: a
  void* out;               // GEMM1: H [tokens][ld_out] FP16; GEMM2: y
  int64_t ld_out;
  int out_f32;
  unsigned* status;
  long long wait_cycles;  // budget of every bounded wait (clock64 cycles)
};

struct __align__(8) PrefillBarriers {
  uint64_t full_a[kMaxStages];  // the 4 expander warps have stored the stage's A
  uint64_t full_b[kMaxStages];  // the TMA tile has landed
  uint64_t empty[kMaxStages];   // the stage's MMAs are done
  uint64_t done;
  uint32_t tmem_addr;
  uint32_t err;
};

__device__ __forceinline__ void tmem_ld16(uint32_t addr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(addr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Cluster helper for the split-K reduction.
__device__ __forceinline__ void st_cluster_f32(float* local, uint32_t rank, float v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(v) : "memory");
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
// Tensor-memory columns: D (BN) then the A ring (stages x 32), rounded up
// to a power of two.
template <int BN>
__host__ __device__ constexpr uint32_t tmem_cols() {
  return (BN + stages<BN>() * 32) <= 256 ? 256u : 512u;
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

// Column scales of stage columns kc .. kc + 63 as 8 groups of 8 FP16
// values, 0 beyond C.
__device__ __forceinline__ void load_colscale(const __half* cs, int64_t kc, int64_t C, uint4 (&out)[8]) {
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int64_t k = kc + 8 * j;
    if (k + 7 < C) {
      out[j] = __ldg(reinterpret_cast<const uint4*>(cs + k));
    } else {
      const uint16_t* c16 = reinterpret_cast<const uint16_t*>(cs);
      uint32_t e[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) e[q] = k + q < C ? c16[k + q] : 0u;
      out[j] = make_uint4(e[0] | (e[1] << 16), e[2] | (e[3] << 16), e[4] | (e[5] << 16), e[6] | (e[7] << 16));
    }
  }
}

// KS > 1: split-K over a cluster of KS CTAs along z. CTA ks runs the stages
// [ks spk, (ks + 1) spk) and the partial tiles are summed through
// distributed shared memory (each CTA finalises 128 / KS rows, summing the
// KS partials in a fixed order), reusing the activation stages as the
// receive buffer once every MMA of the cluster is done.
template <bool GEMM1, int BN, int KS>
__global__ void __launch_bounds__(kThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap act_map, const PrefillArgs a) {
  constexpr int kTileB = tile_b_bytes<BN>();
  constexpr int STAGES = stages<BN>();
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the swizzled operand tiles.
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tileB = smem;
  PrefillBarriers& bar = *reinterpret_cast<PrefillBarriers*>(smem + STAGES * kTileB);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const SignMatrix& tm = a.sm;
  const int f0 = blockIdx.x * BM;  // first feature (row of the sign matrix)
  const int t0 = blockIdx.y * BN;  // first token
  const int nk_all = (int)((tm.C + BK - 1) / BK);
  const int ks = KS > 1 ? (int)blockIdx.z : 0;
  const int spk = (nk_all + KS - 1) / KS;  // stages per CTA (>= 1 for every ks, by the host plan)
  const int it0 = ks * spk;
  const int nk = min(nk_all, it0 + spk) - it0;  // this CTA's stages: it0 .. it0 + nk - 1

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&bar.full_a[s], 4);
      mbar_init(&bar.full_b[s], 1);
      mbar_init(&bar.empty[s], 1);
    }
    mbar_init(&bar.done, 1);
    bar.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&act_map)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&bar.tmem_addr)),
                 "r"(tmem_cols<BN>())
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = bar.tmem_addr;

  if (warp == 0) {
    // ---- activation producer: one TMA copy per stage ---------------------
    griddep_wait();  // the activations are written by the previous kernel
    if (lane == 0) {
      for (int it = 0; it < nk; ++it) {
        const int s = it % STAGES;
        if (it >= STAGES) mbar_wait(&bar.empty[s], ((it / STAGES) & 1) ^ 1, &bar.err, a.wait_cycles);
        mbar_expect_tx(&bar.full_b[s], (uint32_t)kTileB);
        tma_load_2d(tileB + s * kTileB, &act_map, (it0 + it) * BK, t0, &bar.full_b[s]);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA issuer ---------------------------------------------------------
    if (lane == 0) {
      const uint32_t b0 = smem_u32(tileB);
      for (int it = 0; it < nk; ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        mbar_wait(&bar.full_a[s], ph, &bar.err, a.wait_cycles);
        mbar_wait(&bar.full_b[s], ph, &bar.err, a.wait_cycles);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          mma_f16_ts<BN>(tmem, tmem + (uint32_t)(BN + s * 32 + kk * 8), smem_desc(b0 + s * kTileB + kk * 32),
                         it > 0 || kk > 0);
        }
        mma_commit(&bar.empty[s]);
      }
      mma_commit(&bar.done);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---- weight expansion: one feature row per thread --------------------
    const int R = threadIdx.x - 128;  // 0..127 = TMEM lane of this thread
    const int64_t frow = f0 + R;
    const bool row_ok = frow < tm.R;
    // Words of this row: index (rb * 4 NCH + kw) * 128 + R (rows past R are
    // zero words of the padded block). Stage `it` uses words 2 it and
    // 2 it + 1; the next stage's words are loaded while the current stage is
    // expanded.
    const uint32_t* rowp =
        a.signs + (int64_t)blockIdx.x * tm.NCH * kChunkWords * kBlockRows + R + (int64_t)(2 * it0) * kBlockRows;
    uint32_t w0 = __ldg(rowp), w1 = __ldg(rowp + kBlockRows);
    uint4 cs[8];
    if (GEMM1) load_colscale(a.colscale, (int64_t)it0 * BK, tm.C, cs);
    for (int it = 0; it < nk; ++it) {
      const int s = it % STAGES;
      uint32_t n0 = 0u, n1 = 0u;
      uint4 ncs[8];
      if (it + 1 < nk) {
        n0 = __ldg(rowp + (int64_t)(2 * it + 2) * kBlockRows);
        n1 = __ldg(rowp + (int64_t)(2 * it + 3) * kBlockRows);
        if (GEMM1) load_colscale(a.colscale, (int64_t)(it0 + it + 1) * BK, tm.C, ncs);
      }
      uint32_t av[32];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        // Stage columns 8j .. 8j+7 (tensor-memory columns 4j .. 4j+3, two
        // FP16 values each) = columns 4p + e of word j / 4 with p = 2 (j % 4)
        // (first 4) and p + 1 (last 4).
        const uint32_t wd = (j < 4) ? w0 : w1;
        const int p = 2 * (j & 3);
        const uint32_t b01 = __byte_perm(wd, 0u, 0x1404);  // bytes 0,1 -> bytes 1,3 (e = 0, 1)
        const uint32_t b23 = __byte_perm(wd, 0u, 0x3424);  // bytes 2,3 -> bytes 1,3 (e = 2, 3)
        uint4 sv = make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);  // +-1 for GEMM2
        if (GEMM1) sv = cs[j];
        av[4 * j + 0] = signed_pair(b01, p, sv.x);
        av[4 * j + 1] = signed_pair(b23, p, sv.y);
        av[4 * j + 2] = signed_pair(b01, p + 1, sv.z);
        av[4 * j + 3] = signed_pair(b23, p + 1, sv.w);
      }
      // The previous stage's store was left in flight while this stage was
      // expanded: complete it and hand that stage to the MMA issuer.
      if (it > 0) {
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar.full_a[(it - 1) % STAGES]);
      }
      if (it >= STAGES) {
        if (lane == 0) mbar_wait(&bar.empty[s], ((it / STAGES) & 1) ^ 1, &bar.err, a.wait_cycles);
        __syncwarp();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      }
      {
        const uint32_t addr = tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(BN + s * 32);
        asm volatile(
            "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
            "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(addr),
            "r"(av[0]), "r"(av[1]), "r"(av[2]), "r"(av[3]), "r"(av[4]), "r"(av[5]), "r"(av[6]), "r"(av[7]),
            "r"(av[8]), "r"(av[9]), "r"(av[10]), "r"(av[11]), "r"(av[12]), "r"(av[13]), "r"(av[14]), "r"(av[15]),
            "r"(av[16]), "r"(av[17]), "r"(av[18]), "r"(av[19]), "r"(av[20]), "r"(av[21]), "r"(av[22]), "r"(av[23]),
            "r"(av[24]), "r"(av[25]), "r"(av[26]), "r"(av[27]), "r"(av[28]), "r"(av[29]), "r"(av[30]), "r"(av[31])
            : "memory");
      }
      w0 = n0;
      w1 = n1;
      if (GEMM1) {
#pragma unroll
        for (int j = 0; j < 8; ++j) cs[j] = ncs[j];
      }
    }
    if (nk > 0) {
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar.full_a[(nk - 1) % STAGES]);
    }
    // The next kernel may launch once this CTA has expanded its weights: its
    // own expansion needs no input and would otherwise compete with this
    // one's for the SMs. Measured against a trigger right after the
    // tensor-memory allocation: the 2048-token prefill step 4.18 -> 4.04 ms,
    // 64 tokens 4096^2 37.9 -> 31.3 us, 8192^2 56.7 -> 47.9, 1024 x 8192
    // 33.4 -> 26.2, 28672 x 8192 at 128 tokens 179 -> 127; only 28672 x 8192
    // at 64 tokens lost (95 -> 120), where GEMM 1 leaves SMs idle.
    griddep_launch_dependents();
    // ---- epilogue: TMEM -> registers -> global ---------------------------
    if (lane == 0) mbar_wait(&bar.done, 0, &bar.err, a.wait_cycles);
    __syncwarp();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (KS == 1) {
      griddep_wait();  // the output may still be read by the previous kernel until it completes
      const float rsc = row_ok ? __half2float(a.rowscale[frow]) : 0.f;
      const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + (uint32_t)c0, r);
        if (row_ok) {
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int64_t tok = t0 + c0 + q;
            if (tok < a.tokens) {
              const float v = __uint_as_float(r[q]) * rsc;
              if (a.out_f32)
                reinterpret_cast<float*>(a.out)[tok * a.ld_out + frow] = v;
              else
                reinterpret_cast<__half*>(a.out)[tok * a.ld_out + frow] = __float2half_rn(v);
            }
          }
        }
      }
    }
  }

  if (KS > 1) {
    // ---- split-K: partial tiles -> owning CTA through distributed shared
    //      memory. recv[q][i][c ^ (i & 31)] holds CTA q's partial of row i
    //      of this CTA's slice (XOR on the column keeps the row-wise reads of
    //      the final sum free of bank conflicts).
    constexpr int SLICE = BM / KS;
    float* recv = reinterpret_cast<float*>(tileB);  // KS * SLICE * BN floats = STAGES * kTileB bytes
    __syncwarp();
    cluster_sync();  // every MMA of the cluster is done: the activation stages are free
    if (warp >= 4) {
      const int R = threadIdx.x - 128;
      const int owner = R / SLICE, i = R - owner * SLICE;
      const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
      float* row = recv + (size_t)(ks * SLICE + i) * BN;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + (uint32_t)c0, r);
#pragma unroll
        for (int q = 0; q < 16; ++q) st_cluster_f32(row + ((c0 + q) ^ (i & 31)), (uint32_t)owner, __uint_as_float(r[q]));
      }
    }
    cluster_sync();  // all partials have landed
    griddep_wait();  // the output may still be read by the previous kernel until it completes
    for (int idx = threadIdx.x; idx < SLICE * BN; idx += kThreads) {
      const int c = idx / SLICE, i = idx - c * SLICE;  // token column c, slice row i
      const int64_t frow = f0 + ks * SLICE + i;
      const int64_t tok = t0 + c;
      if (frow >= tm.R || tok >= a.tokens) continue;
      float v = 0.f;
#pragma unroll
      for (int q = 0; q < KS; ++q) v += recv[(size_t)(q * SLICE + i) * BN + (c ^ (i & 31))];
      v *= __half2float(a.rowscale[frow]);
      if (a.out_f32)
        reinterpret_cast<float*>(a.out)[tok * a.ld_out + frow] = v;
      else
        reinterpret_cast<__half*>(a.out)[tok * a.ld_out + frow] = __float2half_rn(v);
    }
  }

  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (bar.err != 0 && threadIdx.x == 0) {
    // A wait gave up: let TMA copies that may still be in flight land
    // (bounded) before the CTA exits, and report it.
    for (int s = 0; s < STAGES; ++s) mbar_wait(&bar.full_b[s], 0, &bar.err, a.wait_cycles);
    atomicOr(a.status, kStatusTimeout);
  }
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_cols<BN>()) : "memory");
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
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)bn};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <bool GEMM1, int BN, int KS>
cudaError_t launch_gemm_bn(const PrefillArgs& a, const __half* act, int64_t ld_act, cudaStream_t st) {
  CUtensorMap map;
  cudaError_t e = make_act_map(&map, act, a.tokens, a.sm.C, ld_act, BN);
  if (e != cudaSuccess) return e;
  auto kern = prefill_kernel<GEMM1, BN, KS>;
  // A cluster's CTAs wait for each other while holding tensor memory, so no
  // third CTA may share an SM with two of them (one that blocks in
  // tcgen05.alloc would wait for a CTA that waits for it): with at least
  // 80 KB of shared memory per CTA, at most two CTAs fit on an SM and their
  // tensor memory (<= 256 columns each) always fits.
  constexpr int smem = (KS > 1 && smem_bytes<BN>() < 80 * 1024) ? 80 * 1024 : smem_bytes<BN>();
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.sm.RB, (unsigned)((a.tokens + BN - 1) / BN), (unsigned)KS);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = (unsigned)KS;
  cfg.attrs = attr;
  cfg.numAttrs = KS > 1 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kern, map, a);
}

// Tiling of one GEMM: the smallest token tile of 64 / 128 / 256 that covers
// the pass, made smaller while the grid would leave half the SMs idle; with
// tiles of 64, short passes (few row blocks x token tiles) split K over a
// cluster of 2, 4 or 8 CTAs (every CTA keeps at least two K-stages) while
// the grid fits one CTA per SM, or two per SM for contractions of 256
// K-stages or more (measured: 8192 x 28672 at 64 tokens 164 -> 108 us; the
// same on shorter contractions lost, e.g. 4096^2 31 -> 40 us).
template <bool GEMM1>
cudaError_t launch_gemm(const PrefillArgs& a, const __half* act, int64_t ld_act, int num_sms, cudaStream_t st) {
  const int64_t rb = a.sm.RB;
  int bn = a.tokens > 128 ? 256 : a.tokens > 64 ? 128 : 64;
  while (bn > 64 && rb * ((a.tokens + bn - 1) / bn) < num_sms / 2) bn /= 2;
  if (bn == 256) return launch_gemm_bn<GEMM1, 256, 1>(a, act, ld_act, st);
  if (bn == 128) return launch_gemm_bn<GEMM1, 128, 1>(a, act, ld_act, st);
  const int64_t base = rb * ((a.tokens + 63) / 64);
  const int nk = (int)((a.sm.C + BK - 1) / BK);
  int ks = 1;
  const int64_t room = nk >= 256 ? 2 * (int64_t)num_sms : (int64_t)num_sms;
  while (ks < 8 && base * ks * 2 <= room && nk >= 4 * ks) ks *= 2;
  // every CTA of the split needs at least one stage
  while (ks > 1 && (ks - 1) * ((nk + ks - 1) / ks) >= nk) ks /= 2;
  switch (ks) {
    case 8: return launch_gemm_bn<GEMM1, 64, 8>(a, act, ld_act, st);
    case 4: return launch_gemm_bn<GEMM1, 64, 4>(a, act, ld_act, st);
    case 2: return launch_gemm_bn<GEMM1, 64, 2>(a, act, ld_act, st);
    default: return launch_gemm_bn<GEMM1, 64, 1>(a, act, ld_act, st);
  }
}

}  // namespace

int64_t prefill_h_ld(const af1_layer& L) { return (L.r + 7) / 8 * 8; }

cudaError_t launch_prefill(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y, int64_t ldy,
                           int y_dtype, uint8_t* h_buf, unsigned* status, cudaStream_t st) {
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
    g1.status = status;
    g1.wait_cycles = wait_budget();
    cudaError_t e = launch_gemm<true>(g1, static_cast<const __half*>(x) + t0 * ldx, ldx, L.num_sms, st);
    if (e != cudaSuccess) return e;
    PrefillArgs g2 = {};
    g2.signs = reinterpret_cast<const uint32_t*>(L.signs2);
    g2.sm = L.p2;
    g2.tokens = T;
    g2.colscale = nullptr;
    g2.rowscale = reinterpret_cast<const __half*>(L.a);
    g2.out = static_cast<uint8_t*>(y) + t0 * ldy * ysize;
    g2.ld_out = ldy;
    g2.out_f32 = y_dtype == 0 ? 0 : 1;
    g2.status = status;
    g2.wait_cycles = g1.wait_cycles;
    e = launch_gemm<false>(g2, reinterpret_cast<const __half*>(h_buf), ldh, L.num_sms, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace af1
