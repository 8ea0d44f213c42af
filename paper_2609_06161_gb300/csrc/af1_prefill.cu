// af1_prefill.cu — prefill path (more than 16 tokens): the two sign-matrix
// products of AF1 Eq. final_reconstruction as dense GEMMs on the sm_103a
// tensor cores (tcgen05), with the 1-bit factors expanded on the fly.
//
//   GEMM1: H[t][k] = s_k * sum_j B[k][j] * (b_j x[t][j])    (B = V^T, r x n)
//   GEMM2: y[t][i] = a_i * sum_k U[i][k] * H[t][k]          (U, m x r)
//
// A CTA computes D = A . B^T for 128 features x 128 tokens, D in tensor
// memory (128 lanes x 128 FP32 columns). Per K-stage of 64:
//   * warp 0 copies the 128 x 64 FP16 activation tile with cp.async into the
//     128-byte-swizzled K-major layout the MMA descriptor describes;
//   * warps 4-7 (one feature row per thread) expand the packed signs of the
//     128 x 64 weight tile into FP16 (+-b_j for GEMM1, +-1 for GEMM2: exact)
//     in the same layout;
//   * warp 1 (one lane) issues four tcgen05.mma.kind::f16 (K = 16 each) and
//     commits them to the stage's "empty" mbarrier.
// Warps 4-7 then read D back with tcgen05.ld (warp w owns TMEM lanes
// 32 (w % 4) .. +31), apply the per-feature scale and store FP16 / FP32.
// All mbarrier waits are bounded; a wait that gives up sets the status word.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1_internal.h"
#include "af1_layout.h"

namespace af1 {
namespace {

constexpr int BM = 128;  // features per CTA (MMA M, TMEM lanes)
constexpr int BN = 128;  // tokens per CTA (MMA N, TMEM columns)
constexpr int BK = 64;   // K per stage: one 128-byte swizzle row of FP16
constexpr int STAGES = 4;
constexpr int kThreads = 256;
constexpr int kTileA = BM * BK * 2;  // 16 KB
constexpr int kTileB = BN * BK * 2;  // 16 KB
constexpr long long kWaitCycles = 2000000000ll;
constexpr unsigned kStatusTimeout = 1u;

struct PrefillArgs {
  const uint32_t* signs;  // packed signs, af1_layout.h row-block layout
  SignMatrix sm;          // R = features, C = K
  const __half* act;      // B operand source: [tokens][ld_act] FP16
  int64_t ld_act;
  int tokens;
  const __half* colscale;  // GEMM1: b (length C); GEMM2: nullptr (+-1)
  const __half* rowscale;  // GEMM1: s (length R); GEMM2: a
  void* out;               // GEMM1: H [tokens][ld_out] FP16; GEMM2: y
  int64_t ld_out;
  int out_f32;
  unsigned* status;
};

struct __align__(8) PrefillBarriers {
  uint64_t full_a[STAGES];
  uint64_t full_b[STAGES];
  uint64_t empty[STAGES];
  uint64_t done;
  uint32_t tmem_addr;
  uint32_t err;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}
// Bounded wait; on timeout records the error in the CTA flag and returns.
__device__ __forceinline__ void mbar_wait(uint64_t* bar, uint32_t parity, uint32_t* err) {
  if (mbar_try_wait(bar, parity)) return;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) {
      atomicOr(err, 1u);
      return;
    }
  }
}

__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// 16-byte cp.async with zero fill beyond `src_bytes`.
__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);        // start address
  d |= (uint64_t)1u << 16;                      // leading byte offset (unused for this layout)
  d |= (uint64_t)(1024u >> 4) << 32;            // stride byte offset
  d |= (uint64_t)1u << 46;                      // version
  d |= (uint64_t)2u << 61;                      // 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: D F32, A and B F16, both K-major,
// N = BN, M = BM.
constexpr uint32_t kIdesc = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, bool accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate ? 1u : 0u)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// Byte offset of the 16-byte chunk `j` (0..7) of row `r` in a 128-byte
// swizzled K-major tile.
__device__ __forceinline__ uint32_t swz(int r, int j) { return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4)); }

// Sign bit (bit `p` of bytes b0 and b1 of the selected pair) -> the sign
// positions 15 and 31 of an FP16 pair, then value = +-v (bit 1 keeps v).
__device__ __forceinline__ uint32_t signed_pair(uint32_t pair_bytes, int p, uint32_t v) {
  const uint32_t sh = pair_bytes << (7 - p);
  return v ^ (~sh & 0x80008000u);
}

template <bool GEMM1>
__global__ void __launch_bounds__(kThreads, 1) prefill_kernel(const PrefillArgs a) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the swizzled operand tiles.
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tileA = smem;
  uint8_t* tileB = smem + STAGES * kTileA;
  PrefillBarriers& bar = *reinterpret_cast<PrefillBarriers*>(smem + STAGES * (kTileA + kTileB));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const SignMatrix& tm = a.sm;
  const int f0 = blockIdx.x * BM;  // first feature (row of the sign matrix)
  const int t0 = blockIdx.y * BN;  // first token
  const int nk = (int)((tm.C + BK - 1) / BK);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&bar.full_a[s], 4);
      mbar_init(&bar.full_b[s], 1);
      mbar_init(&bar.empty[s], 1);
    }
    mbar_init(&bar.done, 1);
    bar.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&bar.tmem_addr)),
                 "r"((uint32_t)BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = bar.tmem_addr;

  griddep_launch_dependents();
  griddep_wait();

  if (warp == 0) {
    // ---- activation producer: cp.async into the swizzled B tiles -------
    constexpr int LAG = 2;
    for (int it = 0; it < nk; ++it) {
      const int s = it % STAGES;
      if (it >= STAGES) mbar_wait(&bar.empty[s], ((it / STAGES) & 1) ^ 1, &bar.err);
      uint8_t* dst = tileB + s * kTileB;
      const int64_t k0 = (int64_t)it * BK;
      for (int q = lane; q < BN * 8; q += 32) {
        const int r = q >> 3, j = q & 7;
        const int64_t tok = t0 + r;
        const int64_t k = k0 + j * 8;
        uint32_t bytes = 0;
        const __half* src = a.act;
        if (tok < a.tokens && k < tm.C) {
          const int64_t left = tm.C - k;
          bytes = left >= 8 ? 16u : (uint32_t)(left * 2);
          src = a.act + tok * a.ld_act + k;
        }
        cp_async16(dst + swz(r, j), src, bytes);
      }
      cp_async_commit();
      if (it >= LAG) {
        cp_async_wait<LAG>();
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar.full_b[(it - LAG) % STAGES]);
      }
    }
    cp_async_wait<0>();
    fence_proxy_async();
    __syncwarp();
    if (lane == 0)
      for (int it = nk - LAG < 0 ? 0 : nk - LAG; it < nk; ++it) mbar_arrive(&bar.full_b[it % STAGES]);
  } else if (warp == 1) {
    // ---- MMA issuer ---------------------------------------------------------
    if (lane == 0) {
      const uint32_t a0 = smem_u32(tileA), b0 = smem_u32(tileB);
      for (int it = 0; it < nk; ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        mbar_wait(&bar.full_a[s], ph, &bar.err);
        mbar_wait(&bar.full_b[s], ph, &bar.err);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          mma_f16(tmem, smem_desc(a0 + s * kTileA + kk * 32), smem_desc(b0 + s * kTileB + kk * 32), it > 0 || kk > 0);
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
    // zero words of the padded block).
    const uint32_t* rowp = a.signs + (int64_t)blockIdx.x * tm.NCH * kChunkWords * kBlockRows + R;
    for (int it = 0; it < nk; ++it) {
      const int s = it % STAGES;
      if (it >= STAGES) mbar_wait(&bar.empty[s], ((it / STAGES) & 1) ^ 1, &bar.err);
      // Stage columns 64 it .. 64 it + 63 = words 2 it and 2 it + 1.
      const uint32_t w0 = __ldg(rowp + (int64_t)(2 * it) * kBlockRows);
      const uint32_t w1 = __ldg(rowp + (int64_t)(2 * it + 1) * kBlockRows);
      uint8_t* dst = tileA + s * kTileA;
      const int64_t k0 = (int64_t)it * BK;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        // 16-byte chunk j = stage columns 8j .. 8j+7 = columns 4p + e of word
        // j / 4 with p = 2 (j % 4) (first 4) and p + 1 (last 4).
        const uint32_t wd = (j < 4) ? w0 : w1;
        const int p = 2 * (j & 3);
        const uint32_t b01 = __byte_perm(wd, 0u, 0x1404);  // bytes 0,1 -> bytes 1,3 (e = 0, 1)
        const uint32_t b23 = __byte_perm(wd, 0u, 0x3424);  // bytes 2,3 -> bytes 1,3 (e = 2, 3)
        uint32_t sv[4] = {0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u};  // +-1 for GEMM2
        if (GEMM1) {
          const int64_t kc = k0 + j * 8;
          if (kc + 7 < tm.C) {
            const uint4 bb = __ldg(reinterpret_cast<const uint4*>(a.colscale + kc));
            sv[0] = bb.x;
            sv[1] = bb.y;
            sv[2] = bb.z;
            sv[3] = bb.w;
          } else {
            const uint16_t* cs = reinterpret_cast<const uint16_t*>(a.colscale);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint32_t e0 = kc + 2 * q < tm.C ? cs[kc + 2 * q] : 0u;
              const uint32_t e1 = kc + 2 * q + 1 < tm.C ? cs[kc + 2 * q + 1] : 0u;
              sv[q] = e0 | (e1 << 16);
            }
          }
        }
        uint4 v;
        v.x = signed_pair(b01, p, sv[0]);
        v.y = signed_pair(b23, p, sv[1]);
        v.z = signed_pair(b01, p + 1, sv[2]);
        v.w = signed_pair(b23, p + 1, sv[3]);
        *reinterpret_cast<uint4*>(dst + swz(R, j)) = v;
      }
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar.full_a[s]);
    }
    // ---- epilogue: TMEM -> registers -> global ---------------------------
    mbar_wait(&bar.done, 0, &bar.err);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const float rsc = row_ok ? __half2float(a.rowscale[frow]) : 0.f;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      uint32_t r[16];
      asm volatile(
          "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
          : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
            "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
          : "r"(tmem + lane_base + (uint32_t)c0));
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
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

  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (bar.err != 0 && threadIdx.x == 0) atomicOr(a.status, kStatusTimeout);
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)BN) : "memory");
  }
}

constexpr int kSmemBytes = STAGES * (kTileA + kTileB) + (int)sizeof(PrefillBarriers) + 1024;

template <bool GEMM1>
cudaError_t launch_gemm(const PrefillArgs& a, cudaStream_t st) {
  auto kern = prefill_kernel<GEMM1>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.sm.RB, (unsigned)((a.tokens + BN - 1) / BN), 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
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
    g1.act = static_cast<const __half*>(x) + t0 * ldx;
    g1.ld_act = ldx;
    g1.tokens = T;
    g1.colscale = reinterpret_cast<const __half*>(L.b);
    g1.rowscale = reinterpret_cast<const __half*>(L.s);
    g1.out = h_buf;
    g1.ld_out = ldh;
    g1.out_f32 = 0;
    g1.status = status;
    cudaError_t e = launch_gemm<true>(g1, st);
    if (e != cudaSuccess) return e;
    PrefillArgs g2 = {};
    g2.signs = reinterpret_cast<const uint32_t*>(L.signs2);
    g2.sm = L.p2;
    g2.act = reinterpret_cast<const __half*>(h_buf);
    g2.ld_act = ldh;
    g2.tokens = T;
    g2.colscale = nullptr;
    g2.rowscale = reinterpret_cast<const __half*>(L.a);
    g2.out = static_cast<uint8_t*>(y) + t0 * ldy * ysize;
    g2.ld_out = ldy;
    g2.out_f32 = y_dtype == 0 ? 0 : 1;
    g2.status = status;
    e = launch_gemm<false>(g2, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace af1
