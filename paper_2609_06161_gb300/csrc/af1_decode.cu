// af1_decode.cu — decode path (1..16 tokens per pass) of the forward pass of
// an AF1 binary-factorized linear layer on sm_103a:
//     y = a * (U (s * (V^T (b * x)))),
// the right-to-left evaluation of AF1 Eq. final_reconstruction /
// Eq. double_factor_equiv that never forms the dense W_hat.
//
// Two kernels per pass, chained with programmatic dependent launch (PDL):
//   phase 1: t = B z with B = V^T (r x n) and z = b * x; s' = s * t is
//            written as FP32 to the workspace;
//   phase 2: u = U s' (m x r); y = a * u, stored as FP16 or FP32.
// A phase is an R x C sign matrix (af1_layout.h) times T <= 16 vectors.
// CTA (rb, ks) owns row block rb (128 rows: the M of one tcgen05 MMA) and
// the ks-th slice of CPC column chunks; the KS CTAs of a row block form one
// thread-block cluster and reduce their partial sums through distributed
// shared memory, each CTA finalising 1/KS of the rows by summing the KS
// partials in a fixed order (deterministic, no global atomics).
//
// Inside a CTA (256 threads):
//   * one thread starts bulk copies (cp.async.bulk) of the CTA's packed
//     chunks, 2 KB each, before anything else;
//   * warps 0-3 (thread i = matrix row i = tensor-memory lane i) expand every
//     chunk into e4m3 A values in tensor memory (tcgen05.st) through a ring
//     of A buffers. The signs do not depend on the previous kernel, so this
//     runs while it is still finishing;
//   * warps 4-7 wait for the previous kernel (griddepcontrol.wait), read the
//     CTA's activations and write the B operand (e4m3, N = 16/32/64 rows =
//     4 terms x tokens) to shared memory in the 128-byte-swizzled K-major
//     layout of the MMA descriptor;
//   * lane 0 of warps 4..4+NACC-1 issue the MMAs (tcgen05.mma kind::f8f6f4,
//     A from tensor memory, B from shared memory), each into its own
//     accumulator: one issuing thread sustains about one MMA per 93 cycles
//     whatever N is, so NACC independent issuers multiply the rate;
//   * warps 0-3 read the accumulators back (tcgen05.ld), add terms and
//     accumulators, apply the sign correction and the activation scale and
//     push the partial sums to the cluster CTA that owns each row.
//
// Sign arithmetic. A sign bit becomes an e4m3 byte with one LOP3 per 4 signs:
// (word & mask_p) | base_p puts the bit at a fixed position p of a constant
// byte, giving A = L_p + d_p * bit with L_p, d_p powers of two (mantissa bits,
// exponent bit 0 or the sign bit). With z'_k = z_k / d_k the MMA yields
// D = sum_k L_k z'_k + sum_k bit_k z_k, and since sign = 2 bit - 1,
//     sum_k sign_k z_k = 2 D - Q,   Q = sum_k (L_k + H_k) z'_k  (H = L + d).
// Each z'_k is scaled by a per-(CTA, token) power of two 2^sigma that puts
// the largest magnitude in [128, 256), and split into 4 e4m3 terms
// (z' ~ t1 + t2 + t3 + t4, about 16 significant bits) that occupy 4 of the N
// rows of B. Products are exact and the MMA accumulates in FP32.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1.h"
#include "af1_internal.h"
#include "af1_layout.h"
#include "af1_ptx.cuh"

namespace af1 {
namespace {

constexpr int kThreads = 256;
constexpr int kTmemCols = 256;        // per CTA: two CTAs fit on one SM
constexpr int kMaxCPC = 64;           // column chunks per CTA (one mbarrier each)
constexpr int kMaxKS = 16;            // CTAs per cluster
constexpr int kMinSmem = 80 * 1024;   // at most two CTAs per SM: their tensor memory always fits

// ---------------------------------------------------------------------------
// PTX helpers (hand-written: mbarrier, bulk copy, PDL, cluster, tcgen05, FP8)
// ---------------------------------------------------------------------------

__device__ __forceinline__ void st_cluster_f32(float* local, uint32_t rank, float v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(v) : "memory");
}
// Named barrier of the four builder warps (4..7).
__device__ __forceinline__ void builders_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

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
// D (FP32, tensor memory) [+]= A (e4m3, tensor memory) x B (e4m3, shared
// memory)^T, M = 128, K = 32, N = the template argument.
template <int N>
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, bool accumulate) {
  constexpr uint32_t idesc = (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(kBlockRows >> 4) << 24);
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate ? 1u : 0u)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t addr, const uint32_t (&r)[32], int o) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          addr),
      "r"(r[o + 0]), "r"(r[o + 1]), "r"(r[o + 2]), "r"(r[o + 3]), "r"(r[o + 4]), "r"(r[o + 5]), "r"(r[o + 6]),
      "r"(r[o + 7]), "r"(r[o + 8]), "r"(r[o + 9]), "r"(r[o + 10]), "r"(r[o + 11]), "r"(r[o + 12]), "r"(r[o + 13]),
      "r"(r[o + 14]), "r"(r[o + 15])
      : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t addr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(addr));
}

// Two floats -> two e4m3 bytes (round to nearest even, saturating); `lo`
// lands in bits 0..7.
__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}
// Exact values of two e4m3 bytes (bits 0..7 and 8..15).
__device__ __forceinline__ float2 e4m3x2_value(uint32_t two) {
  uint32_t h2;
  uint16_t in = static_cast<uint16_t>(two);
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(in));
  return __half22float2(*reinterpret_cast<__half2*>(&h2));
}

// Bit position p of a byte (column 4p + e of a word, af1_layout.h): 1 / d_p
// and L_p + H_p.
//   p:        0     1     2     3     4     5     6     7
//   d_p:    1/8   1/4   1/2   1/2   1/4   1/2   1/2    -2
//   L_p:      1     1     1   1/2     1     1   1/2     1
__constant__ float c_inv_delta[8] = {8.f, 4.f, 2.f, 2.f, 4.f, 2.f, 2.f, -0.5f};
__constant__ float c_lph[8] = {2.125f, 2.25f, 2.5f, 1.5f, 2.25f, 2.5f, 1.5f, 0.f};

// One word (32 columns) -> 8 tensor-memory columns of e4m3 A values:
// column p holds columns 4p .. 4p+3 of the word (bit p of each byte).
__device__ __forceinline__ void expand_word(uint32_t w, uint32_t* s) {
  const uint32_t v = w >> 3;
  s[0] = (w & 0x01010101u) | 0x38383838u;  // mantissa bit 0: {1, 1.125}
  s[1] = (w & 0x02020202u) | 0x38383838u;  // mantissa bit 1: {1, 1.25}
  s[2] = (w & 0x04040404u) | 0x38383838u;  // mantissa bit 2: {1, 1.5}
  s[3] = (w & 0x08080808u) | 0x30303030u;  // exponent bit 0: {0.5, 1}
  s[4] = (v & 0x02020202u) | 0x38383838u;  // byte bit 4 -> mantissa bit 1
  s[5] = (v & 0x04040404u) | 0x38383838u;  // byte bit 5 -> mantissa bit 2
  s[6] = (v & 0x08080808u) | 0x30303030u;  // byte bit 6 -> exponent bit 0
  s[7] = (w & 0x80808080u) | 0x38383838u;  // sign bit: {1, -1}
}

// The power of two 2^sigma that brings a positive maximum m into [128, 256),
// read from m's exponent field (m = f 2^e with f in [0.5, 1), sigma = 8 - e).
// Returns 2^sigma in *sc and 2^-sigma in *is; m == 0 gives 1, 1.
__device__ __forceinline__ void pow2_scale(float m, float* sc, float* is) {
  if (!(m > 0.f)) {
    *sc = 1.f;
    *is = 1.f;
    return;
  }
  const int e = (int)((__float_as_uint(m) >> 23) & 0xFFu) - 126;
  const int sigma = max(min(8 - e, 120), -120);
  *sc = __uint_as_float((uint32_t)(127 + sigma) << 23);
  *is = __uint_as_float((uint32_t)(127 - sigma) << 23);
}

// ---------------------------------------------------------------------------
// Kernel arguments and shared-memory plan
// ---------------------------------------------------------------------------

struct DecodeArgs {
  const uint8_t* signs;  // af1_layout.h row-block layout
  SignMatrix sm;
  int KS, CPC;           // cluster size along K, chunks per CTA
  int tokens;            // T (1..N/4)
  const __half* x;       // phase 1 input [T][ldx] (FP16)
  int64_t ldx;
  const float* zin;      // phase 2 input [T][ldz] (FP32)
  int64_t ldz;
  const __half* colscale;  // phase 1: b (C entries)
  const __half* rowscale;  // phase 1: s; phase 2: a (R entries)
  float* sout;             // phase 1 output [T][lds]
  int64_t lds;
  void* y;                 // phase 2 output [T][ldy], FP16 (ydtype 0) or FP32
  int64_t ldy;
  int ydtype;
  unsigned* status;
  long long wait_cycles;  // budget of every bounded wait (clock64 cycles)
  // Prepared B operand (passes of more than 4 tokens): tiles of every chunk
  // (chunk c at c N 128 bytes) and per-(slice, token) {2^-sigma, Q 2^-sigma}
  // at bstats[slice * kMaxPassTokens + t]; written by bprep_kernel, read by
  // decode_kernel<..., true>.
  uint8_t* bbuf;
  float2* bstats;
};

struct __align__(8) DecodeHeader {
  uint64_t wfull[kMaxCPC];  // packed chunk c has landed (bulk copy)
  uint64_t afull[8];        // A buffer holds its chunk (128 expander arrivals)
  uint64_t aempty[8];       // the MMAs that read an A buffer are done (NACC commits)
  uint64_t xfull;           // staged activations have landed (bulk copies)
  uint64_t ddone;           // all MMAs done (NACC commits)
  uint64_t stats;           // per-token 2^-sigma and Q 2^-sigma are published
  uint32_t tmem_base, err;
  uint32_t maxbits[kMaxPassTokens];  // max |z'| per token, as FP32 bits
  float sc[kMaxPassTokens], is[kMaxPassTokens], qis[kMaxPassTokens];
};

struct DecodeSmem {
  int bt, w, act, recv, qpart, rs, hdr, total;  // byte offsets from the 1024-aligned base
};

__host__ __device__ inline int align128(int v) { return (v + 127) & ~127; }
__host__ __device__ inline int slice_rows(int KS) { return (kBlockRows + KS - 1) / KS; }

// Passes of more than 4 tokens stage the CTA's activations in shared memory
// with bulk copies (one per token row) before splitting them.
__host__ __device__ inline bool staged_acts(int N) { return N > 16; }

// prep: the B operand is prepared (bprep_kernel), so no activations are staged.
__host__ __device__ inline DecodeSmem decode_smem(int phase, int N, int CPC, int KS, int T, bool prep) {
  DecodeSmem p;
  int off = 0;
  p.bt = off;
  off += N * 128 * CPC;  // B: chunk c at c N 128, 1024-aligned
  p.w = off;
  off += kChunkBytes * CPC;
  p.act = off;  // T rows of CPC * 128 activations (FP16 phase 1, FP32 phase 2)
  if (staged_acts(N) && !prep) off += T * CPC * kChunkCols * (phase == 1 ? 2 : 4);
  p.recv = off;
  off = align128(off + KS * T * slice_rows(KS) * 4);
  p.qpart = off;
  off = align128(off + T * 128 * 4);
  p.rs = off;
  off = align128(off + slice_rows(KS) * 4);
  p.hdr = off;
  off = align128(off + (int)sizeof(DecodeHeader));
  p.total = off + 1024;  // slack for aligning the base to 1024 bytes
  return p;
}

__host__ __device__ constexpr int nacc_for(int N) { return N <= 32 ? 4 : 2; }
__host__ __device__ constexpr int nbuf_for(int N) { return (kTmemCols - nacc_for(N) * N) / 32; }

// ---------------------------------------------------------------------------
// Kernel
// ---------------------------------------------------------------------------

template <int PHASE>
__device__ __forceinline__ float4 load4(const DecodeArgs& a, int t, int64_t k) {
  // Four consecutive activations of token t from column k (zero beyond C).
  // Written by the kernel this one overlaps through PDL, so read through L2
  // (ld.global.cg), never through the non-coherent L1 path.
  const int64_t C = a.sm.C;
  float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  if (PHASE == 1) {
    const __half* p = a.x + (int64_t)t * a.ldx + k;
    if (k + 3 < C) {
      const uint2 raw = __ldcg(reinterpret_cast<const uint2*>(p));
      const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&raw.x));
      const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&raw.y));
      z = make_float4(f0.x, f0.y, f1.x, f1.y);
    } else {
      if (k < C) z.x = __half2float(__ldcg(p));
      if (k + 1 < C) z.y = __half2float(__ldcg(p + 1));
      if (k + 2 < C) z.z = __half2float(__ldcg(p + 2));
    }
  } else {
    const float* p = a.zin + (int64_t)t * a.ldz + k;
    if (k + 3 < C) {
      z = __ldcg(reinterpret_cast<const float4*>(p));
    } else {
      if (k < C) z.x = __ldcg(p);
      if (k + 1 < C) z.y = __ldcg(p + 1);
      if (k + 2 < C) z.z = __ldcg(p + 2);
    }
  }
  return z;
}

// z'_k = z_k * colscale_k / d_p for the 4 columns k..k+3 (one bit position p).
template <int PHASE>
__device__ __forceinline__ float4 scale4(const DecodeArgs& a, float4 z, int64_t k) {
  const float id = c_inv_delta[(k >> 2) & 7];
  if (PHASE == 1) {
    const int64_t C = a.sm.C;
    float b0 = 0.f, b1 = 0.f, b2 = 0.f, b3 = 0.f;
    if (k + 3 < C) {
      const uint2 raw = __ldg(reinterpret_cast<const uint2*>(a.colscale + k));
      const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&raw.x));
      const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&raw.y));
      b0 = f0.x;
      b1 = f0.y;
      b2 = f1.x;
      b3 = f1.y;
    } else {
      if (k < C) b0 = __half2float(a.colscale[k]);
      if (k + 1 < C) b1 = __half2float(a.colscale[k + 1]);
      if (k + 2 < C) b2 = __half2float(a.colscale[k + 2]);
    }
    z = make_float4(z.x * b0, z.y * b1, z.z * b2, z.w * b3);
  }
  return make_float4(z.x * id, z.y * id, z.z * id, z.w * id);
}

// Four consecutive staged activations of token t at CTA column kl (zero at
// and beyond kv, the CTA's valid columns).
template <int PHASE>
__device__ __forceinline__ float4 act4(const uint8_t* act, int rowlen, int t, int kl, int kv) {
  float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  if (PHASE == 1) {
    const __half* p = reinterpret_cast<const __half*>(act) + (size_t)t * rowlen + kl;
    if (kl + 3 < kv) {
      const uint2 raw = *reinterpret_cast<const uint2*>(p);
      const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&raw.x));
      const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&raw.y));
      z = make_float4(f0.x, f0.y, f1.x, f1.y);
    } else {
      if (kl < kv) z.x = __half2float(p[0]);
      if (kl + 1 < kv) z.y = __half2float(p[1]);
      if (kl + 2 < kv) z.z = __half2float(p[2]);
    }
  } else {
    const float* p = reinterpret_cast<const float*>(act) + (size_t)t * rowlen + kl;
    if (kl + 3 < kv) {
      z = *reinterpret_cast<const float4*>(p);
    } else {
      if (kl < kv) z.x = p[0];
      if (kl + 1 < kv) z.y = p[1];
      if (kl + 2 < kv) z.z = p[2];
    }
  }
  return z;
}

// The B operand of one K slice for T tokens (chunks c0 .. c0 + nch - 1,
// columns from k0), built by 128 threads (bt = 0..127, named barrier 1):
// per-token power-of-two scale from the slice's max |z'|, four e4m3 terms per
// value in the 128-byte-swizzled K-major tile layout at Bt (chunk c at
// c N 128), and per-thread Q partials in qpart[t][bt]. Bt is shared memory in
// the decode kernel and global memory in the prep kernel. The activations
// must be readable (after griddepcontrol.wait).
template <int PHASE, int N>
__device__ __forceinline__ void build_b(const DecodeArgs& a, int T, int nch, int64_t k0, int bt, uint8_t* act,
                                        uint8_t* Bt, float* qpart, uint32_t* maxbits, uint64_t* xfull,
                                        uint32_t* err) {
  constexpr int STASH = 4;         // activation groups a builder thread keeps in registers
  constexpr bool STAGED = N > 16;  // staged_acts(N)
  const int g4 = nch * (kChunkCols / 4);  // groups of 4 columns per token
  const int ngroups = T * g4;
  for (int t = 0; t < T; ++t) qpart[t * 128 + bt] = 0.f;  // own column only
  const int rowlen = a.CPC * kChunkCols;
  const int kv = (int)min((int64_t)nch * kChunkCols, a.sm.C - k0);  // valid columns of this CTA
  if (STAGED) {
    // One bulk copy per token row of its 16-byte-multiple valid prefix; the
    // few remaining columns with plain loads.
    constexpr int ESZ = PHASE == 1 ? 2 : 4;
    const int bulk_cols = ((kv * ESZ) & ~15) / ESZ;
    if (bt == 0) {
      const uint32_t bytes = (uint32_t)(bulk_cols * ESZ);
      if (bytes > 0) {
        mbar_expect_tx(xfull, bytes * (uint32_t)T);
        for (int t = 0; t < T; ++t) {
          const uint8_t* src = PHASE == 1 ? reinterpret_cast<const uint8_t*>(a.x + (int64_t)t * a.ldx + k0)
                                          : reinterpret_cast<const uint8_t*>(a.zin + (int64_t)t * a.ldz + k0);
          bulk_g2s(act + (size_t)t * rowlen * ESZ, src, bytes, xfull);
        }
      } else {
        mbar_arrive(xfull);
      }
    }
    for (int i = bt; i < T * 8; i += 128) {
      const int t = i >> 3, k = bulk_cols + (i & 7);
      if (k < kv) {
        if (PHASE == 1)
          reinterpret_cast<__half*>(act)[(size_t)t * rowlen + k] = __ldcg(a.x + (int64_t)t * a.ldx + k0 + k);
        else
          reinterpret_cast<float*>(act)[(size_t)t * rowlen + k] = __ldcg(a.zin + (int64_t)t * a.ldz + k0 + k);
      }
    }
    mbar_wait(xfull, 0, err, a.wait_cycles);
    builders_sync();  // tail values visible
  }
  // z' of group (t, c4): from the staged activations or straight from L2.
  auto zq = [&](int t, int c4) -> float4 {
    const int64_t k = k0 + 4 * c4;
    const float4 z = STAGED ? act4<PHASE>(act, rowlen, t, 4 * c4, kv) : load4<PHASE>(a, t, k);
    return scale4<PHASE>(a, z, k);
  };
  float4 stash[STASH];
  // Pass 1: maxima of |z'| per token.
  {
    int cur_t = -1;
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < STASH; ++i) stash[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = 0, g = bt; g < ngroups; ++i, g += 128) {
      const int t = g / g4, c4 = g - t * g4;
      const float4 u = zq(t, c4);
      if (i < STASH) {
#pragma unroll
        for (int j = 0; j < STASH; ++j)
          if (j == i) stash[j] = u;
      }
      if (t != cur_t) {
        if (cur_t >= 0 && mx > 0.f) atomicMax(&maxbits[cur_t], __float_as_uint(mx));
        cur_t = t;
        mx = 0.f;
      }
      mx = fmaxf(mx, fmaxf(fmaxf(fabsf(u.x), fabsf(u.y)), fmaxf(fabsf(u.z), fabsf(u.w))));
    }
    if (cur_t >= 0 && mx > 0.f) atomicMax(&maxbits[cur_t], __float_as_uint(mx));
  }
  builders_sync();
  // Pass 2: split into 4 e4m3 terms, write B rows 4t + q, and Q partials.
  {
    int cur_t = -1;
    float sc = 0.f, q = 0.f;
    for (int i = 0, g = bt; g < ngroups; ++i, g += 128) {
      const int t = g / g4, c4 = g - t * g4;
      if (t != cur_t) {
        if (cur_t >= 0) qpart[cur_t * 128 + bt] = q;
        cur_t = t;
        q = 0.f;
        float is_unused;
        pow2_scale(__uint_as_float(maxbits[t]), &sc, &is_unused);
      }
      float4 u;
      if (i < STASH) {
        u = stash[0];
#pragma unroll
        for (int j = 1; j < STASH; ++j)
          if (j == i) u = stash[j];
      } else {
        u = zq(t, c4);
      }
      float4 v = make_float4(u.x * sc, u.y * sc, u.z * sc, u.w * sc);
      const float4 v0 = v;
      const int kl = 4 * c4;  // column within the CTA's range
      const int c = kl >> 7, kin = kl & 127;
      uint8_t* base = Bt + c * (N * 128) + (kin & 15);
      const int j16 = kin >> 4;
#pragma unroll
      for (int term = 0; term < kTerms; ++term) {
        const uint32_t lo = e4m3x2(v.x, v.y), hi = e4m3x2(v.z, v.w);
        const float2 flo = e4m3x2_value(lo), fhi = e4m3x2_value(hi);
        v.x -= flo.x;
        v.y -= flo.y;
        v.z -= fhi.x;
        v.w -= fhi.y;
        const int n = 4 * t + term;
        *reinterpret_cast<uint32_t*>(base + n * 128 + ((j16 ^ (n & 7)) << 4)) = lo | (hi << 16);
      }
      q += c_lph[c4 & 7] * (((v0.x - v.x) + (v0.y - v.y)) + ((v0.z - v.z) + (v0.w - v.w)));
    }
    if (cur_t >= 0) qpart[cur_t * 128 + bt] = q;
  }
}

template <int PHASE, int N, bool PREP>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const DecodeArgs a) {
  constexpr int NACC = nacc_for(N);
  constexpr int NBUF = nbuf_for(N);
  constexpr int DCOL = NBUF * 32;  // first accumulator column

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int T = a.tokens;
  const int KS = a.KS;
  const DecodeSmem sp = decode_smem(PHASE, N, a.CPC, KS, T, PREP);
  constexpr bool STAGED = N > 16;  // staged_acts(N)
  uint8_t* act = smem + sp.act;
  uint8_t* Bt = smem + sp.bt;
  const uint32_t* W = reinterpret_cast<const uint32_t*>(smem + sp.w);
  float* recv = reinterpret_cast<float*>(smem + sp.recv);
  float* qpart = reinterpret_cast<float*>(smem + sp.qpart);
  float* rs = reinterpret_cast<float*>(smem + sp.rs);
  DecodeHeader& h = *reinterpret_cast<DecodeHeader*>(smem + sp.hdr);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = blockIdx.x, ks = blockIdx.y;
  const int nch_total = a.sm.NCH;
  const int c0 = ks * a.CPC;
  const int nch = min(a.CPC, nch_total - c0);  // >= 1 by construction of KS
  const int64_t row0 = (int64_t)rb * kBlockRows;
  const int64_t k0 = (int64_t)c0 * kChunkCols;
  const int slice = slice_rows(KS);
  const int my0 = ks * slice;  // first block row this CTA finalises

  cluster_arrive_relaxed();  // matched by cluster_wait before the first remote store

  if (tid == 128) {
    for (int c = 0; c < nch; ++c) mbar_init(&h.wfull[c], 1);
    for (int b = 0; b < NBUF; ++b) {
      mbar_init(&h.afull[b], 128);
      mbar_init(&h.aempty[b], NACC);
    }
    mbar_init(&h.xfull, 1);
    mbar_init(&h.ddone, NACC);
    mbar_init(&h.stats, 16);
    h.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // Packed chunks of this CTA: contiguous 2 KB blocks of row block rb.
    const uint8_t* src = a.signs + ((int64_t)rb * nch_total + c0) * kChunkBytes;
    for (int c = 0; c < nch; ++c) {
      mbar_expect_tx(&h.wfull[c], kChunkBytes);
      bulk_g2s(smem + sp.w + c * kChunkBytes, src + (int64_t)c * kChunkBytes, kChunkBytes, &h.wfull[c]);
    }
  }
  if (tid < kMaxPassTokens) h.maxbits[tid] = 0u;  // published by the CTA barrier below
  __syncwarp();
  if (warp == 4) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&h.tmem_base)),
                 "r"((uint32_t)kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // Row scales of the rows this CTA finalises (layer constants).
  for (int i = tid; i < slice; i += kThreads) {
    const int64_t row = row0 + my0 + i;
    rs[i] = (my0 + i < kBlockRows && row < a.sm.R) ? __half2float(a.rowscale[row]) : 0.f;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = h.tmem_base;

  if (warp < 4) {
    // ---- A: expand packed chunks into the tensor-memory ring --------------
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    bool ok = true;
    for (int c = 0; c < nch && ok; ++c) {
      const int b = c % NBUF, use = c / NBUF;
      if (use >= 1) {
        ok = mbar_wait(&h.aempty[b], (use - 1) & 1, &h.err, a.wait_cycles);
        tc_fence_after();
      }
      if (ok) ok = mbar_wait(&h.wfull[c], 0, &h.err, a.wait_cycles);
      if (!ok) break;
      uint32_t r[32];
      const uint32_t* wc = W + c * (kChunkBytes / 4);
#pragma unroll
      for (int kw = 0; kw < kChunkWords; ++kw) expand_word(wc[kw * kBlockRows + tid], r + 8 * kw);
      const uint32_t addr = tmem + lane_base + (uint32_t)(b * 32);
      tmem_st16(addr, r, 0);
      tmem_st16(addr + 16, r, 16);
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      tc_fence_before();
      mbar_arrive(&h.afull[b]);
    }
  } else {
    // ---- B: activations -> e4m3 terms in the swizzled B tile --------------
    const int bt = tid - 128;
    griddep_wait();  // activations are written by the previous kernel
    if constexpr (PREP) {
      // Prepared by bprep_kernel for this K slice: one bulk copy per chunk.
      if (bt == 0) {
        mbar_expect_tx(&h.xfull, (uint32_t)(nch * N * 128));
        for (int c = 0; c < nch; ++c)
          bulk_g2s(Bt + c * N * 128, a.bbuf + (int64_t)(c0 + c) * N * 128, (uint32_t)(N * 128), &h.xfull);
      }
      mbar_wait(&h.xfull, 0, &h.err, a.wait_cycles);
    } else {
      build_b<PHASE, N>(a, T, nch, k0, bt, act, Bt, qpart, h.maxbits, &h.xfull, &h.err);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // B is read by the tensor cores
    builders_sync();
    const int ia = warp - 4;
    if (lane == 0 && ia < NACC) {
      // ---- MMA issue: chunk c, K step kk (32 columns) by issuer kk % NACC --
      const uint32_t b0 = smem_u32(Bt);
      bool ok = true;
      for (int c = 0; c < nch && ok; ++c) {
        const int b = c % NBUF, use = c / NBUF;
        ok = mbar_wait(&h.afull[b], use & 1, &h.err, a.wait_cycles);
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int kk = ia; kk < 4; kk += NACC) {
          mma_ts<N>(tmem + (uint32_t)(DCOL + ia * N), tmem + (uint32_t)(b * 32 + kk * 8),
                    smem_desc(b0 + (uint32_t)(c * N * 128 + kk * 32)), c > 0 || kk >= NACC);
        }
        mma_commit(&h.aempty[b]);
      }
      mma_commit(&h.ddone);
    }
    if (bt >= 112) {
      // ---- per-token 2^-sigma and Q 2^-sigma, summed in a fixed order ------
      const int t = bt - 112;
      if (t < T) {
        if constexpr (PREP) {
          const float2 st = __ldcg(a.bstats + ks * kMaxPassTokens + t);
          h.is[t] = st.x;
          h.qis[t] = st.y;
        } else {
          float qs = 0.f;
          for (int j = 0; j < 128; ++j) qs += qpart[t * 128 + j];
          float sc, is;
          pow2_scale(__uint_as_float(h.maxbits[t]), &sc, &is);
          h.is[t] = is;
          h.qis[t] = qs * is;
        }
      }
      mbar_arrive(&h.stats);
    }
    __syncwarp();
  }

  griddep_launch_dependents();
  // ---- epilogue: accumulators -> per-row partial sums -> owner CTA ----------
  griddep_wait();  // outputs may still be read by the previous kernel until it completes
  cluster_wait();  // every CTA of the cluster has started
  if (warp < 4) {
    const bool ok = mbar_wait(&h.ddone, 0, &h.err, a.wait_cycles) && mbar_wait(&h.stats, 0, &h.err, a.wait_cycles);
    tc_fence_after();
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    const int i = tid;  // block row
    const int owner = i / slice;
#pragma unroll
    for (int cb = 0; cb < N / 16; ++cb) {
      float acc[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) acc[j] = 0.f;
#pragma unroll
      for (int d = 0; d < NACC; ++d) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + (uint32_t)(DCOL + d * N + cb * 16), r);
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
        for (int j = 0; j < 16; ++j) acc[j] += __uint_as_float(r[j]);
      }
#pragma unroll
      for (int tt = 0; tt < 4; ++tt) {
        const int t = cb * 4 + tt;
        if (ok && t < T) {
          const float dsum = (acc[4 * tt] + acc[4 * tt + 1]) + (acc[4 * tt + 2] + acc[4 * tt + 3]);
          const float p = 2.f * dsum * h.is[t] - h.qis[t];
          st_cluster_f32(recv + ((ks * T + t) * slice + (i - owner * slice)), (uint32_t)owner, p);
        }
      }
    }
  }
  // All partials of the cluster have landed in their owners' buffers.
  cluster_sync();
  const int cnt = min(slice, kBlockRows - my0);
  for (int idx = tid; idx < T * cnt; idx += kThreads) {
    const int t = idx / cnt;
    const int i = idx - t * cnt;
    const int64_t row = row0 + my0 + i;
    if (row >= a.sm.R) continue;
    float v = 0.f;
    for (int q = 0; q < KS; ++q) v += recv[(q * T + t) * slice + i];
    const float out = v * rs[i];
    if (PHASE == 1) {
      a.sout[(int64_t)t * a.lds + row] = out;
    } else if (a.ydtype == 0) {
      reinterpret_cast<__half*>(a.y)[(int64_t)t * a.ldy + row] = __float2half_rn(out);
    } else {
      reinterpret_cast<float*>(a.y)[(int64_t)t * a.ldy + row] = out;
    }
  }

  // ---- teardown ---------------------------------------------------------------
  tc_fence_before();
  __syncthreads();
  if (tid == 128 && h.err != 0) {
    // Something timed out: let the bulk copies drain (bounded) so that none
    // lands after the CTA has exited, and report it.
    for (int c = 0; c < nch; ++c) mbar_wait(&h.wfull[c], 0, &h.err, a.wait_cycles);
    if (STAGED || PREP) mbar_wait(&h.xfull, 0, &h.err, a.wait_cycles);
    atomicOr(a.status, kStatusTimeout);
  }
  if (warp == 4) {
    tc_fence_after();
    if (lane == 0) mbar_wait(&h.ddone, 0, &h.err, a.wait_cycles);  // no MMA may still read tensor memory
    __syncwarp();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)kTmemCols)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// Decode kernel with 16-bit MMA operands (tcgen05.mma kind::f16), passes of
// up to 16 tokens, and calls of 17..64 tokens on small layers as one pass
// (mid_pass). The signs become exact 16-bit A values in tensor memory:
//   phase 1: A = +-b_j (FP16; the column scale carries the sign), B = x
//            (FP16, N = 16/32/64 rows, row t = token t), so
//            D = sum_j +-b_j x_j;
//   phase 2, up to 16 tokens: A = +-1 (BF16), B = s' split into
//            kS2Terms = 2 BF16 terms hi + lo (N = 16/32 rows, term q of
//            token t in row 2 t + q): BF16 keeps FP32's exponent range, so
//            no scaling is needed, and hi + lo holds the 16 leading
//            significant bits of s' (a relative error of at most 2^-17);
//   phase 2, one pass of 17..64 tokens: A = +-1 (FP16), B = s' rounded to
//            FP16 (N = 32/64 rows), as the prefill path rounds its H.
// Every product is exact and the MMA accumulates in FP32: up to that
// rounding of s', the result is the FP32 signed sum the lookup-table
// kernels form, summed in another order.
// Against the e4m3 kernel above there is no activation split, no power-of-
// two scale and no sign correction, and the B operand is a copy (phase 1) or
// a split (phase 2) that the CTA builds itself, so no preparation
// kernel runs. A chunk of A takes 64 tensor-memory columns (two values per
// column), twice the e4m3 chunk. The CTA structure is the e4m3 kernel's:
// bulk copies of the signs first, warps 0-3 expand, warps 4-7 build B and
// issue the MMAs (K = 16 each) into NACC accumulators, warps 0-3 read them
// back and push the partial sums to the cluster CTA that owns each row.
// ---------------------------------------------------------------------------

// Terms of s' in the phase-2 B operand: 1 = s' rounded to FP16 (with FP16
// +-1 signs), 2 = BF16 terms (with BF16 +-1 signs) that hold its 16 leading
// significant bits. Measured on the 32-layer stack at 16 / 8 tokens (ms per
// step): three BF16 terms (s' exactly) 4.20 / 3.28, two 4.03 / 3.16, one
// 3.87 / 3.14. Two: a relative error of at most 2^-17 per value and FP32's
// exponent range (one FP16 term loses small values to FP16's range; three
// would need an epilogue that sums a token's terms across column blocks).
constexpr int kS2Terms = 2;
// Calls of 17..kMidMaxTokens tokens run as one pass (mid_pass) with s' as
// ONE FP16 term, the rounding their prefill path makes of its H (reading
// R11): two BF16 terms make phase 2's B 128 rows at 64 tokens (32 KB per
// chunk, one CTA per SM). Measured at 32 / 64 tokens (us, two terms -> one):
// 14336x4096 41.9 -> 39.2 / 120 -> 113, 4096x14336 47.4 -> 40.2 / 133 ->
// 131, 8192^2 38.2 -> 33.3 / 115 -> 79.9.
__host__ __device__ constexpr int s2_terms(int T) { return T <= kMaxPassTokens ? kS2Terms : 1; }
// Accumulators (one MMA issuer each) and A-ring depth for N rows of B,
// within the CTA's 256 tensor-memory columns: N 16: 4 and 3; 32: 2 and 3;
// 48 / 64: 2 and 2; 128: 1 and 2.
__host__ __device__ constexpr int hnacc_for(int N) { return N == 16 ? 4 : N <= 64 ? 2 : 1; }
__host__ __device__ constexpr int hnbuf_for(int N) { return (kTmemCols - hnacc_for(N) * N) / 64; }
// B rows of a pass of T tokens (up to kMidMaxTokens): T rows (phase 1) or
// s2_terms(T) T rows (phase 2), rounded up to 16, 32 or 64.
__host__ __device__ constexpr int hround_n(int rows) { return rows <= 16 ? 16 : rows <= 32 ? 32 : 64; }
__host__ __device__ constexpr int hdecode_n(int phase, int T) { return hround_n(phase == 1 ? T : s2_terms(T) * T); }

struct __align__(8) HDecodeHeader {
  uint64_t wfull[kMaxCPC];  // packed chunk c has landed (chunk 0: with the column scales)
  uint64_t afull[4];        // A buffer holds its chunk (128 expander arrivals)
  uint64_t aempty[4];       // the MMAs that read an A buffer are done (NACC commits)
  uint64_t ddone;           // all MMAs done (NACC commits)
  uint32_t tmem_base, err;
};

struct HDecodeSmem {
  int bt, w, cs, recv, rs, hdr, total;  // byte offsets from the 1024-aligned base
};

__host__ __device__ inline HDecodeSmem hdecode_smem(int N, int CPC, int KS, int T) {
  HDecodeSmem p;
  int off = 0;
  p.bt = off;
  off += 2 * N * 128 * CPC;  // B: K half h of chunk c at (2 c + h) N 128, 1024-aligned
  p.w = off;
  off += kChunkBytes * CPC;
  p.cs = off;
  off += CPC * kChunkCols * 2;  // phase 1: the column scales of the CTA's chunks
  p.recv = off;
  off = align128(off + KS * T * slice_rows(KS) * 4);
  p.rs = off;
  off = align128(off + slice_rows(KS) * 4);
  p.hdr = off;
  off = align128(off + (int)sizeof(HDecodeHeader));
  p.total = off + 1024;  // slack for aligning the base to 1024 bytes
  return p;
}

// D (FP32) [+]= A (tensor memory) x B (shared memory)^T, kind::f16, M = 128,
// K = 16, N rows of B; A and B both FP16, or both BF16.
template <int N, bool BF16>
__device__ __forceinline__ void mma_h(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, bool accumulate) {
  constexpr uint32_t fmt = BF16 ? 1u : 0u;
  constexpr uint32_t idesc =
      (1u << 4) | (fmt << 7) | (fmt << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(kBlockRows >> 4) << 24);
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate ? 1u : 0u)
      : "memory");
}

// Sign bits p of bytes 1 and 3 of `pair_bytes` -> the sign bits (15, 31) of
// a 16-bit pair: bit 1 keeps v, bit 0 negates it.
__device__ __forceinline__ uint32_t sign_pair(uint32_t pair_bytes, int p, uint32_t v) {
  return v ^ (~(pair_bytes << (7 - p)) & 0x80008000u);
}

// Word w of a row -> 16 tensor-memory columns of 16-bit A values in K order:
// column 4 jj + u holds columns 8 jj + 2 u, + 1 of the word. Column 4 p + e
// of the word is bit 8 e + p (af1_layout.h); v[jj] holds the magnitudes of
// columns 8 jj .. 8 jj + 7 as four pairs.
__device__ __forceinline__ void expand_word_h(uint32_t w, const uint4 (&v)[4], uint32_t* s) {
  const uint32_t b01 = __byte_perm(w, 0u, 0x1404);  // bytes 0, 1 (e = 0, 1) -> bytes 1, 3
  const uint32_t b23 = __byte_perm(w, 0u, 0x3424);  // bytes 2, 3 (e = 2, 3) -> bytes 1, 3
#pragma unroll
  for (int jj = 0; jj < 4; ++jj) {
    const int p = 2 * jj;
    s[4 * jj + 0] = sign_pair(b01, p, v[jj].x);
    s[4 * jj + 1] = sign_pair(b23, p, v[jj].y);
    s[4 * jj + 2] = sign_pair(b01, p + 1, v[jj].z);
    s[4 * jj + 3] = sign_pair(b23, p + 1, v[jj].w);
  }
}

__device__ __forceinline__ void tmem_st16p(uint32_t addr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          addr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// The TERMS 16-bit terms of v: v rounded to FP16 (one term), or the BF16
// terms hi and lo (v - hi is exact in FP32; lo is it rounded to BF16).
template <int TERMS>
__device__ __forceinline__ void split_terms(float v, uint16_t* t3) {
  if constexpr (TERMS == 1) {
    t3[0] = __half_as_ushort(__float2half_rn(v));
  } else {
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(hi);
    t3[0] = __bfloat16_as_ushort(hi);
    t3[1] = __bfloat16_as_ushort(__float2bfloat16_rn(r1));
  }
}

// The B operand of the CTA's K slice (chunks of columns from k0, kv valid
// columns), built by 128 threads (bt = 0..127): 16-byte units of 8 columns,
// row n of K half h of chunk c at Bt + (2 c + h) N 128 + n 128, unit j at
// (j ^ (n & 7)) 16 (128-byte swizzle, K-major). Columns >= kv are zero. The
// activations come from L2 (written by the previous kernel): each thread
// issues the loads of UB units before it converts and stores any, so a CTA
// waits for about T nu / (128 UB) round trips instead of T nu / 128.
template <int PHASE>
__device__ __forceinline__ void load_unit_h(const DecodeArgs& a, int t, int kl, int64_t k0, int kv, uint4 (&raw)[2]) {
  if (PHASE == 1) {
    const __half* p = a.x + (int64_t)t * a.ldx + k0 + kl;
    if (kl + 7 < kv) {
      raw[0] = __ldcg(reinterpret_cast<const uint4*>(p));
    } else {
      uint16_t e[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) e[q] = kl + q < kv ? __half_as_ushort(__ldcg(p + q)) : (uint16_t)0;
      raw[0] = make_uint4(e[0] | (uint32_t)e[1] << 16, e[2] | (uint32_t)e[3] << 16, e[4] | (uint32_t)e[5] << 16,
                          e[6] | (uint32_t)e[7] << 16);
    }
  } else {
    const float* p = a.zin + (int64_t)t * a.ldz + k0 + kl;
    if (kl + 7 < kv) {
      raw[0] = __ldcg(reinterpret_cast<const uint4*>(p));
      raw[1] = __ldcg(reinterpret_cast<const uint4*>(p + 4));
    } else {
      uint32_t f[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) f[q] = kl + q < kv ? __float_as_uint(__ldcg(p + q)) : 0u;
      raw[0] = make_uint4(f[0], f[1], f[2], f[3]);
      raw[1] = make_uint4(f[4], f[5], f[6], f[7]);
    }
  }
}

template <int PHASE, int N, int TERMS>
__device__ __forceinline__ void build_b_h(const DecodeArgs& a, int T, int nch, int64_t k0, int kv, int bt,
                                          uint8_t* Bt) {
  constexpr int UB = 4;
  const int nu = nch * (kChunkCols / 8);  // 8-column units per token
  const int total = T * nu;
  for (int i0 = bt; i0 < total; i0 += UB * 128) {
    uint4 raw[UB][2];
#pragma unroll
    for (int u = 0; u < UB; ++u) {
      const int i = i0 + u * 128;
      if (i < total) {
        const int t = i / nu;
        load_unit_h<PHASE>(a, t, 8 * (i - t * nu), k0, kv, raw[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < UB; ++u) {
      const int i = i0 + u * 128;
      if (i >= total) break;
      const int t = i / nu, uu = i - t * nu;
      const int c = uu >> 4, hh = (uu >> 3) & 1, j = uu & 7;
      uint8_t* half_base = Bt + (2 * c + hh) * (N * 128);
      if (PHASE == 1) {
        *reinterpret_cast<uint4*>(half_base + t * 128 + ((j ^ (t & 7)) << 4)) = raw[u][0];
      } else {
        const uint32_t fw[8] = {raw[u][0].x, raw[u][0].y, raw[u][0].z, raw[u][0].w,
                                raw[u][1].x, raw[u][1].y, raw[u][1].z, raw[u][1].w};
        uint16_t e[3][8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          uint16_t t3[3];
          split_terms<TERMS>(__uint_as_float(fw[q]), t3);
#pragma unroll
          for (int term = 0; term < TERMS; ++term) e[term][q] = t3[term];
        }
#pragma unroll
        for (int term = 0; term < TERMS; ++term) {
          const int n = TERMS * t + term;
          const uint4 v = make_uint4(e[term][0] | (uint32_t)e[term][1] << 16, e[term][2] | (uint32_t)e[term][3] << 16,
                                     e[term][4] | (uint32_t)e[term][5] << 16, e[term][6] | (uint32_t)e[term][7] << 16);
          *reinterpret_cast<uint4*>(half_base + n * 128 + ((j ^ (n & 7)) << 4)) = v;
        }
      }
    }
  }
}

// TERMS: terms of s' per token in phase 2's B (1: FP16, 2: BF16).
template <int PHASE, int N, int TERMS>
__global__ void __launch_bounds__(kThreads, 1) hdecode_kernel(const DecodeArgs a) {
  constexpr int NACC = hnacc_for(N);
  constexpr int NBUF = hnbuf_for(N);
  constexpr int DCOL = NBUF * 64;  // first accumulator column
  constexpr bool BF16 = PHASE == 2 && TERMS > 1;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int T = a.tokens;
  const int KS = a.KS;
  const HDecodeSmem sp = hdecode_smem(N, a.CPC, KS, T);
  uint8_t* Bt = smem + sp.bt;
  const uint32_t* W = reinterpret_cast<const uint32_t*>(smem + sp.w);
  const uint8_t* cs = smem + sp.cs;
  float* recv = reinterpret_cast<float*>(smem + sp.recv);
  float* rs = reinterpret_cast<float*>(smem + sp.rs);
  HDecodeHeader& h = *reinterpret_cast<HDecodeHeader*>(smem + sp.hdr);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = blockIdx.x, ks = blockIdx.y;
  const int nch_total = a.sm.NCH;
  const int c0 = ks * a.CPC;
  const int nch = min(a.CPC, nch_total - c0);  // >= 1 by construction of KS
  const int64_t row0 = (int64_t)rb * kBlockRows;
  const int64_t k0 = (int64_t)c0 * kChunkCols;
  const int kv = (int)min((int64_t)nch * kChunkCols, a.sm.C - k0);  // valid columns of this CTA
  const int slice = slice_rows(KS);
  const int my0 = ks * slice;  // first block row this CTA finalises

  cluster_arrive_relaxed();  // matched by cluster_wait before the first remote store

  if (tid == 128) {
    for (int c = 0; c < nch; ++c) mbar_init(&h.wfull[c], 1);
    for (int b = 0; b < NBUF; ++b) {
      mbar_init(&h.afull[b], 128);
      mbar_init(&h.aempty[b], NACC);
    }
    mbar_init(&h.ddone, NACC);
    h.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // Packed chunks of this CTA (contiguous 2 KB blocks of row block rb) and,
    // for phase 1, the column scales of its chunks (the layer's b is
    // zero-padded to whole chunks), which land with chunk 0.
    const uint8_t* src = a.signs + ((int64_t)rb * nch_total + c0) * kChunkBytes;
    for (int c = 0; c < nch; ++c) {
      const uint32_t extra = (PHASE == 1 && c == 0) ? (uint32_t)(nch * kChunkCols * 2) : 0u;
      mbar_expect_tx(&h.wfull[c], kChunkBytes + extra);
      bulk_g2s(smem + sp.w + c * kChunkBytes, src + (int64_t)c * kChunkBytes, kChunkBytes, &h.wfull[c]);
      if (extra != 0) bulk_g2s(smem + sp.cs, a.colscale + k0, extra, &h.wfull[0]);
    }
  }
  __syncwarp();
  if (warp == 4) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&h.tmem_base)),
                 "r"((uint32_t)kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // Row scales of the rows this CTA finalises (layer constants).
  for (int i = tid; i < slice; i += kThreads) {
    const int64_t row = row0 + my0 + i;
    rs[i] = (my0 + i < kBlockRows && row < a.sm.R) ? __half2float(a.rowscale[row]) : 0.f;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = h.tmem_base;

  if (warp < 4) {
    // ---- A: expand packed chunks into the tensor-memory ring --------------
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    bool ok = true;
    for (int c = 0; c < nch && ok; ++c) {
      const int b = c % NBUF, use = c / NBUF;
      if (use >= 1) {
        ok = mbar_wait(&h.aempty[b], (use - 1) & 1, &h.err, a.wait_cycles);
        tc_fence_after();
      }
      if (ok) ok = mbar_wait(&h.wfull[c], 0, &h.err, a.wait_cycles);
      if (!ok) break;
      const uint32_t* wc = W + c * (kChunkBytes / 4);
      const uint32_t addr = tmem + lane_base + (uint32_t)(b * 64);
#pragma unroll
      for (int kw = 0; kw < kChunkWords; ++kw) {
        uint4 v[4];
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          if (PHASE == 1)
            v[jj] = *reinterpret_cast<const uint4*>(cs + (c * kChunkCols + 32 * kw + 8 * jj) * 2);
          else
            v[jj] = BF16 ? make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u)   // BF16 pairs of 1
                         : make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);  // FP16 pairs of 1
        }
        uint32_t r[16];
        expand_word_h(wc[kw * kBlockRows + tid], v, r);
        tmem_st16p(addr + (uint32_t)(16 * kw), r);
      }
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      tc_fence_before();
      mbar_arrive(&h.afull[b]);
    }
  } else {
    // ---- B: activations -> the swizzled B tile; then the MMAs -------------
    const int bt = tid - 128;
    griddep_wait();  // activations are written by the previous kernel
    build_b_h<PHASE, N, TERMS>(a, T, nch, k0, kv, bt, Bt);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // B is read by the tensor cores
    builders_sync();
    const int ia = warp - 4;
    if (lane == 0 && ia < NACC) {
      // ---- MMA issue: chunk c, K step kk (16 columns) by issuer kk % NACC --
      const uint32_t b0 = smem_u32(Bt);
      bool ok = true;
      for (int c = 0; c < nch && ok; ++c) {
        const int b = c % NBUF, use = c / NBUF;
        ok = mbar_wait(&h.afull[b], use & 1, &h.err, a.wait_cycles);
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int kk = ia; kk < 8; kk += NACC) {
          mma_h<N, BF16>(tmem + (uint32_t)(DCOL + ia * N), tmem + (uint32_t)(b * 64 + kk * 8),
                         smem_desc(b0 + (uint32_t)((2 * c + (kk >> 2)) * N * 128 + (kk & 3) * 32)),
                         c > 0 || kk >= NACC);
        }
        mma_commit(&h.aempty[b]);
      }
      mma_commit(&h.ddone);
    }
    __syncwarp();
  }

  griddep_launch_dependents();
  // ---- epilogue: accumulators -> per-row partial sums -> owner CTA ----------
  griddep_wait();  // outputs may still be read by the previous kernel until it completes
  cluster_wait();  // every CTA of the cluster has started
  if (warp < 4) {
    const bool ok = mbar_wait(&h.ddone, 0, &h.err, a.wait_cycles);
    tc_fence_after();
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    const int i = tid;  // block row
    const int owner = i / slice;
    // One block of 16 accumulator columns at a time (the accumulators summed
    // in a fixed order), then the tokens whose terms lie in the block.
    constexpr int NT = PHASE == 1 ? 1 : TERMS;  // B rows per token
    static_assert(16 % NT == 0, "a token's terms must lie in one block of 16 columns");
    constexpr int TPB = 16 / NT;  // tokens per block
#pragma unroll
    for (int cb = 0; cb < N / 16; ++cb) {
      if (cb * TPB >= T) break;
      float acc[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) acc[j] = 0.f;
#pragma unroll
      for (int d = 0; d < NACC; ++d) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + (uint32_t)(DCOL + d * N + cb * 16), r);
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
        for (int j = 0; j < 16; ++j) acc[j] += __uint_as_float(r[j]);
      }
      if (ok) {
#pragma unroll
        for (int tl = 0; tl < TPB; ++tl) {
          const int t = cb * TPB + tl;
          if (t < T) {
            float p = acc[NT * tl];
#pragma unroll
            for (int q = 1; q < NT; ++q) p += acc[NT * tl + q];
            st_cluster_f32(recv + ((ks * T + t) * slice + (i - owner * slice)), (uint32_t)owner, p);
          }
        }
      }
    }
  }
  // All partials of the cluster have landed in their owners' buffers.
  cluster_sync();
  const int cnt = min(slice, kBlockRows - my0);
  for (int idx = tid; idx < T * cnt; idx += kThreads) {
    const int t = idx / cnt;
    const int i = idx - t * cnt;
    const int64_t row = row0 + my0 + i;
    if (row >= a.sm.R) continue;
    float v = 0.f;
    for (int q = 0; q < KS; ++q) v += recv[(q * T + t) * slice + i];
    const float out = v * rs[i];
    if (PHASE == 1) {
      a.sout[(int64_t)t * a.lds + row] = out;
    } else if (a.ydtype == 0) {
      reinterpret_cast<__half*>(a.y)[(int64_t)t * a.ldy + row] = __float2half_rn(out);
    } else {
      reinterpret_cast<float*>(a.y)[(int64_t)t * a.ldy + row] = out;
    }
  }

  // ---- teardown ---------------------------------------------------------------
  tc_fence_before();
  __syncthreads();
  if (tid == 128 && h.err != 0) {
    // Something timed out: let the bulk copies drain (bounded) so that none
    // lands after the CTA has exited, and report it.
    for (int c = 0; c < nch; ++c) mbar_wait(&h.wfull[c], 0, &h.err, a.wait_cycles);
    atomicOr(a.status, kStatusTimeout);
  }
  if (warp == 4) {
    tc_fence_after();
    if (lane == 0) mbar_wait(&h.ddone, 0, &h.err, a.wait_cycles);  // no MMA may still read tensor memory
    __syncwarp();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)kTmemCols)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// Prep kernel: the B operand of every K slice of a pass, built once per slice
// instead of once per row block (the split of a pass of T tokens into 4T
// e4m3 terms costs about 40 instructions per value and grows with T, while
// the decode CTAs of one slice all need the same tiles). CTA ks = slice ks,
// 128 threads.
// ---------------------------------------------------------------------------

struct __align__(8) PrepHeader {
  uint64_t xfull;  // staged activations have landed (bulk copies)
  uint32_t err;
  uint32_t maxbits[kMaxPassTokens];
};

struct PrepSmem {
  int act, qpart, hdr, total;
};

__host__ __device__ inline PrepSmem prep_smem(int phase, int CPC, int T) {
  PrepSmem p;
  int off = 0;
  p.act = off;
  off = align128(off + T * CPC * kChunkCols * (phase == 1 ? 2 : 4));
  p.qpart = off;
  off = align128(off + T * 128 * 4);
  p.hdr = off;
  off = align128(off + (int)sizeof(PrepHeader));
  p.total = off + 128;  // slack for aligning the base to 128 bytes
  return p;
}

template <int PHASE, int N>
__global__ void __launch_bounds__(128) bprep_kernel(const DecodeArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 127) & ~(uintptr_t)127);
  const int T = a.tokens;
  const PrepSmem sp = prep_smem(PHASE, a.CPC, T);
  uint8_t* act = smem + sp.act;
  float* qpart = reinterpret_cast<float*>(smem + sp.qpart);
  PrepHeader& h = *reinterpret_cast<PrepHeader*>(smem + sp.hdr);
  const int bt = threadIdx.x, ks = blockIdx.x;
  const int c0 = ks * a.CPC;
  const int nch = min(a.CPC, a.sm.NCH - c0);
  const int64_t k0 = (int64_t)c0 * kChunkCols;
  if (bt == 0) {
    mbar_init(&h.xfull, 1);
    h.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (bt < kMaxPassTokens) h.maxbits[bt] = 0u;
  __syncthreads();
  // The decode kernel that consumes the tiles starts now: its sign copies and
  // expansion into tensor memory do not depend on this kernel.
  griddep_launch_dependents();
  griddep_wait();  // activations are written by the previous kernel
  build_b<PHASE, N>(a, T, nch, k0, bt, act, a.bbuf + (int64_t)c0 * N * 128, qpart, h.maxbits, &h.xfull, &h.err);
  builders_sync();
  if (bt < T) {
    float qs = 0.f;
    for (int j = 0; j < 128; ++j) qs += qpart[bt * 128 + j];
    float sc, is;
    pow2_scale(__uint_as_float(h.maxbits[bt]), &sc, &is);
    a.bstats[ks * kMaxPassTokens + bt] = make_float2(is, qs * is);
  }
  // The tiles are read by bulk copies (async proxy) in the next kernel.
  asm volatile("fence.proxy.async.global;" ::: "memory");
  __syncthreads();
  if (bt == 0 && h.err != 0) {
    if (staged_acts(N)) mbar_wait(&h.xfull, 0, &h.err, a.wait_cycles);
    atomicOr(a.status, kStatusTimeout);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

struct DecodePlan {
  int N = 0, KS = 0, CPC = 0, smem = 0;
  bool ok = false;
};

int n_for_tokens(int T) { return T <= 4 ? 16 : T <= 8 ? 32 : 64; }

constexpr int kTwoPerSmSmem = 110 * 1024;  // at or below this, two CTAs share an SM

// Split of one sign matrix for a pass of T tokens: about one CTA per SM
// (row blocks x KS <= SMs), KS <= 16 CTAs per cluster, and the CTA's chunks
// within the shared-memory budget. The first finer split whose CTAs are
// small enough for two per SM is taken when it lowers waves x chunks per CTA
// (the streaming time of the slowest SM): two CTAs per SM overlap their
// streaming of signs into tensor memory (measured: 28672x8192 at one token
// 62.0 -> 42.1 us, 14336x4096 at 16 tokens 86.3 -> 57.0 us). Then, while a
// CTA streams more chunks than its A ring holds, K is split twice as finely
// (portable clusters, at most two CTAs per SM; 14336x4096 at one token
// 20.9 -> 15.2 us).
DecodePlan plan_decode(int phase, const SignMatrix& sm, int T, int num_sms, int max_smem, bool prep) {
  DecodePlan p;
  p.N = n_for_tokens(T);
  const int sms = num_sms > 0 ? num_sms : kDefaultSms;
  int ks = sms / (sm.RB > 0 ? sm.RB : 1);
  if (ks < 1) ks = 1;
  if (ks > kMaxKS) ks = kMaxKS;
  // One-token calls are latency-bound and usually run beside their sibling
  // linears (q | k | v): portable clusters of at most 8 leave SMs to them
  // (config-1 stack on the DAG schedule 10.88 -> 10.37 us per linear; the
  // k/v shape alone 8.49 -> 8.63 us), unless the CTAs would then stream more
  // chunks than their A ring holds.
  if (T == 1 && ks > 8 && (sm.NCH + 7) / 8 <= nbuf_for(p.N)) ks = 8;
  if (ks > sm.NCH) ks = sm.NCH;
  auto waves = [&](int KS, int need) {
    const int64_t slots = (int64_t)sms * (need <= kTwoPerSmSmem ? 2 : 1);
    return ((int64_t)sm.RB * KS + slots - 1) / slots;
  };
  for (; ks <= kMaxKS; ++ks) {
    const int cpc = (sm.NCH + ks - 1) / ks;
    if (cpc > kMaxCPC) continue;
    const int KS = (sm.NCH + cpc - 1) / cpc;
    const int need = decode_smem(phase, p.N, cpc, KS, T, prep).total;
    if (need <= max_smem) {
      p.KS = KS;
      p.CPC = cpc;
      p.smem = need < kMinSmem ? kMinSmem : need;
      p.ok = true;
      if (need > kTwoPerSmSmem) {
        for (int k2 = ks + 1; k2 <= kMaxKS && k2 <= sm.NCH; ++k2) {
          const int c2 = (sm.NCH + k2 - 1) / k2;
          const int K2 = (sm.NCH + c2 - 1) / c2;
          const int n2 = decode_smem(phase, p.N, c2, K2, T, prep).total;
          if (n2 <= kTwoPerSmSmem) {
            if (waves(K2, n2) * c2 < waves(p.KS, p.smem) * p.CPC) {
              p.KS = K2;
              p.CPC = c2;
              p.smem = n2 < kMinSmem ? kMinSmem : n2;
            }
            // Passes of one to four tokens take the first such split; wider
            // ones (fewer chunks fit) search every finer split.
            if (p.N <= 16) break;
          }
        }
      }
      // CTAs that stream more chunks than their tensor-memory ring holds:
      // split K further (portable clusters) while the CTA count stays within
      // two per SM.
      while (p.CPC > nbuf_for(p.N) && p.KS * 2 <= 8 && (int64_t)sm.RB * p.KS * 2 <= 2 * sms) {
        const int k2 = p.KS * 2;
        const int c2 = (sm.NCH + k2 - 1) / k2;
        const int K2 = (sm.NCH + c2 - 1) / c2;
        const int n2 = decode_smem(phase, p.N, c2, K2, T, prep).total;
        if (n2 > max_smem) break;
        p.KS = K2;
        p.CPC = c2;
        p.smem = n2 < kMinSmem ? kMinSmem : n2;
      }
      return p;
    }
  }
  return p;
}


// Split of one sign matrix for the 16-bit-operand kernel: the same rules as
// plan_decode (about one CTA per SM, KS <= 16, a finer split where it lets
// two CTAs share an SM and lowers waves x chunks per CTA, then K split
// further while a CTA streams more chunks than its A ring holds), with that
// kernel's shared memory and ring depth.
DecodePlan plan_hdecode(int phase, const SignMatrix& sm, int T, int num_sms, int max_smem) {
  DecodePlan p;
  p.N = hdecode_n(phase, T);
  const int sms = num_sms > 0 ? num_sms : kDefaultSms;
  const int nbuf = hnbuf_for(p.N);
  int ks = sms / (sm.RB > 0 ? sm.RB : 1);
  if (ks < 1) ks = 1;
  if (ks > kMaxKS) ks = kMaxKS;
  if (ks > sm.NCH) ks = sm.NCH;
  auto waves = [&](int KS, int need) {
    const int64_t slots = (int64_t)sms * (need <= kTwoPerSmSmem ? 2 : 1);
    return ((int64_t)sm.RB * KS + slots - 1) / slots;
  };
  for (; ks <= kMaxKS; ++ks) {
    const int cpc = (sm.NCH + ks - 1) / ks;
    if (cpc > kMaxCPC) continue;
    const int KS = (sm.NCH + cpc - 1) / cpc;
    const int need = hdecode_smem(p.N, cpc, KS, T).total;
    if (need > max_smem) continue;
    p.KS = KS;
    p.CPC = cpc;
    p.smem = need < kMinSmem ? kMinSmem : need;
    p.ok = true;
    if (need > kTwoPerSmSmem) {
      for (int k2 = ks + 1; k2 <= kMaxKS && k2 <= sm.NCH; ++k2) {
        const int c2 = (sm.NCH + k2 - 1) / k2;
        const int K2 = (sm.NCH + c2 - 1) / c2;
        const int n2 = hdecode_smem(p.N, c2, K2, T).total;
        if (n2 <= kTwoPerSmSmem && waves(K2, n2) * c2 < waves(p.KS, p.smem) * p.CPC) {
          p.KS = K2;
          p.CPC = c2;
          p.smem = n2 < kMinSmem ? kMinSmem : n2;
        }
      }
    }
    while (p.CPC > nbuf && p.KS * 2 <= 8 && (int64_t)sm.RB * p.KS * 2 <= 2 * sms) {
      const int k2 = p.KS * 2;
      const int c2 = (sm.NCH + k2 - 1) / k2;
      const int K2 = (sm.NCH + c2 - 1) / c2;
      const int n2 = hdecode_smem(p.N, c2, K2, T).total;
      if (n2 > max_smem) break;
      p.KS = K2;
      p.CPC = c2;
      p.smem = n2 < kMinSmem ? kMinSmem : n2;
    }
    return p;
  }
  return p;
}

template <int PHASE, int N>
cudaError_t launch_prep(const DecodeArgs& a, const DecodePlan& p, cudaStream_t st) {
  auto kern = bprep_kernel<PHASE, N>;
  const int smem = prep_smem(PHASE, p.CPC, a.tokens).total;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.KS, 1, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int PHASE, int N, bool PREP>
cudaError_t launch_decode_n(const DecodeArgs& a, const DecodePlan& p, cudaStream_t st) {
  if (PREP) {
    cudaError_t e = launch_prep<PHASE, N>(a, p, st);
    if (e != cudaSuccess) return e;
  }
  auto kern = decode_kernel<PHASE, N, PREP>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
  if (e != cudaSuccess) return e;
  if (p.KS > 8) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.sm.RB, (unsigned)p.KS, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)p.smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = (unsigned)p.KS;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

// Passes of more than 4 tokens (N > 16) build the B operand once per K slice
// in bprep_kernel when the caller's workspace holds the tiles (a.bbuf set).
template <int PHASE>
cudaError_t launch_decode(DecodeArgs a, const DecodePlan& p, cudaStream_t st) {
  a.KS = p.KS;
  a.CPC = p.CPC;
  const bool prep = a.bbuf != nullptr && p.N > 16;
  switch (p.N) {
    case 16: return launch_decode_n<PHASE, 16, false>(a, p, st);
    case 32: return prep ? launch_decode_n<PHASE, 32, true>(a, p, st) : launch_decode_n<PHASE, 32, false>(a, p, st);
    default: return prep ? launch_decode_n<PHASE, 64, true>(a, p, st) : launch_decode_n<PHASE, 64, false>(a, p, st);
  }
}

template <int PHASE, int N, int TERMS>
cudaError_t launch_hdecode_n(const DecodeArgs& a, const DecodePlan& p, cudaStream_t st) {
  auto kern = hdecode_kernel<PHASE, N, TERMS>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
  if (e != cudaSuccess) return e;
  if (p.KS > 8) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.sm.RB, (unsigned)p.KS, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)p.smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = (unsigned)p.KS;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int PHASE>
cudaError_t launch_hdecode(DecodeArgs a, const DecodePlan& p, cudaStream_t st) {
  a.KS = p.KS;
  a.CPC = p.CPC;
  if (PHASE == 1 || s2_terms(a.tokens) == 1) {
    switch (p.N) {
      case 16: return launch_hdecode_n<PHASE, 16, 1>(a, p, st);
      case 32: return launch_hdecode_n<PHASE, 32, 1>(a, p, st);
      default: return launch_hdecode_n<PHASE, 64, 1>(a, p, st);
    }
  }
  if constexpr (PHASE == 2) {
    static_assert(kS2Terms == 2, "passes of up to 16 tokens: two BF16 terms, 16 or 32 rows");
    if (p.N == 16) return launch_hdecode_n<2, 16, 2>(a, p, st);
    return launch_hdecode_n<2, 32, 2>(a, p, st);
  }
  return cudaErrorInvalidConfiguration;
}

int64_t align256(int64_t v) { return (v + 255) / 256 * 256; }

LutProblem lut_problem(const DecodeArgs& d) {
  LutProblem q = {};
  q.signs = d.signs;
  q.sm = d.sm;
  q.x = d.x;
  q.ldx = d.ldx;
  q.zin = d.zin;
  q.ldz = d.ldz;
  q.colscale = d.colscale;
  q.rowscale = d.rowscale;
  q.sout = d.sout;
  q.lds = d.lds;
  q.y = d.y;
  q.ldy = d.ldy;
  return q;
}

LutArgs lut_args(const DecodeArgs& d) {
  LutArgs a = {};
  a.count = 1;
  a.tokens = d.tokens;
  a.ydtype = d.ydtype;
  a.status = d.status;
  a.wait_cycles = d.wait_cycles;
  a.late_trigger = many_streams() ? 1 : 0;
  a.prob[0] = lut_problem(d);
  return a;
}

}  // namespace

int64_t decode_ldz(const af1_layer& L) { return (int64_t)L.p2.NCH * kChunkCols; }

int64_t swiglu_ld(const af1_layer& L) { return (L.n + 7) / 8 * 8; }

// Measured per call (us, weights streamed from HBM, one pass of the
// 16-bit-operand kernel vs the prefill kernel) at 17 / 32 / 64 tokens:
// 4096^2 (16.6 M signs) 13.2 / 15.7 / 25.2 vs 24.2 / 24.3 / 30.9;
// 1024x8192 (8.1 M) 11.3 / 13.8 / 21.6 vs 27.7 / 27.2 / 28.3; 14336x4096
// (58 M) 28.4 / 39.2 / 113 vs 41.3 / 41.5 / 45.9; 4096x14336 (58 M) 30.4 /
// 40.2 / 131 vs 42.9 / 43.0 / 47.7; 8192^2 (67 M) 25.3 / 33.3 / 79.9 vs
// 43.1 / 43.3 / 46.6; 28672x8192 (234 M) 103 / 142 / 298 vs 109 / 109 /
// 112; 8192x28672 (234 M) 171 / 227 vs 116 / 116. The one pass wins while
// its expansion of the signs into tensor memory (about 15 signs per clock
// per SM) stays short and, at 64 tokens, on small layers only (its 64-row
// tiles and 64-token epilogue multiply a larger matrix's waves; eight
// activation loads in flight per builder instead of four: 2 %).
constexpr int64_t kMidSignsShort = 70000000;  // up to 32 tokens
constexpr int64_t kMidSignsLong = 20000000;   // up to kMidMaxTokens

bool mid_pass(const af1_layer& L, int64_t tokens, bool prep) {
  if (!prep || tokens <= kMaxPassTokens || tokens > kMidMaxTokens) return false;
  if ((L.flags & (AF1_FLAG_TC_DECODE | AF1_FLAG_LUT_DECODE)) != 0) return false;
  const int64_t signs = L.r * (L.m + L.n);
  if (!((tokens <= 32 && signs <= kMidSignsShort) || signs <= kMidSignsLong)) return false;
  const int T = (int)tokens;
  return plan_hdecode(1, L.p1, T, L.num_sms, L.max_smem).ok && plan_hdecode(2, L.p2, T, L.num_sms, L.max_smem).ok;
}

Workspace plan_workspace(const af1_layer& L, int64_t tokens, bool prep, bool swiglu) {
  Workspace w;
  int64_t off = 0;
  w.status = off;
  off += 256;
  const bool mid = mid_pass(L, tokens, prep);
  w.sbuf = off;
  off += align256((mid ? tokens : (int64_t)kMaxPassTokens) * decode_ldz(L) * 4);
  if (prep && tokens > 4 && tokens <= kMaxPassTokens) {
    // Prepared B operand of the wider decode passes: every chunk's tiles at
    // the widest N (64 rows of 128 bytes) and the per-(slice, token) scales.
    const int nch = L.p1.NCH > L.p2.NCH ? L.p1.NCH : L.p2.NCH;
    w.bbuf = off;
    off += align256((int64_t)nch * 64 * 128);
    w.bstats = off;
    off += align256((int64_t)kMaxKS * kMaxPassTokens * 8);
  }
  w.hbuf = off;
  if (tokens > kMaxPassTokens && !mid) {
    const int64_t t = tokens < kPrefillPassTokens ? tokens : kPrefillPassTokens;
    off += align256(t * prefill_h_ld(L) * 2);
    if (prep) {
      w.pbuf = off;
      off += align256(prefill_part_bytes(L, tokens));
      w.pcnt = off;
      off += align256(prefill_count_bytes(L, tokens));
    }
  }
  if (swiglu) {
    const int64_t t = tokens < kPrefillPassTokens ? tokens : kPrefillPassTokens;
    w.hx = off;
    off += align256(t * swiglu_ld(L) * 2);
  }
  w.total = off;
  return w;
}

namespace {

// Kernel of one phase of a decode pass of T tokens: the e4m3 tensor-core
// kernel (tc, AF1_FLAG_TC_DECODE), the 16-bit-operand tensor-core kernel
// (mma), the streaming CUDA-core kernel (stream.ok) or the clustered one
// (lut.ok); mma also when neither CUDA-core kernel has a plan.
struct PhaseChoice {
  bool tc = false;
  bool mma = false;
  LutPlan lut;
  StreamPlan stream;
};

// Passes of more than kLutMaxTokens tokens take the 16-bit-operand
// tensor-core kernel by default. The lookup tables' work grows with the
// tokens (a table read per 4 signs per token pair, and from 5 tokens on a
// second token group of CTAs that reads every sign tile again), the MMAs'
// hardly does, but expanding signs into tensor memory costs more per sign
// than a lookup. Measured on the 32-layer HiSA-rank stack (decoder DAG, ms
// per step, lookup tables vs MMA): 4 tokens 2.56 vs 2.91, 6 tokens 3.96 vs
// 3.23, 8 tokens 4.05 vs 3.40. (Per call in isolation the MMA kernel already
// wins at 4 tokens on matrices of 8 Mi signs and more, e.g. 14336x4096 21.5
// vs 19.9 us, but loses inside the stack, where it shares the SMs with the
// sibling linears' kernels.)
constexpr int kLutMaxTokens = 4;

PhaseChoice choose_phase(const af1_layer& L, int phase, const SignMatrix& m, int T, const Workspace& W) {
  (void)W;
  PhaseChoice c;
  if ((L.flags & AF1_FLAG_TC_DECODE) != 0) {
    c.tc = true;
    return c;
  }
  if ((L.flags & AF1_FLAG_MMA_DECODE) != 0 || ((L.flags & AF1_FLAG_LUT_DECODE) == 0 && T > kLutMaxTokens)) {
    c.mma = true;
    return c;
  }
  c.lut = plan_lut(&m, 1, T, L.num_sms, L.max_smem);
  if (T <= 2) {
    // The streaming kernel where the clustered split needs more than one
    // wave of CTAs (each wave pays the CTAs' start-up and reduction), or
    // wherever it has a plan when the layer asks for it. (On one-wave
    // matrices it is faster alone but slower when several layers run at once
    // on parallel streams, as a decoder's q|k|v and gate|up do: measured.)
    const bool flag = (L.flags & AF1_FLAG_STREAM_DECODE) != 0;
    bool want = flag || !c.lut.ok;
    if (!want) {
      const int sms = L.num_sms > 0 ? L.num_sms : kDefaultSms;
      int per_sm = 233472 / (c.lut.smem + 1024);
      per_sm = per_sm > 4 ? 4 : per_sm;
      want = (int64_t)m.RB * c.lut.KS > (int64_t)sms * per_sm;
    }
    if (want) c.stream = plan_stream(phase, m, T, L.num_sms, L.max_smem);
  }
  if (!c.stream.ok && !c.lut.ok) c.mma = true;
  return c;
}

}  // namespace

cudaError_t launch_forward(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y,
                           int64_t ldy, int y_dtype, void* ws, cudaStream_t st, bool prep, unsigned* status,
                           const void* x2) {
  const Workspace W = plan_workspace(L, tokens, prep, x2 != nullptr);
  uint8_t* wsb = static_cast<uint8_t*>(ws);
  unsigned* stat = status != nullptr ? status : reinterpret_cast<unsigned*>(wsb + W.status);
  const int ysize = y_dtype == 0 ? 2 : 4;
  const __half* gx = static_cast<const __half*>(x);
  const __half* ux = static_cast<const __half*>(x2);
  __half* hx = x2 != nullptr ? reinterpret_cast<__half*>(wsb + W.hx) : nullptr;
  const int64_t ldh = swiglu_ld(L);
  const bool mid = mid_pass(L, tokens, prep);
  if (tokens > kMaxPassTokens && !mid) {
    // Prefill: two tensor-core GEMMs per pass (af1_prefill.cu); the SwiGLU
    // input is formed first, one pass of tokens at a time.
    float* part = W.pbuf != 0 ? reinterpret_cast<float*>(wsb + W.pbuf) : nullptr;
    unsigned* count = W.pcnt != 0 ? reinterpret_cast<unsigned*>(wsb + W.pcnt) : nullptr;
    if (x2 == nullptr) return launch_prefill(L, x, ldx, tokens, y, ldy, y_dtype, wsb + W.hbuf, part, count, stat, st);
    for (int64_t t0 = 0; t0 < tokens; t0 += kPrefillPassTokens) {
      const int64_t T = (tokens - t0) < kPrefillPassTokens ? (tokens - t0) : kPrefillPassTokens;
      cudaError_t e = launch_swiglu(gx + t0 * ldx, ux + t0 * ldx, ldx, T, L.n, hx, ldh, st);
      if (e == cudaSuccess)
        e = launch_prefill(L, hx, ldh, T, static_cast<uint8_t*>(y) + t0 * ldy * ysize, ldy, y_dtype, wsb + W.hbuf,
                           part, count, stat, st);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  }
  // Widest pass whose plans fit (16 tokens normally; fewer only for very
  // long contractions; a mid pass takes all its tokens at once, its plans
  // checked by mid_pass).
  int pass = mid ? (int)tokens : kMaxPassTokens;
  bool fits = mid;
  for (; !mid;) {
    const int T = (int)(tokens < pass ? tokens : pass);
    fits = plan_decode(1, L.p1, T, L.num_sms, L.max_smem, false).ok &&
           plan_decode(2, L.p2, T, L.num_sms, L.max_smem, false).ok;
    if (fits) {
      // The 16-bit-operand kernel's B tiles grow with the pass (2 T rows in
      // phase 2): its plans must fit too where it would run.
      const PhaseChoice c1 = choose_phase(L, 1, L.p1, T, W), c2 = choose_phase(L, 2, L.p2, T, W);
      if (c1.mma && !plan_hdecode(1, L.p1, T, L.num_sms, L.max_smem).ok) fits = false;
      if (c2.mma && !plan_hdecode(2, L.p2, T, L.num_sms, L.max_smem).ok) fits = false;
    }
    if (fits || pass <= 4) break;
    pass /= 2;
  }
  if (!fits) return cudaErrorInvalidConfiguration;
  for (int64_t t0 = 0; t0 < tokens; t0 += pass) {
    const int T = (int)((tokens - t0) < pass ? (tokens - t0) : pass);
    PhaseChoice c1 = choose_phase(L, 1, L.p1, T, W), c2 = choose_phase(L, 2, L.p2, T, W);
    // When the second phase streams, the first streams too (measured on the
    // LLaMA-70B 28672 x 8192 matrix at one token: 22.5 -> 18.7 us per call;
    // the converse, a streamed first phase pulling the second along, was
    // slower on 8192 x 28672: 21.7 -> 24.1 us).
    if (!c1.tc && !c1.mma && !c1.stream.ok && c2.stream.ok)
      c1.stream = plan_stream(1, L.p1, T, L.num_sms, L.max_smem);
    DecodePlan q1, q2;
    const bool prep = W.bbuf != 0 && n_for_tokens(T) > 16;  // launch_decode prepares B then
    if (c1.tc) q1 = plan_decode(1, L.p1, T, L.num_sms, L.max_smem, prep);
    if (c2.tc) q2 = plan_decode(2, L.p2, T, L.num_sms, L.max_smem, prep);
    if (c1.mma) q1 = plan_hdecode(1, L.p1, T, L.num_sms, L.max_smem);
    if (c2.mma) q2 = plan_hdecode(2, L.p2, T, L.num_sms, L.max_smem);
    if (((c1.tc || c1.mma) && !q1.ok) || ((c2.tc || c2.mma) && !q2.ok)) return cudaErrorInvalidConfiguration;

    DecodeArgs a1 = {};
    a1.signs = L.signs1;
    a1.sm = L.p1;
    a1.tokens = T;
    a1.x = static_cast<const __half*>(x) + t0 * ldx;
    a1.ldx = ldx;
    a1.colscale = reinterpret_cast<const __half*>(L.b);
    a1.rowscale = reinterpret_cast<const __half*>(L.s);
    a1.sout = reinterpret_cast<float*>(wsb + W.sbuf);
    a1.lds = decode_ldz(L);
    a1.status = stat;
    a1.wait_cycles = wait_budget();
    a1.bbuf = W.bbuf != 0 ? wsb + W.bbuf : nullptr;
    a1.bstats = W.bbuf != 0 ? reinterpret_cast<float2*>(wsb + W.bstats) : nullptr;
    cudaError_t e = cudaSuccess;
    // SwiGLU input: the CUDA-core kernels form h while staging; the
    // tensor-core kernel reads it from the workspace.
    const __half* u1 = x2 != nullptr ? ux + t0 * ldx : nullptr;
    if (u1 != nullptr && (c1.tc || c1.mma)) {
      e = launch_swiglu(a1.x, u1, ldx, T, L.n, hx, ldh, st);
      if (e != cudaSuccess) return e;
      a1.x = hx;
      a1.ldx = ldh;
    }
    if (c1.tc) {
      e = launch_decode<1>(a1, q1, st);
    } else if (c1.mma) {
      e = launch_hdecode<1>(a1, q1, st);
    } else if (c1.stream.ok) {
      LutProblem q = lut_problem(a1);
      q.x2 = u1;
      e = launch_stream(1, q, T, 0, c1.stream, stat, st);
    } else {
      LutArgs la = lut_args(a1);
      la.prob[0].x2 = u1;
      e = launch_lut(1, la, c1.lut, st);
    }
    if (e != cudaSuccess) return e;

    DecodeArgs a2 = {};
    a2.signs = L.signs2;
    a2.sm = L.p2;
    a2.tokens = T;
    a2.zin = a1.sout;
    a2.ldz = a1.lds;
    a2.rowscale = reinterpret_cast<const __half*>(L.a);
    a2.y = static_cast<uint8_t*>(y) + t0 * ldy * ysize;
    a2.ldy = ldy;
    a2.ydtype = y_dtype;
    a2.status = a1.status;
    a2.wait_cycles = a1.wait_cycles;
    a2.bbuf = a1.bbuf;
    a2.bstats = a1.bstats;
    e = c2.tc          ? launch_decode<2>(a2, q2, st)
        : c2.mma       ? launch_hdecode<2>(a2, q2, st)
        : c2.stream.ok ? launch_stream(2, lut_problem(a2), T, y_dtype, c2.stream, stat, st)
                       : launch_lut(2, lut_args(a2), c2.lut, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}


}  // namespace af1

extern "C" int af1_mma_plan_dry(int phase, int64_t R, int64_t C, int64_t tokens, int num_sms, int max_smem,
                                int32_t* out) {
  using namespace af1;
  if (out == nullptr || (phase != 1 && phase != 2) || R < 1 || R > ((int64_t)1 << 30) || C < 1 || C > kMaxCols ||
      tokens < 1 || tokens > kMidMaxTokens || num_sms < 1 || max_smem < 1)
    return set_error(AF1_ERR_INVALID_ARG, "af1_mma_plan_dry: argument out of range");
  const SignMatrix sm = make_sign_matrix(R, C);
  const DecodePlan p = plan_hdecode(phase, sm, (int)tokens, num_sms, max_smem);
  const int nacc = hnacc_for(p.N), nbuf = hnbuf_for(p.N);
  const int32_t v[10] = {p.N, nacc, nbuf, nacc * p.N + nbuf * 64, p.KS, p.CPC, p.smem, sm.RB, p.KS, p.ok ? 1 : 0};
  for (int i = 0; i < 10; ++i) out[i] = v[i];
  return AF1_OK;
}

namespace af1 {

int64_t multi_workspace_offset(const af1_layer* const* Ls, int i, int64_t tokens, bool prep) {
  int64_t off = 0;
  for (int j = 0; j < i; ++j) off += align256(plan_workspace(*Ls[j], tokens, prep).total);
  return off;
}

cudaError_t launch_forward_multi(const af1_layer* const* Ls, int count, const void* x, int64_t ldx, int64_t tokens,
                                 void* const* ys, const int64_t* ldys, int y_dtype, void* ws, cudaStream_t st,
                                 bool prep) {
  uint8_t* wsb = static_cast<uint8_t*>(ws);
  unsigned* status = reinterpret_cast<unsigned*>(wsb);  // layer 0's slice starts with its status word
  const int T = (int)tokens;
  // One launch per phase for all layers when every phase of every layer
  // would run on the clustered lookup-table kernel anyway and the group has
  // a plan.
  bool group = tokens <= kMaxPassTokens;
  SignMatrix m1[kMaxGroup], m2[kMaxGroup];
  for (int i = 0; i < count && group; ++i) {
    const af1_layer& L = *Ls[i];
    const Workspace W = plan_workspace(L, tokens, prep);
    const PhaseChoice c1 = choose_phase(L, 1, L.p1, T, W), c2 = choose_phase(L, 2, L.p2, T, W);
    if (c1.tc || c2.tc || c1.mma || c2.mma || c1.stream.ok || c2.stream.ok) group = false;
    m1[i] = L.p1;
    m2[i] = L.p2;
  }
  LutPlan g1, g2;
  if (group) {
    g1 = plan_lut(m1, count, T, Ls[0]->num_sms, Ls[0]->max_smem);
    g2 = plan_lut(m2, count, T, Ls[0]->num_sms, Ls[0]->max_smem);
    group = g1.ok && g2.ok;
  }
  if (!group) {
    // One call per layer, each with its own workspace slice, all reporting to
    // the first slice's status word.
    for (int i = 0; i < count; ++i) {
      const int64_t off = multi_workspace_offset(Ls, i, tokens, prep);
      cudaError_t e = launch_forward(*Ls[i], x, ldx, tokens, ys[i], ldys[i], y_dtype, wsb + off, st, prep, status);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  }
  LutArgs a1 = {}, a2 = {};
  a1.count = a2.count = count;
  a1.tokens = a2.tokens = T;
  a1.ydtype = a2.ydtype = y_dtype;
  a1.status = a2.status = status;
  a1.wait_cycles = a2.wait_cycles = wait_budget();
  a1.late_trigger = a2.late_trigger = many_streams() ? 1 : 0;
  for (int i = 0; i < count; ++i) {
    const af1_layer& L = *Ls[i];
    const Workspace W = plan_workspace(L, tokens, prep);
    float* sbuf = reinterpret_cast<float*>(wsb + multi_workspace_offset(Ls, i, tokens, prep) + W.sbuf);
    LutProblem& q1 = a1.prob[i];
    q1.signs = L.signs1;
    q1.sm = L.p1;
    q1.x = static_cast<const __half*>(x);
    q1.ldx = ldx;
    q1.colscale = reinterpret_cast<const __half*>(L.b);
    q1.rowscale = reinterpret_cast<const __half*>(L.s);
    q1.sout = sbuf;
    q1.lds = decode_ldz(L);
    LutProblem& q2 = a2.prob[i];
    q2.signs = L.signs2;
    q2.sm = L.p2;
    q2.zin = sbuf;
    q2.ldz = decode_ldz(L);
    q2.rowscale = reinterpret_cast<const __half*>(L.a);
    q2.y = ys[i];
    q2.ldy = ldys[i];
  }
  cudaError_t e = launch_lut(1, a1, g1, st);
  if (e != cudaSuccess) return e;
  return launch_lut(2, a2, g2, st);
}

}  // namespace af1
