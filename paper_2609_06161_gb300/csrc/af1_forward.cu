// af1_forward.cu — forward pass of an AF1 binary-factorized linear layer on
// sm_103a: y = a * (U (s * (V^T (b * x)))), the right-to-left evaluation of
// AF1 Eq. final_reconstruction / Eq. double_factor_equiv that never forms the
// dense W_hat.
//
// Two kernels per pass of up to 16 tokens, chained with programmatic
// dependent launch (PDL):
//   phase 1: t = B z with B = V^T (r x n) and z = b * x; then s' = s * t
//            (the rank scale), written as FP32 to the workspace.
//   phase 2: u = U s' (m x r); then y = a * u, stored as FP16 or FP32.
// Each phase is a sign-matrix product over an R x C tile matrix
// (af1_layout.h). A CTA owns a block of RTC row tiles x KTC column tiles; the
// KS CTAs that share a row block form one thread-block cluster and reduce
// their split-K partial sums through distributed shared memory (each CTA
// finalises 1/KS of the rows, summing the KS partials in a fixed order), so
// there are no global atomics and the result is deterministic. Every CTA
// issues bulk copies (cp.async.bulk) of its whole weight block and loads its
// scales before it waits on the previous kernel, so weight streaming overlaps
// the dependency.
//
// Sign contraction on FP8 tensor cores. A sign bit is expanded into an e4m3
// A-fragment byte with one LOP3 per 4 signs: (word & mask_p) | base_p puts
// the bit at a fixed position p of a constant byte, giving A = L_p + d_p * bit
// with L_p, d_p powers of two (mantissa bits 0..2, exponent bit 0, sign bit).
// With z'_k = z_k / d_k the MMA yields D = sum_k L_k z'_k + sum_k bit_k z_k,
// and since sign = 2 bit - 1,
//     sum_k sign_k z_k = 2 D - Q,   Q = sum_k (L_k + H_k) z'_k   (H = L + d).
// Each activation z'_k is scaled by a per-(CTA, token) power of two so that
// the largest magnitude sits in [128, 256), and is split into 4 e4m3 terms
// (z' ~ t1 + t2 + t3 + t4, ~16 significant bits) that occupy the 8 columns of
// an m16n8k32 MMA (2 tokens x 4 terms). Products are exact and the MMA
// accumulates in FP32, so the only rounding is the term split and FP32
// summation.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1_internal.h"
#include "af1_layout.h"

namespace af1 {
namespace {

constexpr long long kWaitCycles = 2000000000ll;  // ~1 s at 2 GHz
constexpr unsigned kStatusTimeout = 1u;
constexpr int kMaxWarps = 16;

// ---------------------------------------------------------------------------
// PTX helpers (hand-written: mbarrier, bulk copy, PDL, cluster, MMA, FP8)
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
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

// Bounded wait: false if the barrier did not complete within kWaitCycles.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) return false;
  }
  return true;
}

__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Split cluster barrier used only to know that every CTA of the cluster has
// started (required before its shared memory may be written remotely).
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.aligned;" ::: "memory"); }

// Cluster-wide barrier with release/acquire semantics for shared memory.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Store a float into the shared memory of CTA `rank` of this cluster, at the
// offset that `local` has in this CTA.
__device__ __forceinline__ void st_cluster_f32(float* local, uint32_t rank, float v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(v) : "memory");
}

__device__ __forceinline__ void mma_e4m3(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
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

// Slot p of a word (see af1_layout.h): 1 / d_p and L_p + H_p.
//   p:        0     1     2     3     4     5     6     7
//   d_p:    1/8   1/4   1/2   1/2   1/4   1/2   1/2    -2
//   L_p:      1     1     1   1/2     1     1   1/2     1
__constant__ float c_inv_delta[8] = {8.f, 4.f, 2.f, 2.f, 4.f, 2.f, 2.f, -0.5f};
__constant__ float c_lph[8] = {2.125f, 2.25f, 2.5f, 1.5f, 2.25f, 2.5f, 1.5f, 0.f};

// Expand one lane word into its 8 e4m3 A-fragment registers.
__device__ __forceinline__ void expand_word(uint32_t w, uint32_t (&s)[8]) {
  const uint32_t v = w >> 3;
  s[0] = (w & 0x01010101u) | 0x38383838u;  // mantissa bit 0: {1, 1.125}
  s[1] = (w & 0x02020202u) | 0x38383838u;  // mantissa bit 1: {1, 1.25}
  s[2] = (w & 0x04040404u) | 0x38383838u;  // mantissa bit 2: {1, 1.5}
  s[3] = (w & 0x08080808u) | 0x30303030u;  // exponent bit 0: {0.5, 1}
  s[4] = (v & 0x02020202u) | 0x38383838u;  // word bit 4 -> mantissa bit 1
  s[5] = (v & 0x04040404u) | 0x38383838u;  // word bit 5 -> mantissa bit 2
  s[6] = (v & 0x08080808u) | 0x30303030u;  // word bit 6 -> exponent bit 0
  s[7] = (w & 0x80808080u) | 0x38383838u;  // sign bit: {1, -1}
}

// ---------------------------------------------------------------------------
// Kernel arguments and shared-memory plan
// ---------------------------------------------------------------------------

struct PhaseArgs {
  const uint8_t* tiles;
  TileMatrix tm;
  int tokens;
  // phase 1 input: z = colscale * x (FP16)
  const __half* x;
  int64_t ldx;
  const __half* colscale;
  // phase 2 input: z = zin (FP32)
  const float* zin;
  int64_t ldz;
  unsigned* status;
  // finalisation: out = rowscale * (sum over the row)
  const __half* rowscale;
  float* sout;  // phase 1
  int64_t lds;
  void* y;  // phase 2
  int64_t ldy;
  int ydtype;
};

struct SmemHeader {
  uint64_t mbar[kMaxKTC];
  float maxv[kMaxPassTokens * kMaxWarps];  // per-warp max |z / d| per token
  float qpart[kMaxPassTokens * kMaxWarps]; // per-warp partial Q per token
  float sc[kMaxPassTokens];                // 2^sigma per token (0 for padding slots)
  float qis[kMaxPassTokens];               // Q * 2^-sigma per token
  float is[kMaxPassTokens];                // 2^-sigma per token
};
constexpr int kHeaderBytes = ((int)sizeof(SmemHeader) + 127) / 128 * 128;

// Rows of a block that each of the KS CTAs of a cluster finalises.
__host__ __device__ inline int slice_rows(int rtc, int ks_count) {
  return (rtc * kTileRows + ks_count - 1) / ks_count;
}

struct SmemPlan {
  int frag, wts, recv, rs, bi, red, total;
};

__host__ __device__ inline int align128(int v) { return (v + 127) / 128 * 128; }

// Shared-memory regions of one CTA; every region starts on a 128-byte
// boundary (bulk-copy destinations and vector accesses need >= 16 bytes).
__host__ __device__ inline SmemPlan smem_plan(const TileMatrix& tm, int ng) {
  SmemPlan p;
  const int slice = slice_rows(tm.RTC, tm.KS);
  int off = kHeaderBytes;
  p.frag = off;
  off = align128(off + tm.KTC * 4 * ng * 256);
  p.wts = off;
  off = align128(off + tm.RTC * tm.KTC * kTileBytes);
  p.recv = off;  // [KS][2 * ng][slice] partial sums pushed by the cluster
  off = align128(off + tm.KS * 2 * ng * slice * 4);
  p.rs = off;
  off = align128(off + slice * 4);
  p.bi = off;
  off = align128(off + tm.KTC * kTileCols * 4);
  p.red = off;  // [WK][2 * ng][rows of the block], WK * rows <= 16 warps x 16 rows
  off = align128(off + kMaxWarps * 2 * ng * kTileRows * 4);
  p.total = off;
  return p;
}

// Four consecutive activations of one token (zero beyond column C). The
// inputs may have been written by the kernel this one overlaps with through
// programmatic dependent launch, so they are read through L2 (ld.global.cg),
// never through the non-coherent L1/texture path.
template <int PHASE>
__device__ __forceinline__ float4 load_z4(const PhaseArgs& a, int tok, int64_t k) {
  const int64_t C = a.tm.C;
  float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  if (PHASE == 1) {
    const __half* p = a.x + (int64_t)tok * a.ldx + k;
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
    const float* p = a.zin + (int64_t)tok * a.ldz + k;
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

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// The power of two 2^sigma that brings a positive maximum m into [128, 256),
// read from m's exponent field (m = f 2^e with f in [0.5, 1), sigma = 8 - e).
// m comes from products of FP16 values, so 127 +- sigma stays a normal
// exponent. Returns 2^sigma in *sc and 2^-sigma in *is; m == 0 gives 1, 1.
__device__ __forceinline__ void pow2_scale(float m, float* sc, float* is) {
  if (!(m > 0.f)) {
    *sc = 1.f;
    *is = 1.f;
    return;
  }
  const int e = (int)((__float_as_uint(m) >> 23) & 0xFFu) - 126;
  const int sigma = min(8 - e, 120);  // FP32-subnormal maxima (not produced by FP16 inputs) stay in range
  *sc = __uint_as_float((uint32_t)(127 + sigma) << 23);
  *is = __uint_as_float((uint32_t)(127 - sigma) << 23);
}

// Build the e4m3 B fragments of this CTA's column range for all token slots
// (2 * NG). bi[kl] holds colscale * (1 / d) (phase 1) or 1 / d (phase 2), and
// 0 beyond column C (staged and published by the caller). Each thread owns
// one group of 4 columns (the block has at most 16 x 128 columns, i.e. 512
// groups, and the CTA has WARPS * 32 >= 512 threads when NG <= 2; with
// 8 warps a thread owns up to two groups). Two CTA barriers: after the
// maxima and after the fragments.
template <int PHASE, int NG, int WARPS>
__device__ void build_fragments(const PhaseArgs& a, SmemHeader& h, uint32_t* frag32, const float* bi, int64_t k0,
                                int ncols) {
  constexpr int NT = 2 * NG;
  constexpr int NTH = WARPS * 32;
  constexpr bool STASH = NT <= 4;  // keep z * bi in registers between the passes
  const int T = a.tokens;
  const int n4 = ncols >> 2;
  const bool one = n4 <= NTH;      // each thread owns at most one group of 4 columns
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float4 zs[STASH ? NT : 1];
#pragma unroll
  for (int tok = 0; tok < NT; ++tok) {
    if (STASH) zs[tok] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (tok < T) {
      float mx = 0.f;
      for (int c4 = threadIdx.x; c4 < n4; c4 += NTH) {
        const float4 z = load_z4<PHASE>(a, tok, k0 + 4 * c4);
        const float4 w = *reinterpret_cast<const float4*>(bi + 4 * c4);
        const float4 zb = make_float4(z.x * w.x, z.y * w.y, z.z * w.z, z.w * w.w);
        if (STASH) zs[tok] = zb;
        mx = fmaxf(mx, fmaxf(fmaxf(fabsf(zb.x), fabsf(zb.y)), fmaxf(fabsf(zb.z), fabsf(zb.w))));
      }
      mx = warp_max(mx);
      if (lane == 0) h.maxv[tok * WARPS + warp] = mx;
    }
  }
  __syncthreads();
  if (threadIdx.x < NT) {
    // One thread per token slot: block maximum -> 2^sigma, 2^-sigma.
    float m = 0.f;
    if ((int)threadIdx.x < T)
      for (int w = 0; w < WARPS; ++w) m = fmaxf(m, h.maxv[threadIdx.x * WARPS + w]);
    float sc, is;
    pow2_scale(m, &sc, &is);
    h.sc[threadIdx.x] = (int)threadIdx.x < T ? sc : 0.f;
    h.is[threadIdx.x] = (int)threadIdx.x < T ? is : 0.f;
  }
  __syncthreads();
#pragma unroll
  for (int tok = 0; tok < NT; ++tok) {
    const float sc = h.sc[tok];
    const int gam = tok >> 1, tb = (tok & 1) * 4;
    float q = 0.f;
    for (int c4 = threadIdx.x; c4 < n4; c4 += NTH) {
      float4 zb = make_float4(0.f, 0.f, 0.f, 0.f);
      if (tok < T) {
        if (STASH && one) {
          zb = zs[tok];
        } else {
          const float4 z = load_z4<PHASE>(a, tok, k0 + 4 * c4);
          const float4 w = *reinterpret_cast<const float4*>(bi + 4 * c4);
          zb = make_float4(z.x * w.x, z.y * w.y, z.z * w.z, z.w * w.w);
        }
      }
      float4 v = make_float4(zb.x * sc, zb.y * sc, zb.z * sc, zb.w * sc);
      const float4 v0 = v;
      const int kt_l = c4 >> 5, mu = (c4 >> 3) & 3, breg = (c4 >> 2) & 1, c = c4 & 3;
      uint32_t* dst = frag32 + ((((kt_l * 4 + mu) * NG + gam) * 32 + 4 * tb + c) * 2 + breg);
#pragma unroll
      for (int term = 0; term < kTerms; ++term) {
        const uint32_t lo = e4m3x2(v.x, v.y), hi = e4m3x2(v.z, v.w);
        const float2 blo = e4m3x2_value(lo), bhi = e4m3x2_value(hi);
        v.x -= blo.x;
        v.y -= blo.y;
        v.z -= bhi.x;
        v.w -= bhi.y;
        dst[term * 4 * 2] = lo | (hi << 16);  // column g = tb + term: 4 lanes per g
      }
      q += c_lph[(c4 >> 2) & 7] * (((v0.x - v.x) + (v0.y - v.y)) + ((v0.z - v.z) + (v0.w - v.w)));
    }
    q = warp_sum(q);
    if (lane == 0) h.qpart[tok * WARPS + warp] = q;
  }
  __syncthreads();
  if (threadIdx.x < NT) {
    float q = 0.f;
    for (int w = 0; w < WARPS; ++w) q += h.qpart[threadIdx.x * WARPS + w];
    h.qis[threadIdx.x] = q * h.is[threadIdx.x];
  }
  __syncthreads();
}

template <int PHASE, int NG, int WARPS, int TPP>
__global__ void __launch_bounds__(WARPS * 32) phase_kernel(const PhaseArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  SmemHeader& h = *reinterpret_cast<SmemHeader*>(smem);
  const TileMatrix& tm = a.tm;
  const SmemPlan sp = smem_plan(tm, NG);
  uint32_t* frag32 = reinterpret_cast<uint32_t*>(smem + sp.frag);
  uint8_t* wts = smem + sp.wts;
  float* recv = reinterpret_cast<float*>(smem + sp.recv);
  float* rs = reinterpret_cast<float*>(smem + sp.rs);
  float* bi = reinterpret_cast<float*>(smem + sp.bi);
  float* red = reinterpret_cast<float*>(smem + sp.red);

  const int rg = blockIdx.x, ks = blockIdx.y, KS = gridDim.y;
  const int rtc = blk_rows(tm, rg), ktc = blk_cols(tm, ks);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t row0 = (int64_t)rg * tm.RTC * kTileRows;
  const int64_t k0 = (int64_t)ks * tm.KTC * kTileCols;
  const int nrows = rtc * kTileRows;       // rows of this block
  const int slice = slice_rows(rtc, KS);   // rows finalised per CTA
  const int my0 = ks * slice;              // first block row this CTA finalises

  cluster_arrive_relaxed();  // this CTA has started (matched by cluster_wait)
  // The block's column tiles arrive in at most kMaxKTC bulk copies (one
  // mbarrier each) of `cpt` column tiles.
  const int cpt = (ktc + kMaxKTC - 1) / kMaxKTC;
  const int nchunks = (ktc + cpt - 1) / cpt;
  if (tid == 0) {
    // Barriers and weight copies; the CTA barrier below publishes the
    // initialised barriers to the other warps.
    const uint32_t per_kt = (uint32_t)rtc * kTileBytes;
    const uint8_t* gblk = a.tiles + blk_base(tm, rg, ks) * kTileBytes;
    for (int i = 0; i < nchunks; ++i) mbar_init(&h.mbar[i], 1);
    fence_barrier_init();
    for (int i = 0; i < nchunks; ++i) {
      const int kts = min(cpt, ktc - i * cpt);
      const uint32_t bytes = per_kt * (uint32_t)kts;
      mbar_expect_tx(&h.mbar[i], bytes);
      bulk_g2s(wts + (size_t)i * cpt * per_kt, gblk + (size_t)i * cpt * per_kt, bytes, &h.mbar[i]);
    }
  }
  // Layer constants: row scales of the rows this CTA finalises, column
  // factors of its column slice.
  for (int i = tid; i < slice; i += WARPS * 32) {
    const int64_t row = row0 + my0 + i;
    rs[i] = (my0 + i < nrows && row < tm.R) ? __half2float(a.rowscale[row]) : 0.f;
  }
  for (int i = tid; i < ktc * kTileCols; i += WARPS * 32) {
    const int64_t k = k0 + i;
    float v = 0.f;
    if (k < tm.C) v = c_inv_delta[(i & 127) >> 4] * (PHASE == 1 ? __half2float(a.colscale[k]) : 1.f);
    bi[i] = v;
  }
  // Everything above is independent of earlier kernels; everything below
  // may read their outputs.
  griddep_launch_dependents();
  griddep_wait();
  __syncthreads();  // rs / bi staged by all warps are read by every warp below

  build_fragments<PHASE, NG, WARPS>(a, h, frag32, bi, k0, ktc * kTileCols);
  // Every CTA of the cluster has started, so partials may be pushed into
  // peers' shared memory from here on.
  cluster_wait();

  const int g = lane >> 2, c = lane & 3;
  const int T = a.tokens;
  // Warps split the block into WR row-tile classes x WK column-tile classes.
  int WK = WARPS / rtc;
  if (WK < 1) WK = 1;
  if (WK > ktc) WK = ktc;
  const int WR = WARPS / WK;
  const int wr = warp / WK, wk = warp - wr * WK;
  const bool wactive = warp < WR * WK;
  // 2^-sigma and Q 2^-sigma of the tokens this lane finalises: 2 gg + (c >> 1).
  float isv[NG], qisv[NG];
#pragma unroll
  for (int gg = 0; gg < NG; ++gg) {
    const int tok = 2 * gg + (c >> 1);
    isv[gg] = h.is[tok];
    qisv[gg] = h.qis[tok];
  }

  bool ok = true;
  const int rt_per_warp = wactive ? (rtc - wr + WR - 1) / WR : 0;
  for (int j0 = 0; j0 < rt_per_warp && ok; j0 += TPP) {
    float acc[TPP][NG][4];
#pragma unroll
    for (int j = 0; j < TPP; ++j)
#pragma unroll
      for (int gg = 0; gg < NG; ++gg) acc[j][gg][0] = acc[j][gg][1] = acc[j][gg][2] = acc[j][gg][3] = 0.f;

    for (int kt_l = wk; kt_l < ktc; kt_l += WK) {
      if (!mbar_wait_bounded(&h.mbar[kt_l / cpt], 0)) {
        ok = false;
        break;
      }
      uint32_t bf[4][NG][2];
#pragma unroll
      for (int mu = 0; mu < 4; ++mu)
#pragma unroll
        for (int gg = 0; gg < NG; ++gg) {
          const uint2 v = *reinterpret_cast<const uint2*>(frag32 + (((kt_l * 4 + mu) * NG + gg) * 32 + lane) * 2);
          bf[mu][gg][0] = v.x;
          bf[mu][gg][1] = v.y;
        }
#pragma unroll
      for (int j = 0; j < TPP; ++j) {
        const int rt_l = wr + WR * (j0 + j);
        if (rt_l < rtc) {
          const uint2 w = *reinterpret_cast<const uint2*>(wts + ((size_t)(kt_l * rtc + rt_l) * kTileBytes) + lane * 8);
          uint32_t lo[8], hi[8];
          expand_word(w.x, lo);
          expand_word(w.y, hi);
#pragma unroll
          for (int mu = 0; mu < 4; ++mu)
#pragma unroll
            for (int gg = 0; gg < NG; ++gg)
              mma_e4m3(acc[j][gg], lo[2 * mu], hi[2 * mu], lo[2 * mu + 1], hi[2 * mu + 1], bf[mu][gg][0],
                       bf[mu][gg][1]);
        }
      }
    }
    if (!ok) break;
    // 2 D 2^-sigma of these row tiles over this warp's column tiles: to the
    // in-CTA reduction buffer (WK > 1) or, minus Q 2^-sigma, straight into
    // the shared memory of the cluster CTA that finalises the row.
#pragma unroll
    for (int j = 0; j < TPP; ++j) {
      const int rt_l = wr + WR * (j0 + j);
      if (rt_l < rtc) {
#pragma unroll
        for (int gg = 0; gg < NG; ++gg) {
          float vlo = acc[j][gg][0] + acc[j][gg][1];
          float vhi = acc[j][gg][2] + acc[j][gg][3];
          vlo += __shfl_xor_sync(0xffffffffu, vlo, 1);
          vhi += __shfl_xor_sync(0xffffffffu, vhi, 1);
          const int tok = 2 * gg + (c >> 1);
          if ((c & 1) == 0 && tok < T) {
#pragma unroll
            for (int half = 0; half < 2; ++half) {
              const int rl = rt_l * kTileRows + g + 8 * half;
              const float p = 2.f * (half ? vhi : vlo) * isv[gg];
              if (WK > 1) {
                red[(wk * 2 * NG + tok) * nrows + rl] = p;
              } else {
                const int owner = rl / slice;
                st_cluster_f32(recv + ((ks * 2 * NG + tok) * slice + (rl - owner * slice)), (uint32_t)owner,
                               p - qisv[gg]);
              }
            }
          }
        }
      }
    }
  }

  const bool all_ok = __syncthreads_and(ok ? 1 : 0) != 0;
  if (!all_ok && tid == 0) {
    // A bulk copy never completed: flag it and let the copies drain
    // (bounded). The cluster barrier is still honoured so that no CTA of the
    // cluster waits on this one.
    atomicOr(a.status, kStatusTimeout);
    for (int i = 0; i < nchunks; ++i) mbar_wait_bounded(&h.mbar[i], 0);
  }
  if (WK > 1 && all_ok) {
    // Sum the WK column-class partials of each row in a fixed order and push.
    for (int idx = tid; idx < T * nrows; idx += WARPS * 32) {
      const int tok = idx / nrows;
      const int rl = idx - tok * nrows;
      float v = 0.f;
      for (int q = 0; q < WK; ++q) v += red[(q * 2 * NG + tok) * nrows + rl];
      const int owner = rl / slice;
      st_cluster_f32(recv + ((ks * 2 * NG + tok) * slice + (rl - owner * slice)), (uint32_t)owner, v - h.qis[tok]);
    }
  }
  // All partials of the cluster have landed in their owners' buffers.
  cluster_sync();
  const int cnt = min(slice, nrows - my0);
  if (all_ok && cnt > 0) {
    for (int idx = tid; idx < T * cnt; idx += WARPS * 32) {
      const int tok = idx / cnt;
      const int i = idx - tok * cnt;
      const int64_t row = row0 + my0 + i;
      if (row >= tm.R) continue;
      float v = 0.f;
      for (int q = 0; q < KS; ++q) v += recv[(q * 2 * NG + tok) * slice + i];
      const float out = v * rs[i];
      if (PHASE == 1) {
        a.sout[(int64_t)tok * a.lds + row] = out;
      } else if (a.ydtype == 0) {
        reinterpret_cast<__half*>(a.y)[(int64_t)tok * a.ldy + row] = __float2half_rn(out);
      } else {
        reinterpret_cast<float*>(a.y)[(int64_t)tok * a.ldy + row] = out;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

// 16 warps per CTA for up to 4 tokens (shorter serial MMA chains per warp);
// 8 warps for 5-16 tokens (register budget of the wider fragments).
template <int NG>
constexpr int warps_for() {
  return NG <= 2 ? 16 : 8;
}
template <int NG>
constexpr int tpp_for() {
  return NG == 1 ? 2 : NG == 2 ? 2 : NG == 4 ? 2 : 1;
}

template <int PHASE, int NG>
cudaError_t launch_phase(const PhaseArgs& a, cudaStream_t st) {
  constexpr int W = warps_for<NG>();
  auto kern = phase_kernel<PHASE, NG, W, tpp_for<NG>()>;
  const int smem = smem_plan(a.tm, NG).total;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  if (a.tm.KS > 8) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.tm.RG, (unsigned)a.tm.KS, 1);
  cfg.blockDim = dim3(W * 32, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = (unsigned)a.tm.KS;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int PHASE>
cudaError_t launch_phase_ng(int ng, const PhaseArgs& a, cudaStream_t st) {
  switch (ng) {
    case 1: return launch_phase<PHASE, 1>(a, st);
    case 2: return launch_phase<PHASE, 2>(a, st);
    case 4: return launch_phase<PHASE, 4>(a, st);
    default: return launch_phase<PHASE, 8>(a, st);
  }
}

int64_t align256(int64_t v) { return (v + 255) / 256 * 256; }

}  // namespace

int forward_smem_bytes(const TileMatrix& t, int ng) { return smem_plan(t, ng).total; }

// Column tiles per CTA of the decode split of K: one tile per CTA up to 8
// tiles, then clusters of 8 CTAs, beyond 64 tiles clusters of up to 16.
int decode_ktc(int KT) {
  if (KT <= 8) return 1;
  int ktc = (KT + 7) / 8;
  if (ktc > 8) ktc = (KT + 15) / 16;
  return ktc;
}

// Launch-time split of K: a cluster of KS CTAs per row group (decode_ktc),
// with a finer split (up to 16 CTAs) when the shared-memory plan of a wide
// pass needs it.
TileMatrix launch_plan(const TileMatrix& layout, int ng, int max_smem) {
  TileMatrix t = layout;
  t.KTC = decode_ktc(layout.KT);
  t.KS = (layout.KT + t.KTC - 1) / t.KTC;
  while (smem_plan(t, ng).total > max_smem && t.KS < 16 && t.KTC > 1) {
    const int ks = t.KS + 1;
    t.KTC = (layout.KT + ks - 1) / ks;
    t.KS = (layout.KT + t.KTC - 1) / t.KTC;
  }
  return t;
}

void plan_tiles(TileMatrix& t, int64_t R, int64_t C, int num_sms, int max_smem) {
  // Pack-time layout: one block per group of RTC row tiles holding all KT
  // column tiles, column-tile major, so that any split of K chosen at launch
  // (launch_plan) gives every CTA one contiguous range of its block.
  t.R = R;
  t.C = C;
  t.RT = (int)((R + kTileRows - 1) / kTileRows);
  t.KT = (int)((C + kTileCols - 1) / kTileCols);
  t.KTC = t.KT;
  t.KS = 1;
  // Row tiles per group: about two CTAs per SM with the decode split of K
  // (decode_ktc), at least 8 (the activation split is amortised over the
  // group's rows), at most 32.
  const int sms = num_sms > 0 ? num_sms : 148;
  const int dk = decode_ktc(t.KT);
  const int ks = (t.KT + dk - 1) / dk;
  int rtc = (int)(((int64_t)t.RT * ks + sms) / (2 * sms));
  if (rtc < 8) rtc = 8;
  if (rtc > 32) rtc = 32;
  if (rtc > t.RT) rtc = t.RT;
  t.RTC = rtc;
  t.RG = (t.RT + t.RTC - 1) / t.RTC;
  // The widest pass (16 tokens) must fit with a split of at most 16 CTAs.
  for (;;) {
    TileMatrix probe = t;
    probe.KTC = (t.KT + 15) / 16;
    probe.KS = (t.KT + probe.KTC - 1) / probe.KTC;
    if (t.RTC <= 1 || smem_plan(probe, 8).total <= max_smem) break;
    t.RTC = (t.RTC + 1) / 2;
    t.RG = (t.RT + t.RTC - 1) / t.RTC;
  }
}

Workspace plan_workspace(const af1_layer& L, int64_t tokens) {
  Workspace w;
  int64_t off = 0;
  w.status = off;
  off += 256;
  w.sbuf = off;
  off += align256((int64_t)kMaxPassTokens * L.p2.KT * kTileCols * 4);
  w.hbuf = off;
  if (tokens > kMaxPassTokens) {
    const int64_t t = tokens < kPrefillPassTokens ? tokens : kPrefillPassTokens;
    off += align256(t * prefill_h_ld(L) * 2);
  }
  w.total = off;
  return w;
}

cudaError_t launch_forward(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y,
                           int64_t ldy, int y_dtype, void* ws, cudaStream_t st) {
  const Workspace W = plan_workspace(L, tokens);
  uint8_t* wsb = static_cast<uint8_t*>(ws);
  if (tokens > kMaxPassTokens) {
    // Prefill: two tensor-core GEMMs per pass (af1_prefill.cu).
    return launch_prefill(L, x, ldx, tokens, y, ldy, y_dtype, wsb + W.hbuf, reinterpret_cast<unsigned*>(wsb + W.status),
                          st);
  }
  const int ysize = y_dtype == 0 ? 2 : 4;
  for (int64_t t0 = 0; t0 < tokens; t0 += kMaxPassTokens) {
    const int T = (int)((tokens - t0) < kMaxPassTokens ? (tokens - t0) : kMaxPassTokens);
    const int ng = T <= 2 ? 1 : T <= 4 ? 2 : T <= 8 ? 4 : 8;

    PhaseArgs p1 = {};
    p1.tiles = L.tiles1;
    p1.tm = launch_plan(L.p1, ng, L.max_smem);
    p1.tokens = T;
    p1.x = static_cast<const __half*>(x) + t0 * ldx;
    p1.ldx = ldx;
    p1.colscale = reinterpret_cast<const __half*>(L.b);
    p1.status = reinterpret_cast<unsigned*>(wsb + W.status);
    p1.rowscale = reinterpret_cast<const __half*>(L.s);
    p1.sout = reinterpret_cast<float*>(wsb + W.sbuf);
    p1.lds = (int64_t)L.p2.KT * kTileCols;
    cudaError_t e = launch_phase_ng<1>(ng, p1, st);
    if (e != cudaSuccess) return e;

    PhaseArgs p2 = {};
    p2.tiles = L.tiles2;
    p2.tm = launch_plan(L.p2, ng, L.max_smem);
    p2.tokens = T;
    p2.zin = p1.sout;
    p2.ldz = p1.lds;
    p2.status = p1.status;
    p2.rowscale = reinterpret_cast<const __half*>(L.a);
    p2.y = static_cast<uint8_t*>(y) + t0 * ldy * ysize;
    p2.ldy = ldy;
    p2.ydtype = y_dtype;
    e = launch_phase_ng<2>(ng, p2, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace af1
