// af1_forward.cu — forward pass of an AF1 binary-factorized linear layer on
// sm_103a: y = a * (U (s * (V^T (b * x)))), the right-to-left evaluation of
// AF1 Eq. final_reconstruction / Eq. double_factor_equiv that never forms the
// dense W_hat.
//
// Two kernels per pass of up to 16 tokens, chained with programmatic
// dependent launch (PDL):
//   phase 1: t = B z with B = V^T (r x n) and z = b * x; the last CTA of each
//            row block applies the rank scale, s' = s * t (fp32, workspace).
//   phase 2: u = U s' (m x r); the last CTA of each row block applies the
//            row scale, y = a * u, and stores FP16 or FP32.
// Each CTA owns a block of sign tiles (af1_layout.h). It issues bulk copies
// (TMA, cp.async.bulk) of its whole block into shared memory before it waits
// on the previous kernel, so weight streaming overlaps the dependency.
//
// Sign contraction on FP8 tensor cores. A sign bit is expanded into an e4m3
// A-fragment byte with one LOP3 per 4 signs: (word & mask_p) | base_p puts
// the bit at a fixed position p of a constant byte, giving A = L_p + d_p * bit
// with L_p, d_p powers of two (mantissa bits 0..2, exponent bit 0, sign bit).
// With z'_k = z_k / d_k the MMA yields D = sum_k L_k z'_k + sum_k bit_k z_k,
// and since sign = 2 bit - 1,
//     sum_k sign_k z_k = 2 D - Q,   Q = sum_k (L_k + H_k) z'_k   (H = L + d).
// Each activation z'_k is scaled by a per-(CTA, token) power of two so that
// its magnitude sits in [128, 256), and is split into 4 e4m3 terms
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

// ---------------------------------------------------------------------------
// PTX helpers (hand-written; mbarrier, bulk copy, PDL, MMA, FP8 conversion)
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

__device__ __forceinline__ void mma_e4m3(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Round a float to e4m3 (nearest even, saturating); returns the byte.
__device__ __forceinline__ uint32_t to_e4m3(float v) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(0.0f), "f"(v));
  return r & 0xFFu;
}
// Exact value of an e4m3 byte.
__device__ __forceinline__ float from_e4m3(uint32_t byte) {
  uint32_t h2;
  uint16_t in = static_cast<uint16_t>(byte);
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(in));
  return __half2float(__ushort_as_half(static_cast<unsigned short>(h2 & 0xFFFFu)));
}

// Slot p of a word (see af1_layout.h): 1 / d_p and L_p + H_p.
//   p:        0     1     2     3     4     5     6     7
//   d_p:    1/8   1/4   1/2   1/2   1/4   1/2   1/2    -2
//   L_p:      1     1     1   1/2     1     1   1/2     1
__constant__ float c_inv_delta[8] = {8.f, 4.f, 2.f, 2.f, 4.f, 2.f, 2.f, -0.5f};
__constant__ float c_lph[8] = {2.125f, 2.25f, 2.5f, 1.5f, 2.25f, 2.5f, 1.5f, 0.f};
__device__ __forceinline__ float slot_inv_delta(int p) { return c_inv_delta[p]; }
__device__ __forceinline__ float slot_lph(int p) { return c_lph[p]; }

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
// Kernel arguments
// ---------------------------------------------------------------------------

struct PhaseArgs {
  const uint8_t* tiles;
  TileMatrix tm;
  int tokens;
  // phase 1 input: z = colscale * x
  const __half* x;
  int64_t ldx;
  const __half* colscale;
  // phase 2 input: z = zin
  const float* zin;
  int64_t ldz;
  // cross-CTA accumulation (zero on entry, left zero)
  float* acc;
  int64_t ldacc;
  unsigned* counters;
  unsigned* status;
  // finalisation
  const __half* rowscale;
  float* sout;  // phase 1: s' = s * t
  int64_t lds;
  void* y;  // phase 2
  int64_t ldy;
  int ydtype;
};

struct SmemHeader {
  uint64_t mbar[kMaxKTC];
  float scale[kMaxPassTokens];   // 2^sigma per token
  float iscale[kMaxPassTokens];  // 2^-sigma
  float q[kMaxPassTokens];
  float red[32 * kMaxPassTokens];
  unsigned flag;
};
constexpr int kHeaderBytes = ((int)sizeof(SmemHeader) + 127) / 128 * 128;

template <int PHASE>
__device__ __forceinline__ float fetch_z(const PhaseArgs& a, int tok, int64_t k) {
  if (PHASE == 1) {
    return __half2float(a.colscale[k]) * __half2float(a.x[(int64_t)tok * a.ldx + k]);
  } else {
    return a.zin[(int64_t)tok * a.ldz + k];
  }
}

// Block-wide reduction of NV values per thread (max or sum), result in hdr.red[0..NV).
template <int NV, bool MAX, int WARPS>
__device__ __forceinline__ void block_reduce(float (&v)[NV], float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      float other = __shfl_xor_sync(0xffffffffu, v[i], o);
      v[i] = MAX ? fmaxf(v[i], other) : v[i] + other;
    }
  }
  __syncthreads();
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < NV; ++i) red[warp * NV + i] = v[i];
  }
  __syncthreads();
  if (threadIdx.x < NV) {
    float r = red[threadIdx.x];
    for (int w = 1; w < WARPS; ++w) {
      float o = red[w * NV + threadIdx.x];
      r = MAX ? fmaxf(r, o) : r + o;
    }
    red[WARPS * NV + threadIdx.x] = r;
  }
  __syncthreads();
}

// Build the e4m3 B fragments of this CTA's column range for all token slots
// (2 * NG), plus the per-token scale 2^sigma and the constant Q.
template <int PHASE, int NG, int WARPS>
__device__ void build_fragments(const PhaseArgs& a, SmemHeader& h, uint8_t* frag, int64_t k0, int ncols) {
  constexpr int NT = 2 * NG;
  const int T = a.tokens;
  const int64_t C = a.tm.C;
  // pass A: max |z / d| per token
  float mx[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) mx[t] = 0.f;
  for (int kl = threadIdx.x; kl < ncols; kl += WARPS * 32) {
    const int64_t k = k0 + kl;
    if (k < C) {
      const float invd = fabsf(slot_inv_delta((kl & 127) >> 4));
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        if (t < T) mx[t] = fmaxf(mx[t], fabsf(fetch_z<PHASE>(a, t, k)) * invd);
      }
    }
  }
  block_reduce<NT, true, WARPS>(mx, h.red);
  if (threadIdx.x < NT) {
    const float m = h.red[WARPS * NT + threadIdx.x];
    int e = 0;
    if (m > 0.f) frexpf(m, &e);  // m = f * 2^e, f in [0.5, 1)
    const int sigma = (m > 0.f) ? 8 - e : 0;  // 2^sigma * m in [128, 256)
    h.scale[threadIdx.x] = ldexpf(1.f, sigma);
    h.iscale[threadIdx.x] = ldexpf(1.f, -sigma);
  }
  __syncthreads();
  // pass B: split into 4 e4m3 terms, scatter into fragment order, sum Q
  float q[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) q[t] = 0.f;
  for (int kl = threadIdx.x; kl < ncols; kl += WARPS * 32) {
    const int64_t k = k0 + kl;
    const int p = (kl & 127) >> 4;
    const float invd = slot_inv_delta(p);
    const float lph = slot_lph(p);
    const int kt_l = kl >> 7, kk = kl & 127, mu = kk >> 5, r32 = kk & 31;
    const int breg = r32 >> 4, c = (r32 & 15) >> 2, e = r32 & 3;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      float rem = 0.f;
      if (t < T && k < C) rem = fetch_z<PHASE>(a, t, k) * invd * h.scale[t];
      const int gamma = t >> 1;
      float tsum = 0.f;
#pragma unroll
      for (int term = 0; term < kTerms; ++term) {
        const uint32_t byte = to_e4m3(rem);
        const float back = from_e4m3(byte);
        rem -= back;
        tsum += back;
        const int g = 4 * (t & 1) + term;
        const int lane_f = 4 * g + c;
        frag[((((kt_l * 4 + mu) * NG + gamma) * 32 + lane_f) * 8) + breg * 4 + e] = (uint8_t)byte;
      }
      q[t] += lph * tsum;
    }
  }
  block_reduce<NT, false, WARPS>(q, h.red);
  if (threadIdx.x < NT) h.q[threadIdx.x] = h.red[WARPS * NT + threadIdx.x];
  __syncthreads();
}

template <int PHASE, int NG, int WARPS, int TPP>
__global__ void __launch_bounds__(WARPS * 32) phase_kernel(const PhaseArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  SmemHeader& h = *reinterpret_cast<SmemHeader*>(smem);
  const TileMatrix& tm = a.tm;
  uint8_t* frag = smem + kHeaderBytes;
  uint8_t* wts = frag + tm.KTC * 4 * NG * 256;

  const int rg = blockIdx.x, ks = blockIdx.y;
  const int rtc = blk_rows(tm, rg), ktc = blk_cols(tm, ks);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t chunk = (uint32_t)rtc * kTileBytes;
  const uint8_t* gblk = a.tiles + blk_base(tm, rg, ks) * kTileBytes;

  if (tid == 0) {
    for (int i = 0; i < ktc; ++i) mbar_init(&h.mbar[i], 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (tid == 0) {
    for (int i = 0; i < ktc; ++i) {
      mbar_expect_tx(&h.mbar[i], chunk);
      bulk_g2s(wts + (size_t)i * chunk, gblk + (size_t)i * chunk, chunk, &h.mbar[i]);
    }
  }
  // The weights do not depend on earlier kernels; everything below does.
  griddep_launch_dependents();
  griddep_wait();

  build_fragments<PHASE, NG, WARPS>(a, h, frag, (int64_t)ks * tm.KTC * kTileCols, ktc * kTileCols);

  const int g = lane >> 2, c = lane & 3;
  const int T = a.tokens;
  bool ok = true;
  const int rt_per_warp = (rtc + WARPS - 1) / WARPS;
  for (int j0 = 0; j0 < rt_per_warp && ok; j0 += TPP) {
    float acc[TPP][NG][4];
#pragma unroll
    for (int j = 0; j < TPP; ++j)
#pragma unroll
      for (int gg = 0; gg < NG; ++gg) acc[j][gg][0] = acc[j][gg][1] = acc[j][gg][2] = acc[j][gg][3] = 0.f;

    for (int kt_l = 0; kt_l < ktc; ++kt_l) {
      if (!mbar_wait_bounded(&h.mbar[kt_l], 0)) {
        ok = false;
        break;
      }
      uint32_t bf[4][NG][2];
#pragma unroll
      for (int mu = 0; mu < 4; ++mu)
#pragma unroll
        for (int gg = 0; gg < NG; ++gg) {
          const uint2 v = *reinterpret_cast<const uint2*>(frag + ((((kt_l * 4 + mu) * NG + gg) * 32 + lane) * 8));
          bf[mu][gg][0] = v.x;
          bf[mu][gg][1] = v.y;
        }
#pragma unroll
      for (int j = 0; j < TPP; ++j) {
        const int rt_l = warp + WARPS * (j0 + j);
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
    // Partial sums of these row tiles -> cross-CTA accumulation buffer.
#pragma unroll
    for (int j = 0; j < TPP; ++j) {
      const int rt_l = warp + WARPS * (j0 + j);
      if (rt_l < rtc) {
        const int64_t row0 = (int64_t)(rg * tm.RTC + rt_l) * kTileRows + g;
#pragma unroll
        for (int gg = 0; gg < NG; ++gg) {
          float vlo = acc[j][gg][0] + acc[j][gg][1];
          float vhi = acc[j][gg][2] + acc[j][gg][3];
          vlo += __shfl_xor_sync(0xffffffffu, vlo, 1);
          vhi += __shfl_xor_sync(0xffffffffu, vhi, 1);
          const int tok = 2 * gg + (c >> 1);
          if ((c & 1) == 0 && tok < T) {
            const float qv = h.q[tok], is = h.iscale[tok];
            if (row0 < tm.R) atomicAdd(a.acc + (int64_t)tok * a.ldacc + row0, (2.f * vlo - qv) * is);
            if (row0 + 8 < tm.R) atomicAdd(a.acc + (int64_t)tok * a.ldacc + row0 + 8, (2.f * vhi - qv) * is);
          }
        }
      }
    }
  }

  if (!__syncthreads_and(ok ? 1 : 0)) {
    // A bulk copy never completed: flag it, let the copies drain (bounded),
    // and leave without touching the shared bookkeeping.
    if (tid == 0) {
      atomicOr(a.status, kStatusTimeout);
      for (int i = 0; i < ktc; ++i) mbar_wait_bounded(&h.mbar[i], 0);
    }
    return;
  }

  if (tid == 0) {
    __threadfence();
    const unsigned old = atomicAdd(a.counters + rg, 1u);
    const unsigned last = (old == gridDim.y - 1) ? 1u : 0u;
    if (last) a.counters[rg] = 0u;
    h.flag = last;
  }
  __syncthreads();
  if (!h.flag) return;
  __threadfence();
  const int nrows = rtc * kTileRows;
  const int64_t r0 = (int64_t)rg * tm.RTC * kTileRows;
  for (int idx = tid; idx < T * nrows; idx += WARPS * 32) {
    const int tok = idx / nrows;
    const int64_t row = r0 + (idx - tok * nrows);
    if (row >= tm.R) continue;
    float* p = a.acc + (int64_t)tok * a.ldacc + row;
    const float v = __ldcg(p);
    __stcg(p, 0.f);
    const float sc = __half2float(a.rowscale[row]);
    if (PHASE == 1) {
      a.sout[(int64_t)tok * a.lds + row] = v * sc;
    } else if (a.ydtype == 0) {
      reinterpret_cast<__half*>(a.y)[(int64_t)tok * a.ldy + row] = __float2half_rn(v * sc);
    } else {
      reinterpret_cast<float*>(a.y)[(int64_t)tok * a.ldy + row] = v * sc;
    }
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

constexpr int kWarps1 = 8, kWarps2 = 4;

template <int NG>
constexpr int tpp_for() {
  return NG == 1 ? 8 : NG == 2 ? 4 : NG == 4 ? 2 : 1;
}

int64_t smem_bytes(const TileMatrix& tm, int ng) {
  return kHeaderBytes + (int64_t)tm.KTC * 4 * ng * 256 + (int64_t)tm.RTC * tm.KTC * kTileBytes;
}

template <int PHASE, int NG>
cudaError_t launch_phase(const PhaseArgs& a, cudaStream_t st) {
  constexpr int W = PHASE == 1 ? kWarps1 : kWarps2;
  auto kern = phase_kernel<PHASE, NG, W, tpp_for<NG>()>;
  const int64_t smem = smem_bytes(a.tm, NG);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.tm.RG, (unsigned)a.tm.KS, 1);
  cfg.blockDim = dim3(W * 32, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
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

void plan_tiles(TileMatrix& t, int64_t R, int64_t C, int rtc_target, int num_sms, int ktc_max) {
  t.R = R;
  t.C = C;
  t.RT = (int)((R + kTileRows - 1) / kTileRows);
  t.KT = (int)((C + kTileCols - 1) / kTileCols);
  t.RTC = t.RT < rtc_target ? t.RT : rtc_target;
  t.RG = (t.RT + t.RTC - 1) / t.RTC;
  const int sms = num_sms > 0 ? num_sms : 148;
  int ktc = (int)((double)t.RG * t.KT / (2.0 * sms) + 0.5);
  if (ktc < 1) ktc = 1;
  if (ktc > ktc_max) ktc = ktc_max;
  if (ktc > t.KT) ktc = t.KT;
  t.KTC = ktc;
  t.KS = (t.KT + t.KTC - 1) / t.KTC;
}

Workspace plan_workspace(const af1_layer& L) {
  Workspace w;
  int64_t off = 0;
  w.status = off;
  off += 256;
  w.counters1 = off;
  off += align256((int64_t)L.p1.RG * 4);
  w.counters2 = off;
  off += align256((int64_t)L.p2.RG * 4);
  w.tacc = off;
  off += align256((int64_t)kMaxPassTokens * L.p1.RT * kTileRows * 4);
  w.sbuf = off;
  off += align256((int64_t)kMaxPassTokens * L.p2.KT * kTileCols * 4);
  w.yacc = off;
  off += align256((int64_t)kMaxPassTokens * L.p2.RT * kTileRows * 4);
  w.total = off;
  return w;
}

cudaError_t launch_forward(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y,
                           int64_t ldy, int y_dtype, void* ws, cudaStream_t st) {
  const Workspace W = plan_workspace(L);
  uint8_t* wsb = static_cast<uint8_t*>(ws);
  const int ysize = y_dtype == 0 ? 2 : 4;
  for (int64_t t0 = 0; t0 < tokens; t0 += kMaxPassTokens) {
    const int T = (int)((tokens - t0) < kMaxPassTokens ? (tokens - t0) : kMaxPassTokens);
    const int ng = T <= 2 ? 1 : T <= 4 ? 2 : T <= 8 ? 4 : 8;

    PhaseArgs p1 = {};
    p1.tiles = L.tiles1;
    p1.tm = L.p1;
    p1.tokens = T;
    p1.x = static_cast<const __half*>(x) + t0 * ldx;
    p1.ldx = ldx;
    p1.colscale = reinterpret_cast<const __half*>(L.b);
    p1.acc = reinterpret_cast<float*>(wsb + W.tacc);
    p1.ldacc = (int64_t)L.p1.RT * kTileRows;
    p1.counters = reinterpret_cast<unsigned*>(wsb + W.counters1);
    p1.status = reinterpret_cast<unsigned*>(wsb + W.status);
    p1.rowscale = reinterpret_cast<const __half*>(L.s);
    p1.sout = reinterpret_cast<float*>(wsb + W.sbuf);
    p1.lds = (int64_t)L.p2.KT * kTileCols;
    cudaError_t e = launch_phase_ng<1>(ng, p1, st);
    if (e != cudaSuccess) return e;

    PhaseArgs p2 = {};
    p2.tiles = L.tiles2;
    p2.tm = L.p2;
    p2.tokens = T;
    p2.zin = p1.sout;
    p2.ldz = p1.lds;
    p2.acc = reinterpret_cast<float*>(wsb + W.yacc);
    p2.ldacc = (int64_t)L.p2.RT * kTileRows;
    p2.counters = reinterpret_cast<unsigned*>(wsb + W.counters2);
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
