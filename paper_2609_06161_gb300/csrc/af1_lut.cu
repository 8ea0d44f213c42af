// af1_lut.cu — decode path (1..16 tokens per pass) on the CUDA cores: each
// sign-matrix x vector product of the forward pass
//     y = a * (U (s * (V^T (b * x))))      (AF1 Eq. final_reconstruction /
//                                          Eq. double_factor_equiv)
// is evaluated with lookup tables of signed sums instead of tensor-core MMAs.
//
// For every group of 4 columns {k_0..k_3} and every token, the 16 sums
//     T[i] = sum_q (bit q of i ? +z_{k_q} : -z_{k_q}),   i = 0..15,
// are built once per CTA in shared memory (FP32). A matrix row then needs one
// table read and one FP32 add per 4 signs: the 4 sign bits of the group are
// the table index. All 32 lanes of a warp (32 rows) read the same 16-entry
// table at the same time, so every read is a conflict-free broadcast. A
// probe of this inner loop on GB300 sustained about 160 signs per ns per SM
// at one token, twice the rate at which signs can be expanded into tensor
// memory and multiplied there.
//
// Groups. In the row-block layout (af1_layout.h) bit 8e + p of word kw is
// column 32 kw + 4p + e, so nibble j = 2e + h of a word (bits 8e + 4h .. +3)
// holds the signs of columns 32 kw + 16h + 4q + e, q = 0..3: the group of
// nibble j. Table index bit q <-> column 32 kw + 16h + 4q + e.
//
// Table addresses. The tables of one 128-column chunk occupy 2 KB per token
// (one token) or 4 KB per token pair (entries are float2 {token 2p, 2p+1}):
// group g = 4j + w (word w of the chunk, nibble j) at g * 64 (one token) or
// g * 128 (pairs). The byte offset of an entry inside its 256-byte window is
// built from the sign word with one shift and one LOP3 for four nibbles at a
// time, and PRMT splices it under the window's upper address bytes, so a
// lookup costs PRMT + LDS + FADD.
//
// Work split (as the tensor-core decode kernel): CTA (rb, ks, tg) owns row
// block rb (128 rows), the ks-th slice of CPC chunks and token group tg (up
// to 4 tokens of the pass); the KS CTAs of a row block and token group form
// a cluster and reduce their partial sums through distributed shared memory
// in a fixed order (deterministic). Two threads per row each take two of the
// four words of every chunk. The packed chunks are fetched with bulk copies
// before the kernel waits for the previous one (programmatic dependent
// launch); the activations of the CTA's columns are staged in shared memory,
// then the tables are built.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "af1_internal.h"
#include "af1_layout.h"

namespace af1 {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxCPC = 32;       // chunks per CTA (one mbarrier each)
constexpr int kMaxKS = 16;        // CTAs per cluster
constexpr int kGroupTokens = 4;   // tokens per CTA: a pass of T tokens runs ceil(T / 4) CTAs per tile
constexpr long long kWaitCycles = 2000000000ll;  // ~1 s at 2 GHz
constexpr unsigned kStatusTimeout = 1u;

// ---------------------------------------------------------------------------
// PTX helpers (mbarrier, bulk copy, PDL, cluster)
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
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
// Bounded wait: false (and the CTA error flag set) if the phase did not
// complete within kWaitCycles.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) {
      atomicOr(err, 1u);
      return false;
    }
  }
  return true;
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.aligned;" ::: "memory"); }

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
// Shared-memory plan
// ---------------------------------------------------------------------------

// Token pairs of a pass: 0 stands for a single token (FP32 entries).
__host__ __device__ constexpr int pairs_for(int T) { return T == 1 ? 0 : (T + 1) / 2; }
// Table bytes of one chunk.
__host__ __device__ constexpr int table_chunk_bytes(int np) { return np == 0 ? 2048 : 4096 * np; }
// Staged activations: column k of the CTA at k + k / 32 (the skew keeps the
// table builders' stride-32 reads on distinct banks).
__host__ __device__ constexpr int zrow_floats(int CPC) { return CPC * kChunkCols + CPC * (kChunkCols / 32); }
__host__ __device__ inline int slice_rows(int KS) { return (kBlockRows + KS - 1) / KS; }
__host__ __device__ inline int align128(int v) { return (v + 127) & ~127; }

struct __align__(8) LutHeader {
  uint64_t red;             // all partial sums for this CTA's rows have landed (st.async)
  uint64_t wfull[kMaxCPC];  // packed chunk c has landed
  uint32_t err;
};

struct LutSmem {
  int tbl, w, z, recv, rs, hdr, total;  // byte offsets from the 1024-aligned base
};

// T tokens of a CTA, tables laid out for np token pairs (pairs_for of the
// pass's first group; a smaller last group leaves its missing tokens zero).
__host__ __device__ inline LutSmem lut_smem(int CPC, int KS, int T, int np) {
  LutSmem p;
  int off = 0;
  p.tbl = off;
  off += table_chunk_bytes(np) * CPC;
  p.w = off;
  off += kChunkBytes * CPC;
  p.z = off;
  off = align128(off + T * zrow_floats(CPC) * 4);
  p.recv = off;  // [2 KS][T][slice]: partials of the two word halves of each CTA
  off = align128(off + 2 * KS * T * slice_rows(KS) * 4);
  p.rs = off;
  off = align128(off + slice_rows(KS) * 4);
  p.hdr = off;
  off = align128(off + (int)sizeof(LutHeader));
  p.total = off + 1024;  // slack for aligning the base to 1024 bytes
  return p;
}

// ---------------------------------------------------------------------------
// Kernel
// ---------------------------------------------------------------------------

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

template <int PHASE, int NP, bool MULTI>
__global__ void __launch_bounds__(kThreads, 4) lut_kernel(const __grid_constant__ LutArgs a) {
  constexpr int NACC = NP == 0 ? 1 : 2 * NP;
  constexpr int TCB = table_chunk_bytes(NP);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  // Problem of this CTA: grid x runs over the row blocks of all problems.
  // (One problem: fixed parameter offsets, no lookup.)
  int pi = 0;
  if (MULTI) {
    for (int i = 1; i < a.count; ++i)
      if ((int)blockIdx.x >= a.prob[i].rb0) pi = i;
  }
  const LutProblem& pb = a.prob[MULTI ? pi : 0];
  // Token group blockIdx.z: tokens tg0 .. tg0 + T - 1 of the pass.
  const int tg0 = (int)blockIdx.z * kGroupTokens;
  const int T = min(kGroupTokens, a.tokens - tg0);
  const __half* xg = PHASE == 1 ? pb.x + (int64_t)tg0 * pb.ldx : nullptr;
  const float* zg = PHASE == 2 ? pb.zin + (int64_t)tg0 * pb.ldz : nullptr;
  const int KS = a.KS, CPC = pb.CPC;
  const LutSmem sp = lut_smem(CPC, KS, T, NP);
  const uint32_t* W = reinterpret_cast<const uint32_t*>(smem + sp.w);
  float* zs = reinterpret_cast<float*>(smem + sp.z);
  float* recv = reinterpret_cast<float*>(smem + sp.recv);
  float* rs = reinterpret_cast<float*>(smem + sp.rs);
  LutHeader& h = *reinterpret_cast<LutHeader*>(smem + sp.hdr);

  const int tid = threadIdx.x;
  const int rb = (int)blockIdx.x - pb.rb0, ks = blockIdx.y;
  const int nch_total = pb.sm.NCH;
  const int c0 = ks * CPC;
  // Chunks of this CTA; 0 for the last CTAs of a problem with fewer chunks
  // than the group's clusters have CTAs (they still finalise their rows).
  const int nch = max(0, min(CPC, nch_total - c0));
  const int64_t row0 = (int64_t)rb * kBlockRows;
  const int64_t k0 = (int64_t)c0 * kChunkCols;
  const int slice = slice_rows(KS);
  const int my0 = ks * slice;  // first block row this CTA finalises
  const int zrow = zrow_floats(CPC);

  const int cnt = min(slice, kBlockRows - my0);  // rows this CTA finalises (may be <= 0)

  if (tid == 0) {
    for (int c = 0; c < nch; ++c) mbar_init(&h.wfull[c], 1);
    // The partial sums of this CTA's rows arrive by st.async from the 2 KS
    // word halves of the cluster, 4 bytes per row and token each.
    mbar_init(&h.red, 1);
    mbar_expect_tx(&h.red, cnt > 0 ? (uint32_t)(2 * KS * T * cnt * 4) : 0u);
    h.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    const uint8_t* src = pb.signs + ((int64_t)rb * nch_total + c0) * kChunkBytes;
    for (int c = 0; c < nch; ++c) {
      mbar_expect_tx(&h.wfull[c], kChunkBytes);
      bulk_g2s(smem + sp.w + c * kChunkBytes, src + (int64_t)c * kChunkBytes, kChunkBytes, &h.wfull[c]);
    }
  }
  // Matched by cluster_wait before the first remote store: a peer's barrier
  // and expected byte count are set up before any partial can reach it.
  cluster_arrive_relaxed();
  // Row scale of row my0 + tid of the block (a layer constant): loaded now,
  // stored to shared memory once the activations are staged.
  const float rs_own = (tid < slice && my0 + tid < kBlockRows && row0 + my0 + tid < pb.sm.R)
                           ? __half2float(pb.rowscale[row0 + my0 + tid])
                           : 0.f;
  __syncthreads();

  // ---- activations of the CTA's columns -> zs[t][k + k / 32] (FP32) -------
  // Written by the previous kernel: read through L2 (ld.global.cg), 8
  // columns per load, a batch of loads per thread in flight at once.
  griddep_wait();
  {
    const int g8 = nch * (kChunkCols / 8);  // 8-column groups per token
    const int ng = T * g8;
    constexpr int kBatch = 2;
    for (int i0 = tid; i0 < ng; i0 += kBatch * kThreads) {
      float v[kBatch][8];
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        const int i = i0 + u * kThreads;
        const int t = i / g8, k = (i - t * g8) * 8;
        const int64_t col = k0 + k;
        if (i < ng && col + 7 < pb.sm.C) {
          if (PHASE == 1) {
            const uint4 xr = __ldcg(reinterpret_cast<const uint4*>(xg + (int64_t)t * pb.ldx + col));
            const uint4 br = __ldg(reinterpret_cast<const uint4*>(pb.colscale + col));
            const uint32_t xw[4] = {xr.x, xr.y, xr.z, xr.w}, bw[4] = {br.x, br.y, br.z, br.w};
#pragma unroll
            for (int h2 = 0; h2 < 4; ++h2) {
              const float2 xf = __half22float2(*reinterpret_cast<const __half2*>(&xw[h2]));
              const float2 bf = __half22float2(*reinterpret_cast<const __half2*>(&bw[h2]));
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
              if (PHASE == 1)
                z = __half2float(__ldcg(xg + (int64_t)t * pb.ldx + col + q)) * __half2float(pb.colscale[col + q]);
              else
                z = __ldcg(zg + (int64_t)t * pb.ldz + col + q);
            }
            v[u][q] = z;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        const int i = i0 + u * kThreads;
        if (i < ng) {
          const int t = i / g8, k = (i - t * g8) * 8;
          float* dst = zs + t * zrow + k + (k >> 5);  // 8 columns within one 32-column block
#pragma unroll
          for (int q = 0; q < 8; ++q) dst[q] = v[u][q];
        }
      }
    }
  }
  if (tid < slice) rs[tid] = rs_own;
  __syncthreads();

  // ---- tables: task (c, j, w, q) writes entries 4q .. 4q + 3 of group 4j + w
  {
    const int npair = NP == 0 ? 1 : NP;
    const int ntask = nch * 128 * npair;
    for (int task = tid; task < ntask; task += kThreads) {
      const int q = task & 3, w = (task >> 2) & 3, j = (task >> 4) & 7;
      const int rest = task >> 7;
      const int p = rest % npair, c = rest / npair;
      const int e = j >> 1, hh = j & 1;
      // columns of index bits 0..3 (CTA-local): c 128 + 32 w + 16 hh + 4 qq + e
      const int kb = c * kChunkCols + 32 * w + 16 * hh + e;
      const int zb = kb + (kb >> 5);  // same 32-column block for all four
      uint8_t* dst = smem + sp.tbl + c * TCB + (NP == 0 ? (4 * j + w) * 64 + q * 16 : p * 4096 + (4 * j + w) * 128 + q * 32);
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
  __syncthreads();

  // ---- lookups: thread (r, g) = row r, words 2g and 2g + 1 of every chunk ---
  const int r = tid & 127, g = tid >> 7;
  float acc[NACC];
#pragma unroll
  for (int i = 0; i < NACC; ++i) acc[i] = 0.f;
  {
    const uint32_t tbl0 = smem_u32(smem + sp.tbl);
    // Entry-offset byte patterns of words 2g and 2g + 1 (their groups'
    // offsets below the 256-byte window).
    const uint32_t pat0 = NP == 0 ? (uint32_t)(2 * g * 64) * 0x01010101u : 0u;
    const uint32_t pat1 = NP == 0 ? (uint32_t)((2 * g + 1) * 64) * 0x01010101u : 0x80808080u;
    bool ok = true;
    for (int c = 0; c < nch; ++c) {
      if (ok) ok = mbar_wait(&h.wfull[c], 0, &h.err);
      const uint32_t tb = tbl0 + (uint32_t)(c * TCB);
      uint32_t base[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) base[j] = tb + (uint32_t)(NP == 0 ? j * 256 : j * 512 + g * 256);
      const uint32_t* wc = W + c * (kChunkBytes / 4) + r;
      const uint32_t w0 = wc[(2 * g) * kBlockRows], w1 = wc[(2 * g + 1) * kBlockRows];
      if constexpr (NP == 0) {
        lookup_word1(w0, pat0, base, acc[0]);
        lookup_word1(w1, pat1, base, acc[0]);
      } else {
        lookup_word2<NP>(w0, pat0, base, acc);
        lookup_word2<NP>(w1, pat1, base, acc);
      }
    }
  }

  // Let the next kernel launch only now: its CTAs would otherwise hold SM
  // slots (waiting for this kernel) that sibling kernels on other streams
  // need, and its sign copies still get the reduction's time as a head start
  // (measured: config-1 stack 7.40 -> 6.53 us per linear on the DAG schedule,
  // trigger at the start vs here).
  griddep_launch_dependents();
  // ---- partial sums -> owner CTA of each row -> final sums -------------------
  cluster_wait();  // every CTA of the cluster has started
  {
    const int owner = r / slice;
    const int src = ks * 2 + g;
#pragma unroll
    for (int t = 0; t < NACC; ++t)
      if (t < T) st_async_f32(recv + ((src * T + t) * slice + (r - owner * slice)), &h.red, (uint32_t)owner, acc[t]);
  }
  // Exit barrier (waited for after the final sums): no CTA leaves while a
  // peer may still store into it.
  cluster_arrive_relaxed();
  mbar_wait(&h.red, 0, &h.err);  // this CTA's partials have all landed
  for (int idx = tid; idx < T * cnt; idx += kThreads) {
    const int t = idx / cnt;
    const int i = idx - t * cnt;
    const int64_t row = row0 + my0 + i;
    if (row >= pb.sm.R) continue;
    // The 2 KS partials in four interleaved chains (fixed order:
    // deterministic), so their reads overlap.
    const float* pr = recv + t * slice + i;
    const int qstride = T * slice;
    float v0 = 0.f, v1 = 0.f, v2 = 0.f, v3 = 0.f;
    int q = 0;
#pragma unroll 2
    for (; q + 4 <= 2 * KS; q += 4) {
      v0 += pr[q * qstride];
      v1 += pr[(q + 1) * qstride];
      v2 += pr[(q + 2) * qstride];
      v3 += pr[(q + 3) * qstride];
    }
    for (; q < 2 * KS; ++q) v0 += pr[q * qstride];
    const float out = ((v0 + v1) + (v2 + v3)) * rs[i];
    if (PHASE == 1) {
      pb.sout[(int64_t)(tg0 + t) * pb.lds + row] = out;
    } else if (a.ydtype == 0) {
      reinterpret_cast<__half*>(pb.y)[(int64_t)(tg0 + t) * pb.ldy + row] = __float2half_rn(out);
    } else {
      reinterpret_cast<float*>(pb.y)[(int64_t)(tg0 + t) * pb.ldy + row] = out;
    }
  }

  cluster_wait();

  // ---- teardown ---------------------------------------------------------------
  __syncthreads();
  if (tid == 0 && h.err != 0) {
    // A wait gave up: let the bulk copies drain (bounded) so that none lands
    // after the CTA has exited, and report it.
    for (int c = 0; c < nch; ++c) mbar_wait(&h.wfull[c], 0, &h.err);
    atomicOr(a.status, kStatusTimeout);
  }
}

template <int PHASE, int NP, bool MULTI>
cudaError_t launch_np(const LutArgs& a, const LutPlan& p, cudaStream_t st) {
  auto kern = lut_kernel<PHASE, NP, MULTI>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
  if (e != cudaSuccess) return e;
  if (p.KS > 8) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  LutArgs b = a;
  b.KS = p.KS;
  int rbs = 0;  // grid x: the row blocks of all problems, in order
  for (int i = 0; i < a.count; ++i) {
    b.prob[i].CPC = p.CPC[i];
    b.prob[i].rb0 = rbs;
    rbs += a.prob[i].sm.RB;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)rbs, (unsigned)p.KS, (unsigned)((a.tokens + kGroupTokens - 1) / kGroupTokens));
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
  return cudaLaunchKernelEx(&cfg, kern, b);
}

}  // namespace

namespace {

// Split of one sign matrix for a pass of T <= 16 tokens, run as ceil(T / 4)
// token groups of CTAs: about two CTAs per SM (row blocks x KS x groups ~
// 2 SMs, KS <= 16 CTAs per cluster), CTAs small enough that three fit on an
// SM, and at most kMaxCPC chunks each. Returns KS (0: no plan), *cpc and
// *smem.
int plan_one(const SignMatrix& sm, int T, int sms, int max_smem, int* cpc_out, int* smem_out) {
  const int Tg = T < kGroupTokens ? T : kGroupTokens;
  const int groups = (T + kGroupTokens - 1) / kGroupTokens;
  const int cap = max_smem / 3 < 72 * 1024 ? max_smem / 3 : 72 * 1024;
  const int64_t tiles = (int64_t)sm.RB * groups;
  int ks = (int)((2 * sms + tiles - 1) / tiles);
  if (ks > kMaxKS) ks = kMaxKS;
  if (ks > sm.NCH) ks = sm.NCH;
  if (ks < 1) ks = 1;
  for (; ks <= kMaxKS && ks <= sm.NCH; ++ks) {
    const int cpc = (sm.NCH + ks - 1) / ks;
    if (cpc > kMaxCPC) continue;
    const int KS = (sm.NCH + cpc - 1) / cpc;
    const int need = lut_smem(cpc, KS, Tg, pairs_for(Tg)).total;
    if (need <= cap || (ks == kMaxKS || ks == sm.NCH)) {
      if (need > max_smem) return 0;
      *cpc_out = cpc;
      *smem_out = need;
      return KS;
    }
  }
  return 0;
}

}  // namespace

// One problem: its own split. Several (layers sharing their input, one
// launch): the largest of their splits' cluster sizes for all, each problem
// cutting its columns into that many slices (the last CTAs of a problem with
// fewer chunks get none).
LutPlan plan_lut(const SignMatrix* sm, int count, int T, int num_sms, int max_smem) {
  LutPlan p;
  if (count < 1 || count > kMaxGroup || T < 1 || T > kMaxPassTokens) return p;
  const int sms = num_sms > 0 ? num_sms : 148;
  const int Tg = T < kGroupTokens ? T : kGroupTokens;
  int KS = 0;
  for (int i = 0; i < count; ++i) {
    if (sm[i].RB < 1 || sm[i].NCH < 1) return p;
    int cpc = 0, smem = 0;
    const int k = plan_one(sm[i], T, sms, max_smem, &cpc, &smem);
    if (k == 0) return p;
    if (k > KS) KS = k;
  }
  int smem = 0;
  for (int i = 0; i < count; ++i) {
    const int cpc = (sm[i].NCH + KS - 1) / KS;
    if (cpc > kMaxCPC) return p;
    const int need = lut_smem(cpc, KS, Tg, pairs_for(Tg)).total;
    if (need > max_smem) return p;
    if (need > smem) smem = need;
    p.CPC[i] = cpc;
  }
  p.KS = KS;
  p.smem = smem;
  p.ok = true;
  return p;
}

template <int PHASE>
cudaError_t launch_phase(const LutArgs& a, const LutPlan& p, cudaStream_t st) {
  const bool multi = a.count > 1;
  switch (pairs_for(a.tokens < kGroupTokens ? a.tokens : kGroupTokens)) {
    case 0: return multi ? launch_np<PHASE, 0, true>(a, p, st) : launch_np<PHASE, 0, false>(a, p, st);
    case 1: return multi ? launch_np<PHASE, 1, true>(a, p, st) : launch_np<PHASE, 1, false>(a, p, st);
    default: return multi ? launch_np<PHASE, 2, true>(a, p, st) : launch_np<PHASE, 2, false>(a, p, st);
  }
}

cudaError_t launch_lut(int phase, const LutArgs& a, const LutPlan& p, cudaStream_t st) {
  return phase == 1 ? launch_phase<1>(a, p, st) : launch_phase<2>(a, p, st);
}

}  // namespace af1
