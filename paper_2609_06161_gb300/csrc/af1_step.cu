// af1_step.cu — a whole decode step (many AF1 linears in dependent levels)
// as ONE persistent kernel launch.
//
// Each linear is the AF1 forward pass y = a * (U (s * (V^T (b * x))))
// (AF1 Sec. 3.1, Eq. final_reconstruction, evaluated right to left as
// Eq. binary_paths): phase 1 contracts B = V^T (r x n) with z = b * x,
// phase 2 contracts U (m x r) with s' = s * t. A decoder layer chains its
// linears (q | k | v, then o, then gate | up, then down), so one decode token
// through a 32-layer model is a chain of 128 levels of two dependent phases.
// Separate kernels pay a kernel boundary per phase; here one cooperative
// launch covers the chain, and a hand-off between phases costs one trip of
// the data through L2.
//
// Work. Each phase of each linear is cut into tiles: G row blocks (128 rows
// each) x a slice of consecutive 128-column chunks (a K slice). The host
// plans the tiles of every stage — (level, phase 1), (level, phase 2),
// (level, output) — and deals them to the CTAs of one resident wave, longest
// first to the least loaded CTA; a CTA runs its tiles in stage order. A
// lookup tile stages its slice of the input in shared memory, builds the
// lookup tables of signed sums (af1_lut_common.cuh), runs the lookups over
// its sign tiles (which a producer warp copies into a ring of shared-memory
// slots with bulk copies, running ahead across tiles and stages: signs are
// constants) and stores its split-K partial sums.
//
// Hand-offs. Partial sums are stored as 8-byte words {FP32 value, run tag},
// each written with one 64-bit store (single-copy atomic), so a consumer
// knows a value is from this run when it reads it: it reads the words of its
// slice and re-reads (bounded) any whose tag is not yet the run's. No
// counter, fence or atomic lies between a producer and its consumers:
//   * phase 2 sums the phase-1 partials of its rank slice in slice order:
//     s'[k] = s[k] * sum_j t_j[k];
//   * a phase-1 input that is the output of an earlier linear (same pointer
//     and row stride, FP16 outputs) is read the same way from that linear's
//     phase-2 partials, rounded as that output is: FP16(a[k] * sum_j u_j[k])
//     (for a SwiGLU input, of both producers, then FP16(SiLU(g) u));
//   * output tiles (stage (level, output)) store y = FP16 or FP32 of
//     a * sum_j u_j, for the caller, and count the row blocks stored on one
//     device-scope counter; a phase-1 input that is NOT produced in the step
//     is read only once every earlier level's outputs are stored (the
//     counter reaches their row-block count), or, at level 0 with
//     AF1_STEP_WAIT_GATE, once the gate word is set.
// The run tag is the workspace's epoch word + 1, read at launch; the last
// CTA to finish advances the epoch and clears the counter, so every run
// starts clean, and partial words left by an earlier run never match.
//
// Results are deterministic: every sum over slices runs in slice order, and
// a chained input is rounded exactly as the stored output. Every wait is
// bounded (af1_set_wait_cycles); one that gives up sets the status word and
// the run's abort word, every other wait then gives up at once, each CTA
// lets its copies in flight land, and the run still ends with the epoch
// advanced and the counter cleared.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <new>
#include <queue>
#include <string>
#include <tuple>
#include <vector>

#include "af1.h"
#include "af1_internal.h"
#include "af1_layout.h"
#include "af1_lut_common.cuh"
#include "af1_ptx.cuh"

namespace af1 {

constexpr int kStepMaxTokens = 4;
constexpr int kStepMaxG = 4;  // row blocks per tile

// One FP16 operand of a phase-1 input: an external buffer, or the output of
// an earlier linear read from its phase-2 partial sums.
struct StepInput {
  const __half* x;           // external: FP16 [T][ldx]
  int64_t ldx;
  int64_t part_off;          // chained (>= 0): workspace offset of the producer's phase-2 partials
  int part_ks;               // the producer's K slices
  int64_t part_ld;           // the producer's padded rows (RB 128)
  const __half* part_scale;  // the producer's row scale a
};

struct StepProblem {
  const uint8_t* signs;  // af1_layout.h row-block layout
  int64_t R, C;
  int RB, NCH;
  int KS;     // K slices: partial sums per output row
  int phase;  // 1 or 2
  int level;
  int swiglu;               // phase 1: the input is h = FP16(SiLU(in) in2)
  int chained;              // phase 1: some operand is read from partial sums
  int external_wait;        // phase 1: some operand is external and level > 0
  unsigned fin_target;      // row blocks of y stored by all earlier levels
  StepInput in, in2;        // phase 1 operands (in2: the SwiGLU up operand)
  const __half* colscale;   // phase 1: b
  const __half* rankscale;  // phase 2: s (applied to the summed phase-1 partials)
  const __half* rowscale;   // phase 2: a
  int64_t pin_off;          // phase 2: workspace offset of phase 1's partials
  int pin_ks;               // phase 2: KS of phase 1
  int64_t pout_off;         // workspace offset of this problem's partials [KS][T][RB 128] (8-byte words)
  void* y;                  // phase 2 output [T][ldy]
  int64_t ldy;
};

// One tile of problem `prob`: row blocks [rb0, rb0 + G). kind 0: lookups
// over chunks [c0, c0 + nch), the ks-th K slice; kind 1 (phase-2
// problems): store those rows of y.
struct StepTask {
  int prob, rb0, G, c0, nch, ks, kind;
};

namespace {

constexpr int kConsumers = 256;                // 8 warps: staging, tables, lookups, sums
constexpr int kStepThreads = kConsumers + 32;  // + the producer warp
constexpr int kMaxSlots = 64;                  // ring slots (one 2 KB sign tile each)
constexpr int kMaxG = kStepMaxG;
constexpr int kBarConsumers = 1;               // named barrier of the 256 consumer threads
constexpr int kSmemBudget = 110 * 1024;        // per CTA: two CTAs per SM

// Workspace header words (uint32 at byte offsets 4 i).
constexpr int kWsStatus = 0;  // sticky status (af1_workspace_status)
constexpr int kWsDone = 1;    // CTAs finished (the last one closes the run)
constexpr int kWsGate = 2;    // AF1_STEP_WAIT_GATE: level 0 waits until nonzero
constexpr int kWsAbort = 3;   // this run gave up somewhere: every wait stops
constexpr int kWsEpoch = 4;   // the last run's tag; this run's tag is epoch + 1
constexpr int kWsStored = 5;  // row blocks of y stored in this run
constexpr int64_t kWsHeader = 256;

struct StepArgs {
  const StepProblem* probs;
  const StepTask* tasks;
  const int* cta_first;  // [P + 1]: tasks of CTA i are [cta_first[i], cta_first[i + 1])
  uint8_t* ws;
  int T, ydtype, nslot, cpc_max, ctas, gate;
  long long wait_cycles;
};

struct __align__(8) StepHeader {
  uint64_t full[kMaxSlots];   // slot holds its sign tile (bulk copy)
  uint64_t empty[kMaxSlots];  // the 8 consumer warps are done with the slot
  uint32_t err;               // a wait of this CTA gave up
  uint32_t stop;              // consumers stopped: the producer stops too
  uint32_t tag;               // this run's tag
  uint32_t issued;            // tiles copied
  uint32_t last_cta;
};

struct StepSmem {
  int tbl, ring, zs, red, hdr, total;
};

__host__ __device__ inline int align256i(int v) { return (v + 255) & ~255; }

__host__ __device__ inline StepSmem step_smem(int cpc_max, int T, int nslot) {
  StepSmem p;
  int off = 0;
  p.tbl = off;  // 256-aligned: the lookups address 256-byte table windows
  off += table_chunk_bytes(pairs_for(T)) * cpc_max;
  p.ring = off;
  off += nslot * kChunkBytes;
  p.zs = off;
  off = align256i(off + T * zrow_floats(cpc_max) * 4);
  p.red = off;
  off = align256i(off + kMaxG * T * kBlockRows * 4);
  p.hdr = off;
  off = align256i(off + (int)sizeof(StepHeader));
  p.total = off + 256;  // slack for aligning the base
  return p;
}

__device__ __forceinline__ bool aborted(const StepArgs& a) {
  return *reinterpret_cast<const volatile unsigned*>(a.ws + 4 * kWsAbort) != 0;
}

// Bounded wait until *p >= target (acquire). Gives up on the budget or when
// the run's abort word is set.
__device__ __forceinline__ bool wait_count(const unsigned* p, unsigned target, const StepArgs& a) {
  if (ld_acquire_gpu(p) >= target) return true;
  const long long t0 = clock64();
  unsigned it = 0;
  while (ld_acquire_gpu(p) < target) {
    nanosleep_ns(100);
    if ((++it & 15u) == 0 && aborted(a)) return false;
    if (clock64() - t0 > a.wait_cycles) return false;
  }
  return true;
}

// Producer's wait for a free slot: gives up when the consumers stopped.
__device__ __forceinline__ bool wait_slot(uint64_t* bar, uint32_t parity, StepHeader& h, long long budget) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (*reinterpret_cast<volatile uint32_t*>(&h.stop) != 0) return false;
    if (clock64() - t0 > budget) {
      atomicOr(&h.err, 1u);
      return false;
    }
  }
  return true;
}

// ---- tagged partial sums ---------------------------------------------------------

__device__ __forceinline__ void st_tagged(uint64_t* p, float v, uint32_t tag) {
  const uint64_t w = (uint64_t)__float_as_uint(v) | ((uint64_t)tag << 32);
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}
__device__ __forceinline__ uint64_t ld_tagged(const uint64_t* p) {
  uint64_t w;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(w) : "l"(p) : "memory");
  return w;
}

// Sum over j < ks of the values at p + j * stride, in j order, each read
// once it carries `tag` (bounded re-reads). On failure `ok` turns false and
// the value is meaningless.
__device__ __forceinline__ float sum_tagged(const uint64_t* p, int64_t stride, int ks, uint32_t tag,
                                            const StepArgs& a, bool& ok) {
  float s = 0.f;
  for (int j0 = 0; j0 < ks; j0 += 8) {
    uint64_t w[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) w[u] = j0 + u < ks ? ld_tagged(p + (j0 + u) * stride) : 0ull;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (j0 + u >= ks) break;
      if ((uint32_t)(w[u] >> 32) != tag && ok) {
        const long long t0 = clock64();
        unsigned it = 0;
        do {
          nanosleep_ns(100);  // leave the load pipe to the lookups of the SM's other CTA
          w[u] = ld_tagged(p + (j0 + u) * stride);
          if (clock64() - t0 > a.wait_cycles || ((++it & 31u) == 0 && aborted(a))) {
            ok = false;
            break;
          }
        } while ((uint32_t)(w[u] >> 32) != tag);
      }
      s += __uint_as_float((uint32_t)w[u]);
    }
  }
  return s;
}

// Value (FP16-exact, as float) of input column k of token t of one operand.
__device__ __forceinline__ float operand_value(const StepInput& in, const uint8_t* ws, int T, int t, int64_t k,
                                               uint32_t tag, const StepArgs& a, bool& ok) {
  if (in.part_off < 0) return __half2float(__ldcg(in.x + (int64_t)t * in.ldx + k));
  const uint64_t* p = reinterpret_cast<const uint64_t*>(ws + in.part_off) + (int64_t)t * in.part_ld + k;
  const float u = sum_tagged(p, (int64_t)T * in.part_ld, in.part_ks, tag, a, ok);
  return __half2float(__float2half_rn(u * __half2float(in.part_scale[k])));
}

// Phase-1 input of columns [k0, k0 + nch 128) when an operand is chained:
// zs[t][k + k / 32] = b[k] * x[t][k] (x the operand, or FP16(SiLU(g) u)).
__device__ __forceinline__ void stage_chained_input(const StepProblem& pb, const uint8_t* ws, int T, int nch,
                                                    int64_t k0, float* zs, int zrow, int tid, uint32_t tag,
                                                    const StepArgs& a, bool& ok) {
  const int cols = nch * kChunkCols;
  for (int i = tid; i < T * cols; i += kConsumers) {
    const int t = i / cols, k = i - t * cols;
    const int64_t col = k0 + k;
    float z = 0.f;
    if (col < pb.C) {
      float xv = operand_value(pb.in, ws, T, t, col, tag, a, ok);
      if (pb.swiglu) xv = swiglu_h(xv, operand_value(pb.in2, ws, T, t, col, tag, a, ok));
      z = xv * __half2float(pb.colscale[col]);
    }
    zs[t * zrow + k + (k >> 5)] = z;
  }
}

// Phase-2 input of columns [k0, k0 + nch 128): s'[t][k] = s[k] * sum_j P1[j][t][k]
// (slices in order), 0 for k >= C.
__device__ __forceinline__ void stage_rank_input(const StepProblem& pb, const uint8_t* ws, int T, int nch, int64_t k0,
                                                 float* zs, int zrow, int tid, uint32_t tag, const StepArgs& a,
                                                 bool& ok) {
  const int cols = nch * kChunkCols;
  const int64_t ldp = (int64_t)pb.NCH * kChunkCols;  // rows of phase 1 (padded) = columns here
  const uint64_t* pin = reinterpret_cast<const uint64_t*>(ws + pb.pin_off);
  for (int i = tid; i < T * cols; i += kConsumers) {
    const int t = i / cols, k = i - t * cols;
    const int64_t col = k0 + k;
    float v = 0.f;
    if (col < pb.C)
      v = __half2float(pb.rankscale[col]) *
          sum_tagged(pin + (int64_t)t * ldp + col, (int64_t)T * ldp, pb.pin_ks, tag, a, ok);
    zs[t * zrow + k + (k >> 5)] = v;
  }
}

// Lookups of one chunk for thread (r, g), as lookup_chunk in
// af1_lut_common.cuh but with every table read of the chunk issued before
// the additions (an add tree per word).
__device__ __forceinline__ float lds_f(uint32_t addr) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ float2 lds_f2(uint32_t addr) {
  float2 v;
  asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
  return v;
}

template <int NP>
__device__ __forceinline__ void lookup_chunk_ilp(uint32_t tb, const uint32_t* wc, int g,
                                                 float (&acc)[NP == 0 ? 1 : 2 * NP]) {
  const uint32_t w0 = wc[(2 * g) * kBlockRows], w1 = wc[(2 * g + 1) * kBlockRows];
  if constexpr (NP == 0) {
    const uint32_t pat0 = (uint32_t)(2 * g * 64) * 0x01010101u, pat1 = (uint32_t)((2 * g + 1) * 64) * 0x01010101u;
    const uint32_t lo0 = ((w0 << 2) & 0x3C3C3C3Cu) | pat0, hi0 = ((w0 >> 2) & 0x3C3C3C3Cu) | pat0;
    const uint32_t lo1 = ((w1 << 2) & 0x3C3C3C3Cu) | pat1, hi1 = ((w1 >> 2) & 0x3C3C3C3Cu) | pat1;
    float v[16];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const uint32_t base = tb + (uint32_t)(j * 256);
      v[j] = lds_f(__byte_perm((j & 1) ? hi0 : lo0, base, 0x7650 | (j >> 1)));
      v[8 + j] = lds_f(__byte_perm((j & 1) ? hi1 : lo1, base, 0x7650 | (j >> 1)));
    }
#pragma unroll
    for (int k = 8; k >= 1; k >>= 1)
#pragma unroll
      for (int j = 0; j < k; ++j) v[j] += v[j + k];
    acc[0] += v[0];
  } else {
    const uint32_t lo0 = ((w0 << 3) & 0x78787878u), hi0 = ((w0 >> 1) & 0x78787878u);
    const uint32_t lo1 = ((w1 << 3) & 0x78787878u) | 0x80808080u, hi1 = ((w1 >> 1) & 0x78787878u) | 0x80808080u;
#pragma unroll
    for (int pp = 0; pp < NP; ++pp) {
      float2 v[16];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t base = tb + (uint32_t)(pp * 4096 + j * 512 + g * 256);
        v[j] = lds_f2(__byte_perm((j & 1) ? hi0 : lo0, base, 0x7650 | (j >> 1)));
        v[8 + j] = lds_f2(__byte_perm((j & 1) ? hi1 : lo1, base, 0x7650 | (j >> 1)));
      }
#pragma unroll
      for (int k = 8; k >= 1; k >>= 1)
#pragma unroll
        for (int j = 0; j < k; ++j) {
          v[j].x += v[j + k].x;
          v[j].y += v[j + k].y;
        }
      acc[2 * pp] += v[0].x;
      acc[2 * pp + 1] += v[0].y;
    }
  }
}

// Lookups of one tile of G row blocks (G a compile-time constant: a runtime
// row-block count behind guards made this loop 2.3x slower in a probe):
// chunk by chunk, wait for the chunk's G sign tiles (ring order: chunk, then
// row block), look them up against the chunk's tables, free the slots.
template <int NP, int G>
__device__ __forceinline__ void lookup_tile(uint32_t tbl0, const uint32_t* ringw, StepHeader& h, int nch, int NSLOT,
                                            int& cs, uint32_t& cpar, bool& ok, long long budget, int r, int g,
                                            int lane, float (&acc)[kMaxG][NP == 0 ? 1 : 2 * NP]) {
  constexpr int TCB = table_chunk_bytes(NP);
  for (int k = 0; k < nch; ++k) {
    const uint32_t tb = tbl0 + (uint32_t)(k * TCB);
    int slot[G];
#pragma unroll
    for (int gi = 0; gi < G; ++gi) {
      slot[gi] = cs;
      // After a wait gave up, the remaining waits are skipped (the tile is
      // abandoned at its end).
      if (ok) ok = mbar_wait(&h.full[cs], cpar, &h.err, budget);
      if (++cs == NSLOT) {
        cs = 0;
        cpar ^= 1u;
      }
    }
#pragma unroll
    for (int gi = 0; gi < G; ++gi)
      lookup_chunk_ilp<NP>(tb, ringw + (size_t)slot[gi] * (kChunkBytes / 4) + r, g, acc[gi]);
    __syncwarp();
    if (lane == 0)
#pragma unroll
      for (int gi = 0; gi < G; ++gi) mbar_arrive(&h.empty[slot[gi]]);
  }
}

template <int NP>
__global__ void __launch_bounds__(kStepThreads, 2) step_kernel(const __grid_constant__ StepArgs a) {
  constexpr int NACC = NP == 0 ? 1 : 2 * NP;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 255) & ~(uintptr_t)255);
  const int T = a.T, NSLOT = a.nslot;
  const StepSmem sp = step_smem(a.cpc_max, T, NSLOT);
  uint8_t* ring = smem + sp.ring;
  float* zs = reinterpret_cast<float*>(smem + sp.zs);
  float* red = reinterpret_cast<float*>(smem + sp.red);
  StepHeader& h = *reinterpret_cast<StepHeader*>(smem + sp.hdr);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int first = a.cta_first[blockIdx.x], end = a.cta_first[blockIdx.x + 1];
  unsigned* wsw = reinterpret_cast<unsigned*>(a.ws);

  if (tid == 0) {
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(&h.full[s], 1);
      mbar_init(&h.empty[s], kConsumers / 32);
    }
    h.err = 0;
    h.stop = 0;
    h.issued = 0;
    h.tag = *reinterpret_cast<volatile unsigned*>(wsw + kWsEpoch) + 1u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();
  const uint32_t tag = h.tag;

  if (warp == kConsumers / 32) {
    // ---- producer: the sign tiles of this CTA's lookup tiles, in order -------
    if (lane == 0) {
      uint32_t issued = 0, par = 1;  // parity of a slot's previous release (after the first lap)
      int s = 0;
      bool ok = true;
      for (int i = first; i < end && ok; ++i) {
        const StepTask tk = a.tasks[i];
        if (tk.kind != 0) continue;
        const uint8_t* base = a.probs[tk.prob].signs;
        const int NCH = a.probs[tk.prob].NCH;
        for (int k = 0; k < tk.nch && ok; ++k)
          for (int gi = 0; gi < tk.G; ++gi) {
            if (issued >= (uint32_t)NSLOT) {
              ok = wait_slot(&h.empty[s], par, h, a.wait_cycles);
              if (!ok) break;
            }
            mbar_expect_tx(&h.full[s], (uint32_t)kChunkBytes);
            bulk_g2s(ring + (size_t)s * kChunkBytes,
                     base + ((int64_t)(tk.rb0 + gi) * NCH + tk.c0 + k) * kChunkBytes, kChunkBytes, &h.full[s]);
            ++issued;
            if (++s == NSLOT) {
              s = 0;
              par ^= 1u;
            }
          }
      }
      h.issued = issued;
    }
    __syncwarp();
  } else {
    // ---- consumers ----------------------------------------------------------
    const int r = tid & (kBlockRows - 1), g = tid >> 7;
    const int zrow = zrow_floats(a.cpc_max);
    const uint32_t tbl0 = smem_u32(smem + sp.tbl);
    const uint32_t* ringw = reinterpret_cast<const uint32_t*>(ring);
    int cs = 0;         // ring slot of the next sign tile
    uint32_t cpar = 0;  // parity of that slot's next fill
    bool ok = true;     // no wait of this thread gave up
    for (int i = first; i < end; ++i) {
      const StepTask tk = a.tasks[i];
      const StepProblem& pb = a.probs[tk.prob];
      const int G = tk.G, nch = tk.nch;
      const int64_t ldp = (int64_t)pb.RB * kBlockRows;
      uint64_t* pout = reinterpret_cast<uint64_t*>(a.ws + pb.pout_off);
      if (tk.kind == 1) {
        // ---- output tile: y rows of [rb0, rb0 + G) --------------------------
        for (int idx = tid; idx < G * T * kBlockRows; idx += kConsumers) {
          const int gi = idx / (T * kBlockRows), rest = idx - gi * T * kBlockRows;
          const int t = rest / kBlockRows, rr = rest - t * kBlockRows;
          const int64_t row = (int64_t)(tk.rb0 + gi) * kBlockRows + rr;
          if (row >= pb.R) continue;
          const float v = __half2float(pb.rowscale[row]) *
                          sum_tagged(pout + (int64_t)t * ldp + row, (int64_t)T * ldp, pb.KS, tag, a, ok);
          if (a.ydtype == AF1_F16)
            reinterpret_cast<__half*>(pb.y)[(int64_t)t * pb.ldy + row] = __float2half_rn(v);
          else
            reinterpret_cast<float*>(pb.y)[(int64_t)t * pb.ldy + row] = v;
        }
        if (!ok) atomicOr(&h.err, 1u);
        named_sync(kBarConsumers, kConsumers);
        if (tid == 0) {
          fence_acq_rel_gpu();  // release: this CTA's y stores before the count
          red_relaxed_gpu(wsw + kWsStored, (unsigned)G);
        }
        if (h.err != 0) break;
        continue;
      }
      // ---- lookup tile -----------------------------------------------------------
      // 1. external inputs exist
      if (pb.phase == 1 && tid == 0) {
        bool w = true;
        if (pb.external_wait) w = wait_count(wsw + kWsStored, pb.fin_target, a);
        else if (pb.level == 0 && a.gate) w = wait_count(wsw + kWsGate, 1u, a);
        if (!w) atomicOr(&h.err, 1u);
      }
      named_sync(kBarConsumers, kConsumers);
      if (h.err != 0) break;
      // 2. stage the slice's input (chained operands and phase-1 partials are
      //    read as soon as their words carry this run's tag)
      const int64_t k0 = (int64_t)tk.c0 * kChunkCols;
      if (pb.phase == 1) {
        if (pb.chained) {
          stage_chained_input(pb, a.ws, T, nch, k0, zs, zrow, tid, tag, a, ok);
        } else {
          LutProblem lp = {};
          lp.sm.C = pb.C;
          lp.ldx = pb.in.ldx;
          lp.colscale = pb.colscale;
          if (pb.swiglu)
            stage_activations<1, kConsumers, true>(lp, pb.in.x, pb.in2.x, nullptr, T, nch, k0, zs, zrow, tid);
          else
            stage_activations<1, kConsumers, false>(lp, pb.in.x, nullptr, nullptr, T, nch, k0, zs, zrow, tid);
        }
      } else {
        stage_rank_input(pb, a.ws, T, nch, k0, zs, zrow, tid, tag, a, ok);
      }
      if (!ok) atomicOr(&h.err, 1u);
      named_sync(kBarConsumers, kConsumers);
      if (h.err != 0) break;
      build_tables<NP, kConsumers>(smem + sp.tbl, zs, zrow, T, nch, tid);
      named_sync(kBarConsumers, kConsumers);
      // 3. lookups over the tile's sign tiles (ring order: chunk, then row block)
      float acc[kMaxG][NACC];
#pragma unroll
      for (int gi = 0; gi < kMaxG; ++gi)
#pragma unroll
        for (int t = 0; t < NACC; ++t) acc[gi][t] = 0.f;
      switch (G) {
        case 1: lookup_tile<NP, 1>(tbl0, ringw, h, nch, NSLOT, cs, cpar, ok, a.wait_cycles, r, g, lane, acc); break;
        case 2: lookup_tile<NP, 2>(tbl0, ringw, h, nch, NSLOT, cs, cpar, ok, a.wait_cycles, r, g, lane, acc); break;
        case 3: lookup_tile<NP, 3>(tbl0, ringw, h, nch, NSLOT, cs, cpar, ok, a.wait_cycles, r, g, lane, acc); break;
        default: lookup_tile<NP, 4>(tbl0, ringw, h, nch, NSLOT, cs, cpar, ok, a.wait_cycles, r, g, lane, acc); break;
      }
      // 4. partial sums of the tile's rows -> workspace (tagged words)
      if (g == 1) {
#pragma unroll
        for (int gi = 0; gi < kMaxG; ++gi)
          if (gi < G)
#pragma unroll
            for (int t = 0; t < NACC; ++t)
              if (t < T) red[(gi * T + t) * kBlockRows + r] = acc[gi][t];
      }
      named_sync(kBarConsumers, kConsumers);
      if (g == 0) {
#pragma unroll
        for (int gi = 0; gi < kMaxG; ++gi)
          if (gi < G)
#pragma unroll
            for (int t = 0; t < NACC; ++t)
              if (t < T)
                st_tagged(pout + ((int64_t)tk.ks * T + t) * ldp + (int64_t)(tk.rb0 + gi) * kBlockRows + r,
                          acc[gi][t] + red[(gi * T + t) * kBlockRows + r], tag);
      }
      named_sync(kBarConsumers, kConsumers);  // red is reused by the next tile
      if (h.err != 0) break;
    }
    named_sync(kBarConsumers, kConsumers);
    if (tid == 0) {
      if (h.err != 0) {
        atomicOr(wsw + kWsStatus, kStatusTimeout);
        atomicOr(wsw + kWsAbort, 1u);
      }
      h.stop = 1;  // the producer issues nothing more
    }
  }
  __syncthreads();

  // ---- teardown --------------------------------------------------------------
  if (tid == 0) {
    // Copies in flight land before the CTA exits: wait for the last copy
    // issued into each slot (after a normal run every one has landed and
    // the waits return at once; after an abort some may still be in flight).
    const uint32_t iss = h.issued;
    const uint32_t lo = iss > (uint32_t)NSLOT ? iss - (uint32_t)NSLOT : 0u;
    for (uint32_t c = lo; c < iss; ++c)
      mbar_wait(&h.full[c % (uint32_t)NSLOT], (c / NSLOT) & 1u, &h.err, a.wait_cycles);
    if (h.err != 0) {
      atomicOr(wsw + kWsStatus, kStatusTimeout);
      atomicOr(wsw + kWsAbort, 1u);
    }
    fence_acq_rel_gpu();
    const unsigned old = atom_add_acq_rel_gpu(wsw + kWsDone, 1u);
    h.last_cta = old == (unsigned)(a.ctas - 1) ? 1u : 0u;
  }
  __syncthreads();
  if (h.last_cta != 0 && tid == 0) {
    // Every other CTA is done: close the run.
    wsw[kWsStored] = 0u;
    wsw[kWsDone] = 0u;
    wsw[kWsAbort] = 0u;
    if (a.gate) wsw[kWsGate] = 0u;
    wsw[kWsEpoch] = tag;  // the next run's tag is tag + 1
  }
}

}  // namespace
}  // namespace af1

// ---------------------------------------------------------------------------
// Host side: the plan
// ---------------------------------------------------------------------------

struct af1_step {
  int device = 0;
  int T = 0, ydtype = 0, nslot = 0, cpc_max = 0, ctas = 0, smem = 0, gate = 0, levels = 0;
  int64_t ws_bytes = 0;
  int ntasks = 0, nprobs = 0, chained = 0;
  void* dev = nullptr;  // one device allocation: problems, tasks, cta_first
  const af1::StepProblem* probs = nullptr;
  const af1::StepTask* tasks = nullptr;
  const int* cta_first = nullptr;
  double model_us = 0.0;  // modelled critical path of the plan (af1_step_info)
};

namespace {

using af1::kStepMaxG;
using af1::StepInput;
using af1::StepProblem;
using af1::StepTask;

int fail(int code, const std::string& msg) { return af1::set_error(code, msg); }

int64_t align256(int64_t v) { return (v + 255) & ~(int64_t)255; }

// Planning cost model (us per tile, on one of the two CTAs of an SM): a fixed
// part (staging the input through L2, the table build's barriers, storing
// partial sums), lookups per 2 KB sign tile and the table build per chunk;
// output tiles read their partial sums and store rows.
constexpr double kTileFixedUs = 2.0;
constexpr double kTileLookupUs = 0.3;
constexpr double kStageWordUs = 0.0;  // per chunk and partial-sum word of its K slice (not modelled)
constexpr double kChunkTableUs = 0.03;
constexpr double kOutFixedUs = 0.8;
constexpr double kOutPerBlockUs = 0.1;
constexpr int kOutG = 4;  // row blocks per output tile
constexpr double kHandoffUs = 1.5;  // a stage's results reach its consumers

struct TileShape {
  int CPC = 1, G = 1;
};

// stage_us: staging cost per chunk of the tile's K slice (reading the
// producers' partial sums, 0 for an external input).
double tile_cost(int G, int nch, double stage_us = 0.0) {
  return kTileFixedUs + kTileLookupUs * G * nch + (kChunkTableUs + stage_us) * nch;
}

// Consumers of a row block's partial sums read one per K slice; a tile
// covers enough chunks that there are at most kMaxSlices of them (where the
// chunk bound allows).
constexpr int kMaxSlices = 8;

// Largest tile (by cost) of a problem whose cost stays <= tau.
TileShape shape_for(const af1::SignMatrix& sm, int cpc_max, double tau, double stage_us) {
  TileShape best;
  best.CPC = std::min(cpc_max, std::min(sm.NCH, (sm.NCH + kMaxSlices - 1) / kMaxSlices));
  double bc = -1.0;
  for (int G = 1; G <= kStepMaxG && G <= sm.RB; G *= 2)
    for (int cpc = best.CPC; cpc <= cpc_max && cpc <= sm.NCH; ++cpc) {
      const double c = tile_cost(G, cpc, stage_us);
      if (c <= tau && c > bc) {
        bc = c;
        best.CPC = cpc;
        best.G = G;
      }
    }
  return best;
}

struct PlanTile {
  int prob, rb0, G, c0, nch, ks, kind;
  double cost;
};

// The tiles of every stage — (level, phase 1), (level, phase 2), (level,
// output) — dealt to `ctas` CTAs by list scheduling on a simulated clock:
// each tile (longest first) goes to the CTA that can start it earliest,
// no earlier than the stage's input is ready. For each lookup stage, every
// tile shape's cost is tried as a bound; each problem then takes its
// largest tile within the bound (K slices of even size), and the bound whose
// stage ends first wins. A CTA's tasks are in stage order, and every tile
// depends only on tiles of earlier stages: with every CTA resident the step
// cannot deadlock.
struct TilePlan {
  std::vector<StepTask> tasks;
  std::vector<int> cta_first;  // [ctas + 1]
  std::vector<int> KS;         // per problem
  double model_us = 0.0;       // modelled end of the step
};

int cpc_max_for(int T) { return T == 1 ? 16 : T == 2 ? 12 : 8; }

// ext_level[L]: level L has a phase-1 input that waits for stored outputs
// (an input not produced in the step, at L > 0). The output tiles of level L
// are dealt after level L + 1's phase-1 tiles unless level L + 1 waits for
// stored outputs (then they must come first in every CTA's order).
// prod_a / prod_b[q]: for a phase-1 problem, the phase-2 problem whose
// partial sums its input (SwiGLU: gate / up operand) is read from, or -1.
TilePlan plan_tiles(const std::vector<af1::SignMatrix>& sms, const std::vector<int>& level,
                    const std::vector<int>& phase, int levels, int cpc_max, int ctas,
                    const std::vector<char>& ext_level, const std::vector<int>& prod_a,
                    const std::vector<int>& prod_b) {
  const int nprob = (int)sms.size();
  TilePlan out;
  out.KS.assign(nprob, 0);
  // Staging cost per chunk of problem q's K slice: the partial-sum words each
  // input column needs (planned earlier: producers come first).
  auto stage_us = [&](int q) {
    int words = 0;
    if (phase[q] == 2) words = out.KS[q - 1];
    else {
      if (prod_a[q] >= 0) words += out.KS[prod_a[q]];
      if (prod_b[q] >= 0) words += out.KS[prod_b[q]];
    }
    return kStageWordUs * words;
  };
  std::vector<std::vector<PlanTile>> per_cta(ctas);
  // Simulated clock: free[c] is when CTA c finishes the tiles dealt to it so
  // far; a stage's tiles can start when its input is ready (the previous
  // lookup stage's end plus a hand-off), on the CTA free first.
  std::vector<double> free_at(ctas, 0.0);
  double ready = 0.0;
  auto make_tiles = [&](const std::vector<int>& sp, double tau) {
    std::vector<PlanTile> tiles;
    for (int q : sp) {
      const double su = stage_us(q);
      const TileShape ts = shape_for(sms[q], cpc_max, tau, su);
      const int KS = (sms[q].NCH + ts.CPC - 1) / ts.CPC;
      for (int rb = 0; rb < sms[q].RB; rb += ts.G)
        for (int ks = 0; ks < KS; ++ks) {
          PlanTile t;
          t.prob = q;
          t.rb0 = rb;
          t.G = std::min(ts.G, sms[q].RB - rb);
          t.c0 = (int)((int64_t)ks * sms[q].NCH / KS);  // even slices
          t.nch = (int)((int64_t)(ks + 1) * sms[q].NCH / KS) - t.c0;
          t.ks = ks;
          t.kind = 0;
          t.cost = tile_cost(t.G, t.nch, su);
          tiles.push_back(t);
        }
    }
    std::stable_sort(tiles.begin(), tiles.end(), [](const PlanTile& x, const PlanTile& y) { return x.cost > y.cost; });
    return tiles;
  };
  using E = std::pair<double, int>;  // (free time, CTA)
  // Deal `tiles` (longest first) from the state `fr`, starting no earlier
  // than `rdy`; returns the last end time. With `assign`, records the tiles.
  auto simulate = [&](const std::vector<PlanTile>& tiles, std::vector<double>& fr, double rdy, bool assign) {
    std::priority_queue<E, std::vector<E>, std::greater<E>> pq;
    for (int c = 0; c < ctas; ++c) pq.push({fr[c], c});
    double end = rdy;
    for (const PlanTile& t : tiles) {
      E top = pq.top();
      pq.pop();
      const double st = std::max(top.first, rdy);
      top.first = st + t.cost;
      fr[top.second] = top.first;
      end = std::max(end, top.first);
      if (assign) per_cta[top.second].push_back(t);
      pq.push(top);
    }
    return end;
  };
  auto output_tiles = [&](int lev) {
    std::vector<PlanTile> outs;
    for (int q = 0; q < nprob; ++q)
      if (level[q] == lev && phase[q] == 2)
        for (int rb = 0; rb < sms[q].RB; rb += kOutG) {
          PlanTile t;
          t.prob = q;
          t.rb0 = rb;
          t.G = std::min(kOutG, sms[q].RB - rb);
          t.c0 = 0;
          t.nch = 0;
          t.ks = 0;
          t.kind = 1;
          t.cost = kOutFixedUs + kOutPerBlockUs * t.G;
          outs.push_back(t);
        }
    return outs;
  };
  std::vector<double> out_ready(levels, 0.0);  // when a level's phase-2 partials exist
  for (int lev = 0; lev < levels; ++lev) {
    for (int ph = 1; ph <= 2; ++ph) {
      std::vector<int> sp;
      for (int q = 0; q < nprob; ++q)
        if (level[q] == lev && phase[q] == ph) sp.push_back(q);
      if (sp.empty()) continue;
      // Candidate bounds: every tile shape's cost for every problem of the stage.
      std::vector<double> cands;
      for (int q : sp)
        for (int G = 1; G <= kStepMaxG; G *= 2)
          for (int cpc = 1; cpc <= cpc_max; ++cpc) cands.push_back(tile_cost(G, cpc, stage_us(q)));
      std::sort(cands.begin(), cands.end());
      cands.erase(std::unique(cands.begin(), cands.end()), cands.end());
      // The bound whose tiles end the stage first from the current state.
      double best_end = -1.0, tau = cands.front();
      for (double cand : cands) {
        std::vector<double> fr = free_at;
        const double e = simulate(make_tiles(sp, cand + 1e-9), fr, ready, false);
        if (best_end < 0.0 || e < best_end - 1e-9) {
          best_end = e;
          tau = cand;
        }
      }
      const std::vector<PlanTile> tiles = make_tiles(sp, tau + 1e-9);
      for (const PlanTile& t : tiles) out.KS[t.prob] = std::max(out.KS[t.prob], t.ks + 1);
      const double end = simulate(tiles, free_at, ready, true);
      ready = end + kHandoffUs;
      if (ph == 2) out_ready[lev] = ready;
      // Output tiles of the previous level, when deferred past this level's
      // phase 1 (they do not hold up the chain).
      if (ph == 1 && lev > 0 && !ext_level[lev]) simulate(output_tiles(lev - 1), free_at, out_ready[lev - 1], true);
    }
    // Output tiles of this level, now if the next level waits for them.
    if (lev + 1 >= levels || ext_level[lev + 1]) {
      const double end = simulate(output_tiles(lev), free_at, out_ready[lev], true);
      if (lev + 1 < levels) ready = std::max(ready, end + kHandoffUs);
    }
  }
  out.model_us = *std::max_element(free_at.begin(), free_at.end());
  out.cta_first.assign(ctas + 1, 0);
  for (int c = 0; c < ctas; ++c) {
    out.cta_first[c] = (int)out.tasks.size();
    for (const PlanTile& t : per_cta[c]) {
      StepTask k;
      k.prob = t.prob;
      k.rb0 = t.rb0;
      k.G = t.G;
      k.c0 = t.c0;
      k.nch = t.nch;
      k.ks = t.ks;
      k.kind = t.kind;
      out.tasks.push_back(k);
    }
  }
  out.cta_first[ctas] = (int)out.tasks.size();
  return out;
}

// Linear indices sorted by level (stable) and the levels renumbered 0..L-1.
int order_levels(const std::vector<int>& lvl, std::vector<int>& order, std::vector<int>& level_of) {
  const int count = (int)lvl.size();
  order.resize(count);
  level_of.resize(count);
  for (int i = 0; i < count; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int p, int q) { return lvl[p] < lvl[q]; });
  int levels = 0;
  for (int j = 0; j < count; ++j) {
    if (j > 0 && lvl[order[j]] != lvl[order[j - 1]]) ++levels;
    level_of[order[j]] = levels;
  }
  return levels + 1;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

}  // namespace

extern "C" {

int af1_step_create(const af1_step_linear* lin, int count, int64_t tokens, int y_dtype, int32_t flags,
                    af1_step** out) {
  using namespace af1;
  if (out == nullptr) return fail(AF1_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (lin == nullptr || count < 1) return fail(AF1_ERR_INVALID_ARG, "need at least one linear");
  if (tokens < 1 || tokens > kStepMaxTokens)
    return fail(AF1_ERR_INVALID_ARG, "tokens must be in 1.." + std::to_string(kStepMaxTokens));
  if (y_dtype != AF1_F16 && y_dtype != AF1_F32) return fail(AF1_ERR_INVALID_ARG, "y_dtype must be AF1_F16 or AF1_F32");
  if ((flags & ~AF1_STEP_WAIT_GATE) != 0) return fail(AF1_ERR_INVALID_ARG, "unknown flags");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  const int T = (int)tokens;
  const int ysize = y_dtype == AF1_F16 ? 2 : 4;
  // ---- validate the linears ---------------------------------------------------
  for (int i = 0; i < count; ++i) {
    const af1_step_linear& l = lin[i];
    const std::string who = "linear " + std::to_string(i) + ": ";
    if (l.layer == nullptr) return fail(AF1_ERR_INVALID_ARG, who + "layer is NULL");
    if (l.layer->device != dev) return fail(AF1_ERR_BAD_POINTER, who + "the layer is not on the current device");
    if (l.level < 0) return fail(AF1_ERR_INVALID_ARG, who + "level must be >= 0");
    if (l.reserved != 0) return fail(AF1_ERR_INVALID_ARG, who + "reserved must be 0");
    if (l.x == nullptr || l.y == nullptr) return fail(AF1_ERR_INVALID_ARG, who + "x and y must not be NULL");
    if (l.ldx < l.layer->n || l.ldy < l.layer->m) return fail(AF1_ERR_INVALID_ARG, who + "ldx < n or ldy < m");
    if (l.ldx % 8 != 0 || (l.ldy * ysize) % 16 != 0)
      return fail(AF1_ERR_MISALIGNED, who + "ldx and ldy * element size must be multiples of 16 bytes");
    if ((reinterpret_cast<uintptr_t>(l.x) & 15) != 0 || (reinterpret_cast<uintptr_t>(l.y) & 15) != 0 ||
        (reinterpret_cast<uintptr_t>(l.x2) & 15) != 0)
      return fail(AF1_ERR_MISALIGNED, who + "x, x2 and y must be 16-byte aligned");
    if (!is_device_ptr(l.x) || !is_device_ptr(l.y) || (l.x2 != nullptr && !is_device_ptr(l.x2)))
      return fail(AF1_ERR_BAD_POINTER, who + "x, x2 or y is not device memory");
  }
  std::vector<int> lvl(count), order, level_of;
  for (int i = 0; i < count; ++i) lvl[i] = lin[i].level;
  const int levels = order_levels(lvl, order, level_of);
  std::vector<int> pos(count);  // position of linear i in level order
  for (int j = 0; j < count; ++j) pos[order[j]] = j;
  // Chained operands: an input that is exactly the FP16 output (pointer and
  // row stride, matching width) of a linear of an earlier level. Any other
  // overlap with an output is read as an external input, after every
  // earlier level's outputs are stored.
  auto producer_of = [&](const void* x, int64_t ldx, int i) -> int {
    if (y_dtype != AF1_F16 || x == nullptr) return -1;
    for (int j = 0; j < count; ++j)
      if (lin[j].y == x && lin[j].ldy == ldx && level_of[j] < level_of[i] && lin[j].layer->m == lin[i].layer->n)
        return j;
    return -1;
  };
  for (int i = 0; i < count; ++i)
    for (int j = 0; j < count; ++j)
      if ((lin[j].y == lin[i].x || (lin[i].x2 != nullptr && lin[j].y == lin[i].x2)) && level_of[j] >= level_of[i])
        return fail(AF1_ERR_INVALID_ARG, "linear " + std::to_string(i) + " reads the output of linear " +
                                             std::to_string(j) + " of the same or a later level");

  // ---- problems: phase 1 and phase 2 of each linear, in level order --------
  const int nprob = 2 * count;
  std::vector<StepProblem> probs(nprob);
  std::vector<SignMatrix> sms(nprob);
  std::vector<int> lv(nprob), ph(nprob);
  for (int j = 0; j < count; ++j) {
    const int i = order[j];
    const af1_step_linear& l = lin[i];
    const af1_layer& L = *l.layer;
    StepProblem& p1 = probs[2 * j];
    StepProblem& p2 = probs[2 * j + 1];
    p1 = {};
    p2 = {};
    p1.signs = L.signs1;
    p1.R = L.p1.R;
    p1.C = L.p1.C;
    p1.RB = L.p1.RB;
    p1.NCH = L.p1.NCH;
    p1.phase = 1;
    p1.level = level_of[i];
    p1.swiglu = l.x2 != nullptr ? 1 : 0;
    p1.in.x = static_cast<const __half*>(l.x);
    p1.in.ldx = l.ldx;
    p1.in.part_off = -1;  // set below for chained operands
    p1.in2.x = static_cast<const __half*>(l.x2);
    p1.in2.ldx = l.ldx;
    p1.in2.part_off = -1;
    p1.colscale = reinterpret_cast<const __half*>(L.b);
    p2.signs = L.signs2;
    p2.R = L.p2.R;
    p2.C = L.p2.C;
    p2.RB = L.p2.RB;
    p2.NCH = L.p2.NCH;
    p2.phase = 2;
    p2.level = p1.level;
    p2.rankscale = reinterpret_cast<const __half*>(L.s);
    p2.rowscale = reinterpret_cast<const __half*>(L.a);
    p2.y = l.y;
    p2.ldy = l.ldy;
    sms[2 * j] = L.p1;
    sms[2 * j + 1] = L.p2;
    lv[2 * j] = lv[2 * j + 1] = p1.level;
    ph[2 * j] = 1;
    ph[2 * j + 1] = 2;
  }

  // ---- CTAs: one resident wave ----------------------------------------------
  const int NP = pairs_for(T);
  const int cpc_max = cpc_max_for(T);
  const int fixed = step_smem(cpc_max, T, 0).total;
  int nslot = (kSmemBudget - fixed) / kChunkBytes;
  nslot = std::min(nslot, kMaxSlots);
  if (nslot < 4) return fail(AF1_ERR_INVALID_ARG, "internal: shared memory plan does not fit");
  const int smem = step_smem(cpc_max, T, nslot).total;
  const void* kern = NP == 0 ? (const void*)step_kernel<0> : NP == 1 ? (const void*)step_kernel<1>
                                                                      : (const void*)step_kernel<2>;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("step kernel attributes: ") + cudaGetErrorString(e));
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kStepThreads, smem);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("occupancy: ") + cudaGetErrorString(e));
  per_sm = std::min(per_sm, 2);
  if (per_sm < 1) return fail(AF1_ERR_CUDA, "the step kernel does not fit on an SM");
  int sms_count = 0;
  e = cudaDeviceGetAttribute(&sms_count, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess || sms_count < 1) return fail(AF1_ERR_CUDA, "cannot read the SM count");
  const int ctas = sms_count * per_sm;

  // ---- tiles ------------------------------------------------------------------
  // Levels with an input that waits for stored outputs (not produced in the step).
  std::vector<char> ext_level(levels, 0);
  for (int i = 0; i < count; ++i) {
    const int L = level_of[i];
    if (L == 0) continue;
    if (producer_of(lin[i].x, lin[i].ldx, i) < 0 || (lin[i].x2 != nullptr && producer_of(lin[i].x2, lin[i].ldx, i) < 0))
      ext_level[L] = 1;
  }
  std::vector<int> prod_a(nprob, -1), prod_b(nprob, -1);
  for (int j = 0; j < count; ++j) {
    const int i = order[j];
    const int pa = producer_of(lin[i].x, lin[i].ldx, i);
    const int pb2 = lin[i].x2 != nullptr ? producer_of(lin[i].x2, lin[i].ldx, i) : -1;
    prod_a[2 * j] = pa >= 0 ? 2 * pos[pa] + 1 : -1;
    prod_b[2 * j] = pb2 >= 0 ? 2 * pos[pb2] + 1 : -1;
  }
  const TilePlan tp = plan_tiles(sms, lv, ph, levels, cpc_max, ctas, ext_level, prod_a, prod_b);
  for (int q = 0; q < nprob; ++q) probs[q].KS = tp.KS[q];

  // ---- workspace layout: header, then the tagged partial sums of every problem
  int64_t off = kWsHeader;
  for (int q = 0; q < nprob; ++q) {
    probs[q].pout_off = off;
    off = align256(off + (int64_t)probs[q].KS * T * probs[q].RB * kBlockRows * 8);
  }
  const int64_t ws_bytes = off;
  std::vector<unsigned> stored_before(levels + 1, 0u);  // row blocks of y stored by levels < L
  for (int q = 0; q < nprob; ++q)
    if (probs[q].phase == 2) stored_before[probs[q].level + 1] += (unsigned)probs[q].RB;
  for (int L = 1; L <= levels; ++L) stored_before[L] += stored_before[L - 1];
  int chained_any = 0;
  for (int j = 0; j < count; ++j) {
    const int i = order[j];
    StepProblem& p1 = probs[2 * j];
    StepProblem& p2 = probs[2 * j + 1];
    p2.pin_off = p1.pout_off;
    p2.pin_ks = p1.KS;
    bool external = false;
    for (int opnd = 0; opnd < (p1.swiglu ? 2 : 1); ++opnd) {
      StepInput& in = opnd == 0 ? p1.in : p1.in2;
      const int pj = producer_of(opnd == 0 ? lin[i].x : lin[i].x2, lin[i].ldx, i);
      if (pj < 0) {
        external = true;
        continue;
      }
      const StepProblem& pp = probs[2 * pos[pj] + 1];
      in.part_off = pp.pout_off;
      in.part_ks = pp.KS;
      in.part_ld = (int64_t)pp.RB * kBlockRows;
      in.part_scale = pp.rowscale;
      p1.chained = 1;
      chained_any = 1;
    }
    p1.external_wait = external && p1.level > 0 ? 1 : 0;
    p1.fin_target = stored_before[p1.level];
  }

  // ---- device copy of the plan -----------------------------------------------
  const std::vector<StepTask>& tasks = tp.tasks;
  const std::vector<int>& cta_first = tp.cta_first;
  const size_t b_probs = sizeof(StepProblem) * probs.size();
  const size_t b_tasks = sizeof(StepTask) * std::max<size_t>(tasks.size(), 1);
  const size_t b_first = sizeof(int) * cta_first.size();
  const size_t o_tasks = (b_probs + 255) & ~(size_t)255;
  const size_t o_first = (o_tasks + b_tasks + 255) & ~(size_t)255;
  const size_t total = o_first + b_first;
  af1_step* S = new (std::nothrow) af1_step();
  if (S == nullptr) return fail(AF1_ERR_INVALID_ARG, "out of host memory");
  e = cudaMalloc(&S->dev, total);
  if (e != cudaSuccess) {
    delete S;
    return fail(AF1_ERR_CUDA, std::string("cudaMalloc(plan): ") + cudaGetErrorString(e));
  }
  uint8_t* d = static_cast<uint8_t*>(S->dev);
  e = cudaMemcpy(d, probs.data(), b_probs, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !tasks.empty())
    e = cudaMemcpy(d + o_tasks, tasks.data(), sizeof(StepTask) * tasks.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(d + o_first, cta_first.data(), b_first, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    cudaFree(S->dev);
    delete S;
    return fail(AF1_ERR_CUDA, std::string("plan upload: ") + cudaGetErrorString(e));
  }
  S->device = dev;
  S->T = T;
  S->ydtype = y_dtype;
  S->nslot = nslot;
  S->cpc_max = cpc_max;
  S->ctas = ctas;
  S->smem = smem;
  S->gate = (flags & AF1_STEP_WAIT_GATE) ? 1 : 0;
  S->levels = levels;
  S->ws_bytes = ws_bytes;
  S->ntasks = (int)tasks.size();
  S->nprobs = nprob;
  S->chained = chained_any;
  S->probs = reinterpret_cast<const StepProblem*>(d);
  S->tasks = reinterpret_cast<const StepTask*>(d + o_tasks);
  S->cta_first = reinterpret_cast<const int*>(d + o_first);
  S->model_us = tp.model_us;
  *out = S;
  return AF1_OK;
}

int af1_step_plan_dry(const int64_t* m, const int64_t* n, const int64_t* r, const int32_t* level,
                      const int32_t* producer, const int32_t* producer2, int count, int64_t tokens, int32_t ctas,
                      int32_t* order_out,
                      int32_t* tasks_out, int64_t max_tasks, int32_t* cta_first_out, int32_t* ks_out, int64_t* ntasks,
                      double* model_us) {
  using namespace af1;
  if (m == nullptr || n == nullptr || r == nullptr || level == nullptr || count < 1)
    return fail(AF1_ERR_INVALID_ARG, "shapes and levels of at least one linear are required");
  if (tokens < 1 || tokens > kStepMaxTokens)
    return fail(AF1_ERR_INVALID_ARG, "tokens must be in 1.." + std::to_string(kStepMaxTokens));
  if (ctas < 1) return fail(AF1_ERR_INVALID_ARG, "ctas must be >= 1");
  std::vector<int> lvl(count), order, level_of;
  for (int i = 0; i < count; ++i) {
    if (m[i] < 1 || n[i] < 1 || r[i] < 1 || n[i] > kMaxCols || r[i] > kMaxCols || level[i] < 0)
      return fail(AF1_ERR_INVALID_ARG, "linear " + std::to_string(i) + ": bad shape or level");
    lvl[i] = level[i];
  }
  const int levels = order_levels(lvl, order, level_of);
  std::vector<SignMatrix> sms(2 * count);
  std::vector<int> lv(2 * count), ph(2 * count);
  for (int j = 0; j < count; ++j) {
    const int i = order[j];
    sms[2 * j] = make_sign_matrix(r[i], n[i]);
    sms[2 * j + 1] = make_sign_matrix(m[i], r[i]);
    lv[2 * j] = lv[2 * j + 1] = level_of[i];
    ph[2 * j] = 1;
    ph[2 * j + 1] = 2;
  }
  std::vector<int> pos(count);
  for (int j = 0; j < count; ++j) pos[order[j]] = j;
  auto valid_producer = [&](const int32_t* pr, int i) {
    return pr != nullptr && pr[i] >= 0 && pr[i] < count && level_of[pr[i]] < level_of[i];
  };
  std::vector<char> ext_level(levels, 0);
  std::vector<int> prod_a(2 * count, -1), prod_b(2 * count, -1);
  for (int i = 0; i < count; ++i) {
    if (level_of[i] > 0 && !valid_producer(producer, i)) ext_level[level_of[i]] = 1;
    if (valid_producer(producer, i)) prod_a[2 * pos[i]] = 2 * pos[producer[i]] + 1;
    if (valid_producer(producer2, i)) prod_b[2 * pos[i]] = 2 * pos[producer2[i]] + 1;
  }
  const TilePlan tp =
      plan_tiles(sms, lv, ph, levels, cpc_max_for((int)tokens), ctas, ext_level, prod_a, prod_b);
  if (ntasks) *ntasks = (int64_t)tp.tasks.size();
  if (model_us) *model_us = tp.model_us;
  if (order_out)
    for (int j = 0; j < count; ++j) order_out[j] = order[j];
  if (ks_out)
    for (int q = 0; q < 2 * count; ++q) ks_out[q] = tp.KS[q];
  if (cta_first_out)
    for (int c = 0; c <= ctas; ++c) cta_first_out[c] = tp.cta_first[c];
  if (tasks_out) {
    if (max_tasks < (int64_t)tp.tasks.size()) return fail(AF1_ERR_INVALID_ARG, "max_tasks is too small");
    for (size_t k = 0; k < tp.tasks.size(); ++k) {
      const StepTask& t = tp.tasks[k];
      int32_t* o = tasks_out + 7 * k;
      o[0] = t.prob;
      o[1] = t.rb0;
      o[2] = t.G;
      o[3] = t.c0;
      o[4] = t.nch;
      o[5] = t.ks;
      o[6] = t.kind;
    }
  }
  return AF1_OK;
}

int64_t af1_step_workspace_bytes(const af1_step* step) {
  if (step == nullptr) return fail(AF1_ERR_INVALID_ARG, "step is NULL");
  return step->ws_bytes;
}

int af1_step_info(const af1_step* step, int64_t* ctas, int64_t* tasks, int64_t* levels, double* model_us) {
  if (step == nullptr) return fail(AF1_ERR_INVALID_ARG, "step is NULL");
  if (ctas) *ctas = step->ctas;
  if (tasks) *tasks = step->ntasks;
  if (levels) *levels = step->levels;
  if (model_us) *model_us = step->model_us;
  return AF1_OK;
}

int af1_step_run(const af1_step* step, void* workspace, int64_t workspace_bytes, void* stream) {
  using namespace af1;
  if (step == nullptr) return fail(AF1_ERR_INVALID_ARG, "step is NULL");
  if (workspace == nullptr) return fail(AF1_ERR_WORKSPACE, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return fail(AF1_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (workspace_bytes < step->ws_bytes)
    return fail(AF1_ERR_WORKSPACE, "workspace too small: need " + std::to_string(step->ws_bytes) + " bytes");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev != step->device) return fail(AF1_ERR_BAD_POINTER, "the current device is not the step's device");
  if (!is_device_ptr(workspace))
    return fail(AF1_ERR_WORKSPACE, "workspace is not device memory of the current device");
  StepArgs a = {};
  a.probs = step->probs;
  a.tasks = step->tasks;
  a.cta_first = step->cta_first;
  a.ws = static_cast<uint8_t*>(workspace);
  a.T = step->T;
  a.ydtype = step->ydtype;
  a.nslot = step->nslot;
  a.cpc_max = step->cpc_max;
  a.ctas = step->ctas;
  a.gate = step->gate;
  a.wait_cycles = wait_budget();
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)step->ctas, 1, 1);
  cfg.blockDim = dim3(kStepThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)step->smem;
  cfg.stream = static_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident: CTAs wait for one another
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const int NP = pairs_for(step->T);
  if (NP == 0) e = cudaLaunchKernelEx(&cfg, step_kernel<0>, a);
  else if (NP == 1) e = cudaLaunchKernelEx(&cfg, step_kernel<1>, a);
  else e = cudaLaunchKernelEx(&cfg, step_kernel<2>, a);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("step launch: ") + cudaGetErrorString(e));
  return AF1_OK;
}

int af1_step_open_gate(void* workspace, void* stream) {
  if (workspace == nullptr) return fail(AF1_ERR_WORKSPACE, "workspace is NULL");
  cudaError_t e = cudaMemsetAsync(static_cast<uint8_t*>(workspace) + 4 * af1::kWsGate, 1, 4,
                                  static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("af1_step_open_gate: ") + cudaGetErrorString(e));
  return AF1_OK;
}

void af1_step_destroy(af1_step* step) {
  if (step == nullptr) return;
  cudaDeviceSynchronize();
  cudaFree(step->dev);
  delete step;
}

}  // extern "C"
