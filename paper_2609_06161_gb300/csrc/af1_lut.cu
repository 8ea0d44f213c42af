// af1_lut.cu — decode path (1..16 tokens per pass) on the CUDA cores: each
// sign-matrix x vector product of the forward pass
//     y = a * (U (s * (V^T (b * x))))      (AF1 Eq. final_reconstruction /
//                                          Eq. double_factor_equiv)
// is evaluated with lookup tables of signed sums instead of tensor-core MMAs.
//
// Tables of signed sums (af1_lut_common.cuh) are built once per CTA in
// shared memory; all 32 lanes of a warp (32 rows) read the same 16-entry
// table at the same time, so every read is a conflict-free broadcast. A
// probe of this inner loop on GB300 sustained about 160 signs per ns per SM
// at one token, twice the rate at which signs can be expanded into tensor
// memory and multiplied there.
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
#include "af1_lut_common.cuh"

namespace af1 {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxCPC = 32;       // chunks per CTA (one mbarrier each)
constexpr int kMaxKS = 16;        // CTAs per cluster
constexpr int kGroupTokens = 4;   // tokens per CTA: a pass of T tokens runs ceil(T / 4) CTAs per tile

// ---------------------------------------------------------------------------
// Shared-memory plan
// ---------------------------------------------------------------------------

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

// SWIGLU (phase 1, one problem): the input is h = FP16(SiLU(x) x2).
template <int PHASE, int NP, bool MULTI, bool SWIGLU>
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
  const __half* x2g = SWIGLU ? pb.x2 + (int64_t)tg0 * pb.ldx : nullptr;
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
  griddep_wait();
  // Phase 1's dependent is the same call's phase 2: let it launch now, so its
  // CTAs copy their U words from HBM while this kernel computes (they hold
  // no input of another call). Measured against launching it after the
  // lookups (below): config-1 stack 6.33 -> 6.22 us per linear on the DAG
  // schedule, 6.42 -> 6.13 grouped, 8.62 -> 8.42 serial. Phase 2 does the
  // same unless the caller runs several streams (AF1_MANY_STREAMS): early
  // wins on one stream (32-layer HiSA-rank step at one token, grouped calls:
  // 1.323 -> 1.277 ms), late on the decoder DAG over three streams (1.480
  // -> 1.437 ms), where the next kernel's waiting CTAs would hold SM slots
  // that the sibling streams' kernels need.
  if (PHASE == 1 || !a.late_trigger) griddep_launch_dependents();
  stage_activations<PHASE, kThreads, SWIGLU>(pb, xg, x2g, zg, T, nch, k0, zs, zrow, tid);
  if (tid < slice) rs[tid] = rs_own;
  __syncthreads();

  // ---- tables of the CTA's chunks -----------------------------------------------
  build_tables<NP, kThreads>(smem + sp.tbl, zs, zrow, T, nch, tid);
  __syncthreads();

  // ---- lookups: thread (r, g) = row r, words 2g and 2g + 1 of every chunk ---
  const int r = tid & 127, g = tid >> 7;
  float acc[NACC];
#pragma unroll
  for (int i = 0; i < NACC; ++i) acc[i] = 0.f;
  {
    const uint32_t tbl0 = smem_u32(smem + sp.tbl);
    bool ok = true;
    for (int c = 0; c < nch; ++c) {
      if (ok) ok = mbar_wait(&h.wfull[c], 0, &h.err, a.wait_cycles);
      lookup_chunk<NP>(tbl0 + (uint32_t)(c * TCB), W + c * (kChunkBytes / 4) + r, g, acc);
    }
  }

  // With several streams (AF1_MANY_STREAMS): phase 2 lets the next kernel
  // launch only now, so its CTAs do not hold SM slots (waiting for this
  // kernel) that sibling kernels on other streams need, and its sign copies
  // still get the reduction's time as a head start (measured: config-1
  // stack 7.40 -> 6.53 us per linear on the DAG schedule, trigger at the
  // start vs here).
  if (PHASE == 2 && a.late_trigger) griddep_launch_dependents();
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
  mbar_wait(&h.red, 0, &h.err, a.wait_cycles);  // this CTA's partials have all landed
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
    for (int c = 0; c < nch; ++c) mbar_wait(&h.wfull[c], 0, &h.err, a.wait_cycles);
    atomicOr(a.status, kStatusTimeout);
  }
}

template <int PHASE, int NP, bool MULTI, bool SWIGLU = false>
cudaError_t launch_np(const LutArgs& a, const LutPlan& p, cudaStream_t st) {
  auto kern = lut_kernel<PHASE, NP, MULTI, SWIGLU>;
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
// token groups of CTAs: about three CTAs per SM when the caller runs one
// stream, two when it runs several (row blocks x KS x groups ~ 3 or 2 SMs,
// KS <= 16 CTAs per cluster), CTAs small enough that three fit on an SM,
// and at most kMaxCPC chunks each. Returns KS (0: no plan), *cpc and *smem.
// Measured on the 32-layer HiSA-rank step at one token (ms per step, two /
// three / four CTAs per SM): one stream, one call per layer 1.850 / 1.747 /
// 1.745, grouped calls (q | k | v and gate | up keep their own one-wave
// split) 1.278 / 1.249 / 1.442; the DAG over three streams 1.436 / 1.478.
int plan_one(const SignMatrix& sm, int T, int sms, int max_smem, int* cpc_out, int* smem_out) {
  const int Tg = T < kGroupTokens ? T : kGroupTokens;
  const int groups = (T + kGroupTokens - 1) / kGroupTokens;
  const int cap = max_smem / 3 < 72 * 1024 ? max_smem / 3 : 72 * 1024;
  const int64_t tiles = (int64_t)sm.RB * groups;
  const int per_sm = many_streams() ? 2 : 3;
  int ks = (int)((per_sm * sms + tiles - 1) / tiles);
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

// Several problems in one launch: the cluster size that keeps every CTA of
// the group resident (one wave), preferably with at least two CTAs per SM
// (the lookups need them to hide their latency: one CTA per SM made the
// gate | up first phase 5 -> 6 us), and minimises the busiest SM's load,
// ceil(CTAs / SMs) x (chunks per CTA + 2, the fixed cost of a CTA in chunk
// units); 0 if no size fits one wave. (Each problem's own split, as for one
// problem, made the gate | up launch of a LLaMA-3-8B layer 672 CTAs for 608
// resident slots: two waves, 12 us for its second phase.)
int plan_group_ks(const SignMatrix* sm, int count, int T, int sms, int max_smem) {
  const int Tg = T < kGroupTokens ? T : kGroupTokens;
  const int groups = (T + kGroupTokens - 1) / kGroupTokens;
  const int64_t per_sm_smem = (int64_t)max_smem + 1024;  // the SM's shared memory (a CTA may take all but 1 KB)
  int best_ks = 0;
  int64_t best = 0;
  bool best_two = false;  // the best so far has at least two CTAs per SM
  for (int ks = 1; ks <= kMaxKS; ++ks) {
    int64_t ctas = 0;
    int cpc_max = 0, need = 0;
    bool ok = true;
    for (int i = 0; i < count; ++i) {
      const int cpc = (sm[i].NCH + ks - 1) / ks;
      if (cpc > kMaxCPC) ok = false;
      const int nd = lut_smem(cpc, ks, Tg, pairs_for(Tg)).total;
      if (nd > need) need = nd;
      if (cpc > cpc_max) cpc_max = cpc;
      ctas += (int64_t)sm[i].RB * groups * ks;
    }
    if (!ok || need > max_smem) continue;
    int64_t resident = per_sm_smem / need;
    if (resident > 4) resident = 4;  // __launch_bounds__(256, 4)
    if (ctas > resident * sms) continue;
    const int64_t load = ((ctas + sms - 1) / sms) * (cpc_max + 2);
    const bool two = ctas >= 2 * (int64_t)sms;
    if (best_ks == 0 || (two && !best_two) || (two == best_two && load < best)) {
      best = load;
      best_ks = ks;
      best_two = two;
    }
  }
  return best_ks;
}

// One problem: its own split. Several (layers sharing their input, one
// launch): the cluster size of plan_group_ks, or failing that the largest of
// their own splits' cluster sizes; each problem cuts its columns into that
// many slices (the last CTAs of a problem with fewer chunks get none).
LutPlan plan_lut(const SignMatrix* sm, int count, int T, int num_sms, int max_smem) {
  LutPlan p;
  if (count < 1 || count > kMaxGroup || T < 1 || T > kMaxPassTokens) return p;
  const int sms = num_sms > 0 ? num_sms : kDefaultSms;
  const int Tg = T < kGroupTokens ? T : kGroupTokens;
  int KS = 0;
  for (int i = 0; i < count; ++i) {
    if (sm[i].RB < 1 || sm[i].NCH < 1) return p;
    int cpc = 0, smem = 0;
    const int k = plan_one(sm[i], T, sms, max_smem, &cpc, &smem);
    if (k == 0) return p;
    if (k > KS) KS = k;
  }
  // (The same choice for one problem was measured too: the 8B shapes gained
  // up to 6 % at one token, the 70B ones at one token and most shapes at four
  // lost 4-6 %; each problem keeps its own split.)
  if (count > 1) {
    const int g = plan_group_ks(sm, count, T, sms, max_smem);
    if (g > 0) KS = g;
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
  if (PHASE == 1 && !multi && a.prob[0].x2 != nullptr) {
    switch (pairs_for(a.tokens < kGroupTokens ? a.tokens : kGroupTokens)) {
      case 0: return launch_np<PHASE, 0, false, true>(a, p, st);
      case 1: return launch_np<PHASE, 1, false, true>(a, p, st);
      default: return launch_np<PHASE, 2, false, true>(a, p, st);
    }
  }
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
