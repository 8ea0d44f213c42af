// af1_stream.cu — decode passes of one or two tokens over sign matrices too
// large for one wave of the clustered kernel, on the CUDA cores.
//
// Each phase of the forward pass (AF1 Eq. final_reconstruction, right to
// left: t = V^T (b x), then y = a (U (s t))) is an R x C sign matrix times
// one vector per token. The clustered kernel (af1_lut.cu) gives every CTA
// one 128-row block and a slice of its columns, with all of the slice's
// signs resident in shared memory; a large matrix then needs several waves
// of CTAs, and every CTA pays its start-up (activation staging, table build)
// and its cluster reduction once per wave.
//
// Here a CTA owns a super row of G = 1, 2 or 4 row blocks and a slice of
// CPC chunks of it, so that the whole matrix fits in one wave: it builds the
// tables of its CPC chunks once (af1_lut_common.cuh) and uses them for all
// G row blocks. A producer warp streams the CTA's chunk tiles (for each
// chunk, the G tiles of 128 rows x 128 columns, 2 KB each) through a ring
// of shared-memory slots with bulk copies, while 8 consumer warps do the
// lookups: thread (r, g) takes row r of every row block of the super row,
// words 2g and 2g + 1 of every chunk. The KS CTAs of a super row form a
// cluster and reduce their partial sums through distributed shared memory
// in a fixed order (deterministic): each row's 2 KS partials reach the CTA
// that finishes the row with st.async onto its mbarrier.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <map>
#include <mutex>
#include <tuple>

#include "af1_internal.h"
#include "af1_layout.h"
#include "af1_lut_common.cuh"

namespace af1 {
namespace {

constexpr int kConsumers = 256;                  // 8 warps: tables, lookups, sums
constexpr int kStreamThreads = kConsumers + 32;  // + the producer warp
constexpr int kMaxRing = 32;                     // ring slots (of G chunk tiles each)
constexpr int kMaxStreamTokens = 2;
constexpr int kMaxStreamKS = 16;  // CTAs per cluster
constexpr int kMaxStreamG = 4;    // row blocks per super row
constexpr int kSmemPerSM = 233472;  // 228 KB of shared memory per SM
constexpr int kSmemPerCTA = 1024;   // reserved by the system per resident CTA
constexpr int kBarConsumers = 1;    // named barrier: the 256 consumer threads
constexpr double kCopyNs = 2000.0;  // a ring slot's bulk copies under load (planning)

__host__ __device__ inline int align128s(int v) { return (v + 127) & ~127; }
// Rows of the super row each CTA of the cluster finishes.
__host__ __device__ inline int stream_slice(int G, int KS) { return (G * kBlockRows + KS - 1) / KS; }

struct __align__(8) StreamHeader {
  uint64_t full[kMaxRing];   // slot s holds its chunk's G tiles (bulk copies)
  uint64_t empty[kMaxRing];  // the 8 consumer warps are done with slot s
  uint64_t red;              // all partial sums of this CTA's rows have landed (st.async)
  uint32_t err;
};

struct StreamSmem {
  int tbl, ring, zr, rs, hdr, total;  // byte offsets from the 256-aligned base
};

// A ring of NSC slots of G chunk tiles. The staged activations (before the
// lookups) and the received partial sums (after them) share one region.
__host__ __device__ inline StreamSmem stream_smem(int CPC, int KS, int T, int G, int NSC) {
  StreamSmem p;
  int off = 0;
  p.tbl = off;
  off += table_chunk_bytes(pairs_for(T)) * CPC;
  p.ring = off;
  off += NSC * G * kChunkBytes;
  p.zr = off;
  const int zb = T * zrow_floats(CPC) * 4, rb = 2 * KS * T * stream_slice(G, KS) * 4;
  off = align128s(off + (zb > rb ? zb : rb));
  p.rs = off;
  off = align128s(off + stream_slice(G, KS) * 4);
  p.hdr = off;
  off = align128s(off + (int)sizeof(StreamHeader));
  p.total = off + 256;  // slack for aligning the base to 256 bytes (table windows)
  return p;
}

struct StreamArgs {
  LutProblem p;        // CPC and rb0 unused
  int tokens, ydtype;  // T (1..2)
  int KS, CPC, NSC;    // CTAs per cluster (grid y), chunks per CTA, ring slots
  unsigned* status;
  long long wait_cycles;  // budget of every bounded wait (clock64 cycles)
};

// SWIGLU (phase 1): the input is h = FP16(SiLU(x) x2).
template <int PHASE, int NP, int G, bool SWIGLU>
__global__ void __launch_bounds__(kStreamThreads, 3) stream_kernel(const __grid_constant__ StreamArgs a) {
  constexpr int NACC = NP == 0 ? 1 : 2 * NP;
  constexpr int TCB = table_chunk_bytes(NP);
  constexpr int SLOTW = G * kChunkBytes / 4;  // words per ring slot
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 255) & ~(uintptr_t)255);
  const LutProblem& pb = a.p;
  const int T = a.tokens, KS = a.KS, CPC = a.CPC, NSC = a.NSC;
  const int NCH = pb.sm.NCH, RB = pb.sm.RB;
  const int srb = blockIdx.x, ks = blockIdx.y;
  const int c0 = ks * CPC;
  const int nch = max(0, min(CPC, NCH - c0));  // chunks of this CTA (0: it only finishes rows)
  const int nrb = min(G, RB - srb * G);        // row blocks of the super row
  const int64_t row0 = (int64_t)srb * G * kBlockRows;
  const int slice = stream_slice(G, KS);
  const int my0 = ks * slice;                        // first super-row row this CTA finishes
  const int cnt = min(slice, G * kBlockRows - my0);  // rows it finishes (may be <= 0)
  const StreamSmem sp = stream_smem(CPC, KS, T, G, NSC);
  uint8_t* ring = smem + sp.ring;
  float* zs = reinterpret_cast<float*>(smem + sp.zr);
  float* recv = reinterpret_cast<float*>(smem + sp.zr);  // [2 KS][T][slice], after the tables
  float* rs = reinterpret_cast<float*>(smem + sp.rs);
  StreamHeader& h = *reinterpret_cast<StreamHeader*>(smem + sp.hdr);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    for (int s = 0; s < NSC; ++s) {
      mbar_init(&h.full[s], 1);
      mbar_init(&h.empty[s], kConsumers / 32);
    }
    // The partial sums of this CTA's rows arrive from the 2 KS word halves
    // of the cluster, 4 bytes per row and token each.
    mbar_init(&h.red, 1);
    mbar_expect_tx(&h.red, cnt > 0 ? (uint32_t)(2 * KS * T * cnt * 4) : 0u);
    h.err = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  // Row scales of the rows this CTA finishes (layer constants).
  for (int i = tid; i < cnt; i += kStreamThreads) {
    const int64_t row = row0 + my0 + i;
    rs[i] = row < pb.sm.R ? __half2float(pb.rowscale[row]) : 0.f;
  }
  __syncthreads();

  if (warp == kConsumers / 32) {
    // ---- producer: the CTA's chunks, in order, into the ring -----------------
    // (Signs are layer constants: copied before the previous kernel ends.)
    if (lane == 0) {
      bool ok = true;
      int s = 0;
      uint32_t par = 0;  // parity of the slot's release to wait for
      const uint8_t* src = pb.signs + ((int64_t)srb * G * NCH + c0) * kChunkBytes;
      for (int k = 0; k < nch; ++k) {
        if (k >= NSC && ok) ok = mbar_wait(&h.empty[s], par, &h.err, a.wait_cycles);
        mbar_expect_tx(&h.full[s], (uint32_t)(nrb * kChunkBytes));
        for (int gi = 0; gi < nrb; ++gi)
          bulk_g2s(ring + (s * G + gi) * kChunkBytes, src + ((int64_t)gi * NCH + k) * kChunkBytes, kChunkBytes,
                   &h.full[s]);
        if (++s == NSC) {
          s = 0;
          if (k >= NSC) par ^= 1u;
        }
      }
    }
    __syncwarp();
    griddep_launch_dependents();
    // The producer warp takes part in both cluster barriers like the others.
    cluster_arrive_relaxed();
    cluster_wait();
    cluster_arrive_relaxed();
    cluster_wait();
    return;
  }

  // ---- consumers: activations of the CTA's chunks, tables --------------------
  griddep_wait();
  const int zrow = zrow_floats(CPC);
  stage_activations<PHASE, kConsumers, SWIGLU>(pb, pb.x, pb.x2, pb.zin, T, nch, (int64_t)c0 * kChunkCols, zs, zrow,
                                               tid);
  named_sync(kBarConsumers, kConsumers);
  build_tables<NP, kConsumers>(smem + sp.tbl, zs, zrow, T, nch, tid);
  named_sync(kBarConsumers, kConsumers);
  // The staged activations are dead: peers may store partial sums into the
  // region once every CTA of the cluster has arrived here (matched by
  // cluster_wait before the first remote store).
  cluster_arrive_relaxed();

  // ---- lookups: chunk by chunk, the G tiles of each --------------------------
  const int r = tid & 127, g = tid >> 7;
  const uint32_t tbl0 = smem_u32(smem + sp.tbl);
  const uint32_t* ringw = reinterpret_cast<const uint32_t*>(ring);
  float acc[G][NACC];
#pragma unroll
  for (int gi = 0; gi < G; ++gi)
#pragma unroll
    for (int t = 0; t < NACC; ++t) acc[gi][t] = 0.f;
  {
    bool ok = true;
    int s = 0;
    uint32_t par = 0;
    for (int k = 0; k < nch; ++k) {
      if (ok) ok = mbar_wait(&h.full[s], par, &h.err, a.wait_cycles);
      const uint32_t tb = tbl0 + (uint32_t)(k * TCB);
#pragma unroll
      for (int gi = 0; gi < G; ++gi)
        if (gi < nrb) lookup_chunk<NP>(tb, ringw + s * SLOTW + gi * (kChunkBytes / 4) + r, g, acc[gi]);
      __syncwarp();
      if (lane == 0) mbar_arrive(&h.empty[s]);
      if (++s == NSC) {
        s = 0;
        par ^= 1u;
      }
    }
  }
  griddep_launch_dependents();  // the next kernel may start its prologue

  // ---- partial sums -> the CTA finishing each row -> final sums ---------------
  cluster_wait();  // every CTA of the cluster has built its tables
  {
    const int src = ks * 2 + g;
#pragma unroll
    for (int gi = 0; gi < G; ++gi) {
      const int rr = gi * kBlockRows + r;
      const int owner = rr / slice;
#pragma unroll
      for (int t = 0; t < NACC; ++t)
        if (t < T)
          st_async_f32(recv + ((src * T + t) * slice + (rr - owner * slice)), &h.red, (uint32_t)owner, acc[gi][t]);
    }
  }
  // Exit barrier (waited for after the final sums): no CTA leaves while a
  // peer may still store into it.
  cluster_arrive_relaxed();
  mbar_wait(&h.red, 0, &h.err, a.wait_cycles);
  for (int idx = tid; idx < T * cnt; idx += kConsumers) {
    const int t = idx / cnt;
    const int i = idx - t * cnt;
    const int64_t row = row0 + my0 + i;
    if (row >= pb.sm.R) continue;
    // The 2 KS partials in four interleaved chains (fixed order).
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
      pb.sout[(int64_t)t * pb.lds + row] = out;
    } else if (a.ydtype == 0) {
      reinterpret_cast<__half*>(pb.y)[(int64_t)t * pb.ldy + row] = __float2half_rn(out);
    } else {
      reinterpret_cast<float*>(pb.y)[(int64_t)t * pb.ldy + row] = out;
    }
  }
  cluster_wait();

  // ---- teardown -----------------------------------------------------------------
  named_sync(kBarConsumers, kConsumers);
  if (tid == 0 && h.err != 0) {
    // A wait gave up: let the copies in flight land (bounded) before the CTA
    // exits, and report it. The last copy into slot s is chunk k_s, the last
    // k < nch with k mod NSC = s.
    for (int s2 = 0; s2 < NSC && s2 < nch; ++s2) {
      const int kl = s2 + ((nch - 1 - s2) / NSC) * NSC;
      mbar_wait(&h.full[s2], (uint32_t)((kl / NSC) & 1), &h.err, a.wait_cycles);
    }
    atomicOr(a.status, kStatusTimeout);
  }
}

// Kernel attributes for a launch with `smem` bytes and clusters of KS.
template <int PHASE, int NP, int G, bool SWIGLU = false>
cudaError_t prepare_kernel(int smem, int KS) {
  auto kern = stream_kernel<PHASE, NP, G, SWIGLU>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess && KS > 8) e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  return e;
}

// Clusters of KS CTAs with `smem` bytes each that the device runs at once.
template <int PHASE, int NP, int G>
int active_clusters(int smem, int KS) {
  if (prepare_kernel<PHASE, NP, G>(smem, KS) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1, (unsigned)KS, 1);
  cfg.blockDim = dim3(kStreamThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = (unsigned)KS;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, stream_kernel<PHASE, NP, G, false>, &cfg) != cudaSuccess) {
    cudaGetLastError();  // clear: the query failing only rules the split out
    return 0;
  }
  return n;
}

// Cached per (device, phase, tokens, G, KS, smem): the query costs a driver
// call.
int max_active_clusters(int phase, int T, int G, int KS, int smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, int, int, int, int>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, phase, T, G, KS, smem);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  int n = 0;
  const bool one = T == 1;
  if (phase == 1) {
    if (G == 1) n = one ? active_clusters<1, 0, 1>(smem, KS) : active_clusters<1, 1, 1>(smem, KS);
    else if (G == 2) n = one ? active_clusters<1, 0, 2>(smem, KS) : active_clusters<1, 1, 2>(smem, KS);
    else n = one ? active_clusters<1, 0, 4>(smem, KS) : active_clusters<1, 1, 4>(smem, KS);
  } else {
    if (G == 1) n = one ? active_clusters<2, 0, 1>(smem, KS) : active_clusters<2, 1, 1>(smem, KS);
    else if (G == 2) n = one ? active_clusters<2, 0, 2>(smem, KS) : active_clusters<2, 1, 2>(smem, KS);
    else n = one ? active_clusters<2, 0, 4>(smem, KS) : active_clusters<2, 1, 4>(smem, KS);
  }
  std::lock_guard<std::mutex> lock(mu);
  cache[key] = n;
  return n;
}

template <int PHASE, int NP, int G, bool SWIGLU>
cudaError_t launch_g(const StreamArgs& a, const StreamPlan& p, cudaStream_t st) {
  auto kern = stream_kernel<PHASE, NP, G, SWIGLU>;
  cudaError_t e = prepare_kernel<PHASE, NP, G, SWIGLU>(p.smem, p.KS);
  if (e != cudaSuccess) return e;
  const int SRB = (a.p.sm.RB + G - 1) / G;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)SRB, (unsigned)p.KS, 1);
  cfg.blockDim = dim3(kStreamThreads, 1, 1);
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

template <int PHASE, int NP, bool SWIGLU = false>
cudaError_t launch_np(const StreamArgs& a, const StreamPlan& p, cudaStream_t st) {
  switch (p.G) {
    case 1: return launch_g<PHASE, NP, 1, SWIGLU>(a, p, st);
    case 2: return launch_g<PHASE, NP, 2, SWIGLU>(a, p, st);
    default: return launch_g<PHASE, NP, 4, SWIGLU>(a, p, st);
  }
}

}  // namespace

// Every (G, KS) split whose SRB clusters the device runs at once (one wave)
// with at most 3 CTAs per SM (the register budget of 288 threads), each CTA
// padded with shared memory so that no SM holds more than its share
// ceil(CTAs / SMs) (the block scheduler would otherwise fill some SMs and
// leave others idle); the padding deepens the ring, up to the whole slice.
// The chosen split has the smallest modelled time on an SM: lookups of G x
// CPC tiles at the measured per-SM rate for that many CTAs, table builds
// (about a twentieth of a tile's lookups per chunk), and the wait for
// refills the slots ahead do not cover (a copy takes about 2 us under load).
// Not ok when no split fits in one wave.
StreamPlan search_stream(int phase, const SignMatrix& sm, int T, int num_sms, int max_smem) {
  StreamPlan p;
  if (T < 1 || T > kMaxStreamTokens || sm.RB < 1 || sm.NCH < 1) return p;
  const int sms = num_sms > 0 ? num_sms : kDefaultSms;
  int64_t best = -1;
  for (int G = 1; G <= kMaxStreamG; G *= 2) {
    const int64_t SRB = (sm.RB + G - 1) / G;
    for (int k = 1; k <= kMaxStreamKS && k <= sm.NCH; ++k) {
      const int CPC = (sm.NCH + k - 1) / k;
      const int KS = (sm.NCH + CPC - 1) / CPC;
      if (KS != k) continue;  // the same split as a smaller k
      const int64_t ctas = SRB * KS;
      const int on_sm = (int)((ctas + sms - 1) / sms);  // CTAs per SM, spread evenly
      if (on_sm > 3) break;                             // larger k only adds CTAs
      // Shared memory per CTA: at most this SM's share, at least enough that
      // one more CTA does not fit.
      int budget = kSmemPerSM / on_sm - kSmemPerCTA;
      budget = budget < max_smem ? budget : max_smem;
      const int floor_smem = on_sm < 3 ? kSmemPerSM / (on_sm + 1) - kSmemPerCTA + 256 : 0;
      // Lookup rate per SM (signs per ns, one token) with 1, 2, >= 3 CTAs
      // of 8 lookup warps: a probe of the inner loop on GB300.
      const double rate = on_sm >= 3 ? 155.0 : on_sm == 2 ? 149.0 : 130.0;
      const double tile_ns = 16384.0 * (double)on_sm / rate * (T == 2 ? 1.35 : 1.0);
      const int base = stream_smem(CPC, KS, T, G, 0).total;
      if (base > budget) continue;
      int NSC = (budget > floor_smem ? floor_smem - base : 0) / (G * kChunkBytes);  // slots the padding pays for
      const int need = (int)(kCopyNs / (G * tile_ns)) + 2;  // slots ahead that cover a copy
      const int fit = (budget - base) / (G * kChunkBytes);
      NSC = NSC > need ? NSC : need;
      NSC = NSC > 4 ? NSC : 4;
      NSC = NSC < fit ? NSC : fit;
      NSC = NSC < CPC ? NSC : CPC;
      NSC = NSC < kMaxRing ? NSC : kMaxRing;
      if (NSC < 2 && NSC < CPC) continue;
      int smem = stream_smem(CPC, KS, T, G, NSC).total;
      smem = smem > floor_smem ? smem : floor_smem;
      if (smem > budget) continue;
      if (SRB > max_active_clusters(phase, T, G, KS, smem)) continue;  // more than one wave
      double ns = (G * CPC + 0.05 * CPC) * tile_ns;
      if (NSC < CPC) {
        const double cover = (NSC - 1) * G * tile_ns;
        if (cover < kCopyNs) ns += (kCopyNs - cover) * ((CPC - 1) / NSC);
      }
      const int64_t score = (int64_t)ns;
      if (best < 0 || score < best) {
        best = score;
        p.G = G;
        p.KS = KS;
        p.CPC = CPC;
        p.NSC = NSC;
        p.smem = smem;
        p.ok = true;
      }
    }
  }
  return p;
}

// Plans are cached per (device, phase, shape, tokens): the search queries the
// driver.
StreamPlan plan_stream(int phase, const SignMatrix& sm, int T, int num_sms, int max_smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, int, int, int, int, int>, StreamPlan> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, phase, sm.RB, sm.NCH, T, num_sms, max_smem);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  const StreamPlan p = search_stream(phase, sm, T, num_sms, max_smem);
  std::lock_guard<std::mutex> lock(mu);
  cache[key] = p;
  return p;
}

cudaError_t launch_stream(int phase, const LutProblem& prob, int tokens, int ydtype, const StreamPlan& p,
                          unsigned* status, cudaStream_t st) {
  if (!p.ok || tokens < 1 || tokens > kMaxStreamTokens) return cudaErrorInvalidConfiguration;
  StreamArgs a = {};
  a.p = prob;
  a.tokens = tokens;
  a.ydtype = ydtype;
  a.KS = p.KS;
  a.CPC = p.CPC;
  a.NSC = p.NSC;
  a.status = status;
  a.wait_cycles = wait_budget();
  if (phase == 1 && prob.x2 != nullptr)
    return tokens == 1 ? launch_np<1, 0, true>(a, p, st) : launch_np<1, 1, true>(a, p, st);
  if (phase == 1) return tokens == 1 ? launch_np<1, 0>(a, p, st) : launch_np<1, 1>(a, p, st);
  return tokens == 1 ? launch_np<2, 0>(a, p, st) : launch_np<2, 1>(a, p, st);
}

}  // namespace af1
