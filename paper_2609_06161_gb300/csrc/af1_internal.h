// af1_internal.h — host-side structures shared by the C-ABI layer and the
// kernel launchers. Not installed; the public interface is include/af1.h.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "af1_layout.h"

struct af1_layer {
  int64_t m = 0, n = 0, r = 0;
  int32_t flags = 0;
  int device = 0;
  int num_sms = 0;
  int max_smem = 0;  // opt-in shared memory per block on this device
  // Phase 1 contracts V (B = V^T, r x n) with z = b * x; phase 2 contracts
  // U (m x r) with s' = s * t.
  af1::SignMatrix p1, p2;
  uint8_t* signs1 = nullptr;  // sign_matrix_bytes(p1)
  uint8_t* signs2 = nullptr;  // sign_matrix_bytes(p2)
  uint16_t* a = nullptr;      // FP16 row scale, m entries
  uint16_t* s = nullptr;      // FP16 rank scale, r entries
  uint16_t* b = nullptr;      // FP16 column scale, n entries
  void* alloc = nullptr;      // single device allocation holding all of the above
  int64_t sign_bytes = 0, scale_bytes = 0;
};

namespace af1 {

// Tokens per prefill pass (calls with more than kMaxPassTokens tokens).
constexpr int64_t kPrefillPassTokens = 2048;
// Longest call that may run as one pass of the 16-bit-operand decode kernel
// instead of the prefill kernel (mid_pass).
constexpr int64_t kMidMaxTokens = 64;
// SM count the planners assume when the caller passes none (a GB300 has 152).
constexpr int kDefaultSms = 152;

// Workspace carve-up for one layer and one forward call of `tokens` tokens.
struct Workspace {
  int64_t status = 0;  // uint32 status word
  int64_t sbuf = 0;    // float[max(kMaxPassTokens, tokens of a mid pass)][decode_ldz]: s' = s * t (decode)
  int64_t bbuf = 0;    // prepared B tiles of decode passes of 5..16 tokens (0: none)
  int64_t bstats = 0;  // float2 [16 slices][16 tokens] of the prepared B (0: none)
  int64_t hbuf = 0;    // FP16 [min(tokens, kPrefillPassTokens)][prefill_h_ld]: H (prefill)
  int64_t hx = 0;      // FP16 [min(tokens, kPrefillPassTokens)][swiglu_ld]: SwiGLU input h (0: none)
  int64_t pbuf = 0;    // FP32 partial tiles of the prefill GEMMs (0: none; one tile per CTA then)
  int64_t pcnt = 0;    // uint32 per prefill tile: contributors arrived (zero between calls)
  int64_t total = 0;
};
// prep = false leaves out the prepared-B region and the prefill's partial
// tiles (and so never uses them: the prefill then runs one CTA per tile);
// swiglu adds the region the SwiGLU entry point forms h in for the kernels
// that cannot form it while staging (tensor-core decode and prefill).
Workspace plan_workspace(const af1_layer& L, int64_t tokens, bool prep = true, bool swiglu = false);
// Whether a call of `tokens` tokens (17..kMidMaxTokens) runs as one pass of
// the 16-bit-operand decode kernel instead of the prefill kernel: the normal
// entry (prep), no decode-kernel flag that excludes it, a layer small enough
// for the width (measured rule in af1_decode.cu), and plans for both phases
// at that width.
bool mid_pass(const af1_layer& L, int64_t tokens, bool prep);
// Row stride (elements) of the SwiGLU input h in the workspace.
int64_t swiglu_ld(const af1_layer& L);
int64_t prefill_h_ld(const af1_layer& L);
// Bytes of the prefill's partial tiles and tile counters for a call of
// `tokens` (> kMaxPassTokens) tokens.
int64_t prefill_part_bytes(const af1_layer& L, int64_t tokens);
int64_t prefill_count_bytes(const af1_layer& L, int64_t tokens);
int64_t decode_ldz(const af1_layer& L);

// Kernel launchers (stream-ordered, asynchronous). Return cudaSuccess or the
// launch error.
cudaError_t launch_pack_signs(const int8_t* src, int64_t rows, int64_t cols, int64_t row_stride,
                              int64_t col_stride, uint32_t* words, int64_t words_per_row,
                              uint32_t* bad_flag, cudaStream_t st);
cudaError_t launch_words_to_blocks(const uint32_t* words, int64_t words_per_row, const SignMatrix& sm,
                                   uint8_t* out, cudaStream_t st);
cudaError_t launch_blocks_to_words(const uint8_t* blocks, const SignMatrix& sm, int64_t wpr, uint32_t* words,
                                   cudaStream_t st);
cudaError_t launch_bf16_to_f16(const uint16_t* src, uint16_t* dst, int64_t count, uint32_t* bad, cudaStream_t st);
// h[t][j] = FP16(SiLU(g[t][j]) u[t][j]) for t < tokens, j < n (rows of g and
// u at stride ldx, of h at ldh).
cudaError_t launch_swiglu(const __half* g, const __half* u, int64_t ldx, int64_t tokens, int64_t n, __half* h,
                          int64_t ldh, cudaStream_t st);
// Budget, in clock64() cycles, of every bounded device-side wait of the
// kernels launched from now on (af1_set_wait_cycles; process-wide). The
// default is about 1 s at the GB300's 2 GHz clock.
constexpr long long kDefaultWaitCycles = 2000000000ll;
long long wait_budget();
// Whether the caller runs layers on several streams at once
// (af1_set_stream_layout(AF1_MANY_STREAMS); process-wide): the lookup-table
// kernels then let their dependents launch late and take fewer CTAs.
bool many_streams();
// Set the calling thread's af1_last_error() message; returns `code`.
int set_error(int code, const std::string& msg);

// Decode on the CUDA cores (af1_lut.cu): the sign-matrix products of one
// phase of a pass of 1..16 tokens through lookup tables of signed sums, for
// up to kMaxGroup independent problems (layers that share their input) in
// one launch.
constexpr int kMaxGroup = 4;
struct LutProblem {
  const uint8_t* signs;  // af1_layout.h row-block layout
  SignMatrix sm;
  const __half* x;       // phase 1 input [T][ldx] (FP16)
  const __half* x2;      // phase 1, SwiGLU input: x is g, x2 is u, the input h = FP16(SiLU(g) u) (nullptr: x)
  int64_t ldx;
  const float* zin;      // phase 2 input [T][ldz] (FP32)
  int64_t ldz;
  const __half* colscale;  // phase 1: b (C entries)
  const __half* rowscale;  // phase 1: s; phase 2: a (R entries)
  float* sout;             // phase 1 output [T][lds]
  int64_t lds;
  void* y;                 // phase 2 output [T][ldy], FP16 (ydtype 0) or FP32
  int64_t ldy;
  int CPC, rb0;            // set by the launcher: chunks per CTA, first grid x of the problem
};
struct LutArgs {
  int count;         // problems (1..kMaxGroup)
  int tokens;        // T (1..16)
  int ydtype;
  int KS;            // set by the launcher: CTAs per cluster, common to all problems
  unsigned* status;
  long long wait_cycles;  // budget of every bounded wait (clock64 cycles)
  int late_trigger;       // phase 2: let the dependent launch after the lookups, not after the input
  LutProblem prob[kMaxGroup];
};
struct LutPlan {
  int KS = 0, smem = 0;
  int CPC[kMaxGroup] = {0, 0, 0, 0};
  bool ok = false;
};
// Plan of one phase for `count` problems (sm[i]) of a pass of T tokens.
LutPlan plan_lut(const SignMatrix* sm, int count, int T, int num_sms, int max_smem);
cudaError_t launch_lut(int phase, const LutArgs& a, const LutPlan& p, cudaStream_t st);

// Decode passes of 1..2 tokens over matrices too large for one wave of the
// clustered kernel (af1_stream.cu): clusters of KS CTAs per super row of G
// row blocks, CPC chunks per CTA, streamed through a ring of NSC slots, in
// one wave.
struct StreamPlan {
  int G = 0, KS = 0, CPC = 0, NSC = 0, smem = 0;
  bool ok = false;
};
// Plan of `phase` for a pass of T tokens over sm on the current device (not
// ok when no split runs in one wave).
StreamPlan plan_stream(int phase, const SignMatrix& sm, int T, int num_sms, int max_smem);
cudaError_t launch_stream(int phase, const LutProblem& prob, int tokens, int ydtype, const StreamPlan& p,
                          unsigned* status, cudaStream_t st);

// part == nullptr: one CTA per output tile (no partial tiles).
cudaError_t launch_prefill(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y, int64_t ldy,
                           int y_dtype, uint8_t* h_buf, float* part, unsigned* count, unsigned* status,
                           cudaStream_t st);
// status: the status word to report to (nullptr: the workspace's own).
// x2 != nullptr: the SwiGLU entry point (x is g, x2 is u; the workspace was
// planned with swiglu = true).
cudaError_t launch_forward(const af1_layer& L, const void* x, int64_t ldx, int64_t tokens, void* y,
                           int64_t ldy, int y_dtype, void* ws, cudaStream_t st, bool prep = true,
                           unsigned* status = nullptr, const void* x2 = nullptr);
// Several layers with the same input x (same n): one lookup-table launch per
// phase for all of them when possible, else one call per layer. The
// workspace holds one single-layer workspace per layer, each 256-aligned,
// in order (multi_workspace_offset); status reports go to the first.
int64_t multi_workspace_offset(const af1_layer* const* Ls, int i, int64_t tokens, bool prep);
cudaError_t launch_forward_multi(const af1_layer* const* Ls, int count, const void* x, int64_t ldx, int64_t tokens,
                                 void* const* ys, const int64_t* ldys, int y_dtype, void* ws, cudaStream_t st,
                                 bool prep);
// af1_linear_forward with all its argument checks; prep = false never uses
// (and does not require) the prepared-B region of the workspace.
int linear_forward_checked(const af1_layer* layer, const void* x, int64_t ldx, int64_t tokens, void* y, int64_t ldy,
                           int y_dtype, void* workspace, int64_t workspace_bytes, void* stream, bool prep,
                           const void* x2 = nullptr);

}  // namespace af1
