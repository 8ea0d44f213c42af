/*
 * af1.h — C ABI of the GB300 (sm_103a) implementation of the AF1
 * binary-factorized linear layer.
 *
 * The layer (AF1, Sec. 3.1, Eq. final_reconstruction; App. "Double-factor
 * binary representation", Eq. double_factor_equiv and Eq. binary_paths) is
 *
 *     W_hat = Diag(a) . U . Diag(s) . V^T . Diag(b)        (d_out x d_in)
 *     y     = x . W_hat^T
 *
 * with U = A_pm1 in {-1,+1}^{m x r}, V = B_pm1^T in {-1,+1}^{n x r}, the row
 * scale a (m), the merged rank scale s = m1 * m2 (r) and the column scale
 * b (n); m = d_out, n = d_in. What is stored per matrix is exactly what
 * App. "Effective Bit-Width" (Eq. app_af1_memory) counts: r(m + n) sign bits
 * plus three 16-bit scale vectors. Scales are FP16 here (the paper stores
 * BF16; both cost 16 bits). The dense W_hat is never formed: a forward call
 * evaluates y = a * (U (s * (V^T (b * x)))) on the GPU.
 *
 * Conventions for every entry point
 *   - Return value: AF1_OK (0) or a negative AF1_ERR_* code; af1_last_error()
 *     then returns a message for the calling thread. No C++ exception crosses
 *     this boundary.
 *   - All data pointers are DEVICE pointers (cudaMalloc, or memory the CUDA
 *     runtime reports as device or managed). A host pointer is rejected with
 *     AF1_ERR_BAD_POINTER before any work is queued.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream). Work is queued on it in stream order.
 *   - FP16 values are passed as their 16-bit patterns (uint16_t).
 *
 * Canonical packed format (the paper prescribes no bit layout; this is the
 * reading this library fixes): each factor is packed along its contraction
 * axis, least significant bit first, bit = 1 for +1 and bit = 0 for -1,
 * 32 signs per uint32 word, each row padded with zero bits to a multiple of
 * 4 words (16 bytes). With W(c) = 4 * ceil(c / 128):
 *   U words: m rows x W(r) words;  bit (k % 32) of word (k / 32) of row i = U[i][k]
 *   V words: r rows x W(n) words;  bit (j % 32) of word (j / 32) of row k = V[j][k]
 * Internally a layer keeps the signs in a row-block layout of its own (same
 * bit count plus block padding); the canonical words are the exchange format.
 */
#ifndef AF1_H
#define AF1_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define AF1_API __attribute__((visibility("default")))
#else
#define AF1_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes -------------------------------------------------------- */
#define AF1_OK 0
#define AF1_ERR_INVALID_ARG (-1)   /* bad size, dtype, flag or NULL where required */
#define AF1_ERR_BAD_POINTER (-2)   /* a pointer that is not device-accessible       */
#define AF1_ERR_MISALIGNED (-3)    /* pointer or leading dimension misaligned       */
#define AF1_ERR_OVER_BUDGET (-4)   /* r above the 1.0-BPW rank of (m, n)            */
#define AF1_ERR_INVALID_SIGN (-5)  /* a sign entry that is not exactly +1 or -1     */
#define AF1_ERR_CUDA (-6)          /* a CUDA runtime error (message has details)    */
#define AF1_ERR_TIMEOUT (-7)       /* a bounded device wait gave up                 */
#define AF1_ERR_WORKSPACE (-8)     /* workspace missing, too small or misaligned    */
#define AF1_ERR_IO (-9)            /* a layer file could not be read or written     */

/* ---- output dtypes for af1_linear_forward -------------------------------- */
#define AF1_F16 0
#define AF1_F32 1

/* ---- layer description flags --------------------------------------------- */
/* Allow r above the exact 1.0-BPW rank (for other budgets such as the
   paper's 2.5-BPW setting). Without it r > af1_rank_for_budget(m, n, 1, 1)
   is rejected with AF1_ERR_OVER_BUDGET. */
#define AF1_FLAG_ANY_RANK 1
/* Run decode passes (1..16 tokens) on the tensor-core kernel (tcgen05 MMAs on
   e4m3 sign and activation terms) instead of the default CUDA-core kernel
   (lookup tables of signed sums). Both compute the same products within the
   library's tolerance; the default is faster at every measured shape. */
#define AF1_FLAG_TC_DECODE 2
/* The scale vectors a, s, b passed to af1_pack_layer / af1_load_packed_layer
   are BF16 bit patterns (the paper's storage type) instead of FP16. The layer
   converts them to FP16 on the device, exactly; a value FP16 cannot hold
   exactly (beyond +-65504, nonzero below 2^-24, more significant bits than
   FP16 has at that magnitude, NaN) fails the call with AF1_ERR_INVALID_ARG.
   Both types cost 16 bits, so the bit budget is unchanged. */
#define AF1_FLAG_BF16_SCALES 4
/* Run decode passes of 1 or 2 tokens on the streaming CUDA-core kernel (one
   wave of CTAs, each streaming an equal share of the sign chunks) whenever it
   has a plan. Without the flag it runs only where its plan beats the default
   clustered kernel (matrices whose clustered split needs more than one wave
   of CTAs). Results agree within the library's tolerance. */
#define AF1_FLAG_STREAM_DECODE 8
/* Run every decode pass (1..16 tokens) on the tensor-core kernel with 16-bit
   operands (tcgen05 MMAs on exact +-b_j FP16 or +-1 BF16 sign values, the
   activations as FP16, and the rank intermediate s' as two BF16 terms that
   hold its 16 leading significant bits). Without a decode flag the library
   takes this kernel for passes of more than 4 tokens and the lookup-table
   kernels for passes of 1 to 4 tokens; calls of 17 to 64 tokens on small
   layers (up to 32 tokens below 70 M signs r (m + n), up to 64 below 20 M)
   run as one pass of it, with s' rounded to FP16 as the prefill kernel
   rounds its intermediate, unless AF1_FLAG_TC_DECODE or AF1_FLAG_LUT_DECODE
   is set. Results agree within the library's tolerance. */
#define AF1_FLAG_MMA_DECODE 16
/* Run every decode pass (1..16 tokens) on the CUDA-core lookup-table kernels
   (clustered or streaming), never on a tensor-core kernel. At most one of
   AF1_FLAG_TC_DECODE, AF1_FLAG_MMA_DECODE and AF1_FLAG_LUT_DECODE may be set. */
#define AF1_FLAG_LUT_DECODE 32

/* The launch plan of one phase of the 16-bit-operand tensor-core decode
 * kernel (AF1_FLAG_MMA_DECODE; by default passes of 5 to 16 tokens and
 * one-pass calls of 17 to 64), computed on the host alone (no GPU needed):
 * an R x C sign matrix (phase 1: r x n; phase 2: m x r) times `tokens`
 * vectors (1..64) on a GPU with num_sms SMs and max_smem bytes of opt-in
 * shared memory per block. out[0..9] = {rows N of the B operand,
 * accumulators (one MMA issuer each), A-ring depth in 128-column chunks,
 * tensor-memory columns used (of the 256 a CTA allocates), CTAs per cluster
 * along K, 128-column chunks per CTA, dynamic shared memory per CTA in
 * bytes, grid x (row blocks of 128), grid y (CTAs per cluster), 1 if a plan
 * exists else 0}. Errors: INVALID_ARG (phase not 1 or 2, R or C outside
 * 1..2^30 / 1..32768, tokens outside 1..64, num_sms < 1, max_smem < 1,
 * out NULL). */
AF1_API int af1_mma_plan_dry(int phase, int64_t R, int64_t C, int64_t tokens, int num_sms, int max_smem,
                             int32_t* out);

typedef struct af1_layer_desc {
  int64_t m;       /* d_out: rows of W_hat, length of a, length of y rows */
  int64_t n;       /* d_in: columns of W_hat, length of b and of x rows   */
  int64_t r;       /* rank: length of s, inner dimension of U and V       */
  int32_t flags;   /* AF1_FLAG_* */
  int32_t reserved;/* must be 0 */
} af1_layer_desc;

typedef struct af1_layer af1_layer; /* opaque, owns its device buffers */

/* Exact rank for a storage budget of (budget_num / budget_den) bits per
 * weight: the largest r with r(m+n) + 16(m+r+n) <= budget * m * n
 * (App. "Effective Bit-Width", Eq. app_af1_memory, read as a hard cap on the
 * full storage; App. A.3 rounds the sign bits only). Writes 0 when not even
 * rank 1 fits. Host-only, no GPU needed. Errors: INVALID_ARG for m, n <= 0,
 * budget_den <= 0, budget_num < 0, r_out NULL, or overflow. */
AF1_API int af1_rank_for_budget(int64_t m, int64_t n, int64_t budget_num, int64_t budget_den,
                        int64_t* r_out);

/* Bits one layer stores (App. "Effective Bit-Width", Eq. app_af1_memory):
 * r(m + n) sign bits plus 16 bits per FP16 scale, m + r + n of them. This is
 * the count the 1.0-BPW budget caps; a rank allocation over several layers
 * (HiSA) sums it. Host-only. Errors: INVALID_ARG for m, n, r <= 0, m or n
 * above 2^31, r above 2^31, or bits_out NULL. */
AF1_API int af1_storage_bits(int64_t m, int64_t n, int64_t r, int64_t* bits_out);

/* Build a layer from sign matrices (the factors NABF produces, Sec. 3.1).
 *   U:   int8 [m x r] row-major, entries exactly +1 or -1
 *   V:   int8 [n x r] row-major (V = B_pm1^T), entries exactly +1 or -1
 *   a:   FP16 bits [m]; s: FP16 bits [r]; b: FP16 bits [n]
 *   out_U, out_V: optional (may be NULL) device buffers that receive the
 *        canonical packed words, [m x W(r)] and [r x W(n)] uint32.
 * All inputs are device pointers read on `stream`; the layer takes its own
 * copies, so the caller may free them once this call returns (the call
 * synchronizes `stream` to validate the signs). On success *out owns the
 * layer (release with af1_free). Errors: INVALID_ARG, BAD_POINTER,
 * OVER_BUDGET, INVALID_SIGN (nothing is created), CUDA. */
AF1_API int af1_pack_layer(const af1_layer_desc* desc, const int8_t* U, const int8_t* V,
                   const uint16_t* a, const uint16_t* s, const uint16_t* b,
                   uint32_t* out_U, uint32_t* out_V, void* stream, af1_layer** out);

/* Build a layer from canonical packed words (the deployable format), e.g. a
 * saved checkpoint. U_words [m x W(r)], V_words [r x W(n)] uint32, device.
 * Padding bits are ignored. Same ownership, synchronization and errors as
 * af1_pack_layer (no INVALID_SIGN: every bit is a valid sign). */
AF1_API int af1_load_packed_layer(const af1_layer_desc* desc, const uint32_t* U_words,
                          const uint32_t* V_words, const uint16_t* a, const uint16_t* s,
                          const uint16_t* b, void* stream, af1_layer** out);

/* The layer's factors and scales in the exchange format: canonical packed
 * words U [m x W(r)] and V [r x W(n)] (uint32) and FP16 bit patterns of a, s,
 * b (for a layer made from BF16 scales: their exact FP16 values). Every output
 * is an optional device pointer (NULL skips it). Stream-ordered, asynchronous.
 * Errors: INVALID_ARG, BAD_POINTER, CUDA. */
AF1_API int af1_export_layer(const af1_layer* layer, uint32_t* U_words, uint32_t* V_words, uint16_t* a,
                             uint16_t* s, uint16_t* b, void* stream);

/* Layer files. Layout (little-endian): the 40-byte header below, then U words
 * (m x W(r) uint32), V words (r x W(n) uint32), a (m FP16), s (r FP16), b
 * (n FP16), with no padding between the arrays. flags holds the layer's
 * AF1_FLAG_ANY_RANK / AF1_FLAG_TC_DECODE / AF1_FLAG_STREAM_DECODE bits. */
#define AF1_FILE_MAGIC "AF1LAYER"
#define AF1_FILE_VERSION 1u
typedef struct af1_file_header {
  char magic[8];     /* AF1_FILE_MAGIC, no terminating NUL */
  uint32_t version;  /* AF1_FILE_VERSION */
  uint32_t flags;
  int64_t m, n, r;
} af1_file_header;

/* Write a layer to `path` (host file). Synchronizes the device work it
 * queues (on the legacy default stream). Errors: INVALID_ARG, CUDA, IO. */
AF1_API int af1_save_layer(const af1_layer* layer, const char* path);

/* Read a layer file and build the layer (as af1_load_packed_layer, on
 * `stream`, which is synchronized). Errors: INVALID_ARG, OVER_BUDGET, CUDA,
 * IO (missing, truncated or foreign file). */
AF1_API int af1_load_layer(const char* path, void* stream, af1_layer** out);

/* Copy the description of a layer into *desc. */
AF1_API int af1_layer_get_desc(const af1_layer* layer, af1_layer_desc* desc);

/* Device bytes the layer holds for its signs (row-block layout) and its scales. */
AF1_API int af1_layer_device_bytes(const af1_layer* layer, int64_t* sign_bytes, int64_t* scale_bytes);

/* Bytes of workspace one af1_linear_forward call with `tokens` rows needs
 * (>= 256). Returns a negative AF1_ERR_* code on bad arguments. */
AF1_API int64_t af1_workspace_bytes(const af1_layer* layer, int64_t tokens);

/* y = x . W_hat^T for `tokens` rows (AF1 Eq. final_reconstruction applied
 * right to left).
 *   x:  FP16 [tokens x n], row stride ldx elements (ldx >= n, ldx % 8 == 0),
 *       16-byte aligned device pointer.
 *   y:  [tokens x m], row stride ldy >= m elements, 16-byte aligned; y_dtype
 *       AF1_F16 (ldy % 8 == 0) or AF1_F32 (ldy % 4 == 0). Only the first m
 *       entries of each row are written.
 *   workspace: device scratch of at least af1_workspace_bytes(layer, tokens)
 *       bytes, 256-byte aligned, owned by the caller. It must be zero-filled
 *       before its first use; every completed call leaves its bookkeeping
 *       words at zero again, so one workspace serves any sequence of calls
 *       on one stream, for any layer. Calls that may overlap on the GPU
 *       (different streams) need different workspaces.
 * Asynchronous and stream-ordered: nothing is synchronized. tokens == 0 is a
 * no-op returning AF1_OK. Launch errors are returned at once; a device-side
 * wait that gave up is reported by af1_workspace_status. The layer is not
 * modified, so several streams may use one layer concurrently, each with its
 * own workspace. Errors: INVALID_ARG, BAD_POINTER, MISALIGNED, WORKSPACE,
 * CUDA. */
AF1_API int af1_linear_forward(const af1_layer* layer, const void* x, int64_t ldx, int64_t tokens,
                       void* y, int64_t ldy, int y_dtype, void* workspace,
                       int64_t workspace_bytes, void* stream);

/* ---- NABF: the factorization that produces an AF1 layer ---------------------
 * Algorithm NABF (Null-space-Aware Binary Factorization; App. "ADMM-SVID
 * Framework in DBF", "Adaptive Residual-Energy Cutoff") on the GPU: the
 * surrogate W' = o * W * i^T is factorized as A B with A = a * A_pm1 * m1^T,
 * B = m2 * B_pm1 * b^T by alternating ADMM proxies, SVID projections (signs
 * and a rank-1 magnitude fit by power iteration), null-space compensation and
 * closed-form scale fits. Readings: initialization by a randomized range
 * finder (W' Omega, Omega +-1 from SplitMix64(seed, j r + k), top bit -> -1,
 * then the right proxy with a zero prior and SVID of both), Sign(0) = +1,
 * power iteration from the all-ones vector with the singular value split
 * evenly, duals updated with the compensated factors. Dense products,
 * Cholesky / triangular solves and symmetric eigendecompositions use cuBLAS
 * and cuSOLVER, loaded at run time (AF1_ERR_CUDA if they cannot be loaded). */
typedef struct af1_nabf_params {
  int32_t iters;        /* T: alternating iterations, >= 0 */
  int32_t power_iters;  /* power iterations per SVID projection, >= 1 */
  double rho;           /* ADMM penalty, > 0 */
  double eta;           /* residual-energy cutoff of the null-space projector, in [0, 1) (paper: 0.01) */
  double eps;           /* stabilizer of the cutoff fraction and of the scale fits, >= 0 */
  uint64_t seed;        /* seed of the initial +-1 draw */
  int32_t compensate;   /* 1: NABF; 0: plain ADMM-SVID (no compensation) */
  int32_t reserved;     /* must be 0 */
} af1_nabf_params;

/* Factorize W (device, FP32, row-major m x n) at rank r (0 < r <= min(m, n)).
 *   in_scale (n) / out_scale (m): the surrogate's i and o (device FP32), or
 *       NULL for ones.
 *   Outputs, device: U (int8 +-1, row-major m x r) = A_pm1, V (int8 +-1,
 *       row-major n x r) = B_pm1^T, a (m), s (r) = m1 * m2, b (n) as FP32,
 *       with the surrogate scaling undone (a / o, b / i): the AF1 layer
 *       W_hat = Diag(a) U Diag(s) V^T Diag(b) (pack with af1_pack_layer after
 *       converting the scales to FP16).
 *   history (host, may be NULL): 3 (iters + 1) doubles: the relative
 *       objective |W' - A B|_F^2 / |W'|_F^2 after the initialization and after
 *       each iteration, then the numbers of trailing eigenvectors the left and
 *       right null-space projectors kept per iteration (0 at index 0).
 * Synchronizes the stream; allocates and frees its own scratch. Errors:
 * INVALID_ARG, CUDA (including a proxy that is not positive definite). */
AF1_API int af1_nabf_factorize(const float* W, int64_t m, int64_t n, int64_t r, const float* in_scale,
                               const float* out_scale, const af1_nabf_params* params, int8_t* U, int8_t* V,
                               float* a, float* s, float* b, double* history, void* stream);

/* SwiGLU input of a down projection (the MLP of the LLaMA models the paper
 * compresses): y = h . W_hat^T with h = FP16(SiLU(g) * u) elementwise,
 * SiLU(z) = z / (1 + e^-z) in FP32, from the outputs g and u of the gate and
 * up projections, without h in memory where the kernel allows it.
 *   g, u: FP16 [tokens x n], both with row stride ldx, each under the rules
 *       of x in af1_linear_forward (16-byte aligned, ldx % 8 == 0).
 *   workspace: at least af1_workspace_bytes_swiglu(layer, tokens) bytes.
 * Other arguments, stream semantics and errors as af1_linear_forward
 * (u NULL: INVALID_ARG). Decode passes on the CUDA-core kernels form h while
 * they stage their activations; the tensor-core kernels (AF1_FLAG_TC_DECODE,
 * wide passes, prefill) first write h into the workspace. Both give the same
 * h. */
AF1_API int64_t af1_workspace_bytes_swiglu(const af1_layer* layer, int64_t tokens);
AF1_API int af1_linear_forward_swiglu(const af1_layer* layer, const void* g, const void* u, int64_t ldx,
                                      int64_t tokens, void* y, int64_t ldy, int y_dtype, void* workspace,
                                      int64_t workspace_bytes, void* stream);

/* Several layers applied to the same input, e.g. the q, k and v projections
 * of a decoder layer (or gate and up): y_i = x . W_hat_i^T for i < count.
 * The paper has no counterpart; it is the batching of a decoder layer's
 * V-contractions that share x. Decode passes (up to 16 tokens) run as one
 * launch per phase for all layers when every phase of every layer would use
 * the CUDA-core decode kernel; otherwise, and for longer calls, the layers run
 * one after another. Results equal af1_linear_forward per layer within the
 * library's tolerance (count == 1: bit-identical).
 *   layers: count (1..4) layers with the same n, on the current device.
 *   x, ldx, tokens: as af1_linear_forward (shared by all layers).
 *   ys[i], ldys[i]: output of layer i, as y and ldy of af1_linear_forward.
 *   workspace: at least af1_workspace_bytes_multi(layers, count, tokens)
 *       bytes, 256-byte aligned, zero-filled before first use, as for
 *       af1_linear_forward; af1_workspace_status reports on it.
 * Errors: INVALID_ARG (count out of range, NULL entries, different n or
 * devices), BAD_POINTER, MISALIGNED, WORKSPACE, CUDA. */
AF1_API int64_t af1_workspace_bytes_multi(const af1_layer* const* layers, int count, int64_t tokens);
AF1_API int af1_linear_forward_multi(const af1_layer* const* layers, int count, const void* x, int64_t ldx,
                                     int64_t tokens, void* const* ys, const int64_t* ldys, int y_dtype,
                                     void* workspace, int64_t workspace_bytes, void* stream);

/* af1_linear_forward for callers that cannot allocate device memory when
 * they run a layer: for example a runtime that reserves all GPU memory at
 * start-up and forbids later cudaMalloc calls, or a plugin whose host owns
 * the allocator and hands it no scratch buffer. The paper has no counterpart;
 * this is a deployment convenience.
 * Same arguments as af1_linear_forward minus the workspace: the scratch is a
 * 1 MiB array compiled into the library, present on every GPU that loads it
 * until the process exits. Nothing is allocated by this call. Calls whose
 * scratch need (af1_workspace_bytes(layer, tokens)) exceeds 1 MiB are
 * rejected with AF1_ERR_WORKSPACE: with up to 16 tokens every shape with
 * r <= 16256 fits; longer calls also hold min(tokens, 2048) x r FP16 rank
 * intermediates, so they fit only for short passes of small-rank layers.
 * Passes of 8-16 tokens over large sign matrices run here without the
 * prepared tensor-core operand that af1_linear_forward keeps in its
 * workspace (the CUDA-core kernel takes them), so they can be slower.
 * The first call on a device looks up the array's device address (once per
 * device); make that first call before any stream capture. All calls share
 * the array and leave their intermediate results in it, so calls that may
 * overlap on the GPU (different streams or devices' contexts racing on one
 * device) corrupt each other: issue them in one stream. */
AF1_API int af1_linear_forward_static(const af1_layer* layer, const void* x, int64_t ldx, int64_t tokens,
                                      void* y, int64_t ldy, int y_dtype, void* stream);

/* Status of the built-in scratch array of af1_linear_forward_static on the
 * current device: synchronizes `stream`, then returns AF1_OK, or
 * AF1_ERR_TIMEOUT if a bounded device-side wait of a static call gave up
 * since the last check. On AF1_ERR_TIMEOUT the whole array is zeroed again
 * (status word and bookkeeping), so the next static call starts clean.
 * Allocates nothing. Errors: CUDA. */
AF1_API int af1_static_status(void* stream);

/* Synchronize `stream` and report the status word the kernels keep in a
 * workspace: AF1_OK, or AF1_ERR_TIMEOUT if a bounded device-side wait gave
 * up since the workspace was last cleared (the word is then reset to 0).
 * After AF1_ERR_TIMEOUT the outputs of the calls since the last check are
 * undefined and other bookkeeping words (the prefill's per-tile counters)
 * may be left non-zero: zero-fill the whole workspace before reusing it. */
AF1_API int af1_workspace_status(void* workspace, void* stream);

/* Budget of every bounded device-side wait (mbarrier phases, dependency
 * counters), in clock64() cycles, for the kernels launched after this call
 * on any thread (default 2e9, about 1 s at 2 GHz). A launch captured in a
 * CUDA graph keeps the budget it was captured with. A wait that exceeds it
 * gives up and the call reports AF1_ERR_TIMEOUT through its status word.
 * Errors: INVALID_ARG (cycles < 1). */
AF1_API int af1_set_wait_cycles(int64_t cycles);
AF1_API int64_t af1_get_wait_cycles(void);

/* How the caller runs its layers' calls, which the lookup-table decode
 * kernels (passes of 1 to 4 tokens) adapt to:
 *   AF1_ONE_STREAM (default): one call after another on one stream. The
 *     second kernel of a call lets the next kernel of the stream launch
 *     (programmatic dependent launch) as soon as it has read its input, so
 *     the next kernel's CTAs fetch their sign words meanwhile, and a single
 *     call spreads each phase over about three CTAs per SM.
 *   AF1_MANY_STREAMS: several streams run layers at once (e.g. q | k | v of
 *     a decoder layer on three streams). The next kernel launches only after
 *     the lookups, and a call takes about two CTAs per SM, which leaves SM
 *     slots to the kernels of the other streams.
 * Measured on a 32-layer decode step at one token: grouped calls on one
 * stream 1.323 ms (many-stream settings) -> 1.249 ms (one-stream settings);
 * the decoder's dependency DAG over three streams 1.478 -> 1.436 ms the
 * other way round. Both give results within the library's tolerance (the
 * K split of a call, and so the order of its FP32 sums, can differ).
 * Process-wide, for calls made after this one on any thread; a launch
 * captured in a CUDA graph keeps the setting it was captured with.
 * Errors: INVALID_ARG (another value). */
#define AF1_ONE_STREAM 0
#define AF1_MANY_STREAMS 1
AF1_API int af1_set_stream_layout(int layout);
AF1_API int af1_get_stream_layout(void);

/* ---- A decode step as one launch ---------------------------------------------
 * Many linears (e.g. the 7 of each decoder layer of a model) in dependent
 * levels, run by ONE persistent kernel. Each linear computes
 * y = x . W_hat^T (AF1 Sec. 3.1, Eq. final_reconstruction, right to left);
 * the paper has no counterpart for the batching, which removes the kernel
 * boundary per phase that separate calls pay.
 * Dependencies: an input that is exactly the output of a linear of an
 * earlier level (same pointer and row stride, matching width, FP16 outputs)
 * is chained: the consumer reads the producer's results as soon as they
 * exist, rounded exactly as the stored output (so a decoder's o projection
 * can read q's output and down can read gate's and up's through x2). Any
 * other input of a linear at level L > 0 is read only after every linear of
 * the levels below L has stored its output, as kernels in stream order
 * would. An input may not be the output of the same or a later level.
 * Results agree with af1_linear_forward per linear within the library's
 * tolerance; with integer-exact inputs they are identical. */
typedef struct af1_step_linear {
  const af1_layer* layer;
  const void* x;    /* FP16 [tokens x n], row stride ldx (ldx >= n, ldx % 8 == 0), 16-byte aligned */
  const void* x2;   /* NULL, or FP16 u of the same shape: the input is then h = FP16(SiLU(x) u),
                       SiLU(z) = z / (1 + e^-z) in FP32 (x is the gate output g) */
  int64_t ldx;
  void* y;          /* [tokens x m] of the step's y_dtype, row stride ldy, 16-byte aligned */
  int64_t ldy;
  int32_t level;    /* >= 0; linears of one level are independent of each other */
  int32_t reserved; /* must be 0 */
} af1_step_linear;

/* Level 0 waits until af1_step_open_gate has set the workspace's gate word
 * (a hand-off from another stream without an event); each run closes the
 * gate again when it ends. */
#define AF1_STEP_WAIT_GATE 1

typedef struct af1_step af1_step; /* opaque plan, owns a small device table */

/* Plan a step over `count` linears for `tokens` rows (1..4) with outputs of
 * y_dtype (AF1_F16 or AF1_F32). The pointers in lin are baked into the plan:
 * each run reads the x buffers and writes the y buffers given here. Layers
 * must outlive the plan. Allocates the plan's device table (synchronous).
 * Errors: INVALID_ARG, BAD_POINTER, MISALIGNED, CUDA. */
AF1_API int af1_step_create(const af1_step_linear* lin, int count, int64_t tokens, int y_dtype, int32_t flags,
                            af1_step** out);

/* The schedule af1_step_create would build, computed on the host alone (no
 * GPU needed): for linears of shapes (m[i], n[i], r[i]) at level[i], `tokens`
 * rows and `ctas` CTAs. producer[i] >= 0 names the linear (of an earlier
 * level) whose output is linear i's input, producer2[i] >= 0 the one whose
 * output is its SwiGLU up operand; -1 (or a NULL array) means none: an
 * external input. Problem 2j is phase 1 (t = V^T (b x), an r x n sign
 * matrix) and 2j + 1 phase 2 (u = U s', m x r) of linear order_out[j] (the
 * linears sorted by level, stably). Tile k is tasks_out[7k .. 7k + 6] =
 * {problem, first row block, row blocks G, first 128-column chunk, chunks,
 * K slice, kind}: kind 0 computes partial sums over the chunks, kind 1 (on
 * phase-2 problems, chunks 0) stores the G row blocks of y; a level's kind-1
 * tiles run after the next level's phase-1 tiles when every linear of that
 * level has a producer, else before them. CTA c runs tiles
 * cta_first_out[c] .. cta_first_out[c + 1] - 1 in that order; ks_out[q] is
 * the number of K slices of problem q. Every output
 * pointer may be NULL (tasks_out needs max_tasks >= *ntasks). Errors:
 * INVALID_ARG. */
AF1_API int af1_step_plan_dry(const int64_t* m, const int64_t* n, const int64_t* r, const int32_t* level,
                              const int32_t* producer, const int32_t* producer2, int count, int64_t tokens,
                              int32_t ctas, int32_t* order_out, int32_t* tasks_out, int64_t max_tasks,
                              int32_t* cta_first_out, int32_t* ks_out, int64_t* ntasks, double* model_us);

/* Workspace bytes af1_step_run needs (>= 256: a header of run bookkeeping
 * and the split-K partial sums of every phase, 8 bytes each). */
AF1_API int64_t af1_step_workspace_bytes(const af1_step* step);

/* Plan summary: CTAs of the launch, tiles, levels and the planner's modelled
 * critical path in microseconds (any pointer may be NULL). */
AF1_API int af1_step_info(const af1_step* step, int64_t* ctas, int64_t* tasks, int64_t* levels, double* model_us);

/* Run the step on `stream`: one cooperative kernel launch (every CTA of the
 * launch is resident). workspace: device memory of af1_step_workspace_bytes,
 * 256-byte aligned, zero-filled before its first use; every completed run
 * leaves the header ready for the next one, so one workspace serves any
 * sequence of runs on one stream. Runs that may overlap on the GPU need
 * different workspaces. A bounded wait that gave up is reported by
 * af1_workspace_status(workspace, stream) (the run's bookkeeping is closed
 * even then, so the workspace stays usable). Asynchronous; errors:
 * INVALID_ARG, WORKSPACE, BAD_POINTER, CUDA. */
AF1_API int af1_step_run(const af1_step* step, void* workspace, int64_t workspace_bytes, void* stream);

/* Open the gate of a step created with AF1_STEP_WAIT_GATE (stream-ordered
 * write of the workspace's gate word). Errors: WORKSPACE, CUDA. */
AF1_API int af1_step_open_gate(void* workspace, void* stream);

/* Release a plan (synchronizes the device first). NULL is a no-op. */
AF1_API void af1_step_destroy(af1_step* step);

/* Release a layer and its device buffers. NULL is a no-op. Synchronizes the
 * device before freeing, so queued work that reads the layer completes. */
AF1_API void af1_free(af1_layer* layer);

/* HiSA budget arithmetic (AF1 Sec. 3.2, "Hierarchical Shapley Allocation"),
 * host-only, from Shapley scores the caller estimated (which needs a model
 * and calibration data, outside this library). The paper has these as
 * formulas; these functions state them once, in double precision.
 *
 * Layer budgets, Eq. hisa_layer_budget:
 *   B_out[l] = B_total exp(phi[l] / tau) / sum_j exp(phi[j] / tau).
 * With equal-size layers and a per-layer budget in bits per weight, B_total
 * is L times the target average (e.g. L for 1.0 BPW). Errors: INVALID_ARG
 * (L <= 0, tau <= 0, non-finite inputs, NULL). */
AF1_API int af1_hisa_layer_budgets(const double* phi, int64_t L, double B_total, double tau, double* B_out);

/* Module budgets within one layer (Eq. hisa_mad_norm, the logistic map and
 * Soft-OR fusion, Eq. hisa_module_budget): for the N submodules with
 * directional and magnitude Shapley scores phi_dir[i], phi_mag[i] and
 * parameter counts params[i],
 *   z_c = (phi_c - median) / (1.4826 MAD + eps),  P_c = 1 / (1 + exp(-z_c)),
 *   v = 1 - (1 - P_dir)(1 - P_mag),  w = (v / params + eps)^alpha,
 *   b_out[i] = B_l (sum_k params[k]) w_i / sum_j params[j] w_j,
 * so that the parameter-weighted mean of b_out is B_l (bits per weight).
 * The paper's defaults: alpha = 0.2; eps is not given (1e-8 is a reading).
 * Errors: INVALID_ARG. */
AF1_API int af1_hisa_module_budgets(const double* phi_dir, const double* phi_mag, const int64_t* params,
                                    int64_t N, double B_l, double alpha, double eps, double* b_out);

/* Budget-to-rank conversion (App. "Budget-to-rank conversion"):
 * r = Round(b m n / (m + n)) (round half up; dominant sign bits only),
 * clipped to [1, 32768]. For the exact storage rule use
 * af1_rank_for_budget. Errors: INVALID_ARG. */
AF1_API int af1_budget_to_rank(double b, int64_t m, int64_t n, int64_t* r_out);

/* Message for the last error on the calling thread ("" if none). */
AF1_API const char* af1_last_error(void);

/* Library version string. */
AF1_API const char* af1_version(void);

#ifdef __cplusplus
}
#endif

#endif /* AF1_H */
