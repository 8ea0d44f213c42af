// af1_nabf.cu — NABF (Null-space-Aware Binary Factorization, Algorithm NABF;
// App. "ADMM-SVID Framework in DBF") on the GPU: the offline step that turns
// a weight matrix W (m x n) into the AF1 layer's signs and scales.
//
//     W' = o * W * i^T,   W' ~ A B,  A = a * A_pm1 * m1^T,  B = m2 * B_pm1 * b^T
//
// Per iteration: the ADMM proxies A_hat = (W' B^T + rho (A - U_A))
// (B B^T + rho I)^-1 and B_hat = (A^T A + rho I)^-1 (A^T W' + rho (B - U_B)),
// their SVID projections (signs and a rank-1 magnitude fit by power
// iteration), the null-space compensation (Sec. 3.1: the projection
// residual A_hat - A_q is removed along P_B, the projector onto the trailing
// eigenvectors of B B^T carrying at most eta of its spectral energy) and the
// closed-form scale fits gamma* / eta* (Eq. gamma_solution) folded into
// m1 / m2, then the dual updates.
//
// The dense linear algebra goes to the vendor libraries, loaded at run time
// (the rest of the library does not depend on them): SGEMM (cuBLAS), the
// Cholesky factorization and triangular solves of the SPD proxies (cuSOLVER
// potrf, cuBLAS trsm) and the symmetric eigendecomposition of the r x r
// covariances (cuSOLVER syevd). This file's kernels do everything else:
// the surrogate scaling, the initial +-1 draw (SplitMix64), SVID (signs,
// power iteration), the compensation, the scale fits, the factor and dual
// updates, the objective and the output in AF1 form. Matrices are stored
// column-major (the libraries' convention); FP32 arithmetic, FP64 sums for
// the objective and the energy cutoff.
#include <cublas_v2.h>
#include <cuda_runtime.h>
#include <cusolverDn.h>
#include <dlfcn.h>
#include <stdint.h>

#include <cmath>
#include <mutex>
#include <string>
#include <vector>

#include "af1.h"
#include "af1_internal.h"

namespace af1 {
namespace {

// ---------------------------------------------------------------------------
// Vendor linear algebra, loaded once
// ---------------------------------------------------------------------------

struct LinAlg {
  bool ok = false;
  std::string why;
  decltype(&cublasCreate_v2) blas_create = nullptr;
  decltype(&cublasDestroy_v2) blas_destroy = nullptr;
  decltype(&cublasSetStream_v2) blas_set_stream = nullptr;
  decltype(&cublasSgemm_v2) sgemm = nullptr;
  decltype(&cublasStrsm_v2) strsm = nullptr;
  decltype(&cusolverDnCreate) sol_create = nullptr;
  decltype(&cusolverDnDestroy) sol_destroy = nullptr;
  decltype(&cusolverDnSetStream) sol_set_stream = nullptr;
  decltype(&cusolverDnSpotrf_bufferSize) potrf_buf = nullptr;
  decltype(&cusolverDnSpotrf) potrf = nullptr;
  decltype(&cusolverDnSsyevd_bufferSize) syevd_buf = nullptr;
  decltype(&cusolverDnSsyevd) syevd = nullptr;
};

void* open_first(const char* const* names) {
  for (int i = 0; names[i] != nullptr; ++i) {
    void* h = dlopen(names[i], RTLD_NOW | RTLD_GLOBAL);
    if (h != nullptr) return h;
  }
  return nullptr;
}

template <class F>
bool sym(void* h, const char* name, F& out) {
  out = reinterpret_cast<F>(dlsym(h, name));
  return out != nullptr;
}

const LinAlg& linalg() {
  static LinAlg L;
  static std::once_flag once;
  std::call_once(once, [] {
    static const char* blas_names[] = {"libcublas.so.13", "libcublas.so", "/usr/local/cuda/lib64/libcublas.so",
                                       nullptr};
    static const char* sol_names[] = {"libcusolver.so.12", "libcusolver.so.13", "libcusolver.so",
                                      "/usr/local/cuda/lib64/libcusolver.so", nullptr};
    void* hb = open_first(blas_names);
    void* hs = hb != nullptr ? open_first(sol_names) : nullptr;
    if (hb == nullptr || hs == nullptr) {
      L.why = std::string("cannot load ") + (hb == nullptr ? "cuBLAS" : "cuSOLVER") + ": " + dlerror();
      return;
    }
    const bool all = sym(hb, "cublasCreate_v2", L.blas_create) && sym(hb, "cublasDestroy_v2", L.blas_destroy) &&
                     sym(hb, "cublasSetStream_v2", L.blas_set_stream) && sym(hb, "cublasSgemm_v2", L.sgemm) &&
                     sym(hb, "cublasStrsm_v2", L.strsm) && sym(hs, "cusolverDnCreate", L.sol_create) &&
                     sym(hs, "cusolverDnDestroy", L.sol_destroy) && sym(hs, "cusolverDnSetStream", L.sol_set_stream) &&
                     sym(hs, "cusolverDnSpotrf_bufferSize", L.potrf_buf) && sym(hs, "cusolverDnSpotrf", L.potrf) &&
                     sym(hs, "cusolverDnSsyevd_bufferSize", L.syevd_buf) && sym(hs, "cusolverDnSsyevd", L.syevd);
    if (!all) {
      L.why = "a cuBLAS / cuSOLVER entry point is missing";
      return;
    }
    L.ok = true;
  });
  return L;
}

// ---------------------------------------------------------------------------
// Kernels (column-major: element (i, j) of an R x C matrix at i + j R)
// ---------------------------------------------------------------------------

constexpr int kT = 256;

inline unsigned blocks_for(int64_t n) { return (unsigned)((n + kT - 1) / kT); }

// W' = o * W * i^T, from row-major W (m x n) to column-major.
__global__ void surrogate_kernel(const float* __restrict__ W, int64_t m, int64_t n, const float* __restrict__ o,
                                 const float* __restrict__ in, float* __restrict__ Wc) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= m * n) return;
  const int64_t i = idx % m, j = idx / m;
  float v = W[i * n + j];
  if (o != nullptr) v *= o[i];
  if (in != nullptr) v *= in[j];
  Wc[idx] = v;
}

// Omega (n x r): +-1 from SplitMix64(seed, index j r + k), top bit -> -1.
__global__ void rademacher_kernel(uint64_t seed, int64_t n, int64_t r, float* __restrict__ Om) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n * r) return;
  const int64_t j = idx % n, k = idx / n;
  uint64_t z = seed + (uint64_t)(j * r + k + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  z = z ^ (z >> 31);
  Om[idx] = (z >> 63) ? -1.f : 1.f;
}

// y = alpha * (x1 + beta * x2) elementwise.
// (y may be x1 or x2: each element is read before it is written.)
__global__ void combine_kernel(const float* x1, const float* x2, float alpha, float beta, int64_t count, float* y) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx < count) y[idx] = alpha * (x1[idx] + beta * (x2 != nullptr ? x2[idx] : 0.f));
}

__global__ void add_diag_kernel(float* __restrict__ S, int64_t r, float v) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < r) S[i + i * r] += v;
}

// u[i] = sum_j |Z(i, j)| v[j]  (rows x cols).
// Columns per block of the row pass (a thread per row looping over every
// column left most SMs idle: 16 blocks for 4096 rows, 30 % of an iteration).
constexpr int kRowChunk = 64;

// part[c][i] = sum over the columns j of chunk c (blockIdx.y) of |Z(i, j)| v[j].
__global__ void absmv_rows_part_kernel(const float* __restrict__ Z, int64_t rows, int64_t cols,
                                       const float* __restrict__ v, float* __restrict__ part) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= rows) return;
  const int64_t j0 = (int64_t)blockIdx.y * kRowChunk;
  const int64_t j1 = j0 + kRowChunk < cols ? j0 + kRowChunk : cols;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  int64_t j = j0;
  for (; j + 4 <= j1; j += 4) {
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] += fabsf(Z[i + (j + q) * rows]) * v[j + q];
  }
  for (; j < j1; ++j) acc[0] += fabsf(Z[i + j * rows]) * v[j];
  part[(int64_t)blockIdx.y * rows + i] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
}

// u[i] = sum over the chunks of part[c][i], in chunk order.
__global__ void sum_parts_kernel(const float* __restrict__ part, int64_t chunks, int64_t rows,
                                 float* __restrict__ u) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= rows) return;
  float acc = 0.f;
  for (int64_t c = 0; c < chunks; ++c) acc += part[c * rows + i];
  u[i] = acc;
}

// v[j] = sum_i |Z(i, j)| u[i]: one block per column.
__global__ void absmv_cols_kernel(const float* __restrict__ Z, int64_t rows, int64_t cols, const float* __restrict__ u,
                                  float* __restrict__ v) {
  __shared__ float part[kT / 32];
  const int64_t j = blockIdx.x;
  float acc = 0.f;
  for (int64_t i = threadIdx.x; i < rows; i += blockDim.x) acc += fabsf(Z[i + j * rows]) * u[i];
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < kT / 32; ++w) t += part[w];
    v[j] = t;
  }
}

// x <- x / |x| in one block; out_norm (if set) <- |x|.
__global__ void normalize_kernel(float* __restrict__ x, int64_t count, float* __restrict__ out_norm) {
  __shared__ double part[kT / 32];
  __shared__ float nrm;
  double acc = 0.0;
  for (int64_t i = threadIdx.x; i < count; i += blockDim.x) acc += (double)x[i] * (double)x[i];
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < kT / 32; ++w) t += part[w];
    nrm = (float)sqrt(t);
    if (out_norm != nullptr) *out_norm = nrm;
  }
  __syncthreads();
  const float s = nrm > 0.f ? 1.f / nrm : 1.f;
  for (int64_t i = threadIdx.x; i < count; i += blockDim.x) x[i] *= s;
}

__global__ void fill_kernel(float* __restrict__ x, int64_t count, float v) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < count) x[i] = v;
}

// SVID assembly: rs = sqrt(sigma) u, cs = sqrt(sigma) v (in place), and
// Zq(i, j) = rs[i] Sign(Z(i, j)) cs[j] with Sign(0) = +1.
__global__ void svid_scales_kernel(float* __restrict__ u, int64_t rows, float* __restrict__ v, int64_t cols,
                                   const float* __restrict__ sigma) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const float q = sqrtf(*sigma);
  if (i < rows) u[i] *= q;
  if (i < cols) v[i] *= q;
}

__global__ void svid_assemble_kernel(const float* __restrict__ Z, int64_t rows, int64_t cols,
                                     const float* __restrict__ rs, const float* __restrict__ cs,
                                     float* __restrict__ Zq) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * cols) return;
  const int64_t i = idx % rows, j = idx / rows;
  const float m = rs[i] * cs[j];
  Zq[idx] = Z[idx] < 0.f ? -m : m;
}

// gamma[j] = <Aq(:, j), At(:, j)> / (<Aq(:, j), Aq(:, j)> + eps), then
// cs[j] *= gamma[j] (one block per column).
__global__ void col_fit_kernel(const float* __restrict__ Aq, const float* __restrict__ At, int64_t rows, float eps,
                               float* __restrict__ cs) {
  __shared__ double pn[kT / 32], pd[kT / 32];
  const int64_t j = blockIdx.x;
  double num = 0.0, den = 0.0;
  for (int64_t i = threadIdx.x; i < rows; i += blockDim.x) {
    const double q = Aq[i + j * rows], t = At[i + j * rows];
    num += q * t;
    den += q * q;
  }
  for (int o = 16; o > 0; o >>= 1) {
    num += __shfl_xor_sync(0xffffffffu, num, o);
    den += __shfl_xor_sync(0xffffffffu, den, o);
  }
  if ((threadIdx.x & 31) == 0) {
    pn[threadIdx.x >> 5] = num;
    pd[threadIdx.x >> 5] = den;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double a = 0.0, b = 0.0;
    for (int w = 0; w < kT / 32; ++w) {
      a += pn[w];
      b += pd[w];
    }
    cs[j] = (float)((double)cs[j] * (a / (b + (double)eps)));
  }
}

// eta[i] = <Bq(i, :), Bt(i, :)> / (<Bq(i, :), Bq(i, :)> + eps), then
// rs[i] *= eta[i] (one thread per row).
__global__ void row_fit_kernel(const float* __restrict__ Bq, const float* __restrict__ Bt, int64_t rows, int64_t cols,
                               float eps, float* __restrict__ rs) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= rows) return;
  double num = 0.0, den = 0.0;
  for (int64_t j = 0; j < cols; ++j) {
    const double q = Bq[i + j * rows], t = Bt[i + j * rows];
    num += q * t;
    den += q * q;
  }
  rs[i] = (float)((double)rs[i] * (num / (den + (double)eps)));
}

// X(i, j) = rs[i] Sign(Z(i, j)) cs[j]: a scaled factor from its SVID input.
__global__ void scaled_factor_kernel(const float* __restrict__ Z, int64_t rows, int64_t cols,
                                     const float* __restrict__ rs, const float* __restrict__ cs,
                                     float* __restrict__ X) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * cols) return;
  const int64_t i = idx % rows, j = idx / rows;
  const float m = rs[i] * cs[j];
  X[idx] = Z[idx] < 0.f ? -m : m;
}

// sum(x .* y) in FP64, accumulated into *out (one block per 64 K elements).
__global__ void dot_kernel(const float* __restrict__ x, const float* __restrict__ y, int64_t count,
                           double* __restrict__ out) {
  __shared__ double part[kT / 32];
  double acc = 0.0;
  const int64_t base = (int64_t)blockIdx.x * 65536;
  const int64_t end = base + 65536 < count ? base + 65536 : count;
  for (int64_t i = base + threadIdx.x; i < end; i += blockDim.x) acc += (double)x[i] * (double)y[i];
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < kT / 32; ++w) t += part[w];
    atomicAdd(out, t);
  }
}

// Outputs in AF1 form: signs as int8 (U = A_pm1 row-major m x r from
// column-major Z_A; V = B_pm1^T row-major n x r, the same memory order as
// column-major Z_B), and the scales with the surrogate undone.
__global__ void signs_u_kernel(const float* __restrict__ ZA, int64_t m, int64_t r, int8_t* __restrict__ U) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= m * r) return;
  const int64_t i = idx / r, k = idx % r;
  U[idx] = ZA[i + k * m] < 0.f ? (int8_t)-1 : (int8_t)1;
}

__global__ void signs_v_kernel(const float* __restrict__ ZB, int64_t count, int8_t* __restrict__ V) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx < count) V[idx] = ZB[idx] < 0.f ? (int8_t)-1 : (int8_t)1;
}

__global__ void out_scales_kernel(const float* __restrict__ rsA, const float* __restrict__ o, int64_t m,
                                  const float* __restrict__ csA, const float* __restrict__ rsB, int64_t r,
                                  const float* __restrict__ csB, const float* __restrict__ in, int64_t n,
                                  float* __restrict__ a, float* __restrict__ s, float* __restrict__ b) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx < m) a[idx] = o != nullptr ? rsA[idx] / o[idx] : rsA[idx];
  if (idx < r) s[idx] = csA[idx] * rsB[idx];
  if (idx < n) b[idx] = in != nullptr ? csB[idx] / in[idx] : csB[idx];
}

// ---------------------------------------------------------------------------
// Host orchestration
// ---------------------------------------------------------------------------

// Device buffers freed on every exit path.
struct Buffers {
  std::vector<void*> ptrs;
  bool failed = false;
  ~Buffers() {
    for (void* p : ptrs) cudaFree(p);
  }
  template <class T>
  T* get(int64_t count) {
    void* p = nullptr;
    if (cudaMalloc(&p, (size_t)(count > 0 ? count : 1) * sizeof(T)) != cudaSuccess) {
      failed = true;
      return nullptr;
    }
    ptrs.push_back(p);
    return static_cast<T*>(p);
  }
};

struct Handles {
  const LinAlg& L;
  cublasHandle_t blas = nullptr;
  cusolverDnHandle_t sol = nullptr;
  explicit Handles(const LinAlg& l) : L(l) {}
  ~Handles() {
    if (blas != nullptr) L.blas_destroy(blas);
    if (sol != nullptr) L.sol_destroy(sol);
  }
};

class Run {
 public:
  Run(const LinAlg& L, cudaStream_t st) : L_(L), h_(L), st_(st) {}
  // Scratch of the SVID row pass: ceil(max cols / kRowChunk) x max rows floats.
  void set_svid_scratch(float* p) { part_ = p; }

  int fail(int code, const std::string& msg) { return set_error(code, "af1_nabf_factorize: " + msg); }
  bool blas_ok(cublasStatus_t s) { return s == CUBLAS_STATUS_SUCCESS; }

  int init() {
    if (!blas_ok(L_.blas_create(&h_.blas)) || !blas_ok(L_.blas_set_stream(h_.blas, st_)))
      return fail(AF1_ERR_CUDA, "cuBLAS handle");
    if (L_.sol_create(&h_.sol) != CUSOLVER_STATUS_SUCCESS || L_.sol_set_stream(h_.sol, st_) != CUSOLVER_STATUS_SUCCESS)
      return fail(AF1_ERR_CUDA, "cuSOLVER handle");
    return AF1_OK;
  }

  // C (M x N) = alpha op(A) op(B) + beta C, column-major.
  bool gemm(bool ta, bool tb, int64_t M, int64_t N, int64_t K, float alpha, const float* A, int64_t lda,
            const float* B, int64_t ldb, float beta, float* C, int64_t ldc) {
    return blas_ok(L_.sgemm(h_.blas, ta ? CUBLAS_OP_T : CUBLAS_OP_N, tb ? CUBLAS_OP_T : CUBLAS_OP_N, (int)M, (int)N,
                            (int)K, &alpha, A, (int)lda, B, (int)ldb, &beta, C, (int)ldc));
  }

  // Cholesky S = L L^T (lower, in place); false if not positive definite.
  bool potrf(float* S, int64_t r, float* work, int lwork, int* info) {
    if (L_.potrf(h_.sol, CUBLAS_FILL_MODE_LOWER, (int)r, S, (int)r, work, lwork, info) != CUSOLVER_STATUS_SUCCESS)
      return false;
    int hinfo = 0;
    if (cudaMemcpyAsync(&hinfo, info, sizeof(int), cudaMemcpyDeviceToHost, st_) != cudaSuccess) return false;
    if (cudaStreamSynchronize(st_) != cudaSuccess) return false;
    return hinfo == 0;
  }

  // X <- X (L L^T)^-1 (X: rows x r) or X <- (L L^T)^-1 X (X: r x cols).
  bool solve_right(const float* Lf, int64_t r, float* X, int64_t rows) {
    const float one = 1.f;
    return blas_ok(L_.strsm(h_.blas, CUBLAS_SIDE_RIGHT, CUBLAS_FILL_MODE_LOWER, CUBLAS_OP_T, CUBLAS_DIAG_NON_UNIT,
                            (int)rows, (int)r, &one, Lf, (int)r, X, (int)rows)) &&
           blas_ok(L_.strsm(h_.blas, CUBLAS_SIDE_RIGHT, CUBLAS_FILL_MODE_LOWER, CUBLAS_OP_N, CUBLAS_DIAG_NON_UNIT,
                            (int)rows, (int)r, &one, Lf, (int)r, X, (int)rows));
  }
  bool solve_left(const float* Lf, int64_t r, float* X, int64_t cols) {
    const float one = 1.f;
    return blas_ok(L_.strsm(h_.blas, CUBLAS_SIDE_LEFT, CUBLAS_FILL_MODE_LOWER, CUBLAS_OP_N, CUBLAS_DIAG_NON_UNIT,
                            (int)r, (int)cols, &one, Lf, (int)r, X, (int)r)) &&
           blas_ok(L_.strsm(h_.blas, CUBLAS_SIDE_LEFT, CUBLAS_FILL_MODE_LOWER, CUBLAS_OP_T, CUBLAS_DIAG_NON_UNIT,
                            (int)r, (int)cols, &one, Lf, (int)r, X, (int)r));
  }

  // SVID of Z (rows x cols): rs, cs = sqrt(sigma) u, sqrt(sigma) v after
  // `iters` power iterations on |Z| from the all-ones vector; Zq (if set) =
  // rs Sign(Z) cs^T.
  void svid(const float* Z, int64_t rows, int64_t cols, int iters, float* rs, float* cs, float* Zq, float* sigma) {
    fill_kernel<<<blocks_for(cols), kT, 0, st_>>>(cs, cols, 1.f / sqrtf((float)cols));
    for (int it = 0; it < (iters > 0 ? iters : 1); ++it) {
      const int64_t chunks = (cols + kRowChunk - 1) / kRowChunk;
      absmv_rows_part_kernel<<<dim3((unsigned)blocks_for(rows), (unsigned)chunks), kT, 0, st_>>>(Z, rows, cols, cs,
                                                                                                part_);
      sum_parts_kernel<<<blocks_for(rows), kT, 0, st_>>>(part_, chunks, rows, rs);
      normalize_kernel<<<1, kT, 0, st_>>>(rs, rows, nullptr);
      absmv_cols_kernel<<<(unsigned)cols, kT, 0, st_>>>(Z, rows, cols, rs, cs);
      normalize_kernel<<<1, kT, 0, st_>>>(cs, cols, sigma);
    }
    svid_scales_kernel<<<blocks_for(rows > cols ? rows : cols), kT, 0, st_>>>(rs, rows, cs, cols, sigma);
    if (Zq != nullptr) svid_assemble_kernel<<<blocks_for(rows * cols), kT, 0, st_>>>(Z, rows, cols, rs, cs, Zq);
  }

  // Null-space projector (App. "Adaptive Residual-Energy Cutoff"): P = U_hat U_hat^T over
  // the q trailing eigenvectors of the symmetric C whose residual-energy
  // fraction is <= eta. Returns q, or -1 on a library failure.
  int64_t null_projector(const float* C, int64_t r, double eta, double eps, float* EV, float* w, float* work,
                         int lwork, int* info, float* P) {
    if (cudaMemcpyAsync(EV, C, (size_t)(r * r) * 4, cudaMemcpyDeviceToDevice, st_) != cudaSuccess) return -1;
    if (L_.syevd(h_.sol, CUSOLVER_EIG_MODE_VECTOR, CUBLAS_FILL_MODE_LOWER, (int)r, EV, (int)r, w, work, lwork, info) !=
        CUSOLVER_STATUS_SUCCESS)
      return -1;
    std::vector<float> hw((size_t)r);
    int hinfo = 0;
    if (cudaMemcpyAsync(hw.data(), w, (size_t)r * 4, cudaMemcpyDeviceToHost, st_) != cudaSuccess ||
        cudaMemcpyAsync(&hinfo, info, sizeof(int), cudaMemcpyDeviceToHost, st_) != cudaSuccess ||
        cudaStreamSynchronize(st_) != cudaSuccess || hinfo != 0)
      return -1;
    // Eigenvalues come ascending; pre[j] = sum of the j smallest. k = the
    // first index with sum_{i > k} lambda_i / (total + eps) <= eta, where the
    // sum over i > k (descending order) is the r - k smallest: pre[r - k].
    std::vector<double> pre((size_t)r + 1, 0.0);
    for (int64_t i = 0; i < r; ++i) pre[(size_t)i + 1] = pre[(size_t)i] + (double)hw[(size_t)i];
    const double total = pre[(size_t)r];
    int64_t q = 0;
    for (int64_t k = 0; k <= r; ++k) {
      if (pre[(size_t)(r - k)] / (total + eps) <= eta) {
        q = r - k;
        break;
      }
    }
    if (q > 0 && !gemm(false, true, r, r, q, 1.f, EV, r, EV, r, 0.f, P, r)) return -1;
    return q;
  }

  double dot(const float* x, const float* y, int64_t count, double* acc) {
    double h = 0.0;
    if (cudaMemsetAsync(acc, 0, sizeof(double), st_) != cudaSuccess) return NAN;
    dot_kernel<<<(unsigned)((count + 65535) / 65536), kT, 0, st_>>>(x, y, count, acc);
    if (cudaMemcpyAsync(&h, acc, sizeof(double), cudaMemcpyDeviceToHost, st_) != cudaSuccess) return NAN;
    if (cudaStreamSynchronize(st_) != cudaSuccess) return NAN;
    return h;
  }

  const LinAlg& L_;
  Handles h_;
  cudaStream_t st_;
  float* part_ = nullptr;
};

// Algorithm NABF; see the file comment and the oracle's readings.
int nabf_run(const float* W, int64_t m, int64_t n, int64_t r, const float* in_scale, const float* out_scale,
             const af1_nabf_params& P, int8_t* Uo, int8_t* Vo, float* ao, float* so, float* bo, double* history,
             cudaStream_t st) {
  const LinAlg& L = linalg();
  if (!L.ok) return set_error(AF1_ERR_CUDA, "af1_nabf_factorize: " + L.why);
  Run run(L, st);
  int rc = run.init();
  if (rc != AF1_OK) return rc;
  Buffers buf;
  {
    // SVIDs run on m x r (A) and r x n (B).
    const int64_t max_cols = n > r ? n : r, max_rows = m > r ? m : r;
    run.set_svid_scratch(buf.get<float>((max_cols + kRowChunk - 1) / kRowChunk * max_rows));
  }
  float* Wc = buf.get<float>(m * n);
  float *ZA = buf.get<float>(m * r), *Ah = buf.get<float>(m * r), *A = buf.get<float>(m * r),
        *UA = buf.get<float>(m * r), *Aq = buf.get<float>(m * r), *Et = buf.get<float>(m * r),
        *At = buf.get<float>(m * r);
  float *ZB = buf.get<float>(r * n), *Bh = buf.get<float>(r * n), *B = buf.get<float>(r * n),
        *UB = buf.get<float>(r * n), *Bq = buf.get<float>(r * n), *Eb = buf.get<float>(r * n),
        *Bt = buf.get<float>(r * n), *G = buf.get<float>(r * n);
  float *CB = buf.get<float>(r * r), *CA = buf.get<float>(r * r), *S = buf.get<float>(r * r),
        *EV = buf.get<float>(r * r), *Pm = buf.get<float>(r * r);
  float *rsA = buf.get<float>(m), *csA = buf.get<float>(r), *rsB = buf.get<float>(r), *csB = buf.get<float>(n),
        *w = buf.get<float>(r), *sigma = buf.get<float>(1);
  double* acc = buf.get<double>(1);
  int* info = buf.get<int>(1);
  if (buf.failed) return run.fail(AF1_ERR_CUDA, "out of device memory");
  int lw1 = 0, lw2 = 0;
  if (L.potrf_buf(run.h_.sol, CUBLAS_FILL_MODE_LOWER, (int)r, S, (int)r, &lw1) != CUSOLVER_STATUS_SUCCESS ||
      L.syevd_buf(run.h_.sol, CUSOLVER_EIG_MODE_VECTOR, CUBLAS_FILL_MODE_LOWER, (int)r, EV, (int)r, w, &lw2) !=
          CUSOLVER_STATUS_SUCCESS)
    return run.fail(AF1_ERR_CUDA, "cuSOLVER workspace query");
  const int lwork = lw1 > lw2 ? lw1 : lw2;
  float* work = buf.get<float>(lwork);
  if (buf.failed) return run.fail(AF1_ERR_CUDA, "out of device memory");
  const float rho = (float)P.rho;
  const int pit = P.power_iters;
  const int64_t mr = m * r, rn = r * n, rr = r * r;

  // Surrogate and initialization.
  surrogate_kernel<<<blocks_for(m * n), kT, 0, st>>>(W, m, n, out_scale, in_scale, Wc);
  rademacher_kernel<<<blocks_for(rn), kT, 0, st>>>(P.seed, n, r, G);  // Omega (n x r) in G
  if (!run.gemm(false, false, m, r, n, 1.f, Wc, m, G, n, 0.f, ZA, m)) return run.fail(AF1_ERR_CUDA, "SGEMM");
  if (!run.gemm(true, false, r, r, m, 1.f, ZA, m, ZA, m, 0.f, S, r) ||
      !run.gemm(true, false, r, n, m, 1.f, ZA, m, Wc, m, 0.f, ZB, r))
    return run.fail(AF1_ERR_CUDA, "SGEMM");
  add_diag_kernel<<<blocks_for(r), kT, 0, st>>>(S, r, rho);
  if (!run.potrf(S, r, work, lwork, info)) return run.fail(AF1_ERR_CUDA, "A0^T A0 + rho I is not positive definite");
  if (!run.solve_left(S, r, ZB, n)) return run.fail(AF1_ERR_CUDA, "TRSM");
  run.svid(ZA, m, r, pit, rsA, csA, nullptr, sigma);
  scaled_factor_kernel<<<blocks_for(mr), kT, 0, st>>>(ZA, m, r, rsA, csA, A);
  run.svid(ZB, r, n, pit, rsB, csB, nullptr, sigma);
  scaled_factor_kernel<<<blocks_for(rn), kT, 0, st>>>(ZB, r, n, rsB, csB, B);
  if (cudaMemsetAsync(UA, 0, (size_t)mr * 4, st) != cudaSuccess || cudaMemsetAsync(UB, 0, (size_t)rn * 4, st) != cudaSuccess)
    return run.fail(AF1_ERR_CUDA, "memset");

  // |W' - A B|^2 = |W'|^2 - 2 <A^T W', B> + <A^T A, B B^T> (relative).
  const double wn2 = run.dot(Wc, Wc, m * n, acc);
  auto objective = [&]() -> double {
    if (!run.gemm(true, false, r, n, m, 1.f, A, m, Wc, m, 0.f, G, r) ||
        !run.gemm(true, false, r, r, m, 1.f, A, m, A, m, 0.f, CA, r) ||
        !run.gemm(false, true, r, r, n, 1.f, B, r, B, r, 0.f, CB, r))
      return NAN;
    return (wn2 - 2.0 * run.dot(G, B, rn, acc) + run.dot(CA, CB, rr, acc)) / wn2;
  };
  const int T = P.iters;
  if (history != nullptr) {
    history[0] = objective();
    history[T + 1] = 0.0;
    history[2 * (T + 1)] = 0.0;
  } else if (!run.gemm(false, true, r, r, n, 1.f, B, r, B, r, 0.f, CB, r)) {
    return run.fail(AF1_ERR_CUDA, "SGEMM");
  }

  for (int t = 1; t <= T; ++t) {
    // ---- left factor (B fixed; CB = B B^T) ----
    if (cudaMemcpyAsync(S, CB, (size_t)rr * 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
      return run.fail(AF1_ERR_CUDA, "copy");
    add_diag_kernel<<<blocks_for(r), kT, 0, st>>>(S, r, rho);
    combine_kernel<<<blocks_for(mr), kT, 0, st>>>(A, UA, rho, -1.f, mr, Ah);  // rho (A - U_A)
    if (!run.gemm(false, true, m, r, n, 1.f, Wc, m, B, r, 1.f, Ah, m)) return run.fail(AF1_ERR_CUDA, "SGEMM");
    if (!run.potrf(S, r, work, lwork, info)) return run.fail(AF1_ERR_CUDA, "B B^T + rho I is not positive definite");
    if (!run.solve_right(S, r, Ah, m)) return run.fail(AF1_ERR_CUDA, "TRSM");
    combine_kernel<<<blocks_for(mr), kT, 0, st>>>(Ah, UA, 1.f, 1.f, mr, ZA);  // A_hat + U_A
    run.svid(ZA, m, r, pit, rsA, csA, Aq, sigma);
    int64_t ql = 0;
    if (P.compensate) {
      combine_kernel<<<blocks_for(mr), kT, 0, st>>>(Ah, Aq, 1.f, -1.f, mr, Et);  // residual A_hat - A_q
      ql = run.null_projector(CB, r, P.eta, P.eps, EV, w, work, lwork, info, Pm);
      if (ql < 0) return run.fail(AF1_ERR_CUDA, "eigendecomposition of B B^T");
      if (cudaMemcpyAsync(At, Ah, (size_t)mr * 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return run.fail(AF1_ERR_CUDA, "copy");
      if (ql > 0 && !run.gemm(false, false, m, r, r, -1.f, Et, m, Pm, r, 1.f, At, m))
        return run.fail(AF1_ERR_CUDA, "SGEMM");
      col_fit_kernel<<<(unsigned)r, kT, 0, st>>>(Aq, At, m, (float)P.eps, csA);
    }
    scaled_factor_kernel<<<blocks_for(mr), kT, 0, st>>>(ZA, m, r, rsA, csA, A);

    // ---- right factor (A fixed) ----
    if (!run.gemm(true, false, r, r, m, 1.f, A, m, A, m, 0.f, CA, r) ||
        !run.gemm(true, false, r, n, m, 1.f, A, m, Wc, m, 0.f, G, r))
      return run.fail(AF1_ERR_CUDA, "SGEMM");
    if (cudaMemcpyAsync(S, CA, (size_t)rr * 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
      return run.fail(AF1_ERR_CUDA, "copy");
    add_diag_kernel<<<blocks_for(r), kT, 0, st>>>(S, r, rho);
    combine_kernel<<<blocks_for(rn), kT, 0, st>>>(B, UB, rho, -1.f, rn, Bh);  // rho (B - U_B)
    combine_kernel<<<blocks_for(rn), kT, 0, st>>>(Bh, G, 1.f, 1.f, rn, Bh);   // + A^T W'
    if (!run.potrf(S, r, work, lwork, info)) return run.fail(AF1_ERR_CUDA, "A^T A + rho I is not positive definite");
    if (!run.solve_left(S, r, Bh, n)) return run.fail(AF1_ERR_CUDA, "TRSM");
    combine_kernel<<<blocks_for(rn), kT, 0, st>>>(Bh, UB, 1.f, 1.f, rn, ZB);  // B_hat + U_B
    run.svid(ZB, r, n, pit, rsB, csB, Bq, sigma);
    int64_t qr = 0;
    if (P.compensate) {
      combine_kernel<<<blocks_for(rn), kT, 0, st>>>(Bh, Bq, 1.f, -1.f, rn, Eb);  // residual B_hat - B_q
      qr = run.null_projector(CA, r, P.eta, P.eps, EV, w, work, lwork, info, Pm);
      if (qr < 0) return run.fail(AF1_ERR_CUDA, "eigendecomposition of A^T A");
      if (cudaMemcpyAsync(Bt, Bh, (size_t)rn * 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return run.fail(AF1_ERR_CUDA, "copy");
      if (qr > 0 && !run.gemm(false, false, r, n, r, -1.f, Pm, r, Eb, r, 1.f, Bt, r))
        return run.fail(AF1_ERR_CUDA, "SGEMM");
      row_fit_kernel<<<blocks_for(r), kT, 0, st>>>(Bq, Bt, r, n, (float)P.eps, rsB);
    }
    scaled_factor_kernel<<<blocks_for(rn), kT, 0, st>>>(ZB, r, n, rsB, csB, B);

    // ---- duals (with the compensated factors) ----
    combine_kernel<<<blocks_for(mr), kT, 0, st>>>(UA, Ah, 1.f, 1.f, mr, UA);
    combine_kernel<<<blocks_for(mr), kT, 0, st>>>(UA, A, 1.f, -1.f, mr, UA);
    combine_kernel<<<blocks_for(rn), kT, 0, st>>>(UB, Bh, 1.f, 1.f, rn, UB);
    combine_kernel<<<blocks_for(rn), kT, 0, st>>>(UB, B, 1.f, -1.f, rn, UB);

    if (history != nullptr) {
      history[t] = objective();  // also leaves CB = B B^T for the next left update
      history[(T + 1) + t] = (double)ql;
      history[2 * (T + 1) + t] = (double)qr;
    } else if (!run.gemm(false, true, r, r, n, 1.f, B, r, B, r, 0.f, CB, r)) {
      return run.fail(AF1_ERR_CUDA, "SGEMM");
    }
  }

  // ---- the AF1 layer ----
  signs_u_kernel<<<blocks_for(mr), kT, 0, st>>>(ZA, m, r, Uo);
  signs_v_kernel<<<blocks_for(rn), kT, 0, st>>>(ZB, rn, Vo);
  const int64_t mx = m > n ? (m > r ? m : r) : (n > r ? n : r);
  out_scales_kernel<<<blocks_for(mx), kT, 0, st>>>(rsA, out_scale, m, csA, rsB, r, csB, in_scale, n, ao, so, bo);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return run.fail(AF1_ERR_CUDA, cudaGetErrorString(e));
  return AF1_OK;
}

}  // namespace
}  // namespace af1

extern "C" {

int af1_nabf_factorize(const float* W, int64_t m, int64_t n, int64_t r, const float* in_scale, const float* out_scale,
                       const af1_nabf_params* params, int8_t* U, int8_t* V, float* a, float* s, float* b,
                       double* history, void* stream) {
  if (params == nullptr) return af1::set_error(AF1_ERR_INVALID_ARG, "params is NULL");
  const af1_nabf_params& P = *params;
  if (m <= 0 || n <= 0 || r <= 0 || r > (m < n ? m : n) || m > (int64_t)1 << 20 || n > (int64_t)1 << 20)
    return af1::set_error(AF1_ERR_INVALID_ARG, "need 0 < r <= min(m, n) and m, n <= 2^20");
  if (P.iters < 0 || P.power_iters < 1 || !(P.rho > 0.0) || !(P.eta >= 0.0 && P.eta < 1.0) || !(P.eps >= 0.0) ||
      (P.compensate != 0 && P.compensate != 1) || P.reserved != 0)
    return af1::set_error(AF1_ERR_INVALID_ARG,
                          "need iters >= 0, power_iters >= 1, rho > 0, 0 <= eta < 1, eps >= 0, compensate 0 or 1");
  if (W == nullptr || U == nullptr || V == nullptr || a == nullptr || s == nullptr || b == nullptr)
    return af1::set_error(AF1_ERR_INVALID_ARG, "W, U, V, a, s and b must be device pointers");
  return af1::nabf_run(W, m, n, r, in_scale, out_scale, P, U, V, a, s, b, history, static_cast<cudaStream_t>(stream));
}

}  // extern "C"
