// af1_api.cu — the C ABI declared in include/af1.h: argument validation,
// layer ownership and dispatch to the kernels. No C++ exception crosses the
// boundary; every failure returns an AF1_ERR_* code and sets a thread-local
// message.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>

#include "af1.h"
#include "af1_internal.h"
#include "af1_layout.h"

namespace {

thread_local std::string g_err;

int fail(int code, const std::string& msg) {
  g_err = msg;
  return code;
}

int fail_cuda(cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
  return fail(AF1_ERR_CUDA, m);
}

int64_t words_per_row(int64_t cols) { return 4 * ((cols + 127) / 128); }
int64_t align256(int64_t v) { return (v + 255) / 256 * 256; }

// Exact floor((B - 16(m+n)) / (m+n+16)) with B = num * m * n / den, in
// 128-bit integer arithmetic: the largest r with r(m+n) + 16(m+r+n) <= B.
int rank_rule(int64_t m, int64_t n, int64_t num, int64_t den, int64_t* r) {
  if (m <= 0 || n <= 0 || den <= 0 || num < 0 || r == nullptr)
    return fail(AF1_ERR_INVALID_ARG, "af1_rank_for_budget: m, n, den must be > 0, num >= 0, r_out non-NULL");
  if (m > (int64_t)1 << 31 || n > (int64_t)1 << 31 || num > (int64_t)1 << 20 || den > (int64_t)1 << 20)
    return fail(AF1_ERR_INVALID_ARG, "af1_rank_for_budget: arguments out of range");
  // r <= (num*m*n - 16*den*(m+n)) / (den*(m+n+16))
  __int128 top = (__int128)num * m * n - (__int128)16 * den * (m + n);
  __int128 bot = (__int128)den * (m + n + 16);
  if (top < bot) {
    *r = 0;
    return AF1_OK;
  }
  *r = (int64_t)(top / bot);
  return AF1_OK;
}

int check_device_ptr(const void* p, const char* name, int device) {
  if (p == nullptr) return fail(AF1_ERR_INVALID_ARG, std::string(name) + " is NULL");
  cudaPointerAttributes at;
  cudaError_t e = cudaPointerGetAttributes(&at, p);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(AF1_ERR_BAD_POINTER, std::string(name) + " is not a CUDA pointer");
  }
  if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged)
    return fail(AF1_ERR_BAD_POINTER, std::string(name) + " is not device memory");
  if (at.type == cudaMemoryTypeDevice && at.device != device)
    return fail(AF1_ERR_BAD_POINTER, std::string(name) + " lives on another device");
  return AF1_OK;
}

int check_desc(const af1_layer_desc* d) {
  if (d == nullptr) return fail(AF1_ERR_INVALID_ARG, "desc is NULL");
  if (d->m <= 0 || d->n <= 0 || d->r <= 0) return fail(AF1_ERR_INVALID_ARG, "m, n and r must be positive");
  if (d->m > ((int64_t)1 << 30) || d->n > af1::kMaxCols || d->r > af1::kMaxCols)
    return fail(AF1_ERR_INVALID_ARG, "m must be <= 2^30 and n, r <= " + std::to_string(af1::kMaxCols));
  if (d->reserved != 0 || (d->flags & ~(AF1_FLAG_ANY_RANK | AF1_FLAG_TC_DECODE | AF1_FLAG_BF16_SCALES |
                                                AF1_FLAG_STREAM_DECODE | AF1_FLAG_MMA_DECODE |
                                                AF1_FLAG_LUT_DECODE)) != 0)
    return fail(AF1_ERR_INVALID_ARG, "unknown flags or non-zero reserved field");
  {
    const int kernel_flags = d->flags & (AF1_FLAG_TC_DECODE | AF1_FLAG_MMA_DECODE | AF1_FLAG_LUT_DECODE);
    if ((kernel_flags & (kernel_flags - 1)) != 0)
      return fail(AF1_ERR_INVALID_ARG, "at most one of AF1_FLAG_TC_DECODE, AF1_FLAG_MMA_DECODE, AF1_FLAG_LUT_DECODE");
  }
  if (!(d->flags & AF1_FLAG_ANY_RANK)) {
    int64_t rmax = 0;
    int rc = rank_rule(d->m, d->n, 1, 1, &rmax);
    if (rc != AF1_OK) return rc;
    if (d->r > rmax)
      return fail(AF1_ERR_OVER_BUDGET, "r = " + std::to_string(d->r) + " exceeds the 1.0-BPW rank " +
                                           std::to_string(rmax) + " of this shape");
  }
  return AF1_OK;
}

// Allocate a layer in the row-block layout; buffers zero-filled on `st`.
int create_layer(const af1_layer_desc* d, cudaStream_t st, af1_layer** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  int sms = 0;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaDeviceGetAttribute");
  af1_layer* L = new (std::nothrow) af1_layer();
  if (L == nullptr) return fail(AF1_ERR_CUDA, "host allocation failed");
  L->m = d->m;
  L->n = d->n;
  L->r = d->r;
  L->flags = d->flags;
  L->device = dev;
  L->num_sms = sms;
  int max_smem = 0;
  e = cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) {
    delete L;
    return fail_cuda(e, "cudaDeviceGetAttribute");
  }
  L->max_smem = max_smem;
  L->p1 = af1::make_sign_matrix(d->r, d->n);
  L->p2 = af1::make_sign_matrix(d->m, d->r);
  const int64_t t1 = af1::sign_matrix_bytes(L->p1);
  const int64_t t2 = af1::sign_matrix_bytes(L->p2);
  // Each scale array is zero-padded to a multiple of 256 bytes: the prefill
  // kernel copies column scales in whole 64-column stages.
  const int64_t sa = align256(2 * d->m), ss = align256(2 * d->r), sb = align256(2 * d->n);
  const int64_t total = align256(t1) + align256(t2) + sa + ss + sb;
  e = cudaMalloc(&L->alloc, (size_t)total);
  if (e != cudaSuccess) {
    delete L;
    return fail_cuda(e, "cudaMalloc(layer)");
  }
  uint8_t* base = static_cast<uint8_t*>(L->alloc);
  L->signs1 = base;
  L->signs2 = base + align256(t1);
  L->a = reinterpret_cast<uint16_t*>(L->signs2 + align256(t2));
  L->s = reinterpret_cast<uint16_t*>(reinterpret_cast<uint8_t*>(L->a) + sa);
  L->b = reinterpret_cast<uint16_t*>(reinterpret_cast<uint8_t*>(L->s) + ss);
  L->sign_bytes = t1 + t2;
  L->scale_bytes = 2 * (d->m + d->r + d->n);
  e = cudaMemsetAsync(L->alloc, 0, (size_t)total, st);
  if (e != cudaSuccess) {
    cudaFree(L->alloc);
    delete L;
    return fail_cuda(e, "cudaMemsetAsync(layer)");
  }
  *out = L;
  return AF1_OK;
}

void destroy_layer(af1_layer* L) {
  if (L == nullptr) return;
  cudaDeviceSynchronize();
  if (L->alloc) cudaFree(L->alloc);
  delete L;
}

// The layer keeps FP16 scales. BF16 inputs (AF1_FLAG_BF16_SCALES) are
// converted exactly; a value FP16 cannot hold sets *bad.
int copy_scales(af1_layer* L, const uint16_t* a, const uint16_t* s, const uint16_t* b, cudaStream_t st,
                uint32_t* bad) {
  cudaError_t e;
  if (L->flags & AF1_FLAG_BF16_SCALES) {
    e = af1::launch_bf16_to_f16(a, L->a, L->m, bad, st);
    if (e == cudaSuccess) e = af1::launch_bf16_to_f16(s, L->s, L->r, bad, st);
    if (e == cudaSuccess) e = af1::launch_bf16_to_f16(b, L->b, L->n, bad, st);
  } else {
    e = cudaMemcpyAsync(L->a, a, 2 * L->m, cudaMemcpyDeviceToDevice, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(L->s, s, 2 * L->r, cudaMemcpyDeviceToDevice, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(L->b, b, 2 * L->n, cudaMemcpyDeviceToDevice, st);
  }
  if (e != cudaSuccess) return fail_cuda(e, "copying the scales");
  return AF1_OK;
}

const char* kBf16Msg = "a BF16 scale has no exact FP16 value (out of range or below its resolution)";

int check_scales(const uint16_t* a, const uint16_t* s, const uint16_t* b, int dev) {
  int rc = check_device_ptr(a, "a", dev);
  if (rc == AF1_OK) rc = check_device_ptr(s, "s", dev);
  if (rc == AF1_OK) rc = check_device_ptr(b, "b", dev);
  return rc;
}

}  // namespace

namespace {
std::atomic<long long> g_wait_cycles{af1::kDefaultWaitCycles};
std::atomic<int> g_stream_layout{AF1_ONE_STREAM};
}  // namespace

namespace af1 {
// Record a failure in the calling thread's af1_last_error() message.
int set_error(int code, const std::string& msg) { return fail(code, msg); }
long long wait_budget() { return g_wait_cycles.load(std::memory_order_relaxed); }
bool many_streams() { return g_stream_layout.load(std::memory_order_relaxed) == AF1_MANY_STREAMS; }
}  // namespace af1

extern "C" {

int af1_rank_for_budget(int64_t m, int64_t n, int64_t budget_num, int64_t budget_den, int64_t* r_out) {
  return rank_rule(m, n, budget_num, budget_den, r_out);
}

int af1_storage_bits(int64_t m, int64_t n, int64_t r, int64_t* bits_out) {
  if (m <= 0 || n <= 0 || r <= 0 || bits_out == nullptr)
    return fail(AF1_ERR_INVALID_ARG, "af1_storage_bits: m, n, r must be > 0 and bits_out non-NULL");
  if (m > (int64_t)1 << 31 || n > (int64_t)1 << 31 || r > (int64_t)1 << 31)
    return fail(AF1_ERR_INVALID_ARG, "af1_storage_bits: arguments out of range");
  *bits_out = r * (m + n) + 16 * (m + r + n);
  return AF1_OK;
}

int af1_pack_layer(const af1_layer_desc* desc, const int8_t* U, const int8_t* V, const uint16_t* a,
                   const uint16_t* s, const uint16_t* b, uint32_t* out_U, uint32_t* out_V, void* stream,
                   af1_layer** out) {
  if (out == nullptr) return fail(AF1_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  int rc = check_desc(desc);
  if (rc != AF1_OK) return rc;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  if ((rc = check_device_ptr(U, "U", dev)) != AF1_OK) return rc;
  if ((rc = check_device_ptr(V, "V", dev)) != AF1_OK) return rc;
  if ((rc = check_scales(a, s, b, dev)) != AF1_OK) return rc;
  if (out_U && (rc = check_device_ptr(out_U, "out_U", dev)) != AF1_OK) return rc;
  if (out_V && (rc = check_device_ptr(out_V, "out_V", dev)) != AF1_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int64_t m = desc->m, n = desc->n, r = desc->r;
  const int64_t wu = words_per_row(r), wv = words_per_row(n);

  // Scratch for canonical words the caller did not ask for, plus a flag.
  int64_t need = 256 + (out_U ? 0 : align256(4 * m * wu)) + (out_V ? 0 : align256(4 * r * wv));
  uint8_t* scratch = nullptr;
  e = cudaMalloc(&scratch, (size_t)need);
  if (e != cudaSuccess) return fail_cuda(e, "cudaMalloc(pack scratch)");
  uint32_t* flag = reinterpret_cast<uint32_t*>(scratch);
  uint8_t* cur = scratch + 256;
  uint32_t* Uw = out_U;
  uint32_t* Vw = out_V;
  if (!Uw) {
    Uw = reinterpret_cast<uint32_t*>(cur);
    cur += align256(4 * m * wu);
  }
  if (!Vw) Vw = reinterpret_cast<uint32_t*>(cur);

  af1_layer* L = nullptr;
  rc = create_layer(desc, st, &L);
  if (rc != AF1_OK) {
    cudaFree(scratch);
    return rc;
  }
  e = cudaMemsetAsync(flag, 0, 8, st);
  // U: m rows of r signs, row-major. V^T: r rows of n signs read from the
  // n x r row-major V (row stride 1, column stride r).
  if (e == cudaSuccess) e = af1::launch_pack_signs(U, m, r, r, 1, Uw, wu, flag, st);
  if (e == cudaSuccess) e = af1::launch_pack_signs(V, r, n, 1, r, Vw, wv, flag, st);
  if (e == cudaSuccess) e = af1::launch_words_to_blocks(Vw, wv, L->p1, L->signs1, st);
  if (e == cudaSuccess) e = af1::launch_words_to_blocks(Uw, wu, L->p2, L->signs2, st);
  if (e != cudaSuccess) {
    destroy_layer(L);
    cudaFree(scratch);
    return fail_cuda(e, "pack kernels");
  }
  rc = copy_scales(L, a, s, b, st, flag + 1);
  uint32_t hflag[2] = {0, 0};
  if (rc == AF1_OK) {
    e = cudaMemcpyAsync(hflag, flag, 8, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) rc = fail_cuda(e, "pack synchronize");
  }
  cudaFree(scratch);
  if (rc == AF1_OK && hflag[0] != 0) rc = fail(AF1_ERR_INVALID_SIGN, "a sign entry is not exactly +1 or -1");
  if (rc == AF1_OK && hflag[1] != 0) rc = fail(AF1_ERR_INVALID_ARG, kBf16Msg);
  if (rc != AF1_OK) {
    destroy_layer(L);
    return rc;
  }
  *out = L;
  g_err.clear();
  return AF1_OK;
}

int af1_load_packed_layer(const af1_layer_desc* desc, const uint32_t* U_words, const uint32_t* V_words,
                          const uint16_t* a, const uint16_t* s, const uint16_t* b, void* stream, af1_layer** out) {
  if (out == nullptr) return fail(AF1_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  int rc = check_desc(desc);
  if (rc != AF1_OK) return rc;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  if ((rc = check_device_ptr(U_words, "U_words", dev)) != AF1_OK) return rc;
  if ((rc = check_device_ptr(V_words, "V_words", dev)) != AF1_OK) return rc;
  if ((rc = check_scales(a, s, b, dev)) != AF1_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  af1_layer* L = nullptr;
  rc = create_layer(desc, st, &L);
  if (rc != AF1_OK) return rc;
  e = af1::launch_words_to_blocks(V_words, words_per_row(desc->n), L->p1, L->signs1, st);
  if (e == cudaSuccess) e = af1::launch_words_to_blocks(U_words, words_per_row(desc->r), L->p2, L->signs2, st);
  if (e != cudaSuccess) {
    destroy_layer(L);
    return fail_cuda(e, "pack kernels");
  }
  uint32_t* bad = nullptr;
  if (desc->flags & AF1_FLAG_BF16_SCALES) {
    e = cudaMalloc(&bad, 256);
    if (e == cudaSuccess) e = cudaMemsetAsync(bad, 0, 4, st);
    if (e != cudaSuccess) {
      if (bad) cudaFree(bad);
      destroy_layer(L);
      return fail_cuda(e, "cudaMalloc(flag)");
    }
  }
  rc = copy_scales(L, a, s, b, st, bad);
  uint32_t hbad = 0;
  if (rc == AF1_OK) {
    e = bad ? cudaMemcpyAsync(&hbad, bad, 4, cudaMemcpyDeviceToHost, st) : cudaSuccess;
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) rc = fail_cuda(e, "load synchronize");
  }
  if (bad) cudaFree(bad);
  if (rc == AF1_OK && hbad != 0) rc = fail(AF1_ERR_INVALID_ARG, kBf16Msg);
  if (rc != AF1_OK) {
    destroy_layer(L);
    return rc;
  }
  *out = L;
  g_err.clear();
  return AF1_OK;
}

int af1_layer_get_desc(const af1_layer* layer, af1_layer_desc* desc) {
  if (layer == nullptr || desc == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer or desc is NULL");
  desc->m = layer->m;
  desc->n = layer->n;
  desc->r = layer->r;
  desc->flags = layer->flags;
  desc->reserved = 0;
  return AF1_OK;
}

int af1_layer_device_bytes(const af1_layer* layer, int64_t* sign_bytes, int64_t* scale_bytes) {
  if (layer == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer is NULL");
  if (sign_bytes) *sign_bytes = layer->sign_bytes;
  if (scale_bytes) *scale_bytes = layer->scale_bytes;
  return AF1_OK;
}

int af1_export_layer(const af1_layer* layer, uint32_t* U_words, uint32_t* V_words, uint16_t* a, uint16_t* s,
                     uint16_t* b, void* stream) {
  if (layer == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer is NULL");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  if (dev != layer->device) return fail(AF1_ERR_BAD_POINTER, "the current device is not the layer's device");
  int rc;
  if (U_words && (rc = check_device_ptr(U_words, "U_words", dev)) != AF1_OK) return rc;
  if (V_words && (rc = check_device_ptr(V_words, "V_words", dev)) != AF1_OK) return rc;
  if (a && (rc = check_device_ptr(a, "a", dev)) != AF1_OK) return rc;
  if (s && (rc = check_device_ptr(s, "s", dev)) != AF1_OK) return rc;
  if (b && (rc = check_device_ptr(b, "b", dev)) != AF1_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  e = cudaSuccess;
  if (U_words) e = af1::launch_blocks_to_words(layer->signs2, layer->p2, words_per_row(layer->r), U_words, st);
  if (e == cudaSuccess && V_words)
    e = af1::launch_blocks_to_words(layer->signs1, layer->p1, words_per_row(layer->n), V_words, st);
  if (e == cudaSuccess && a) e = cudaMemcpyAsync(a, layer->a, 2 * layer->m, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && s) e = cudaMemcpyAsync(s, layer->s, 2 * layer->r, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && b) e = cudaMemcpyAsync(b, layer->b, 2 * layer->n, cudaMemcpyDeviceToDevice, st);
  if (e != cudaSuccess) return fail_cuda(e, "export");
  g_err.clear();
  return AF1_OK;
}

int af1_save_layer(const af1_layer* layer, const char* path) {
  if (layer == nullptr || path == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer or path is NULL");
  const int64_t m = layer->m, n = layer->n, r = layer->r;
  const int64_t nu = m * words_per_row(r), nv = r * words_per_row(n);
  const int64_t bytes = 4 * (nu + nv) + 2 * (m + r + n);
  uint8_t* d = nullptr;
  cudaError_t e = cudaMalloc(&d, (size_t)(bytes + 1024));
  if (e != cudaSuccess) return fail_cuda(e, "cudaMalloc(save)");
  uint32_t* dU = reinterpret_cast<uint32_t*>(d);
  uint32_t* dV = dU + nu;
  uint16_t* da = reinterpret_cast<uint16_t*>(dV + nv);
  uint16_t* ds = da + m;
  uint16_t* db = ds + r;
  int rc = af1_export_layer(layer, dU, dV, da, ds, db, nullptr);
  std::string host((size_t)bytes, '\0');
  if (rc == AF1_OK) {
    e = cudaMemcpy(&host[0], d, (size_t)bytes, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) rc = fail_cuda(e, "cudaMemcpy(save)");
  }
  cudaFree(d);
  if (rc != AF1_OK) return rc;
  af1_file_header hdr = {};
  std::memcpy(hdr.magic, AF1_FILE_MAGIC, 8);
  hdr.version = AF1_FILE_VERSION;
  hdr.flags = (uint32_t)(layer->flags & ~AF1_FLAG_BF16_SCALES);  // the file stores FP16 scales
  hdr.m = m;
  hdr.n = n;
  hdr.r = r;
  FILE* f = std::fopen(path, "wb");
  if (f == nullptr) return fail(AF1_ERR_IO, std::string("cannot open ") + path + " for writing");
  const bool ok = std::fwrite(&hdr, sizeof(hdr), 1, f) == 1 && std::fwrite(host.data(), 1, host.size(), f) == host.size();
  const bool closed = std::fclose(f) == 0;
  if (!ok || !closed) return fail(AF1_ERR_IO, std::string("writing ") + path + " failed");
  g_err.clear();
  return AF1_OK;
}

int af1_load_layer(const char* path, void* stream, af1_layer** out) {
  if (out == nullptr || path == nullptr) return fail(AF1_ERR_INVALID_ARG, "path or out is NULL");
  *out = nullptr;
  FILE* f = std::fopen(path, "rb");
  if (f == nullptr) return fail(AF1_ERR_IO, std::string("cannot open ") + path);
  af1_file_header hdr = {};
  if (std::fread(&hdr, sizeof(hdr), 1, f) != 1 || std::memcmp(hdr.magic, AF1_FILE_MAGIC, 8) != 0 ||
      hdr.version != AF1_FILE_VERSION) {
    std::fclose(f);
    return fail(AF1_ERR_IO, std::string(path) + " is not an AF1 layer file of version " +
                                std::to_string(AF1_FILE_VERSION));
  }
  af1_layer_desc desc = {hdr.m, hdr.n, hdr.r, (int32_t)hdr.flags, 0};
  int rc = check_desc(&desc);
  if (rc != AF1_OK || (desc.flags & AF1_FLAG_BF16_SCALES)) {
    std::fclose(f);
    return rc != AF1_OK ? rc : fail(AF1_ERR_IO, std::string(path) + ": invalid flags");
  }
  const int64_t m = hdr.m, n = hdr.n, r = hdr.r;
  const int64_t nu = m * words_per_row(r), nv = r * words_per_row(n);
  const int64_t bytes = 4 * (nu + nv) + 2 * (m + r + n);
  std::string host((size_t)bytes, '\0');
  const bool ok = std::fread(&host[0], 1, host.size(), f) == host.size();
  std::fclose(f);
  if (!ok) return fail(AF1_ERR_IO, std::string(path) + " is truncated");
  uint8_t* d = nullptr;
  cudaError_t e = cudaMalloc(&d, (size_t)(bytes + 1024));
  if (e != cudaSuccess) return fail_cuda(e, "cudaMalloc(load)");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  e = cudaMemcpyAsync(d, host.data(), (size_t)bytes, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // `host` is pageable and freed on return
  if (e != cudaSuccess) {
    cudaFree(d);
    return fail_cuda(e, "cudaMemcpyAsync(load)");
  }
  const uint32_t* dU = reinterpret_cast<const uint32_t*>(d);
  const uint32_t* dV = dU + nu;
  const uint16_t* da = reinterpret_cast<const uint16_t*>(dV + nv);
  const uint16_t* ds = da + m;
  const uint16_t* db = ds + r;
  rc = af1_load_packed_layer(&desc, dU, dV, da, ds, db, stream, out);  // synchronizes `stream`
  cudaFree(d);
  return rc;
}

int64_t af1_workspace_bytes(const af1_layer* layer, int64_t tokens) {
  if (layer == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer is NULL");
  if (tokens < 0) return fail(AF1_ERR_INVALID_ARG, "tokens must be >= 0");
  return af1::plan_workspace(*layer, tokens).total;
}

int af1_linear_forward(const af1_layer* layer, const void* x, int64_t ldx, int64_t tokens, void* y, int64_t ldy,
                       int y_dtype, void* workspace, int64_t workspace_bytes, void* stream) {
  return af1::linear_forward_checked(layer, x, ldx, tokens, y, ldy, y_dtype, workspace, workspace_bytes, stream, true);
}

}  // extern "C"

namespace af1 {

int linear_forward_checked(const af1_layer* layer, const void* x, int64_t ldx, int64_t tokens, void* y, int64_t ldy,
                           int y_dtype, void* workspace, int64_t workspace_bytes, void* stream, bool prep,
                           const void* x2) {
  if (layer == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer is NULL");
  if (tokens < 0) return fail(AF1_ERR_INVALID_ARG, "tokens must be >= 0");
  if (y_dtype != AF1_F16 && y_dtype != AF1_F32) return fail(AF1_ERR_INVALID_ARG, "y_dtype must be AF1_F16 or AF1_F32");
  if (tokens == 0) {
    g_err.clear();
    return AF1_OK;
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  if (dev != layer->device) return fail(AF1_ERR_BAD_POINTER, "the current device is not the layer's device");
  int rc;
  if ((rc = check_device_ptr(x, x2 != nullptr ? "g" : "x", dev)) != AF1_OK) return rc;
  if (x2 != nullptr && (rc = check_device_ptr(x2, "u", dev)) != AF1_OK) return rc;
  if (x2 != nullptr && (reinterpret_cast<uintptr_t>(x2) & 15) != 0)
    return fail(AF1_ERR_MISALIGNED, "u must be 16-byte aligned");
  if ((rc = check_device_ptr(y, "y", dev)) != AF1_OK) return rc;
  if (workspace == nullptr) return fail(AF1_ERR_WORKSPACE, "workspace is NULL");
  if (check_device_ptr(workspace, "workspace", dev) != AF1_OK)
    return fail(AF1_ERR_WORKSPACE, "workspace is not device memory of the current device");
  if (ldx < layer->n) return fail(AF1_ERR_INVALID_ARG, "ldx < n");
  if (ldy < layer->m) return fail(AF1_ERR_INVALID_ARG, "ldy < m");
  if ((reinterpret_cast<uintptr_t>(x) & 15) != 0 || (reinterpret_cast<uintptr_t>(y) & 15) != 0)
    return fail(AF1_ERR_MISALIGNED, "x and y must be 16-byte aligned");
  if (ldx % 8 != 0) return fail(AF1_ERR_MISALIGNED, "ldx must be a multiple of 8");
  if (ldy % (y_dtype == AF1_F16 ? 8 : 4) != 0)
    return fail(AF1_ERR_MISALIGNED, "ldy * element size must be a multiple of 16 bytes");
  if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return fail(AF1_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  const int64_t need = af1::plan_workspace(*layer, tokens, prep, x2 != nullptr).total;
  if (workspace_bytes < need)
    return fail(AF1_ERR_WORKSPACE, "workspace too small: need " + std::to_string(need) + " bytes");
  e = af1::launch_forward(*layer, x, ldx, tokens, y, ldy, y_dtype, workspace, static_cast<cudaStream_t>(stream), prep,
                          nullptr, x2);
  if (e != cudaSuccess) return fail_cuda(e, "forward launch");
  g_err.clear();
  return AF1_OK;
}

}  // namespace af1

extern "C" {

int64_t af1_workspace_bytes_swiglu(const af1_layer* layer, int64_t tokens) {
  if (layer == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer is NULL");
  if (tokens < 0) return fail(AF1_ERR_INVALID_ARG, "tokens must be >= 0");
  return af1::plan_workspace(*layer, tokens, true, true).total;
}

int af1_linear_forward_swiglu(const af1_layer* layer, const void* g, const void* u, int64_t ldx, int64_t tokens,
                              void* y, int64_t ldy, int y_dtype, void* workspace, int64_t workspace_bytes,
                              void* stream) {
  if (u == nullptr) return fail(AF1_ERR_INVALID_ARG, "u is NULL");
  return af1::linear_forward_checked(layer, g, ldx, tokens, y, ldy, y_dtype, workspace, workspace_bytes, stream, true,
                                     u);
}

int64_t af1_workspace_bytes_multi(const af1_layer* const* layers, int count, int64_t tokens) {
  if (layers == nullptr || count < 1 || count > af1::kMaxGroup)
    return fail(AF1_ERR_INVALID_ARG, "layers must hold 1.." + std::to_string(af1::kMaxGroup) + " layers");
  for (int i = 0; i < count; ++i)
    if (layers[i] == nullptr) return fail(AF1_ERR_INVALID_ARG, "layers[" + std::to_string(i) + "] is NULL");
  if (tokens < 0) return fail(AF1_ERR_INVALID_ARG, "tokens must be >= 0");
  return af1::multi_workspace_offset(layers, count, tokens, true);
}

int af1_linear_forward_multi(const af1_layer* const* layers, int count, const void* x, int64_t ldx, int64_t tokens,
                             void* const* ys, const int64_t* ldys, int y_dtype, void* workspace,
                             int64_t workspace_bytes, void* stream) {
  if (layers == nullptr || count < 1 || count > af1::kMaxGroup)
    return fail(AF1_ERR_INVALID_ARG, "layers must hold 1.." + std::to_string(af1::kMaxGroup) + " layers");
  if (ys == nullptr || ldys == nullptr) return fail(AF1_ERR_INVALID_ARG, "ys and ldys must not be NULL");
  for (int i = 0; i < count; ++i) {
    if (layers[i] == nullptr) return fail(AF1_ERR_INVALID_ARG, "layers[" + std::to_string(i) + "] is NULL");
    if (layers[i]->n != layers[0]->n) return fail(AF1_ERR_INVALID_ARG, "the layers' n (d_in) differ");
    if (layers[i]->device != layers[0]->device) return fail(AF1_ERR_INVALID_ARG, "the layers live on different devices");
  }
  if (tokens < 0) return fail(AF1_ERR_INVALID_ARG, "tokens must be >= 0");
  if (y_dtype != AF1_F16 && y_dtype != AF1_F32) return fail(AF1_ERR_INVALID_ARG, "y_dtype must be AF1_F16 or AF1_F32");
  if (tokens == 0) {
    g_err.clear();
    return AF1_OK;
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  if (dev != layers[0]->device) return fail(AF1_ERR_BAD_POINTER, "the current device is not the layers' device");
  int rc;
  if ((rc = check_device_ptr(x, "x", dev)) != AF1_OK) return rc;
  if (ldx < layers[0]->n) return fail(AF1_ERR_INVALID_ARG, "ldx < n");
  if ((reinterpret_cast<uintptr_t>(x) & 15) != 0) return fail(AF1_ERR_MISALIGNED, "x must be 16-byte aligned");
  if (ldx % 8 != 0) return fail(AF1_ERR_MISALIGNED, "ldx must be a multiple of 8");
  for (int i = 0; i < count; ++i) {
    const std::string yi = "ys[" + std::to_string(i) + "]";
    if ((rc = check_device_ptr(ys[i], yi.c_str(), dev)) != AF1_OK) return rc;
    if (ldys[i] < layers[i]->m) return fail(AF1_ERR_INVALID_ARG, "ldys[" + std::to_string(i) + "] < m");
    if ((reinterpret_cast<uintptr_t>(ys[i]) & 15) != 0) return fail(AF1_ERR_MISALIGNED, yi + " must be 16-byte aligned");
    if (ldys[i] % (y_dtype == AF1_F16 ? 8 : 4) != 0)
      return fail(AF1_ERR_MISALIGNED, "ldys[i] * element size must be a multiple of 16 bytes");
  }
  if (workspace == nullptr) return fail(AF1_ERR_WORKSPACE, "workspace is NULL");
  if (check_device_ptr(workspace, "workspace", dev) != AF1_OK)
    return fail(AF1_ERR_WORKSPACE, "workspace is not device memory of the current device");
  if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
    return fail(AF1_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  const int64_t need = af1::multi_workspace_offset(layers, count, tokens, true);
  if (workspace_bytes < need)
    return fail(AF1_ERR_WORKSPACE, "workspace too small: need " + std::to_string(need) + " bytes");
  e = af1::launch_forward_multi(layers, count, x, ldx, tokens, ys, ldys, y_dtype, workspace,
                                static_cast<cudaStream_t>(stream), true);
  if (e != cudaSuccess) return fail_cuda(e, "forward launch");
  g_err.clear();
  return AF1_OK;
}

int af1_workspace_status(void* workspace, void* stream) {
  if (workspace == nullptr) return fail(AF1_ERR_WORKSPACE, "workspace is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t h = 0;
  cudaError_t e = cudaMemcpyAsync(&h, workspace, 4, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail_cuda(e, "af1_workspace_status");
  if (h != 0) {
    cudaMemsetAsync(workspace, 0, 4, st);
    cudaStreamSynchronize(st);
    return fail(AF1_ERR_TIMEOUT, "a bounded device-side wait gave up; re-zero the workspace before reuse");
  }
  g_err.clear();
  return AF1_OK;
}

int af1_set_wait_cycles(int64_t cycles) {
  if (cycles < 1) return fail(AF1_ERR_INVALID_ARG, "cycles must be >= 1");
  g_wait_cycles.store(cycles, std::memory_order_relaxed);
  g_err.clear();
  return AF1_OK;
}

int64_t af1_get_wait_cycles(void) { return g_wait_cycles.load(std::memory_order_relaxed); }

int af1_set_stream_layout(int layout) {
  if (layout != AF1_ONE_STREAM && layout != AF1_MANY_STREAMS)
    return fail(AF1_ERR_INVALID_ARG, "layout must be AF1_ONE_STREAM or AF1_MANY_STREAMS");
  g_stream_layout.store(layout, std::memory_order_relaxed);
  g_err.clear();
  return AF1_OK;
}

int af1_get_stream_layout(void) { return g_stream_layout.load(std::memory_order_relaxed); }

void af1_free(af1_layer* layer) { destroy_layer(layer); }

const char* af1_last_error(void) { return g_err.c_str(); }

const char* af1_version(void) { return "af1-gb300 0.1.0 (sm_103a)"; }

}  // extern "C"
