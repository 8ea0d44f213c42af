// af1_noalloc.cu — af1_linear_forward_static: the forward pass with its
// scratch memory in a fixed device array compiled into this library, for
// callers that cannot call cudaMalloc (or hand out device memory) when they
// run a layer.
//
// The scratch is one file-scope __device__ array of kStaticScratchBytes per
// GPU, reserved when the library is loaded on that device and kept until the
// process exits. Host code cannot use the array's name as a device address,
// so the address is looked up once per device with cudaGetSymbolAddress.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>
#include <string>

#include "af1.h"
#include "af1_internal.h"

namespace {

constexpr int64_t kStaticScratchBytes = int64_t(1) << 20;  // 1 MiB per device
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

int fail(int code, const std::string& msg) { return af1::set_error(code, msg); }

// Device address of the scratch array on the current device, looked up on
// the first call for that device.
int scratch_address(int dev, void** out) {
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess || p == nullptr) {
      return fail(AF1_ERR_CUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
    }
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return AF1_OK;
}

}  // namespace

extern "C" {

int af1_linear_forward_static(const af1_layer* layer, const void* x, int64_t ldx, int64_t tokens, void* y,
                              int64_t ldy, int y_dtype, void* stream) {
  if (layer == nullptr) return fail(AF1_ERR_INVALID_ARG, "layer is NULL");
  if (tokens < 0) return fail(AF1_ERR_INVALID_ARG, "tokens must be >= 0");
  if (y_dtype != AF1_F16 && y_dtype != AF1_F32) return fail(AF1_ERR_INVALID_ARG, "y_dtype must be AF1_F16 or AF1_F32");
  if (tokens == 0) return AF1_OK;
  const int64_t need = af1::plan_workspace(*layer, tokens, false).total;
  if (need > kStaticScratchBytes)
    return fail(AF1_ERR_WORKSPACE, "layer needs " + std::to_string(need) + " bytes of scratch; the built-in array holds " +
                                       std::to_string(kStaticScratchBytes));
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(AF1_ERR_CUDA, "device index out of range");
  void* scratch = nullptr;
  int rc = scratch_address(dev, &scratch);
  if (rc != AF1_OK) return rc;
  // Same argument checks and kernels as af1_linear_forward, with the
  // built-in array as the workspace (without its prepared-B region: wide
  // decode passes build their B operand in every CTA instead).
  return af1::linear_forward_checked(layer, x, ldx, tokens, y, ldy, y_dtype, scratch, kStaticScratchBytes, stream,
                                     false);
}

// Status word of the built-in array (offset 0 of the array, where every
// forward call keeps its workspace status). A timeout leaves the array's
// bookkeeping undefined, so the whole array is zeroed after reporting one.
int af1_static_status(void* stream) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(AF1_ERR_CUDA, "device index out of range");
  void* scratch = nullptr;
  int rc = scratch_address(dev, &scratch);
  if (rc != AF1_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t word = 0;
  e = cudaMemcpyAsync(&word, scratch, 4, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("af1_static_status: ") + cudaGetErrorString(e));
  if (word != 0) {
    e = cudaMemsetAsync(scratch, 0, (size_t)kStaticScratchBytes, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return fail(AF1_ERR_CUDA, std::string("af1_static_status: ") + cudaGetErrorString(e));
    return fail(AF1_ERR_TIMEOUT, "a bounded device-side wait of a static call gave up; the built-in array was reset");
  }
  af1::set_error(AF1_OK, "");
  return AF1_OK;
}

}  // extern "C"
