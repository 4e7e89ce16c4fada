// status.cu -- the device-side error word that kernels latch (first error wins) and
// pifa_device_status() reads and clears. One int per device, in this library's static device data.
#include <mutex>

#include <cuda_runtime.h>

#include "pifa_internal.h"

namespace {
__device__ int g_pifa_status_word = 0;

constexpr int kMaxDevices = 64;
int* g_word_addr[kMaxDevices] = {};
std::mutex g_word_mu;
}  // namespace

int* pifa_status_word(cudaError_t* err) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    if (err) *err = (e != cudaSuccess) ? e : cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_word_mu);
  if (!g_word_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_pifa_status_word);
    if (e != cudaSuccess) {
      if (err) *err = e;
      return nullptr;
    }
    g_word_addr[dev] = static_cast<int*>(p);
  }
  return g_word_addr[dev];
}
