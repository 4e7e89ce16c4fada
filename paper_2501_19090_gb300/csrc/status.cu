// status.cu -- the device-side error word that kernels latch (first error wins) and
// pifa_device_status() reads and clears. One int per device, in this library's static device data.
#include <atomic>
#include <mutex>

#include <cuda_runtime.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {
__device__ int g_pifa_status_word = 0;

std::atomic<int64_t> g_launches{0};

constexpr int kMaxDevices = 64;
int* g_word_addr[kMaxDevices] = {};
std::mutex g_word_mu;
}  // namespace

void pifa_count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

extern "C" int64_t pifa_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

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

namespace {
// Waits, with the library's bound, on an mbarrier that nothing ever arrives on, then latches
// PIFA_ERR_TIMEOUT: the failure-detection path of every bounded wait, exercised on its own.
__global__ void wait_timeout_selftest(int* status, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    pifa::mbar_init(&bar, 1);
    pifa::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !pifa::mbar_wait(&bar, 0, limit_ns)) pifa::latch_status(status, PIFA_ERR_TIMEOUT);
  __syncthreads();
}
}  // namespace

extern "C" int pifa_selftest_wait_timeout(void* cuda_stream) {
  pifa_clear_error();
  cudaError_t e = cudaSuccess;
  int* status = pifa_status_word(&e);
  if (!status) return pifa_fail_cuda("device status word", e);
  wait_timeout_selftest<<<1, 32, 0, reinterpret_cast<cudaStream_t>(cuda_stream)>>>(status, pifa_wait_timeout_ns());
  e = cudaGetLastError();
  if (e != cudaSuccess) return pifa_fail_cuda("wait-timeout self-test launch", e);
  pifa_count_launch();
  return PIFA_OK;
}
