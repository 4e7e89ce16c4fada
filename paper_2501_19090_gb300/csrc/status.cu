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

// ---- side streams: independent products of one call, run concurrently --------------------------
// Per host thread and device, two non-blocking streams and three events, made on first use and
// kept for the thread's life (CUDA releases them with the context). A side stream first waits for
// everything enqueued on the caller's stream so far (PifaSides::fork), and the caller's stream
// waits for it before the call returns (the destructor), so the call behaves as one stream's work:
// under stream capture the side streams join the capture through these event waits and rejoin it.
namespace {
struct SideState {
  bool ready = false;
  cudaStream_t s[2] = {};
  cudaEvent_t fork = nullptr;
  cudaEvent_t join[2] = {};
};
thread_local SideState g_side[kMaxDevices];

SideState* side_state(cudaError_t* err) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *err = e != cudaSuccess ? e : cudaErrorInvalidDevice;
    return nullptr;
  }
  SideState& st = g_side[dev];
  if (!st.ready) {
    for (int i = 0; i < 2 && e == cudaSuccess; ++i) e = cudaStreamCreateWithFlags(&st.s[i], cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&st.fork, cudaEventDisableTiming);
    for (int i = 0; i < 2 && e == cudaSuccess; ++i) e = cudaEventCreateWithFlags(&st.join[i], cudaEventDisableTiming);
    if (e != cudaSuccess) {
      *err = e;
      return nullptr;
    }
    st.ready = true;
  }
  return &st;
}
}  // namespace

PifaSides::~PifaSides() {
  // the caller's stream waits for every side stream that was given work, even after a failure
  for (int i = 0; i < 2; ++i)
    if (forked_[i]) {
      SideState* st = static_cast<SideState*>(state_);
      if (cudaEventRecord(st->join[i], st->s[i]) == cudaSuccess) cudaStreamWaitEvent(main_, st->join[i], 0);
    }
}

int PifaSides::fork(int i, cudaStream_t* side) {
  cudaError_t e = cudaSuccess;
  SideState* st = state_ ? static_cast<SideState*>(state_) : side_state(&e);
  if (!st) return pifa_fail_cuda("side stream", e);
  state_ = st;
  if ((e = cudaEventRecord(st->fork, main_)) != cudaSuccess || (e = cudaStreamWaitEvent(st->s[i], st->fork, 0)) != cudaSuccess)
    return pifa_fail_cuda("side stream fork", e);
  forked_[i] = true;
  *side = st->s[i];
  return PIFA_OK;
}
