// decode.cu -- PIFA forward for small token counts (T <= 16): Algorithm 2 as two HBM-streaming
// GEMV phases.
//
//   phase 1: Y_p = X W_p^T   (r rows of W_p streamed once)   -> y_p fp32 in the workspace,
//            Y[:, I[j]] = bf16(Y_p[:, j])                     (Algorithm 2, steps 2 and 4)
//   phase 2: Y_np = Y_p C^T  (m - r rows of C streamed once)  -> Y[:, I^c[i]] = bf16(Y_np[:, i])
//                                                              (Algorithm 2, steps 3 and 5)
//
// The work is memory bound: every weight byte is read exactly once, x and y_p are tiny and stay in
// L1/L2. One CTA owns 16 consecutive weight rows (one m16 MMA fragment); its warps split the K
// dimension. Each lane issues 128-bit streaming loads straight into registers: for a 32-wide K
// chunk, lane (g = lane/4, c = lane%4) loads 8 consecutive elements of rows g and g+8 at offset
// 8c. Those registers are used directly as the A fragments of two m16n8k16 MMAs by permuting K
// consistently in both operands (a dot product does not depend on the order of its terms): MMA
// step s takes elements 4s..4s+3 of each lane's 8. Each lane loads the matching 8 activations
// of token g (B fragment). Warps then reduce their partial 16 x 8 tiles through shared memory.
//
// Phase 2 is launched with programmatic dependent launch: its CTAs start while phase 1 streams
// W_p, prefetch their rows of C into L2, then block in griddepcontrol.wait until phase 1 has
// completed. y_p enters the second contraction as a bf16 hi + bf16 lo pair (16 significant bits):
// C has large entries and Y_np = C Y_p cancels, so rounding y_p to bf16 alone would amplify its
// rounding error several-fold.
#include <mutex>

#include <cuda_bf16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

constexpr int kRows = 16;   // weight rows per CTA
constexpr int kChunk = 32;  // K elements per warp step (two k16 MMAs)
constexpr int kUnroll = 4;  // chunks in flight per warp

__device__ __forceinline__ uint32_t pack2(uint16_t a, uint16_t b) { return (uint32_t)a | ((uint32_t)b << 16); }

// 8 consecutive bf16 of `row` starting at column k; zero beyond column K or for an invalid row.
template <bool kStream>
__device__ __forceinline__ uint4 load8_bf16(const bf16* __restrict__ base, int64_t ld, int64_t row,
                                            bool row_ok, int k, int K) {
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (!row_ok || k >= K) return v;
  const bf16* p = base + row * ld + k;
  if (k + 8 <= K) {
    if (kStream) return ld_stream_16(p);
    return __ldg(reinterpret_cast<const uint4*>(p));
  }
  uint16_t e[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) e[i] = (k + i < K) ? __bfloat16_as_ushort(p[i]) : (uint16_t)0;
  v.x = pack2(e[0], e[1]);
  v.y = pack2(e[2], e[3]);
  v.z = pack2(e[4], e[5]);
  v.w = pack2(e[6], e[7]);
  return v;
}

// 8 consecutive fp32 y_p values of token t at column k, split into bf16 hi and lo words.
__device__ __forceinline__ void load8_split(const float* __restrict__ yp, bool t_ok, int k, int K, uint4& hi,
                                            uint4& lo) {
  float f[8];
  if (t_ok && k + 8 <= K) {
    const float4 a = __ldcg(reinterpret_cast<const float4*>(yp + k));
    const float4 b = __ldcg(reinterpret_cast<const float4*>(yp + k + 4));
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
    f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) f[i] = (t_ok && k + i < K) ? __ldcg(yp + k + i) : 0.0f;
  }
  uint16_t h[8], l[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const bf16 bh = __float2bfloat16_rn(f[i]);
    const bf16 bl = __float2bfloat16_rn(f[i] - __bfloat162float(bh));
    h[i] = __bfloat16_as_ushort(bh);
    l[i] = __bfloat16_as_ushort(bl);
  }
  hi = make_uint4(pack2(h[0], h[1]), pack2(h[2], h[3]), pack2(h[4], h[5]), pack2(h[6], h[7]));
  lo = make_uint4(pack2(l[0], l[1]), pack2(l[2], l[3]), pack2(l[4], l[5]), pack2(l[6], l[7]));
}

// Cross-warp reduction of the per-warp 16 x (8*NT) partial tiles; returns via shared memory.
template <int NT, int WARPS>
__device__ __forceinline__ void stash_partials(float (*red)[kRows][8 * NT], const float (&acc)[NT][4],
                                               int warp, int g, int c) {
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    red[warp][g][nt * 8 + 2 * c] = acc[nt][0];
    red[warp][g][nt * 8 + 2 * c + 1] = acc[nt][1];
    red[warp][g + 8][nt * 8 + 2 * c] = acc[nt][2];
    red[warp][g + 8][nt * 8 + 2 * c + 1] = acc[nt][3];
  }
}

// ---- phase 1: Y_p = X W_p^T -------------------------------------------------------------------
template <int NT, int WARPS>
__global__ void __launch_bounds__(WARPS * 32) decode_pivot_rows(
    const bf16* __restrict__ X, int T, int n, int64_t ldx, const bf16* __restrict__ Wp, int r, int64_t ldwp,
    const int32_t* __restrict__ piv, int m, bf16* __restrict__ Y, int64_t ldy, float* __restrict__ yp,
    int64_t ldyp, int* status) {
  pdl_launch_dependents();  // let phase 2 start prefetching C right away
  __shared__ float red[WARPS][kRows][8 * NT];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int64_t row0 = (int64_t)blockIdx.x * kRows;
  const bool ok0 = row0 + g < r, ok1 = row0 + g + 8 < r;
  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.0f;

  const int nchunks = (n + kChunk - 1) / kChunk;
  for (int base = warp; base < nchunks; base += WARPS * kUnroll) {
    uint4 wa[kUnroll], wb[kUnroll], xv[kUnroll][NT];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int ch = base + u * WARPS;
      const int k = ch * kChunk + 8 * c;
      const bool in = ch < nchunks;
      wa[u] = load8_bf16<true>(Wp, ldwp, row0 + g, in && ok0, k, n);
      wb[u] = load8_bf16<true>(Wp, ldwp, row0 + g + 8, in && ok1, k, n);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int t = nt * 8 + g;
        xv[u][nt] = load8_bf16<false>(X, ldx, t, in && t < T, k, n);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        mma_m16n8k16_bf16(acc[nt], wa[u].x, wb[u].x, wa[u].y, wb[u].y, xv[u][nt].x, xv[u][nt].y);
        mma_m16n8k16_bf16(acc[nt], wa[u].z, wb[u].z, wa[u].w, wb[u].w, xv[u][nt].z, xv[u][nt].w);
      }
    }
  }
  stash_partials<NT, WARPS>(red, acc, warp, g, c);
  __syncthreads();
  for (int idx = threadIdx.x; idx < kRows * 8 * NT; idx += WARPS * 32) {
    const int row = idx / (8 * NT), t = idx % (8 * NT);
    const int64_t j = row0 + row;
    if (t >= T || j >= r) continue;
    float s = 0.0f;
#pragma unroll
    for (int w = 0; w < WARPS; ++w) s += red[w][row][t];
    yp[(int64_t)t * ldyp + j] = s;
    const int col = piv[j];
    if ((unsigned)col >= (unsigned)m) {
      latch_status(status, PIFA_ERR_DEVICE_INDEX);
      continue;
    }
    Y[(int64_t)t * ldy + col] = __float2bfloat16_rn(s);
  }
}

// ---- phase 2: Y_np = Y_p C^T ------------------------------------------------------------------
template <int NT, int WARPS>
__global__ void __launch_bounds__(WARPS * 32) decode_nonpivot_rows(
    const float* __restrict__ yp, int64_t ldyp, int T, int r, const bf16* __restrict__ C, int mr, int64_t ldc,
    const int32_t* __restrict__ nonpiv, int m, bf16* __restrict__ Y, int64_t ldy, int* status) {
  __shared__ float red[WARPS][kRows][8 * NT];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int64_t row0 = (int64_t)blockIdx.x * kRows;
  if (threadIdx.x < kRows && row0 + threadIdx.x < mr) {
    const uint32_t bytes = ((uint32_t)r * 2u + 15u) & ~15u;  // within the 16-byte row pitch
    prefetch_l2_bulk(C + (row0 + threadIdx.x) * ldc, bytes);
  }
  pdl_wait_primary();  // phase 1 finished; y_p is complete and visible

  const bool ok0 = row0 + g < mr, ok1 = row0 + g + 8 < mr;
  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.0f;
  const int nchunks = (r + kChunk - 1) / kChunk;
  for (int base = warp; base < nchunks; base += WARPS * kUnroll) {
    uint4 ca[kUnroll], cb[kUnroll], hi[kUnroll][NT], lo[kUnroll][NT];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int ch = base + u * WARPS;
      const int k = ch * kChunk + 8 * c;
      const bool in = ch < nchunks;
      ca[u] = load8_bf16<true>(C, ldc, row0 + g, in && ok0, k, r);
      cb[u] = load8_bf16<true>(C, ldc, row0 + g + 8, in && ok1, k, r);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int t = nt * 8 + g;
        const bool t_ok = in && t < T && k < r;
        load8_split(yp + (int64_t)(t < T ? t : 0) * ldyp, t_ok, k, r, hi[u][nt], lo[u][nt]);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        mma_m16n8k16_bf16(acc[nt], ca[u].x, cb[u].x, ca[u].y, cb[u].y, hi[u][nt].x, hi[u][nt].y);
        mma_m16n8k16_bf16(acc[nt], ca[u].x, cb[u].x, ca[u].y, cb[u].y, lo[u][nt].x, lo[u][nt].y);
        mma_m16n8k16_bf16(acc[nt], ca[u].z, cb[u].z, ca[u].w, cb[u].w, hi[u][nt].z, hi[u][nt].w);
        mma_m16n8k16_bf16(acc[nt], ca[u].z, cb[u].z, ca[u].w, cb[u].w, lo[u][nt].z, lo[u][nt].w);
      }
    }
  }
  stash_partials<NT, WARPS>(red, acc, warp, g, c);
  __syncthreads();
  for (int idx = threadIdx.x; idx < kRows * 8 * NT; idx += WARPS * 32) {
    const int row = idx / (8 * NT), t = idx % (8 * NT);
    const int64_t i = row0 + row;
    if (t >= T || i >= mr) continue;
    float s = 0.0f;
#pragma unroll
    for (int w = 0; w < WARPS; ++w) s += red[w][row][t];
    const int col = nonpiv[i];
    if ((unsigned)col >= (unsigned)m) {
      latch_status(status, PIFA_ERR_DEVICE_INDEX);
      continue;
    }
    Y[(int64_t)t * ldy + col] = __float2bfloat16_rn(s);
  }
}

// Phase 1 runs W1 warps per CTA, phase 2 W2: small enough together that a phase-2 CTA fits in the
// registers an SM has left beside a phase-1 CTA, so the two phases overlap under PDL.
template <int NT, int W1, int W2>
int launch_decode_t(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream) {
  const int T = (int)s.T, n = (int)s.n, r = (int)s.r, m = (int)s.m, mr = (int)(s.m - s.r);
  float* yp = reinterpret_cast<float*>(p.ws);
  const int64_t ldyp = (s.r + 7) / 8 * 8;  // 32-byte row pitch keeps the 16-byte loads aligned
  decode_pivot_rows<NT, W1><<<dim3((r + kRows - 1) / kRows), dim3(W1 * 32), 0, stream>>>(
      reinterpret_cast<const bf16*>(p.X), T, n, s.ldx, reinterpret_cast<const bf16*>(p.Wp), r, s.ldwp, p.piv, m,
      reinterpret_cast<bf16*>(p.Y), s.ldy, yp, ldyp, status);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return pifa_fail_cuda("decode phase 1 launch", err);
  if (mr == 0) return PIFA_OK;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((mr + kRows - 1) / kRows);
  cfg.blockDim = dim3(W2 * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = cudaLaunchKernelEx(&cfg, decode_nonpivot_rows<NT, W2>, (const float*)yp, ldyp, T, r,
                           reinterpret_cast<const bf16*>(p.C), mr, (int64_t)s.ldc, p.nonpiv, m,
                           reinterpret_cast<bf16*>(p.Y), (int64_t)s.ldy, status);
  if (err != cudaSuccess) return pifa_fail_cuda("decode phase 2 launch", err);
  return PIFA_OK;
}

}  // namespace

int64_t decode_workspace_bytes(const PifaShape& s) {
  // y_p, fp32, T rows of pitch round_up(r, 8), rounded up to 256 bytes
  return ((s.T * ((s.r + 7) / 8 * 8) * 4 + 255) / 256) * 256;
}

int launch_decode(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream) {
  if (s.T <= 8) return launch_decode_t<1, 16, 8>(s, p, status, stream);
  return launch_decode_t<2, 8, 8>(s, p, status, stream);
}

// ---- allocation-free decode entry point -------------------------------------------------------
// For callers that cannot allocate device memory at all: for example an inference runtime that
// plans every device byte ahead of time and forbids libraries from calling cudaMalloc, or code
// running where an allocation would synchronize the device in the middle of a latency-critical
// decode loop. Such callers cannot provide the workspace pifa_forward asks for, so this entry
// point keeps the decode scratch (y_p, fp32, T rows of pitch round_up(r, 8)) in a fixed array in
// the library's static device data instead. The array exists once per GPU that loads the
// library and stays allocated until the process exits.
namespace {

constexpr int64_t kNoAllocScratchBytes = int64_t(1) << 20;  // 1 MiB: T * round_up(r, 8) * 4 bytes
__device__ __align__(256) unsigned char g_decode_scratch[kNoAllocScratchBytes];

constexpr int kNoAllocMaxDevices = 64;
void* g_decode_scratch_addr[kNoAllocMaxDevices] = {};
std::mutex g_decode_scratch_mu;

bool noalloc_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" int pifa_forward_decode_noalloc(const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp,
                                           int64_t r, int64_t ldwp, const void* C, int64_t m, int64_t ldc,
                                           const int32_t* pivot_idx, const int32_t* nonpivot_idx, void* Y,
                                           int64_t ldy, void* cuda_stream) {
  pifa_clear_error();
  if (T < 0 || m < 1 || n < 1 || r < 1 || r > m || r > n || m >= (int64_t(1) << 30) || n >= (int64_t(1) << 30))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "need T >= 0 and 1 <= r <= min(m, n) < 2^30");
  if (T == 0) return PIFA_OK;
  if (T > 16) return pifa_fail(PIFA_ERR_UNSUPPORTED, "pifa_forward_decode_noalloc needs T <= 16");
  const bool has_np = m > r;
  if (!X || !Wp || !pivot_idx || !Y || (has_np && (!C || !nonpivot_idx)))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "null X, Wp, C, pivot_idx, nonpivot_idx or Y");
  if (ldx < n || ldwp < n || ldy < m || (has_np && ldc < r))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row length");
  if (!noalloc_aligned16(X) || !noalloc_aligned16(Wp) || !noalloc_aligned16(Y) || (has_np && !noalloc_aligned16(C)))
    return pifa_fail(PIFA_ERR_ALIGNMENT, "X, Wp, C and Y must be 16-byte aligned");
  if ((ldx | ldwp | ldy | (has_np ? ldc : 0)) & 7)
    return pifa_fail(PIFA_ERR_ALIGNMENT, "ldx, ldwp, ldc and ldy must be multiples of 8 elements");
  const PifaShape s = {T, m, n, r, ldx, ldwp, has_np ? ldc : r, ldy};
  const int64_t need = decode_workspace_bytes(s);
  if (need > kNoAllocScratchBytes)
    return pifa_fail(PIFA_ERR_WORKSPACE,
                     "T * round_up(r, 8) * 4 bytes exceeds the 1 MiB static scratch of pifa_forward_decode_noalloc");

  // Set-up, once per device, with that device current: the device address of the static array.
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaGetDevice", e);
  if (dev < 0 || dev >= kNoAllocMaxDevices) return pifa_fail(PIFA_ERR_UNSUPPORTED, "device ordinal >= 64");
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_decode_scratch_mu);
    if (!g_decode_scratch_addr[dev]) {
      void* ptr = nullptr;
      e = cudaGetSymbolAddress(&ptr, g_decode_scratch);
      if (e != cudaSuccess) return pifa_fail_cuda("cudaGetSymbolAddress(decode scratch)", e);
      g_decode_scratch_addr[dev] = ptr;
    }
    scratch = g_decode_scratch_addr[dev];
  }
  int* status = pifa_status_word(&e);
  if (!status) return pifa_fail_cuda("device status word", e);
  // y_p is written in full by the first phase before the second reads it, so nothing in the
  // shared array has to start at zero.
  const PifaPointers p = {X, Wp, has_np ? C : nullptr, pivot_idx, has_np ? nonpivot_idx : nullptr, Y, scratch,
                          kNoAllocScratchBytes};
  return launch_decode(s, p, status, reinterpret_cast<cudaStream_t>(cuda_stream));
}
