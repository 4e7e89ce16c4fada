// decode.cu -- PIFA forward for small token counts (T <= 16): Algorithm 2 as two HBM-streaming
// GEMV phases.
//
//   phase 1: Y_p = X W_p^T   (r rows of W_p streamed once)   -> y_p fp32 in the workspace,
//            Y[:, I[j]] = bf16(Y_p[:, j])                     (Algorithm 2, steps 2 and 4)
//   phase 2: Y_np = Y_p C^T  (m - r rows of C streamed once)  -> Y[:, I^c[i]] = bf16(Y_np[:, i])
//                                                              (Algorithm 2, steps 3 and 5)
//
// The work is memory bound: every weight byte is read exactly once; x and y_p are tiny and stay in
// L1/L2. One CTA (16 warps) owns 16 consecutive weight rows (one m16 MMA fragment); its warps split
// the K dimension. For a 32-wide K step, lane (g = lane/4, c = lane%4) holds 8 consecutive elements
// of rows g and g+8 at offset 8c and uses them directly as the A fragments of two m16n8k16 MMAs,
// permuting K identically in both operands (a dot product does not depend on the order of its
// terms): MMA step s takes elements 4s..4s+3. The lane loads the matching 8 activations of token g
// as the B fragment. Warps then reduce their 16 x 8 partial tiles through shared memory.
//
// Both phases are launched with programmatic dependent launch (PDL) and start their weight traffic
// before waiting on the previous kernel: phase 1 bulk-prefetches its W_p rows into L2 and then
// streams them with 128-bit loads straight into registers; phase 2 -- launched while phase 1 still
// runs -- bulk-copies its rows of C into shared memory (rows 64 bytes apart beyond their length, so
// fragment loads hit eight different bank groups per quarter warp). Only after griddepcontrol.wait
// do they read X or y_p or write outputs. The next call's phase 1 likewise starts pulling its W_p
// while this call's phase 2 computes.
// y_p enters the second contraction as a hi + lo pair of C's storage type (bf16 or fp16): C has
// large entries and Y_np = C Y_p cancels, so rounding y_p to one bf16 alone would amplify its
// rounding error several-fold.
#include <mutex>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

constexpr int kRows = 16;       // weight rows per CTA
constexpr int kChunk = 32;      // K elements per warp step (two k16 MMAs)
constexpr int kRowPad = 64;     // bytes between consecutive rows of a stage beyond their length

__device__ __forceinline__ uint32_t pack2(uint16_t a, uint16_t b) { return (uint32_t)a | ((uint32_t)b << 16); }

// 8 consecutive bf16 of `row` starting at column k; zero beyond column K or for an invalid row.
// kStream: weights read exactly once, not allocated in L1.
// kCoherent: data another kernel may have just written (L2 only, never a stale L1 line).
template <bool kStream = false, bool kCoherent = false>
__device__ __forceinline__ uint4 load8_bf16(const bf16* __restrict__ base, int64_t ld, int64_t row, bool row_ok,
                                            int k, int K) {
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (!row_ok || k >= K) return v;
  const bf16* p = base + row * ld + k;
  if (k + 8 <= K) {
    if (kStream) return ld_stream_16(p);
    if (kCoherent) return __ldcg(reinterpret_cast<const uint4*>(p));
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

// 8 weights of one staged row at local column kl; elements at or beyond `len` are zeroed (the
// stage may hold stale bytes there, which must not reach the MMA even as NaN * 0).
__device__ __forceinline__ uint4 lds8_masked(const uint8_t* rowp, int kl, int len, bool row_ok) {
  if (!row_ok || kl >= len) return make_uint4(0u, 0u, 0u, 0u);
  uint4 v = *reinterpret_cast<const uint4*>(rowp + kl * 2);
  if (kl + 8 > len) {
    const int keep = len - kl;  // 1..7 valid elements
    uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e0 = 2 * i, e1 = 2 * i + 1;
      const uint32_t m0 = e0 < keep ? 0x0000FFFFu : 0u, m1 = e1 < keep ? 0xFFFF0000u : 0u;
      w[i] &= (m0 | m1);
    }
    v = make_uint4(w[0], w[1], w[2], w[3]);
  }
  return v;
}

// hi + lo split of an fp32 value in bf16 (kF16 = false) or fp16 (kF16 = true). fp16 saturates at
// +-65504 and reports the overflow through `range_err`.
template <bool kF16>
__device__ __forceinline__ void split2(float f, uint16_t& h, uint16_t& l, bool& range_err) {
  if (kF16) {
    if (fabsf(f) > 65504.0f) {
      range_err = true;
      f = copysignf(65504.0f, f);
    }
    const __half bh = __float2half_rn(f);
    h = __half_as_ushort(bh);
    l = __half_as_ushort(__float2half_rn(f - __half2float(bh)));
  } else {
    const bf16 bh = __float2bfloat16_rn(f);
    h = __bfloat16_as_ushort(bh);
    l = __bfloat16_as_ushort(__float2bfloat16_rn(f - __bfloat162float(bh)));
  }
}

// 8 consecutive fp32 y_p values of one token at column k (zero beyond K), split into hi and lo.
template <bool kF16>
__device__ __forceinline__ void load8_split(const float* __restrict__ yp, bool t_ok, int k, int K, uint4& hi,
                                            uint4& lo, bool& range_err) {
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
  for (int i = 0; i < 8; ++i) split2<kF16>(f[i], h[i], l[i], range_err);
  hi = make_uint4(pack2(h[0], h[1]), pack2(h[2], h[3]), pack2(h[4], h[5]), pack2(h[6], h[7]));
  lo = make_uint4(pack2(l[0], l[1]), pack2(l[2], l[3]), pack2(l[4], l[5]), pack2(l[6], l[7]));
}

// 8 consecutive fp32 y_p values of one token at column k from its staged row in shared memory
// (zero beyond K or for an absent token), split into hi and lo.
template <bool kF16>
__device__ __forceinline__ void lds8_split(const float* row, bool t_ok, int k, int K, uint4& hi, uint4& lo,
                                           bool& range_err) {
  float f[8];
  if (t_ok && k + 8 <= K) {
    const float4 a = *reinterpret_cast<const float4*>(row + k);
    const float4 b = *reinterpret_cast<const float4*>(row + k + 4);
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
    f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) f[i] = (t_ok && k + i < K) ? row[k + i] : 0.0f;
  }
  uint16_t h[8], l[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) split2<kF16>(f[i], h[i], l[i], range_err);
  hi = make_uint4(pack2(h[0], h[1]), pack2(h[2], h[3]), pack2(h[4], h[5]), pack2(h[6], h[7]));
  lo = make_uint4(pack2(l[0], l[1]), pack2(l[2], l[3]), pack2(l[4], l[5]), pack2(l[6], l[7]));
}

struct DecodeArgs {
  const uint16_t* A;     // weight rows (W_p for phase 1, C for phase 2), 2-byte elements
  int64_t lda;
  int R, K;              // rows and columns of A
  const bf16* X;         // phase 1: activations T x K
  int64_t ldx;
  float* yp;             // y_p, T rows of pitch ldyp (phase 1 writes it, phase 2 reads it)
  int64_t ldyp;
  const int32_t* cols;   // output column of each weight row (I or I^c)
  int m;
  bf16* Y;
  int64_t ldy;
  int T;
  int kc;                // phase 2: K columns per shared-memory stage (multiple of 32)
  int stages;            // phase 2: 1 (all of K resident) or 2
  int* status;
  uint64_t timeout_ns;
};

constexpr int kWarps = 16;                 // phase 1 warps per CTA
// Phase 2 runs 8 warps so that one of its CTAs fits in the registers an SM has left beside a
// phase-1 CTA: phase 2 can then launch (PDL) and pull its C rows while phase 1 still streams W_p.
constexpr int kWarps2 = 8;
template <int NT>
constexpr int kUnroll2 = 2;  // phase 2: 32-column steps in flight per warp
// phase 1: 32-column steps in flight per warp (fewer with two token tiles, to stay in 64 registers)
template <int NT>
constexpr int kUnroll1 = NT == 1 ? 4 : 2;

// Cross-warp reduction of the per-warp 16 x (8*NT) partial tiles, then the outputs of this CTA's
// 16 rows: y_p (phase 1 only) and the bf16 values in their output columns of Y.
template <int NT, int PHASE, int WARPS>
__device__ __forceinline__ void reduce_and_store(const DecodeArgs& a, float (*red)[kRows][8 * NT],
                                                 const float (&acc)[NT][4], int64_t row0, int nrows,
                                                 const int* s_cols) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    red[warp][g][nt * 8 + 2 * c] = acc[nt][0];
    red[warp][g][nt * 8 + 2 * c + 1] = acc[nt][1];
    red[warp][g + 8][nt * 8 + 2 * c] = acc[nt][2];
    red[warp][g + 8][nt * 8 + 2 * c + 1] = acc[nt][3];
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < kRows * 8 * NT; idx += WARPS * 32) {
    const int row = idx / (8 * NT), t = idx % (8 * NT);
    if (t >= a.T || row >= nrows) continue;
    float sum = 0.0f;
#pragma unroll
    for (int w = 0; w < WARPS; ++w) sum += red[w][row][t];
    const int64_t i = row0 + row;
    if (PHASE == 1) a.yp[(int64_t)t * a.ldyp + i] = sum;
    const int col = s_cols[row];
    if ((unsigned)col >= (unsigned)a.m) {
      latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
      continue;
    }
    a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(sum);
  }
}

// The output columns of this CTA's rows are layer constants: read them at launch, before waiting
// on the previous kernel, so no dependent global load is left for the end of the kernel.
__device__ __forceinline__ void load_cols(const DecodeArgs& a, int64_t row0, int nrows, int* s_cols) {
  if (threadIdx.x < kRows) s_cols[threadIdx.x] = threadIdx.x < nrows ? a.cols[row0 + threadIdx.x] : 0;
}

// ---- phase 1: Y_p = X W_p^T, streamed with 128-bit loads straight into MMA fragments ----------
template <int NT>
__global__ void __launch_bounds__(kWarps * 32) decode_pivot_rows(DecodeArgs a) {
  __shared__ float red[kWarps][kRows][8 * NT];
  __shared__ int s_cols[kRows];
  pdl_launch_dependents();  // phase 2 may launch now and start pulling its rows of C
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
  const int64_t row0 = (int64_t)blockIdx.x * kRows;
  const int nrows = (int)((int64_t)a.R - row0 < kRows ? (int64_t)a.R - row0 : kRows);
  if (threadIdx.x < nrows)  // start this CTA's W_p rows towards L2 before waiting on anything
    prefetch_l2_bulk(a.A + (row0 + threadIdx.x) * a.lda, ((uint32_t)a.K * 2u + 15u) & ~15u);
  load_cols(a, row0, nrows, s_cols);
  // One thread waits for the previous kernel (X valid, y_p and Y free) while the other warps park
  // in the CTA barrier: warps waiting on the previous grid would otherwise compete for issue slots
  // with the CTAs that are still working on this SM.
  if (threadIdx.x == 0) pdl_wait_primary();
  __syncthreads();
  const bf16* W = reinterpret_cast<const bf16*>(a.A);
  const bool ok0 = g < nrows, ok1 = g + 8 < nrows;
  // one accumulator per unrolled step: independent MMA chains instead of one long dependent one
  float accu[kUnroll1<NT>][NT][4];
#pragma unroll
  for (int u = 0; u < kUnroll1<NT>; ++u)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) accu[u][nt][0] = accu[u][nt][1] = accu[u][nt][2] = accu[u][nt][3] = 0.0f;
  const int nchunks = (a.K + kChunk - 1) / kChunk;
  for (int base = warp; base < nchunks; base += kWarps * kUnroll1<NT>) {
    uint4 wa[kUnroll1<NT>], wb[kUnroll1<NT>], xv[kUnroll1<NT>][NT];
#pragma unroll
    for (int u = 0; u < kUnroll1<NT>; ++u) {
      const int ch = base + u * kWarps;
      const int k = ch * kChunk + 8 * c;
      const bool in = ch < nchunks;
      wa[u] = load8_bf16<true>(W, a.lda, row0 + g, in && ok0, k, a.K);
      wb[u] = load8_bf16<true>(W, a.lda, row0 + g + 8, in && ok1, k, a.K);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int t = nt * 8 + g;
        xv[u][nt] = load8_bf16<false, true>(a.X, a.ldx, t, in && t < a.T, k, a.K);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll1<NT>; ++u) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        mma_m16n8k16_bf16(accu[u][nt], wa[u].x, wb[u].x, wa[u].y, wb[u].y, xv[u][nt].x, xv[u][nt].y);
        mma_m16n8k16_bf16(accu[u][nt], wa[u].z, wb[u].z, wa[u].w, wb[u].w, xv[u][nt].z, xv[u][nt].w);
      }
    }
  }
  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float v = 0.0f;
#pragma unroll
      for (int u = 0; u < kUnroll1<NT>; ++u) v += accu[u][nt][i];
      acc[nt][i] = v;
    }
  reduce_and_store<NT, 1, kWarps>(a, red, acc, row0, nrows, s_cols);
}

// ---- phase 2: Y_np = Y_p C^T from C rows staged in shared memory -------------------------------
// At launch (before waiting on phase 1) thread 0 bulk-copies the CTA's 16 rows of C into shared
// memory -- all of K when it fits, else K-chunks through two stages refilled after each is used.
template <int NT, bool kF16C, bool kYs>
__global__ void __launch_bounds__(kWarps2 * 32) decode_nonpivot_rows(DecodeArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t pitch = (uint32_t)(a.kc * 2 + kRowPad);
  const uint32_t stage_bytes = (uint32_t)kRows * pitch;
  // y_p staged in shared memory: T rows of ldyp floats, 16 bytes apart beyond their length so that
  // the two float4 loads of a quarter warp fall into distinct bank groups
  const uint32_t ypitch = (uint32_t)a.ldyp * 4u + 16u;
  float* ys = reinterpret_cast<float*>(smem + a.stages * stage_bytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + a.stages * stage_bytes + (kYs ? (uint32_t)a.T * ypitch : 0u));
  uint64_t* ybar = full + 2;
  float(*red)[kRows][8 * NT] = reinterpret_cast<float(*)[kRows][8 * NT]>(full + 3);
  __shared__ int s_cols[kRows];
  pdl_launch_dependents();  // the next call's phase 1 may launch and prefetch its W_p
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
  const int64_t row0 = (int64_t)blockIdx.x * kRows;
  const int nrows = (int)((int64_t)a.R - row0 < kRows ? (int64_t)a.R - row0 : kRows);
  const int nchunks = (a.K + a.kc - 1) / a.kc;
  auto issue = [&](int j) {  // thread 0: chunk j into stage j % stages
    const int s = j % a.stages;
    const int len = min(a.kc, a.K - j * a.kc);
    const uint32_t bytes = (uint32_t)((len + 7) & ~7) * 2u;  // stays inside the 16-byte row pitch
    mbar_arrive_expect_tx(&full[s], bytes * (uint32_t)nrows);
    uint8_t* st = smem + s * stage_bytes;
    for (int rr = 0; rr < nrows; ++rr)
      bulk_copy_g2s(smem_u32(st + rr * pitch), a.A + (row0 + rr) * a.lda + (int64_t)j * a.kc, bytes, &full[s]);
  };
  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) mbar_init(&full[s], 1);
    mbar_init(ybar, 1);
    fence_mbar_init();
    for (int j = 0; j < a.stages && j < nchunks; ++j) issue(j);
  }
  load_cols(a, row0, nrows, s_cols);
  if (threadIdx.x == 0) pdl_wait_primary();  // phase 1 has completed: y_p is valid (see phase 1)
  if (kYs && threadIdx.x == 0) {  // all of y_p into shared memory in T bulk copies
    const uint32_t ybytes = (uint32_t)a.ldyp * 4u;
    mbar_arrive_expect_tx(ybar, ybytes * (uint32_t)a.T);
    for (int t = 0; t < a.T; ++t)
      bulk_copy_g2s(smem_u32(reinterpret_cast<uint8_t*>(ys) + t * ypitch), a.yp + (int64_t)t * a.ldyp, ybytes, ybar);
  }
  __syncthreads();  // barriers initialised before anyone waits on them
  const bool ok0 = g < nrows, ok1 = g + 8 < nrows;
  bool range_err = false, dead = false;
  // separate accumulators per unrolled step and per hi / lo pass: short independent MMA chains
  float accu[kUnroll2<NT>][2][NT][4];
#pragma unroll
  for (int u = 0; u < kUnroll2<NT>; ++u)
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) accu[u][h][nt][0] = accu[u][h][nt][1] = accu[u][h][nt][2] = accu[u][h][nt][3] = 0.0f;
  if (kYs && !mbar_wait(ybar, 0, a.timeout_ns)) {
    latch_status(a.status, PIFA_ERR_TIMEOUT);
    dead = true;
  }
  for (int j = 0; j < nchunks; ++j) {
    const int s = j % a.stages;
    const int len = min(a.kc, a.K - j * a.kc);
    const int steps = (len + kChunk - 1) / kChunk;
    if (!mbar_wait(&full[s], (uint32_t)(j / a.stages) & 1u, a.timeout_ns)) {
      latch_status(a.status, PIFA_ERR_TIMEOUT);
      dead = true;
    }
    if (!dead) {
      const uint8_t* st = smem + s * stage_bytes;
      for (int base = warp; base < steps; base += kWarps2 * kUnroll2<NT>) {
        uint4 hi[kUnroll2<NT>][NT], lo[kUnroll2<NT>][NT], wa[kUnroll2<NT>], wb[kUnroll2<NT>];
#pragma unroll
        for (int u = 0; u < kUnroll2<NT>; ++u) {  // several steps' y_p loads in flight together
          const int stp = base + u * kWarps2;
          const int kl = stp * kChunk + 8 * c;
          const bool in = stp < steps;
          wa[u] = lds8_masked(st + g * pitch, kl, len, in && ok0);
          wb[u] = lds8_masked(st + (g + 8) * pitch, kl, len, in && ok1);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int t = nt * 8 + g;
            if (kYs)
              lds8_split<kF16C>(reinterpret_cast<const float*>(reinterpret_cast<const uint8_t*>(ys) +
                                                              (t < a.T ? t : 0) * ypitch),
                                in && t < a.T, j * a.kc + kl, a.K, hi[u][nt], lo[u][nt], range_err);
            else
              load8_split<kF16C>(a.yp + (int64_t)(t < a.T ? t : 0) * a.ldyp, in && t < a.T, j * a.kc + kl, a.K,
                                 hi[u][nt], lo[u][nt], range_err);
          }
        }
#pragma unroll
        for (int u = 0; u < kUnroll2<NT>; ++u) {
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            if (kF16C) {
              mma_m16n8k16_f16(accu[u][0][nt], wa[u].x, wb[u].x, wa[u].y, wb[u].y, hi[u][nt].x, hi[u][nt].y);
              mma_m16n8k16_f16(accu[u][1][nt], wa[u].x, wb[u].x, wa[u].y, wb[u].y, lo[u][nt].x, lo[u][nt].y);
              mma_m16n8k16_f16(accu[u][0][nt], wa[u].z, wb[u].z, wa[u].w, wb[u].w, hi[u][nt].z, hi[u][nt].w);
              mma_m16n8k16_f16(accu[u][1][nt], wa[u].z, wb[u].z, wa[u].w, wb[u].w, lo[u][nt].z, lo[u][nt].w);
            } else {
              mma_m16n8k16_bf16(accu[u][0][nt], wa[u].x, wb[u].x, wa[u].y, wb[u].y, hi[u][nt].x, hi[u][nt].y);
              mma_m16n8k16_bf16(accu[u][1][nt], wa[u].x, wb[u].x, wa[u].y, wb[u].y, lo[u][nt].x, lo[u][nt].y);
              mma_m16n8k16_bf16(accu[u][0][nt], wa[u].z, wb[u].z, wa[u].w, wb[u].w, hi[u][nt].z, hi[u][nt].w);
              mma_m16n8k16_bf16(accu[u][1][nt], wa[u].z, wb[u].z, wa[u].w, wb[u].w, lo[u][nt].z, lo[u][nt].w);
            }
          }
        }
      }
    }
    if (j + a.stages < nchunks) {  // refill stage s once every warp is done with it
      __syncthreads();
      if (threadIdx.x == 0 && !dead) issue(j + a.stages);
    }
  }
  if (threadIdx.x == 0) {
    // nothing may still be landing in shared memory when the CTA exits
    for (int j = nchunks > a.stages ? nchunks - a.stages : 0; j < nchunks; ++j)
      if (!mbar_wait(&full[j % a.stages], (uint32_t)(j / a.stages) & 1u, 100000000ull))
        latch_status(a.status, PIFA_ERR_TIMEOUT);
    if (kYs && !mbar_wait(ybar, 0, 100000000ull)) latch_status(a.status, PIFA_ERR_TIMEOUT);
  }
  if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float v = 0.0f;
#pragma unroll
      for (int u = 0; u < kUnroll2<NT>; ++u) v += accu[u][0][nt][i] + accu[u][1][nt][i];
      acc[nt][i] = v;
    }
  reduce_and_store<NT, 2, kWarps2>(a, red, acc, row0, nrows, s_cols);
}

template <typename Kern>
int launch_pdl(Kern kernel, unsigned grid, unsigned threads, size_t smem, cudaStream_t stream,
               const DecodeArgs& args, const char* what) {
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return pifa_fail_cuda(what, e);
  }

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args);
  if (e != cudaSuccess) return pifa_fail_cuda(what, e);
  return PIFA_OK;
}

template <int NT>
int launch_decode_t(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream) {
  DecodeArgs a = {};
  a.A = reinterpret_cast<const uint16_t*>(p.Wp);
  a.lda = s.ldwp;
  a.R = (int)s.r;
  a.K = (int)s.n;
  a.X = reinterpret_cast<const bf16*>(p.X);
  a.ldx = s.ldx;
  a.yp = reinterpret_cast<float*>(p.ws);
  a.ldyp = (s.r + 7) / 8 * 8;  // 32-byte row pitch keeps the 16-byte loads aligned
  a.cols = p.piv;
  a.m = (int)s.m;
  a.Y = reinterpret_cast<bf16*>(p.Y);
  a.ldy = s.ldy;
  a.T = (int)s.T;
  a.status = status;
  a.timeout_ns = pifa_wait_timeout_ns();
  int st = launch_pdl(decode_pivot_rows<NT>, (unsigned)((s.r + kRows - 1) / kRows), kWarps * 32, 0, stream, a,
                      "decode phase 1 launch");
  if (st != PIFA_OK || s.m == s.r) return st;
  DecodeArgs b = a;
  b.A = reinterpret_cast<const uint16_t*>(p.C);
  b.lda = s.ldc;
  b.R = (int)(s.m - s.r);
  b.K = (int)s.r;
  b.X = nullptr;
  b.cols = p.nonpiv;
  // Shared memory: C all of K in one stage and y_p staged whole when both fit in ~190 KB; else C
  // alone in one stage (y_p read from L2); else C in 2048-column chunks through 2 stages.
  const size_t ys_bytes = (size_t)s.T * (size_t)(b.ldyp * 4 + 16);
  const size_t tail = 32 + (size_t)kWarps2 * kRows * 8 * NT * 4;
  const int kc_all = (b.K + kChunk - 1) / kChunk * kChunk;
  const size_t c_all = (size_t)kRows * (kc_all * 2 + kRowPad);
  bool ys = false;
  if (c_all + ys_bytes + tail <= 190 * 1024) {
    b.kc = kc_all;
    b.stages = 1;
    ys = true;
  } else if (c_all + tail <= 190 * 1024) {
    b.kc = kc_all;
    b.stages = 1;
  } else {
    b.kc = 2048;
    b.stages = 2;
  }
  const size_t smem = (size_t)b.stages * kRows * (b.kc * 2 + kRowPad) + (ys ? ys_bytes : 0) + tail;
  const unsigned grid2 = (unsigned)((s.m - s.r + kRows - 1) / kRows);
  const bool f16 = s.c_dtype == PIFA_DTYPE_FP16;
  const unsigned th = kWarps2 * 32;
  const char* what = "decode phase 2 launch";
  if (f16 && ys) return launch_pdl(decode_nonpivot_rows<NT, true, true>, grid2, th, smem, stream, b, what);
  if (f16) return launch_pdl(decode_nonpivot_rows<NT, true, false>, grid2, th, smem, stream, b, what);
  if (ys) return launch_pdl(decode_nonpivot_rows<NT, false, true>, grid2, th, smem, stream, b, what);
  return launch_pdl(decode_nonpivot_rows<NT, false, false>, grid2, th, smem, stream, b, what);
}

}  // namespace

int64_t decode_workspace_bytes(const PifaShape& s) {
  // y_p, fp32, T rows of pitch round_up(r, 8), rounded up to 256 bytes
  return ((s.T * ((s.r + 7) / 8 * 8) * 4 + 255) / 256) * 256;
}

int launch_decode(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream) {
  if (s.T <= 8) return launch_decode_t<1>(s, p, status, stream);
  return launch_decode_t<2>(s, p, status, stream);
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

constexpr int64_t kNoAllocScratchBytes = int64_t(1) << 20;  // 1 MiB: 256 + T * round_up(r, 8) * 4 bytes
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
  const PifaShape s = {T, m, n, r, ldx, ldwp, has_np ? ldc : r, ldy, PIFA_DTYPE_BF16};
  const int64_t need = kWorkspaceReserve + decode_workspace_bytes(s);
  if (need > kNoAllocScratchBytes)
    return pifa_fail(PIFA_ERR_WORKSPACE,
                     "256 + T * round_up(r, 8) * 4 bytes exceeds the 1 MiB static scratch of "
                     "pifa_forward_decode_noalloc");

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
  // The array starts zeroed (static device data). Its first kWorkspaceReserve bytes hold the
  // decode kernel's grid-barrier words, which every completed call leaves at zero; y_p after them
  // is written in full before it is read.
  const PifaPointers p = {X,
                          Wp,
                          has_np ? C : nullptr,
                          pivot_idx,
                          has_np ? nonpivot_idx : nullptr,
                          Y,
                          static_cast<uint8_t*>(scratch) + kWorkspaceReserve,
                          kNoAllocScratchBytes - kWorkspaceReserve,
                          static_cast<unsigned*>(scratch)};
  return launch_decode(s, p, status, reinterpret_cast<cudaStream_t>(cuda_stream));
}
