// backward.cu -- the gradients of a PIFA layer (fine-tuning after compression, Sec. 5.1; the layer
// is differentiable, Sec. 6) and the online accumulators of the M reconstruction (Sec. 4; the
// accumulation steps of Algorithm 3), as tensor-core contractions (gemm_tc.cu) plus a column split.
//
// Backward, tokens as rows (Y = X W'^T, Y_p = X W_p^T, Y_np = Y_p C^T), given dY = dL/dY:
//   dY_I = dY[:, I], dY_np = dY[:, I^c]      one pass over dY       (Algorithm 2, steps 4-5, reversed)
//   dY_p  = dY_I + dY_np C                   T x r,  K = m - r      (steps 4 and 3, reversed)
//   dX    = dY_p W_p                         T x n,  K = r          (step 2, reversed)
// dY_p and Y_p are kept as hi + lo pairs of bf16 planes: in exact arithmetic dX = dY W', and the
// route through dY_p (amplified by C, then contracted with W_p) would otherwise lose the bits that
// cancel -- the same effect that makes the forward pass carry Y_p as hi + lo; dW_p and dC show it
// in their small entries.
//   dW_p  = dY_p^T X                         r x n,  K = T
//   dC    = dY_np^T Y_p,  Y_p = X W_p^T      (m - r) x r,  K = T    (step 3, reversed)
// M accumulators for one calibration batch (X_o the dense data flow, X_u the low-rank one):
//   Y_t  = (lambda X_o + (1 - lambda) X_u) W^T          T x m   (the mixed target, Eq. 6)
// The mixed input and Y_t are carried as hi + lo bf16 pairs: each feeds a contraction whose sums
// cancel, and a single bf16 rounding of them shows in Y_t X^T's small entries.
//   XXt += X_u^T X_u                                    n x n   (x x^T summed over the batch)
//   YtXt += Y_t^T X_u                                   m x n   (Y_t X^T summed over the batch)
#include <cuda_bf16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

int64_t pad8(int64_t v) { return (v + 7) / 8 * 8; }
int64_t a256(int64_t b) { return (b + 255) / 256 * 256; }

// dY's columns split into its pivot and non-pivot parts (bf16): outp[t][j] = in[t][piv[j]] for
// j < r and outnp[t][i] = in[t][nonpiv[i]] for i < nnp; an index outside [0, bound) writes 0 and
// latches PIFA_ERR_DEVICE_INDEX. A thread owns one output column (its index read once, the lanes
// of a warp on consecutive columns) and walks the rows of its y-block's share, so that the loads of
// consecutive rows are independent and many are in flight.
__global__ void split_cols(const bf16* in, int64_t ldin, const int32_t* piv, int r, const int32_t* nonpiv, int nnp,
                           int bound, int T, bf16* outp, int64_t ldp, bf16* outnp, int64_t ldnp, int* status) {
  pdl_launch_dependents();
  pdl_wait_primary();
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= r + nnp) return;
  const bool pv = j < r;
  const int c = __ldg(pv ? piv + j : nonpiv + (j - r));
  bf16* out = pv ? outp + j : outnp + (j - r);
  const int64_t ldo = pv ? ldp : ldnp;
  const bool ok = (unsigned)c < (unsigned)bound;
  if (!ok) latch_status(status, PIFA_ERR_DEVICE_INDEX);
  const bf16 zero = __float2bfloat16_rn(0.0f);
#pragma unroll 8
  for (int t = blockIdx.y; t < T; t += gridDim.y) out[(int64_t)t * ldo] = ok ? in[(int64_t)t * ldin + c] : zero;
}

// out = a * x + b * y elementwise over T rows of n (bf16 in, fp32 arithmetic), written as a hi +
// lo pair of bf16 planes. A thread owns 8 consecutive columns of a row (16-byte loads and stores:
// every pitch is a multiple of 8 elements and every base 16-byte aligned), scalar at a ragged end.
// Rows across the y grid, column groups across x.
__global__ void axpby_rows(const bf16* x, const bf16* y, int64_t ld, int T, int n, float a, float b, bf16* out,
                           bf16* out_lo, int64_t ldout) {
  pdl_launch_dependents();
  pdl_wait_primary();
  const int ng = (n + 7) / 8;
  for (int t = blockIdx.y; t < T; t += gridDim.y)
    for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < ng; g += gridDim.x * blockDim.x) {
      const int c = 8 * g;
      const bf16* xr = x + (int64_t)t * ld + c;
      const bf16* yr = y + (int64_t)t * ld + c;
      bf16* hr = out + (int64_t)t * ldout + c;
      bf16* lr = out_lo + (int64_t)t * ldout + c;
      if (c + 8 <= n) {
        uint4 xv = *reinterpret_cast<const uint4*>(xr), yv = *reinterpret_cast<const uint4*>(yr), hv, lv;
        const bf16* xe = reinterpret_cast<const bf16*>(&xv);
        const bf16* ye = reinterpret_cast<const bf16*>(&yv);
        bf16* he = reinterpret_cast<bf16*>(&hv);
        bf16* le = reinterpret_cast<bf16*>(&lv);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float v = a * __bfloat162float(xe[e]) + b * __bfloat162float(ye[e]);
          he[e] = __float2bfloat16_rn(v);
          le[e] = __float2bfloat16_rn(v - __bfloat162float(he[e]));
        }
        *reinterpret_cast<uint4*>(hr) = hv;
        *reinterpret_cast<uint4*>(lr) = lv;
      } else {
        for (int e = 0; c + e < n; ++e) {
          const float v = a * __bfloat162float(xr[e]) + b * __bfloat162float(yr[e]);
          const bf16 h = __float2bfloat16_rn(v);
          hr[e] = h;
          lr[e] = __float2bfloat16_rn(v - __bfloat162float(h));
        }
      }
    }
}

// out (cols x rows) = in (rows x cols)^T, bf16, through 64 x 64 shared-memory tiles: each thread
// loads 8 consecutive elements of an input row and stores 8 consecutive elements of an output row
// (16-byte accesses: both pitches are multiples of 8 elements and both bases 16-byte aligned;
// scalar at ragged edges). The tile's 8-element groups are stored XOR-swizzled by the row's group
// (group g of row k at g ^ (k / 8 % 8)), so that the column reads of 8 rows 8 apart hit 8 different
// banks. Block (8, 32); grid (ceil(cols / 64), ceil(rows / 64)).
__global__ void transpose_bf16(const bf16* in, int64_t ldin, int rows, int cols, bf16* out, int64_t ldout) {
  __shared__ __align__(16) bf16 t[64][64];
  pdl_launch_dependents();
  pdl_wait_primary();
  const int c0 = blockIdx.x * 64, r0 = blockIdx.y * 64;
  const int tx = threadIdx.x, ty = threadIdx.y;  // 8 x 32
  for (int k = ty; k < 64; k += 32) {  // input row r0 + k, columns c0 + 8 tx .. + 7
    const int r = r0 + k, c = c0 + 8 * tx;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (r < rows && c + 8 <= cols) {
      v = *reinterpret_cast<const uint4*>(in + (int64_t)r * ldin + c);
    } else if (r < rows) {
      bf16* ve = reinterpret_cast<bf16*>(&v);
      for (int e = 0; e < 8 && c + e < cols; ++e) ve[e] = in[(int64_t)r * ldin + c + e];
    }
    *reinterpret_cast<uint4*>(&t[k][8 * (tx ^ ((k >> 3) & 7))]) = v;
  }
  __syncthreads();
  for (int k = ty; k < 64; k += 32) {  // output row c0 + k (input column), rows r0 + 8 tx .. + 7
    const int c = c0 + k, r = r0 + 8 * tx;
    if (c >= cols) continue;
    uint4 v;
    bf16* ve = reinterpret_cast<bf16*>(&v);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int kr = 8 * tx + e;  // tile row; its group (k >> 3) sits at (k >> 3) ^ tx
      ve[e] = t[kr][8 * ((k >> 3) ^ ((kr >> 3) & 7)) + (k & 7)];
    }
    if (r + 8 <= rows) {
      *reinterpret_cast<uint4*>(out + (int64_t)c * ldout + r) = v;
    } else {
      for (int e = 0; r + e < rows; ++e) out[(int64_t)c * ldout + r + e] = ve[e];
    }
  }
}

// A row-wise elementwise kernel over `rows` rows of `cols` columns: rows on the y grid (at most
// 65535, the kernel loops beyond), columns on x.
int launch_small(const void* fn, void** args, int64_t rows, int64_t cols, cudaStream_t stream, const char* what) {
  cudaLaunchConfig_t cfg = {};
  const int64_t bx = (cols + 255) / 256;
  cfg.gridDim = dim3((unsigned)(bx < 8 ? (bx > 0 ? bx : 1) : 8), (unsigned)(rows < 65535 ? (rows > 0 ? rows : 1) : 65535));
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelExC(&cfg, fn, args);
  if (e == cudaSuccess) pifa_count_launch();
  return e == cudaSuccess ? PIFA_OK : pifa_fail_cuda(what, e);
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct BwdLayout {
  int64_t dynp, dyi, yp, yp_lo, dyp, dyp_lo, total;
};

BwdLayout bwd_layout(int64_t T, int64_t m, int64_t r) {
  BwdLayout L;
  int64_t o = 0;
  L.dynp = o;
  o += a256(T * pad8(m - r > 0 ? m - r : 1) * 2);
  L.dyi = o;
  o += a256(T * pad8(r) * 2);
  L.yp = o;
  o += a256(T * pad8(r) * 2);
  L.yp_lo = o;
  o += a256(T * pad8(r) * 2);
  L.dyp = o;
  o += a256(T * pad8(r) * 2);
  L.dyp_lo = o;
  o += a256(T * pad8(r) * 2);
  L.total = o;
  return L;
}

struct MaccLayout {
  int64_t xut, xmix, xmix_lo, ytt, ytt_lo, total;
};

// X_u^T (n x pad8(T)), the mixed input's hi and lo planes (T x pad8(n)), Y_t^T's hi and lo planes
// (m x pad8(T)), all bf16
MaccLayout macc_layout(int64_t T, int64_t m, int64_t n) {
  MaccLayout L;
  int64_t o = 0;
  L.xut = o;
  o += a256(n * pad8(T) * 2);
  L.xmix = o;
  o += a256(T * pad8(n) * 2);
  L.xmix_lo = o;
  o += a256(T * pad8(n) * 2);
  L.ytt = o;
  o += a256(m * pad8(T) * 2);
  L.ytt_lo = o;
  o += a256(m * pad8(T) * 2);
  L.total = o;
  return L;
}

}  // namespace

extern "C" int64_t pifa_backward_workspace_size(int64_t T, int64_t m, int64_t n, int64_t r) {
  pifa_clear_error();
  if (T < 0 || m < 1 || n < 1 || r < 1 || r > m || r > n) return pifa_fail(PIFA_ERR_INVALID_ARG, "need T >= 0 and 1 <= r <= min(m, n)");
  return bwd_layout(T, m, r).total;
}

extern "C" int pifa_backward(const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp, int64_t r, int64_t ldwp,
                             const void* C, int64_t m, int64_t ldc, const int32_t* pivot_idx,
                             const int32_t* nonpivot_idx, const void* dY, int64_t lddy, void* dX, int64_t lddx,
                             float* dWp, int64_t lddwp, float* dC, int64_t lddc, void* workspace,
                             int64_t workspace_bytes, void* cuda_stream) {
  pifa_clear_error();
  if (T < 0 || m < 1 || n < 1 || r < 1 || r > m || r > n || T >= (1 << 30) || m >= (1 << 30) || n >= (1 << 30))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "need T >= 0 and 1 <= r <= min(m, n) < 2^30");
  const bool has_np = m > r;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(cuda_stream);
  if (!Wp || !pivot_idx || (has_np && (!C || !nonpivot_idx)))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "null Wp, C, pivot_idx or nonpivot_idx");
  if (ldwp < n || (has_np && ldc < r)) return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row");
  if ((dX && lddx < n) || (dWp && lddwp < n) || (dC && lddc < r))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "output leading dimension smaller than the row");
  if (T == 0) {  // no tokens: zero weight gradients
    cudaError_t e = cudaSuccess;
    if (dWp) e = cudaMemset2DAsync(dWp, lddwp * 4, 0, n * 4, r, s);
    if (e == cudaSuccess && dC && has_np) e = cudaMemset2DAsync(dC, lddc * 4, 0, r * 4, m - r, s);
    return e == cudaSuccess ? PIFA_OK : pifa_fail_cuda("backward: zero gradients", e);
  }
  if (!X || !dY) return pifa_fail(PIFA_ERR_INVALID_ARG, "null X or dY");
  if (ldx < n || lddy < m) return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row");
  if (!al16(X) || !al16(Wp) || !al16(dY) || (has_np && !al16(C)) || (dX && !al16(dX)) || (dWp && !al16(dWp)) ||
      (dC && !al16(dC)) || ((ldx | ldwp | lddy | (has_np ? ldc : 0) | (dX ? lddx : 0)) & 7) ||
      ((dWp ? lddwp : 0) & 3) || ((dC ? lddc : 0) & 3))
    return pifa_fail(PIFA_ERR_ALIGNMENT, "16-byte aligned buffers and 16-byte row pitches required");
  const BwdLayout Ly = bwd_layout(T, m, r);
  if (!workspace || workspace_bytes < Ly.total) return pifa_fail(PIFA_ERR_WORKSPACE, "workspace missing or too small");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return pifa_fail(PIFA_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  cudaError_t ce = cudaSuccess;
  int* status = pifa_status_word(&ce);
  if (!status) return pifa_fail_cuda("device status word", ce);
  const uint64_t tmo = pifa_wait_timeout_ns();
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  bf16* dYnp = reinterpret_cast<bf16*>(ws + Ly.dynp);
  bf16* Yp = reinterpret_cast<bf16*>(ws + Ly.yp);
  bf16* Yp_lo = reinterpret_cast<bf16*>(ws + Ly.yp_lo);
  bf16* dYp = reinterpret_cast<bf16*>(ws + Ly.dyp);
  bf16* dYp_lo = reinterpret_cast<bf16*>(ws + Ly.dyp_lo);
  const int64_t ldnp = pad8(m - r > 0 ? m - r : 1), ldr = pad8(r);
  int st;
  bf16* dYi = reinterpret_cast<bf16*>(ws + Ly.dyi);
  {  // dY_I = dY[:, I] and dY_np = dY[:, I^c] in one pass over dY (dY_I straight into dY_p when r = m)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((m + 255) / 256), (unsigned)(T < 64 ? T : 64));
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    const cudaError_t e = pifa_launch_ex(&cfg, split_cols, reinterpret_cast<const bf16*>(dY), lddy, pivot_idx, (int)r,
                                         nonpivot_idx, (int)(m - r), (int)m, (int)T, has_np ? dYi : dYp, ldr, dYnp,
                                         ldnp, status);
    if (e != cudaSuccess) return pifa_fail_cuda("backward: split dY", e);
  }
  // Independent products run concurrently: Y_p and then dC on side stream 0 (after the split),
  // dY_p and then dX on the caller's stream, dW_p on side stream 1 once dY_p is done. Each product
  // alone fills one or two waves of the GPU; together they keep it busy (the side streams rejoin
  // the caller's stream before this call returns, also on failure).
  PifaSides sides(s);
  cudaStream_t s_yp = s, s_dw = s;
  // Y_p = X W_p^T as hi + lo planes (only dC needs it)
  if (dC && has_np) {
    if ((st = sides.fork(0, &s_yp)) != PIFA_OK) return st;
    GemmTc g = {T, r, n, X, ldx, false, Wp, ldwp, false, Yp, ldr, 3, 1.0f, nullptr, nullptr, 0, 0};
    g.D2 = Yp_lo;
    if ((st = gemm_tc(g, status, tmo, s_yp)) != PIFA_OK) return st;
  }
  // dY_p = dY_I + dY_np C, as hi + lo planes (dY_p = dY_I when r = m)
  if (has_np) {
    GemmTc g = {T, r, m - r, dYnp, ldnp, false, C, ldc, true, dYp, ldr, 3, 1.0f, dYi, nullptr, ldr, r};
    g.D2 = dYp_lo;
    if ((st = gemm_tc(g, status, tmo, s)) != PIFA_OK) return st;
  }
  if (dWp) {  // dW_p = (dY_p,hi + dY_p,lo)^T X
    if ((st = sides.fork(1, &s_dw)) != PIFA_OK) return st;
    GemmTc g = {r, n, T, dYp, ldr, true, X, ldx, true, dWp, lddwp, 1, 1.0f, nullptr, nullptr, 0, 0};
    if (has_np) g.A2 = dYp_lo;
    if ((st = gemm_tc(g, status, tmo, s_dw)) != PIFA_OK) return st;
  }
  if (dX) {  // dX = (dY_p,hi + dY_p,lo) W_p  (dY_p exact in bf16 when r == m)
    GemmTc g = {T, n, r, dYp, ldr, false, Wp, ldwp, true, dX, lddx, 0, 1.0f, nullptr, nullptr, 0, 0};
    if (has_np) g.A2 = dYp_lo;
    if ((st = gemm_tc(g, status, tmo, s)) != PIFA_OK) return st;
  }
  if (dC && has_np) {  // dC = dY_np^T (Y_p,hi + Y_p,lo), after Y_p on its side stream
    GemmTc g = {m - r, r, T, dYnp, ldnp, true, Yp, ldr, true, dC, lddc, 1, 1.0f, nullptr, nullptr, 0, 0};
    g.B2 = Yp_lo;
    if ((st = gemm_tc(g, status, tmo, s_yp)) != PIFA_OK) return st;
  }
  return PIFA_OK;
}

extern "C" int64_t pifa_m_accumulate_workspace_size(int64_t T, int64_t m, int64_t n) {
  pifa_clear_error();
  if (T < 0 || m < 1 || n < 1) return pifa_fail(PIFA_ERR_INVALID_ARG, "need T >= 0, m >= 1, n >= 1");
  return macc_layout(T, m, n).total;
}

extern "C" int pifa_m_accumulate(const void* Xo, const void* Xu, int64_t T, int64_t n, int64_t ldx, const void* W,
                                 int64_t m, int64_t ldw, float lambda, float* XXt, int64_t ldxx, float* YtXt,
                                 int64_t ldyx, void* workspace, int64_t workspace_bytes, void* cuda_stream) {
  pifa_clear_error();
  if (T < 0 || m < 1 || n < 1 || T >= (1 << 30) || m >= (1 << 30) || n >= (1 << 30))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "need T >= 0 and 1 <= m, n < 2^30");
  if (!(lambda >= 0.0f && lambda <= 1.0f)) return pifa_fail(PIFA_ERR_INVALID_ARG, "lambda must be in [0, 1]");
  if (T == 0) return PIFA_OK;  // nothing to accumulate
  if (!Xu || !XXt || (YtXt && (!W || !Xo))) return pifa_fail(PIFA_ERR_INVALID_ARG, "null Xu, XXt, or W / Xo with YtXt");
  if (ldx < n || ldxx < n || (YtXt && (ldw < n || ldyx < n)))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row");
  if (!al16(Xu) || !al16(XXt) || (YtXt && (!al16(Xo) || !al16(W) || !al16(YtXt))) || (ldx & 7) || (ldxx & 3) ||
      (YtXt && ((ldw & 7) || (ldyx & 3))))
    return pifa_fail(PIFA_ERR_ALIGNMENT, "16-byte aligned buffers and 16-byte row pitches required");
  const MaccLayout Ly = macc_layout(T, m, n);
  if (!workspace || workspace_bytes < Ly.total) return pifa_fail(PIFA_ERR_WORKSPACE, "workspace missing or too small");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return pifa_fail(PIFA_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  cudaError_t ce = cudaSuccess;
  int* status = pifa_status_word(&ce);
  if (!status) return pifa_fail_cuda("device status word", ce);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(cuda_stream);
  const uint64_t tmo = pifa_wait_timeout_ns();
  int st;
  // Every product runs with both operands K-major (measured twice as fast as the transposed forms):
  // X_u^T is formed once, and Y_t^T comes out of W X_mix^T directly.
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  bf16* XuT = reinterpret_cast<bf16*>(ws + Ly.xut);
  const int64_t ldT = pad8(T), ldn = pad8(n);
  {  // X_u^T
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((n + 63) / 64), (unsigned)((T + 63) / 64));
    cfg.blockDim = dim3(8, 32);
    cfg.stream = s;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    const cudaError_t e = pifa_launch_ex(&cfg, transpose_bf16, reinterpret_cast<const bf16*>(Xu), ldx, (int)T,
                                             (int)n, XuT, ldT);
    if (e != cudaSuccess) return pifa_fail_cuda("m_accumulate: transpose", e);
  }
  // X X^T on the caller's stream and, concurrently, the mix, Y_t^T and Y_t X^T on a side stream
  // (both read X_u^T; the side stream rejoins before this call returns, also on failure)
  PifaSides sides(s);
  if (YtXt) {
    cudaStream_t s2 = s;
    if ((st = sides.fork(0, &s2)) != PIFA_OK) return st;
    bf16* Xmix = reinterpret_cast<bf16*>(ws + Ly.xmix);
    bf16* Xmix_lo = reinterpret_cast<bf16*>(ws + Ly.xmix_lo);
    bf16* YtT = reinterpret_cast<bf16*>(ws + Ly.ytt);
    bf16* YtT_lo = reinterpret_cast<bf16*>(ws + Ly.ytt_lo);
    {  // X_mix = lambda X_o + (1 - lambda) X_u, as hi + lo planes
      int Ti = (int)T, ni = (int)n;
      float a = lambda, b = 1.0f - lambda;
      void* args[] = {(void*)&Xo, (void*)&Xu, (void*)&ldx, (void*)&Ti, (void*)&ni, (void*)&a, (void*)&b, (void*)&Xmix,
                      (void*)&Xmix_lo, (void*)&ldn};
      if ((st = launch_small((const void*)axpby_rows, args, T, (n + 7) / 8, s2, "m_accumulate: mix")) != PIFA_OK)
        return st;
    }
    {  // Y_t^T = W (X_mix,hi + X_mix,lo)^T, as hi + lo planes (m x T)
      GemmTc g = {m, T, n, W, ldw, false, Xmix, ldn, false, YtT, ldT, 3, 1.0f, nullptr, nullptr, 0, 0};
      g.B2 = Xmix_lo;
      g.D2 = YtT_lo;
      if ((st = gemm_tc(g, status, tmo, s2)) != PIFA_OK) return st;
    }
    {  // YtXt += (Y_t^T,hi + Y_t^T,lo) X_u
      GemmTc g = {m, n, T, YtT, ldT, false, XuT, ldT, false, YtXt, ldyx, 2, 1.0f, nullptr, nullptr, 0, 0};
      g.A2 = YtT_lo;
      if ((st = gemm_tc(g, status, tmo, s2)) != PIFA_OK) return st;
    }
  }
  {  // XXt += X_u^T X_u, its upper triangle (the product is symmetric: half the tiles)
    GemmTc g = {n, n, T, XuT, ldT, false, XuT, ldT, false, XXt, ldxx, 2, 1.0f, nullptr, nullptr, 0, 0};
    g.upper = true;
    if ((st = gemm_tc(g, status, tmo, s)) != PIFA_OK) return st;
  }
  return PIFA_OK;
}
