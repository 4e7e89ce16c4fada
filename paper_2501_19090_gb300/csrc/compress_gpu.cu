// compress_gpu.cu -- the float64 set-up steps on the GPU: pifa_compress_device (Algorithm 1,
// Sec. 3.2) and pifa_m_reconstruct (the two solves of the M reconstruction, Sec. 4, at the end).
//
// Route (all device-resident, float64; the caller's workspace holds every temporary):
//   1. G = V^T V (r x r) and its Cholesky factor L (G = L L^T). Then Z = U L (m x r) has the row
//      inner products of W' = U V^T: z_i . z_j = u_i G u_j^T = w_i . w_j, so QR with column
//      pivoting on W'^T (Algorithm 1, step 1) selects the same rows when run on Z^T, whose columns
//      are r long instead of n.
//   2. r greedy Businger-Golub steps on the rows of Z: step k picks the unchosen row of largest
//      residual norm (norms recomputed from the reflected rows every step, no downdating; ties to
//      the lowest index), builds the Householder reflector that maps the pivot row's residual onto
//      e_k, and applies it to every unchosen row. After r steps a chosen row holds its column of
//      the triangular factor R (selection order) and every other row i holds c_i = Q^T z_i.
//   3. Eq. 2 in Z-space: Z_np = C Z_p, with Z_p = R^T Q^T and Z_np = Cmat Q^T (rows c_i), so
//      C = Cmat R^{-T} -- one GEMM against the explicit inverse of R (computed by doubling:
//      inverted 32 x 32 diagonal blocks, then off-diagonal blocks -A^{-1} B D^{-1} level by level).
//      Columns go from selection order to ascending I as they are written.
//   4. W_p = U[I, :] V^T (Eq. 1).
// FP64 runs on the CUDA cores (tensor-core FP64 is no faster on this part); every kernel here is
// bound by FP64 issue rate or by streaming Z, and none waits on another CTA.
#include <cmath>
#include <cstdio>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "pifa.h"
#include "pifa_internal.h"

namespace {

// ---- generic float64 GEMM --------------------------------------------------------------------
// C[crow(i), ccol(j)] = beta C + alpha sum_k A(i, k) B(k, j), with
//   A(i, k) = A[arow(i) * sa_i + k * sa_k],  arow(i) = aidx ? aidx[i] : i
//   B(k, j) = B[k * sb_k + j * sb_j]
//   C at C[i * ldc + (cidx ? cidx[j] : j)]
// and a batch index z (blockIdx.z) offsetting A, B and C by za, zb, zc elements. `tri`: 1 = B is
// lower triangular (B(k, j) = 0 for k < j), 2 = B is upper triangular (B(k, j) = 0 for k > j);
// the k loop then skips the zero blocks.
struct GemmF64 {
  int M, N, K;
  const double* A;
  const int32_t* aidx;
  int64_t sa_i, sa_k;
  const double* B;
  int64_t sb_k, sb_j;
  double* C;
  const int32_t* cidx;
  int64_t ldc;
  double alpha, beta;
  int tri;
  int64_t za, zb, zc;
};

constexpr int GT = 64, GK = 16;  // output tile 64 x 64, k step 16; 256 threads, 4 x 4 outputs each

__global__ void __launch_bounds__(256) gemm_f64(GemmF64 p) {
  __shared__ double As[GK][GT + 1];
  __shared__ double Bs[GK][GT + 1];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int i0 = blockIdx.y * GT, j0 = blockIdx.x * GT;
  const double* A = p.A + blockIdx.z * p.za;
  const double* B = p.B + blockIdx.z * p.zb;
  double* C = p.C + blockIdx.z * p.zc;
  int kbeg = 0, kend = p.K;
  if (p.tri == 1) kbeg = (j0 / GK) * GK;
  if (p.tri == 2) kend = min(p.K, j0 + GT);
  double acc[4][4] = {};
  for (int k0 = kbeg; k0 < kend; k0 += GK) {
    for (int e = threadIdx.x; e < GT * GK; e += 256) {
      const int ii = e % GT, kk = e / GT;  // consecutive threads: consecutive rows of the A tile
      const int i = i0 + ii, k = k0 + kk;
      double va = 0.0;
      if (i < p.M && k < p.K) {
        const int64_t row = p.aidx ? (int64_t)p.aidx[i] : (int64_t)i;
        va = A[row * p.sa_i + (int64_t)k * p.sa_k];
      }
      As[kk][ii] = va;
      const int jj = e % GT, j = j0 + jj;
      double vb = 0.0;
      if (j < p.N && k < p.K) vb = B[(int64_t)k * p.sb_k + (int64_t)j * p.sb_j];
      Bs[kk][jj] = vb;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GK; ++kk) {
      double a[4], b[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        a[u] = As[kk][ty + 16 * u];
        b[u] = Bs[kk][tx + 16 * u];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fma(a[u], b[v], acc[u][v]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int i = i0 + ty + 16 * u;
    if (i >= p.M) continue;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int j = j0 + tx + 16 * v;
      if (j >= p.N) continue;
      double* c = C + (int64_t)i * p.ldc + (p.cidx ? (int64_t)p.cidx[j] : (int64_t)j);
      *c = (p.beta != 0.0 ? p.beta * *c : 0.0) + p.alpha * acc[u][v];
    }
  }
}

int run_gemm_f64(const GemmF64& p, int batch, cudaStream_t s) {
  if (p.M <= 0 || p.N <= 0 || batch <= 0) return PIFA_OK;
  dim3 grid((unsigned)((p.N + GT - 1) / GT), (unsigned)((p.M + GT - 1) / GT), (unsigned)batch);
  gemm_f64<<<grid, 256, 0, s>>>(p);
  pifa_count_launch();
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? PIFA_OK : pifa_fail_cuda("compress: gemm launch", e);
}

// ---- Cholesky of G (r x r, lower triangle used), one column per launch -----------------------
// Step j: L[i][j] = G[i][j] / sqrt(G[j][j]) for i >= j, and the trailing lower triangle
// G[i][l] -= G[i][j] G[l][j] / G[j][j] for j < l <= i. Column j of G is only read in step j, so
// the two parts need no ordering between threads. A non-positive pivot flags `bad`.
__global__ void chol_step(double* G, double* L, int r, int j, int* bad) {
  const int i = j + blockIdx.y * 16 + (threadIdx.x >> 4);
  const int l = j + blockIdx.x * 16 + (threadIdx.x & 15);
  if (i >= r || l > i) return;
  const double d = G[(int64_t)j * r + j];
  if (!(d > 0.0)) {
    if (i == j && l == j) atomicExch(bad, 1);
    return;
  }
  const double gij = G[(int64_t)i * r + j];
  if (l == j) {
    L[(int64_t)i * r + j] = gij / sqrt(d);
  } else {
    G[(int64_t)i * r + l] -= gij * G[(int64_t)l * r + j] / d;
  }
}

// ---- greedy pivoted QR on the rows of Z -------------------------------------------------------
// Best and runner-up residual norms (squared) with their rows; larger norm first, then the lower
// index: the selection rule of Algorithm 1, step 1 with ties to the lowest index.
struct Top2 {
  double v1;
  int i1;
  double v2;
  int i2;
};

__device__ __forceinline__ bool better(double va, int ia, double vb, int ib) {
  return va > vb || (va == vb && ia < ib);
}

__device__ __forceinline__ void top2_add(Top2& t, double v, int i) {
  if (i < 0) return;
  if (t.i1 < 0 || better(v, i, t.v1, t.i1)) {
    t.v2 = t.v1;
    t.i2 = t.i1;
    t.v1 = v;
    t.i1 = i;
  } else if (t.i2 < 0 || better(v, i, t.v2, t.i2)) {
    t.v2 = v;
    t.i2 = i;
  }
}

__device__ __forceinline__ Top2 top2_empty() { return Top2{0.0, -1, 0.0, -1}; }

__device__ __forceinline__ void top2_merge(Top2& a, const Top2& b) {
  top2_add(a, b.v1, b.i1);
  top2_add(a, b.v2, b.i2);
}

__device__ Top2 warp_top2(Top2 t) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Top2 u;
    u.v1 = __shfl_xor_sync(0xffffffffu, t.v1, o);
    u.i1 = __shfl_xor_sync(0xffffffffu, t.i1, o);
    u.v2 = __shfl_xor_sync(0xffffffffu, t.v2, o);
    u.i2 = __shfl_xor_sync(0xffffffffu, t.i2, o);
    top2_merge(t, u);
  }
  return t;
}

// Block-wide Top2 (blockDim.x = 256): every thread gets the block's result.
__device__ Top2 block_top2(Top2 t) {
  __shared__ Top2 sw[8];
  t = warp_top2(t);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) sw[w] = t;
  __syncthreads();
  Top2 r = top2_empty();
  for (int k = 0; k < 8; ++k) top2_merge(r, sw[k]);
  return r;
}

__device__ double block_sum(double v) {
  __shared__ double sw[8];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) sw[w] = v;
  __syncthreads();
  double s = 0.0;
  for (int k = 0; k < 8; ++k) s += sw[k];  // fixed order: the same value in every block
  return s;
}

struct Greedy {
  double* Z;        // m x r, row-major
  int m, r;
  int32_t* sel;     // m flags: chosen in an earlier step
  Top2* blk;        // 2 x nblk per-block results (ping-pong by step parity)
  int nblk;
  int32_t* order;   // r: row chosen at step k
  double* rdiag;    // r: R_kk of the pivoted QR
  double* gap;      // r: (best - runner-up) / best of the residual norms at step k
};

// Initial squared row norms of Z and each block's best two.
__global__ void __launch_bounds__(256) greedy_init(Greedy g) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  Top2 t = top2_empty();
  for (int i = blockIdx.x * 8 + warp; i < g.m; i += gridDim.x * 8) {
    const double* z = g.Z + (int64_t)i * g.r;
    double s = 0.0;
    for (int c = lane; c < g.r; c += 32) s = fma(z[c], z[c], s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) top2_add(t, s, i);
  }
  t = block_top2(t);
  if (threadIdx.x == 0) g.blk[blockIdx.x] = t;
}

// Step k: every block reduces step k - 1's per-block results to the pivot p (all blocks reach the
// same p), forms the reflector from row p's residual (coordinates k..r-1) in shared memory, and
// reflects its share of the unchosen rows, recomputing their residual norms (coordinates k+1..).
// Row p itself is left as it is (other blocks read it during this launch): its column of R is
// its coordinates 0..k-1 plus rdiag[k].
__global__ void __launch_bounds__(256) greedy_step(Greedy g, int k) {
  extern __shared__ double v[];  // r - k entries
  __shared__ int s_p;
  const Top2* in = g.blk + (k & 1) * g.nblk;
  Top2* out = g.blk + ((k + 1) & 1) * g.nblk;
  Top2 t = top2_empty();
  for (int b = threadIdx.x; b < g.nblk; b += 256) top2_merge(t, in[b]);
  t = block_top2(t);
  if (threadIdx.x == 0) s_p = t.i1;
  __syncthreads();
  const int p = s_p;
  const int len = g.r - k;
  if (p < 0 || p >= g.m) return;  // cannot happen for m >= r; guards the row read
  const double* zp = g.Z + (int64_t)p * g.r + k;
  double ss = 0.0;
  for (int c = threadIdx.x; c < len; c += 256) {
    const double x = zp[c];
    v[c] = x;
    ss = fma(x, x, ss);
  }
  const double nx2 = block_sum(ss);  // also orders the v[] writes before the reads below
  const double nx = sqrt(nx2);
  const double x0 = v[0];
  const double alpha = -copysign(nx, x0 != 0.0 ? x0 : 1.0);
  __syncthreads();
  if (threadIdx.x == 0) v[0] = x0 - alpha;
  __syncthreads();
  double vs = 0.0;
  for (int c = threadIdx.x; c < len; c += 256) vs = fma(v[c], v[c], vs);
  const double vn2 = block_sum(vs);
  const double tau = vn2 > 0.0 ? 2.0 / vn2 : 0.0;  // H = I - tau v v^T
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    g.order[k] = p;
    g.rdiag[k] = alpha;
    const double b1 = sqrt(fmax(t.v1, 0.0)), b2 = t.i2 >= 0 ? sqrt(fmax(t.v2, 0.0)) : 0.0;
    g.gap[k] = b1 > 0.0 ? (b1 - b2) / b1 : 0.0;
    g.sel[p] = 1;  // read only by later launches
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  Top2 mine = top2_empty();
  for (int i = blockIdx.x * 8 + warp; i < g.m; i += gridDim.x * 8) {
    if (i == p || g.sel[i]) continue;  // warp-uniform
    double* z = g.Z + (int64_t)i * g.r + k;
    double d = 0.0;
    for (int c = lane; c < len; c += 32) d = fma(z[c], v[c], d);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
    const double s = tau * d;
    double nr = 0.0;
    for (int c = lane; c < len; c += 32) {
      const double y = fma(-s, v[c], z[c]);
      z[c] = y;
      if (c > 0) nr = fma(y, y, nr);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) nr += __shfl_xor_sync(0xffffffffu, nr, o);
    if (lane == 0) top2_add(mine, nr, i);
  }
  mine = block_top2(mine);
  if (threadIdx.x == 0) out[blockIdx.x] = mine;
}

// ---- R, its inverse, the index sets -----------------------------------------------------------
// R (rp x rp, row-major, upper triangular, selection order): R[c][k] = Z[order[k]][c] for c < k,
// R[k][k] = rdiag[k]; identity on the padding k >= r.
__global__ void build_r(const Greedy g, double* R, int rp) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= (int64_t)rp * rp) return;
  const int c = (int)(e / rp), k = (int)(e % rp);
  double val = 0.0;
  if (k >= g.r) {
    val = c == k ? 1.0 : 0.0;
  } else if (c < k) {
    val = g.Z[(int64_t)g.order[k] * g.r + c];
  } else if (c == k) {
    val = g.rdiag[k];
  }
  R[e] = val;
}

// Inverses of the 32 x 32 diagonal blocks of R into Rinv (whose other entries are zeroed): thread
// j of block b solves R_bb y = e_j by back substitution.
__global__ void inv_diag32(const double* R, double* Rinv, int rp) {
  __shared__ double Rb[32][33];
  __shared__ double Y[32][33];
  const int b = blockIdx.x, j = threadIdx.x;
  const int64_t base = (int64_t)b * 32;
  for (int i = 0; i < 32; ++i) Rb[i][j] = R[(base + i) * rp + base + j];
  __syncthreads();
  for (int i = 31; i >= 0; --i) {
    double s = (i == j) ? 1.0 : 0.0;
    for (int l = i + 1; l <= j; ++l) s -= Rb[i][l] * Y[l][j];
    Y[i][j] = i <= j ? s / Rb[i][i] : 0.0;
  }
  __syncthreads();
  for (int i = 0; i < 32; ++i) Rinv[(base + i) * rp + base + j] = Y[i][j];
}

// Ascending I and I^c from the chosen-row flags, and for every selection step k the position of
// its row in ascending I (one block of 1024 threads, chunked prefix sums).
__global__ void __launch_bounds__(1024) index_sets(const int32_t* sel, int m, const int32_t* order, int r,
                                                   int32_t* piv, int32_t* nonpiv, int32_t* pos, int32_t* asc) {
  __shared__ int s_cnt[1024];
  __shared__ int s_base;
  if (threadIdx.x == 0) s_base = 0;
  __syncthreads();
  for (int c0 = 0; c0 < m; c0 += 1024) {
    const int i = c0 + threadIdx.x;
    const int f = (i < m && sel[i]) ? 1 : 0;
    s_cnt[threadIdx.x] = f;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {  // inclusive scan
      const int v = threadIdx.x >= o ? s_cnt[threadIdx.x - o] : 0;
      __syncthreads();
      s_cnt[threadIdx.x] += v;
      __syncthreads();
    }
    if (i < m) {
      const int before = s_base + s_cnt[threadIdx.x] - f;  // chosen rows before i
      pos[i] = before;
      if (f) {
        if (before < r) piv[before] = i;
      } else if (i - before < m - r) {
        nonpiv[i - before] = i;
      }
    }
    __syncthreads();
    if (threadIdx.x == 1023) s_base += s_cnt[1023];
    __syncthreads();
  }
  for (int k = threadIdx.x; k < r; k += 1024) asc[k] = pos[order[k]];
}

// max |C| over the (m - r) x r block (non-negative doubles order like their bit patterns).
__global__ void max_abs(const double* C, int64_t rows, int64_t cols, int64_t ldc, unsigned long long* out) {
  double mx = 0.0;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < rows * cols; e += (int64_t)gridDim.x * blockDim.x)
    mx = fmax(mx, fabs(C[(e / cols) * ldc + e % cols]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((threadIdx.x & 31) == 0) atomicMax(out, (unsigned long long)__double_as_longlong(mx));
}

// Rinv = R^{-1} for an upper-triangular R (rp x rp, rp = 32 * 2^k; identity on any padding), by
// doubling: the 32 x 32 diagonal blocks inverted directly, then, level by level, for every pair
// of sz-blocks [[A, B], [0, D]] along the diagonal the off-diagonal block -A^{-1} (B D^{-1}).
// Tt: scratch of rp * rp / 4 doubles.
int upper_inverse(const double* R, double* Rinv, double* Tt, int rp, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(Rinv, 0, (size_t)rp * rp * 8, s);
  if (e != cudaSuccess) return pifa_fail_cuda("upper inverse: memset", e);
  inv_diag32<<<rp / 32, 32, 0, s>>>(R, Rinv, rp);
  pifa_count_launch();
  e = cudaGetLastError();
  if (e != cudaSuccess) return pifa_fail_cuda("upper inverse: launch", e);
  int st;
  for (int sz = 32; sz < rp; sz *= 2) {
    const int pairs = rp / (2 * sz);
    const int64_t step = (int64_t)2 * sz * rp + 2 * sz;  // next pair along the diagonal
    GemmF64 a = {};
    a.M = sz; a.N = sz; a.K = sz;
    a.A = R + sz; a.sa_i = rp; a.sa_k = 1;                        // B block
    a.B = Rinv + (int64_t)sz * rp + sz; a.sb_k = rp; a.sb_j = 1;  // D^{-1}
    a.C = Tt; a.ldc = sz; a.alpha = 1.0; a.beta = 0.0;
    a.za = step; a.zb = step; a.zc = (int64_t)sz * sz;
    if ((st = run_gemm_f64(a, pairs, s)) != PIFA_OK) return st;
    GemmF64 b = {};
    b.M = sz; b.N = sz; b.K = sz;
    b.A = Rinv; b.sa_i = rp; b.sa_k = 1;                          // A^{-1}
    b.B = Tt; b.sb_k = sz; b.sb_j = 1;
    b.C = Rinv + sz; b.ldc = rp; b.alpha = -1.0; b.beta = 0.0;
    b.za = step; b.zb = (int64_t)sz * sz; b.zc = step;
    if ((st = run_gemm_f64(b, pairs, s)) != PIFA_OK) return st;
  }
  return PIFA_OK;
}

// Workspace layout (bytes, each part 256-aligned).
struct Layout {
  int64_t G, L, Z, R, Rinv, T, blk, order, rdiag, gap, sel, pos, asc, flags, total;
  int rp, nblk;
};

int64_t a256(int64_t b) { return (b + 255) / 256 * 256; }

Layout layout(int64_t m, int64_t r) {
  Layout L = {};
  int rp = 32;
  while (rp < r) rp *= 2;
  L.rp = rp;
  L.nblk = 4 * 152;
  int64_t o = 0;
  auto take = [&](int64_t bytes) {
    const int64_t at = o;
    o += a256(bytes);
    return at;
  };
  L.G = take(r * r * 8);
  L.L = take(r * r * 8);
  L.Z = take(m * r * 8);
  L.R = take((int64_t)rp * rp * 8);
  L.Rinv = take((int64_t)rp * rp * 8);
  L.T = take((int64_t)rp * rp / 4 * 8 + 8);
  L.blk = take(2 * (int64_t)L.nblk * (int64_t)sizeof(Top2));
  L.order = take(r * 4);
  L.rdiag = take(r * 8);
  L.gap = take(r * 8);
  L.sel = take(m * 4);
  L.pos = take(m * 4);
  L.asc = take(r * 4);
  L.flags = take(64);
  L.total = o;
  return L;
}

constexpr int64_t kMaxRank = 16384;  // the reflector lives in shared memory (r doubles)

}  // namespace

extern "C" int64_t pifa_compress_device_workspace_size(int64_t m, int64_t n, int64_t r) {
  pifa_clear_error();
  if (m < 1 || n < 1 || r < 1 || r > m || r > n) return pifa_fail(PIFA_ERR_INVALID_ARG, "need 1 <= r <= min(m, n)");
  if (r > kMaxRank || m >= ((int64_t)1 << 30) || n >= ((int64_t)1 << 30))
    return pifa_fail(PIFA_ERR_UNSUPPORTED, "pifa_compress_device needs r <= 16384 and m, n < 2^30");
  return layout(m, r).total;
}

extern "C" int pifa_compress_device(const double* U, const double* V, int64_t m, int64_t n, int64_t r,
                                    int32_t* pivot_idx, int32_t* nonpivot_idx, double* Wp, int64_t ldwp,
                                    double* C, int64_t ldc, void* workspace, int64_t workspace_bytes,
                                    pifa_compress_info* info, void* cuda_stream) {
  const int64_t need = pifa_compress_device_workspace_size(m, n, r);
  if (need < 0) return (int)need;
  pifa_clear_error();
  const bool has_np = m > r;
  if (!U || !V || !pivot_idx || !Wp || (has_np && (!nonpivot_idx || !C)))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "null U, V, pivot_idx, Wp, nonpivot_idx or C");
  if (ldwp < n || (has_np && ldc < r)) return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row");
  if (!workspace || workspace_bytes < need) return pifa_fail(PIFA_ERR_WORKSPACE, "workspace missing or too small");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return pifa_fail(PIFA_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(cuda_stream);
  const Layout Ly = layout(m, r);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  double* G = reinterpret_cast<double*>(ws + Ly.G);
  double* L = reinterpret_cast<double*>(ws + Ly.L);
  double* Z = reinterpret_cast<double*>(ws + Ly.Z);
  double* R = reinterpret_cast<double*>(ws + Ly.R);
  double* Rinv = reinterpret_cast<double*>(ws + Ly.Rinv);
  double* Tt = reinterpret_cast<double*>(ws + Ly.T);
  int* flags = reinterpret_cast<int*>(ws + Ly.flags);  // [0] Cholesky failure, [2..3] max |C| bits
  Greedy g;
  g.Z = Z;
  g.m = (int)m;
  g.r = (int)r;
  g.sel = reinterpret_cast<int32_t*>(ws + Ly.sel);
  g.blk = reinterpret_cast<Top2*>(ws + Ly.blk);
  g.nblk = Ly.nblk;
  g.order = reinterpret_cast<int32_t*>(ws + Ly.order);
  g.rdiag = reinterpret_cast<double*>(ws + Ly.rdiag);
  g.gap = reinterpret_cast<double*>(ws + Ly.gap);
  int32_t* pos = reinterpret_cast<int32_t*>(ws + Ly.pos);
  int32_t* asc = reinterpret_cast<int32_t*>(ws + Ly.asc);
  const int ri = (int)r, mi = (int)m, ni = (int)n, rp = Ly.rp;
  cudaError_t e;
  int st;
#define PIFA_CK(call, what)                          \
  do {                                               \
    if ((e = (call)) != cudaSuccess) return pifa_fail_cuda(what, e); \
  } while (0)
  PIFA_CK(cudaMemsetAsync(flags, 0, 64, s), "compress: memset");
  PIFA_CK(cudaMemsetAsync(g.sel, 0, m * 4, s), "compress: memset");
  PIFA_CK(cudaMemsetAsync(L, 0, r * r * 8, s), "compress: memset");
  // every index a later kernel gathers through starts valid, whatever the selection does
  PIFA_CK(cudaMemsetAsync(g.order, 0, r * 4, s), "compress: memset");
  PIFA_CK(cudaMemsetAsync(pivot_idx, 0, r * 4, s), "compress: memset");
  if (has_np) PIFA_CK(cudaMemsetAsync(nonpivot_idx, 0, (m - r) * 4, s), "compress: memset");

  // 1. G = V^T V, L = chol(G), Z = U L
  GemmF64 q = {};
  q.M = ri; q.N = ri; q.K = ni;
  q.A = V; q.sa_i = 1; q.sa_k = r;
  q.B = V; q.sb_k = r; q.sb_j = 1;
  q.C = G; q.ldc = r; q.alpha = 1.0; q.beta = 0.0;
  if ((st = run_gemm_f64(q, 1, s)) != PIFA_OK) return st;
  for (int j = 0; j < ri; ++j) {
    const int t = (ri - j + 15) / 16;
    chol_step<<<dim3(t, t), 256, 0, s>>>(G, L, ri, j, flags);
    pifa_count_launch();
  }
  PIFA_CK(cudaGetLastError(), "compress: cholesky launch");
  q = GemmF64{};
  q.M = mi; q.N = ri; q.K = ri;
  q.A = U; q.sa_i = r; q.sa_k = 1;
  q.B = L; q.sb_k = r; q.sb_j = 1;
  q.C = Z; q.ldc = r; q.alpha = 1.0; q.beta = 0.0; q.tri = 1;
  if ((st = run_gemm_f64(q, 1, s)) != PIFA_OK) return st;

  // 2. r greedy steps
  greedy_init<<<Ly.nblk, 256, 0, s>>>(g);
  pifa_count_launch();
  PIFA_CK(cudaGetLastError(), "compress: greedy init launch");
  const size_t vsm = (size_t)r * 8;
  PIFA_CK(cudaFuncSetAttribute(greedy_step, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)vsm),
          "compress: greedy smem attribute");
  for (int k = 0; k < ri; ++k) {
    greedy_step<<<Ly.nblk, 256, (size_t)(r - k) * 8, s>>>(g, k);
    pifa_count_launch();
  }
  PIFA_CK(cudaGetLastError(), "compress: greedy step launch");

  // 3. index sets, R, R^{-1}, C = Z[I^c] R^{-T} in ascending-I columns
  index_sets<<<1, 1024, 0, s>>>(g.sel, mi, g.order, ri, pivot_idx, has_np ? nonpivot_idx : pos, pos, asc);
  pifa_count_launch();
  PIFA_CK(cudaGetLastError(), "compress: index sets launch");
  {
    const int64_t tot = (int64_t)rp * rp;
    build_r<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(g, R, rp);
    pifa_count_launch();
    if ((st = upper_inverse(R, Rinv, Tt, rp, s)) != PIFA_OK) return st;
  }
  if (has_np) {
    // C[a][asc[j]] = sum_{k >= j} Z[I^c[a]][k] Rinv[j][k]
    GemmF64 c = {};
    c.M = (int)(m - r); c.N = ri; c.K = ri;
    c.A = Z; c.aidx = nonpivot_idx; c.sa_i = r; c.sa_k = 1;
    c.B = Rinv; c.sb_k = 1; c.sb_j = rp;
    c.C = C; c.cidx = asc; c.ldc = ldc; c.alpha = 1.0; c.beta = 0.0; c.tri = 1;
    if ((st = run_gemm_f64(c, 1, s)) != PIFA_OK) return st;
    max_abs<<<4 * 152, 256, 0, s>>>(C, m - r, r, ldc, reinterpret_cast<unsigned long long*>(flags + 2));
    pifa_count_launch();
    PIFA_CK(cudaGetLastError(), "compress: max launch");
  }
  // 4. W_p = U[I] V^T
  {
    GemmF64 w = {};
    w.M = ri; w.N = ni; w.K = ri;
    w.A = U; w.aidx = pivot_idx; w.sa_i = r; w.sa_k = 1;
    w.B = V; w.sb_k = 1; w.sb_j = r;
    w.C = Wp; w.ldc = ldwp; w.alpha = 1.0; w.beta = 0.0;
    if ((st = run_gemm_f64(w, 1, s)) != PIFA_OK) return st;
  }

  // results for the rank check and the diagnostics
  int hflags[4] = {0, 0, 0, 0};
  double rd0 = 0.0, rdl = 0.0;
  PIFA_CK(cudaMemcpyAsync(hflags, flags, sizeof hflags, cudaMemcpyDeviceToHost, s), "compress: read back");
  PIFA_CK(cudaMemcpyAsync(&rd0, g.rdiag, 8, cudaMemcpyDeviceToHost, s), "compress: read back");
  PIFA_CK(cudaMemcpyAsync(&rdl, g.rdiag + (r - 1), 8, cudaMemcpyDeviceToHost, s), "compress: read back");
  double* hgap = nullptr;
  PIFA_CK(cudaMallocHost(&hgap, r * 8), "compress: host buffer");
  e = cudaMemcpyAsync(hgap, g.gap, r * 8, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  double min_gap = 1.0;
  if (e == cudaSuccess)
    for (int64_t k = 0; k < r; ++k) min_gap = hgap[k] < min_gap ? hgap[k] : min_gap;
  cudaFreeHost(hgap);
  if (e != cudaSuccess) return pifa_fail_cuda("compress: synchronize", e);
#undef PIFA_CK
  double cmax = 0.0;
  {
    unsigned long long bits = (unsigned long long)(unsigned)hflags[2] | ((unsigned long long)(unsigned)hflags[3] << 32);
    memcpy(&cmax, &bits, 8);
  }
  if (info) {
    info->min_pivot_gap = min_gap;
    info->r_ratio = rd0 != 0.0 ? std::fabs(rdl) / std::fabs(rd0) : 0.0;
    info->max_abs_c = cmax;
    info->threads = 0;
  }
  if (hflags[0] || !(std::fabs(rdl) >= 1e-8 * std::fabs(rd0)) || rd0 == 0.0)
    return pifa_fail(PIFA_ERR_RANK_DEFICIENT, "W' = U V^T has fewer than r independent rows (|R_rr| < 1e-8 |R_00|)");
  return PIFA_OK;
}

// ---- the M reconstruction solves (Sec. 4, Eqs. 4 and 8; Algorithm 3, part 1) ------------------
namespace {

// dst (rows x cols, pitch lddst, fp64) = src (fp32, pitch ldsrc)
__global__ void f32_to_f64(const float* src, int64_t ldsrc, int64_t rows, int64_t cols, double* dst, int64_t lddst) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < rows * cols; e += (int64_t)gridDim.x * blockDim.x)
    dst[(e / cols) * lddst + e % cols] = (double)src[(e / cols) * ldsrc + e % cols];
}

// dst (rows x cols, fp64) += alpha * W (bf16, pitch ldw)
__global__ void add_scaled_bf16(const __nv_bfloat16* W, int64_t ldw, int64_t rows, int64_t cols, double alpha,
                                double* dst, int64_t lddst) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < rows * cols; e += (int64_t)gridDim.x * blockDim.x)
    dst[(e / cols) * lddst + e % cols] += alpha * (double)__bfloat162float(W[(e / cols) * ldw + e % cols]);
}

// A[i][j] = A[j][i] for i > j (n x n, pitch lda): the lower triangle from the upper.
__global__ void mirror_upper(double* A, int64_t n, int64_t lda) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n * n; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = e / n, j = e % n;
    if (i > j) A[i * lda + j] = A[j * lda + i];
  }
}

__global__ void add_diag(double* A, int64_t k, int64_t lda, double alpha) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < k; i += (int64_t)gridDim.x * blockDim.x)
    A[i * lda + i] += alpha;
}

// R (rp x rp) = L^T for a lower-triangular L (k x k, pitch k), identity on the padding i >= k.
__global__ void transpose_pad_lower(const double* L, int64_t k, double* R, int rp) {
  const int64_t tot = (int64_t)rp * rp;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < tot; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = e / rp, j = e % rp;
    double v = 0.0;
    if (i < k && j < k)
      v = i <= j ? L[j * k + i] : 0.0;
    else if (i == j)
      v = 1.0;
    R[e] = v;
  }
}

int grid_for(int64_t work) {
  const int64_t b = (work + 255) / 256;
  return (int)(b < 4 * 152 ? (b > 0 ? b : 1) : 4 * 152);
}

int pad_pow2_32(int64_t k) {
  int rp = 32;
  while (rp < k) rp *= 2;
  return rp;
}

// Scratch of spd_inverse for k: a copy of S, L, R and R^{-1} (rp x rp), and the doubling's T.
int64_t spd_scratch_doubles(int64_t k) {
  const int64_t rp = pad_pow2_32(k);
  return 2 * k * k + 2 * rp * rp + rp * rp / 4 + 64;
}

// Sinv = S^{-1} for a symmetric positive definite S (k x k, pitch k): S = L L^T (Cholesky, one
// column per launch), R = L^T, S^{-1} = R^{-1} R^{-T}. `bad` is set when a pivot is not positive.
int spd_inverse(const double* S, int64_t k, double* Sinv, double* scratch, int* bad, cudaStream_t s) {
  const int rp = pad_pow2_32(k);
  double* G = scratch;
  double* L = G + k * k;
  double* R = L + k * k;
  double* Rinv = R + (int64_t)rp * rp;
  double* Tt = Rinv + (int64_t)rp * rp;
  cudaError_t e = cudaMemcpyAsync(G, S, (size_t)k * k * 8, cudaMemcpyDeviceToDevice, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(L, 0, (size_t)k * k * 8, s);
  if (e != cudaSuccess) return pifa_fail_cuda("spd inverse: copy", e);
  for (int j = 0; j < (int)k; ++j) {
    const int t = ((int)k - j + 15) / 16;
    chol_step<<<dim3(t, t), 256, 0, s>>>(G, L, (int)k, j, bad);
    pifa_count_launch();
  }
  transpose_pad_lower<<<grid_for((int64_t)rp * rp), 256, 0, s>>>(L, k, R, rp);
  pifa_count_launch();
  e = cudaGetLastError();
  if (e != cudaSuccess) return pifa_fail_cuda("spd inverse: launch", e);
  int st = upper_inverse(R, Rinv, Tt, rp, s);
  if (st != PIFA_OK) return st;
  GemmF64 g = {};  // Sinv[i][j] = sum_t Rinv[i][t] Rinv[j][t]
  g.M = (int)k; g.N = (int)k; g.K = (int)k;
  g.A = Rinv; g.sa_i = rp; g.sa_k = 1;
  g.B = Rinv; g.sb_k = 1; g.sb_j = rp;
  g.C = Sinv; g.ldc = k; g.alpha = 1.0; g.beta = 0.0;
  return run_gemm_f64(g, 1, s);
}

}  // namespace

extern "C" int64_t pifa_m_reconstruct_workspace_size(int64_t m, int64_t n, int64_t r) {
  pifa_clear_error();
  if (m < 1 || n < 1 || r < 1 || r > n || r > m) return pifa_fail(PIFA_ERR_INVALID_ARG, "need 1 <= r <= min(m, n)");
  if (n > 16384 || m >= ((int64_t)1 << 30)) return pifa_fail(PIFA_ERR_UNSUPPORTED, "pifa_m_reconstruct needs n <= 16384");
  const int64_t d = 2 * n * n + m * n + n * r + m * r + 4 * r * r + 2 * r * n + spd_scratch_doubles(n > r ? n : r) + 64;
  return d * 8 + 256;
}

extern "C" int pifa_m_reconstruct(const float* XXt, int64_t ldxx, const float* YtXt, int64_t ldyx, const double* V,
                                  const void* W, int64_t ldw, int64_t m, int64_t n, int64_t r, double alpha,
                                  double* U_r, double* V_r, void* workspace, int64_t workspace_bytes,
                                  void* cuda_stream) {
  const int64_t need = pifa_m_reconstruct_workspace_size(m, n, r);
  if (need < 0) return (int)need;
  pifa_clear_error();
  if (!XXt || !YtXt || !V || !U_r || !V_r || (alpha != 0.0 && !W))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "null XXt, YtXt, V, U_r, V_r, or W with alpha != 0");
  if (!(alpha >= 0.0)) return pifa_fail(PIFA_ERR_INVALID_ARG, "alpha must be >= 0");
  if (ldxx < n || ldyx < n || (W && ldw < n)) return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row");
  if (!workspace || workspace_bytes < need) return pifa_fail(PIFA_ERR_WORKSPACE, "workspace missing or too small");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return pifa_fail(PIFA_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(cuda_stream);
  double* A = static_cast<double*>(workspace);  // X X^T (n x n), later X X^T + alpha I
  double* B = A + n * n;                         // Y_t X^T (m x n), later + alpha W
  double* T1 = B + m * n;                        // X X^T V (n x r)
  double* Sm = T1 + n * r;                       // V^T X X^T V (r x r)
  double* B1 = Sm + r * r;                       // Y_t X^T V (m x r)
  double* Sinv = B1 + m * r;
  double* Pm = Sinv + r * r;                     // U_r^T U_r
  double* Pinv = Pm + r * r;
  double* Rhs = Pinv + r * r;                    // U_r^T (Y_t X^T + alpha W) (r x n)
  double* Q = Rhs + r * n;                       // (U_r^T U_r)^{-1} Rhs (r x n)
  double* Ginv = Q + r * n;                      // (X X^T + alpha I)^{-1}
  int* bad = reinterpret_cast<int*>(Ginv + n * n);
  double* scratch = reinterpret_cast<double*>(bad) + 8;
  cudaError_t e = cudaMemsetAsync(bad, 0, 8, s);
  if (e != cudaSuccess) return pifa_fail_cuda("reconstruct: memset", e);
  f32_to_f64<<<grid_for(n * n), 256, 0, s>>>(XXt, ldxx, n, n, A, n);
  pifa_count_launch();
  mirror_upper<<<grid_for(n * n), 256, 0, s>>>(A, n, n);  // pifa_m_accumulate keeps the upper triangle
  pifa_count_launch();
  f32_to_f64<<<grid_for(m * n), 256, 0, s>>>(YtXt, ldyx, m, n, B, n);
  pifa_count_launch();
  e = cudaGetLastError();
  if (e != cudaSuccess) return pifa_fail_cuda("reconstruct: launch", e);
  const int ni = (int)n, mi = (int)m, ri = (int)r;
  int st;
  auto gemm = [&](int M, int N, int K, const double* Ap, int64_t sai, int64_t sak, const double* Bp, int64_t sbk,
                  int64_t sbj, double* Cp, int64_t ldc) {
    GemmF64 g = {};
    g.M = M; g.N = N; g.K = K;
    g.A = Ap; g.sa_i = sai; g.sa_k = sak;
    g.B = Bp; g.sb_k = sbk; g.sb_j = sbj;
    g.C = Cp; g.ldc = ldc; g.alpha = 1.0; g.beta = 0.0;
    return run_gemm_f64(g, 1, s);
  };
  // Eq. 4: U_r = (Y_t X^T) V (V^T (X X^T) V)^{-1}
  if ((st = gemm(ni, ri, ni, A, n, 1, V, r, 1, T1, r)) != PIFA_OK) return st;
  if ((st = gemm(ri, ri, ni, V, 1, r, T1, r, 1, Sm, r)) != PIFA_OK) return st;   // V^T T1
  if ((st = gemm(mi, ri, ni, B, n, 1, V, r, 1, B1, r)) != PIFA_OK) return st;
  if ((st = spd_inverse(Sm, r, Sinv, scratch, bad, s)) != PIFA_OK) return st;
  if ((st = gemm(mi, ri, ri, B1, r, 1, Sinv, r, 1, U_r, r)) != PIFA_OK) return st;
  // Eq. 8: V_r^T = (U_r^T U_r)^{-1} U_r^T (Y_t X^T + alpha W) (X X^T + alpha I)^{-1}
  if ((st = gemm(ri, ri, mi, U_r, 1, r, U_r, r, 1, Pm, r)) != PIFA_OK) return st;   // U_r^T U_r
  if ((st = spd_inverse(Pm, r, Pinv, scratch, bad, s)) != PIFA_OK) return st;
  if (alpha != 0.0) {
    add_scaled_bf16<<<grid_for(m * n), 256, 0, s>>>(static_cast<const __nv_bfloat16*>(W), ldw, m, n, alpha, B, n);
    pifa_count_launch();
    add_diag<<<grid_for(n), 256, 0, s>>>(A, n, n, alpha);
    pifa_count_launch();
    e = cudaGetLastError();
    if (e != cudaSuccess) return pifa_fail_cuda("reconstruct: launch", e);
  }
  if ((st = gemm(ri, ni, mi, U_r, 1, r, B, n, 1, Rhs, n)) != PIFA_OK) return st;   // U_r^T B
  if ((st = gemm(ri, ni, ri, Pinv, r, 1, Rhs, n, 1, Q, n)) != PIFA_OK) return st;
  if ((st = spd_inverse(A, n, Ginv, scratch, bad, s)) != PIFA_OK) return st;
  // V_r = (Q Ginv)^T = Ginv Q^T (Ginv symmetric)
  if ((st = gemm(ni, ri, ni, Ginv, n, 1, Q, 1, n, V_r, r)) != PIFA_OK) return st;
  int hbad = 0;
  e = cudaMemcpyAsync(&hbad, bad, sizeof(int), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return pifa_fail_cuda("reconstruct: synchronize", e);
  if (hbad) return pifa_fail(PIFA_ERR_RANK_DEFICIENT, "a matrix of the reconstruction is not positive definite");
  return PIFA_OK;
}
