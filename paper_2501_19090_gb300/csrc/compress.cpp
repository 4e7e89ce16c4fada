// compress.cpp -- pifa_compress: Algorithm 1 (Sec. 3.2) on the host in float64.
//
// Route. W' = U V^T has rank r. With V = Q_V R_V (thin Householder QR, Q_V orthonormal columns),
// W' = (U R_V^T) Q_V^T, so the rows of Z = U R_V^T (m x r) have exactly the inner products of the
// rows of W'. QR with column pivoting on W'^T (Algorithm 1, step 1; Businger-Golub) therefore
// selects the same rows when run on Z^T, whose columns are only r long instead of n:
//   step k: pick the unchosen column of largest residual norm (norms recomputed from the
//           reflected columns every step -- no downdating; ties to the lowest index), reflect it
//           onto e_k with a Householder transform, apply the transform to every unchosen column.
// After r steps Z^T P = Q [R11 R12]; the chosen columns satisfy Z_np^T = Z_p^T R11^{-1} R12, so the
// coefficient matrix of Eq. 2 is C = (R11^{-1} R12)^T in the greedy order, permuted to ascending I.
// Finally W_p = U[I, :] V^T (Eq. 1).
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include <omp.h>

#include "pifa.h"
#include "pifa_internal.h"

namespace {

// C[i][j] = sum_k A[i][k] * B[j][k]  (A: M x K, B: N x K, both row-major, k contiguous).
void gemm_nt(int64_t M, int64_t N, int64_t K, const double* A, int64_t lda, const double* B,
             int64_t ldb, double* C, int64_t ldc) {
  const int64_t BI = 32, BJ = 32, BK = 512;
  const int64_t ni = (M + BI - 1) / BI, nj = (N + BJ - 1) / BJ;
#pragma omp parallel for schedule(dynamic, 1) collapse(2)
  for (int64_t bi = 0; bi < ni; ++bi) {
    for (int64_t bj = 0; bj < nj; ++bj) {
      const int64_t i0 = bi * BI, i1 = std::min(M, i0 + BI);
      const int64_t j0 = bj * BJ, j1 = std::min(N, j0 + BJ);
      double acc[BI][BJ];
      for (int64_t i = 0; i < i1 - i0; ++i)
        for (int64_t j = 0; j < j1 - j0; ++j) acc[i][j] = 0.0;
      for (int64_t k0 = 0; k0 < K; k0 += BK) {
        const int64_t k1 = std::min(K, k0 + BK);
        for (int64_t i = i0; i < i1; ++i) {
          const double* a = A + i * lda;
          for (int64_t j = j0; j < j1; ++j) {
            const double* b = B + j * ldb;
            double s = 0.0;
            for (int64_t k = k0; k < k1; ++k) s += a[k] * b[k];
            acc[i - i0][j - j0] += s;
          }
        }
      }
      for (int64_t i = i0; i < i1; ++i)
        for (int64_t j = j0; j < j1; ++j) C[i * ldc + j] = acc[i - i0][j - j0];
    }
  }
}

// Householder reflector for x (len entries): returns alpha (x -> alpha e_0) and writes the unit
// vector v (v = (x - alpha e_0) / ||x - alpha e_0||); v is all zero when x is already zero.
double make_reflector(const double* x, int64_t len, double* v) {
  double ss = 0.0;
  for (int64_t i = 0; i < len; ++i) ss += x[i] * x[i];
  const double nx = std::sqrt(ss);
  const double alpha = -std::copysign(nx, x[0] != 0.0 ? x[0] : 1.0);
  for (int64_t i = 0; i < len; ++i) v[i] = x[i];
  v[0] -= alpha;
  double vs = 0.0;
  for (int64_t i = 0; i < len; ++i) vs += v[i] * v[i];
  const double vn = std::sqrt(vs);
  if (vn > 0.0)
    for (int64_t i = 0; i < len; ++i) v[i] /= vn;
  else
    for (int64_t i = 0; i < len; ++i) v[i] = 0.0;
  return alpha;
}

}  // namespace

extern "C" int pifa_compress(const double* U, const double* V, int64_t m, int64_t n, int64_t r,
                             int32_t* pivot_idx, int32_t* nonpivot_idx, double* Wp, int64_t ldwp,
                             double* C, int64_t ldc, pifa_compress_info* info) {
  pifa_clear_error();
  if (!U || !V || !pivot_idx || !Wp) return pifa_fail(PIFA_ERR_INVALID_ARG, "pifa_compress: null pointer");
  if (m < 1 || n < 1 || r < 1 || r > std::min(m, n))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "pifa_compress: need 1 <= r <= min(m, n)");
  if (m > INT32_MAX) return pifa_fail(PIFA_ERR_INVALID_ARG, "pifa_compress: m exceeds int32 indices");
  if (ldwp < n) return pifa_fail(PIFA_ERR_INVALID_ARG, "pifa_compress: ldwp < n");
  if (m > r && (!C || !nonpivot_idx || ldc < r))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "pifa_compress: C / nonpivot_idx missing or ldc < r");

  // --- thin QR of V (n x r): columns stored contiguously, Householder, keep R_V -------------
  std::vector<double> Vc((size_t)r * n);
  for (int64_t i = 0; i < n; ++i)
    for (int64_t j = 0; j < r; ++j) Vc[(size_t)j * n + i] = V[i * r + j];
  std::vector<double> Rv((size_t)r * r, 0.0);  // row-major r x r, upper triangular
  {
    std::vector<double> v(n);
    for (int64_t k = 0; k < r; ++k) {
      double* colk = &Vc[(size_t)k * n];
      const double alpha = make_reflector(colk + k, n - k, v.data());
      Rv[k * r + k] = alpha;
#pragma omp parallel for schedule(static)
      for (int64_t j = k + 1; j < r; ++j) {
        double* col = &Vc[(size_t)j * n + k];
        double s = 0.0;
        for (int64_t i = 0; i < n - k; ++i) s += v[i] * col[i];
        s *= 2.0;
        for (int64_t i = 0; i < n - k; ++i) col[i] -= s * v[i];
      }
      for (int64_t j = k + 1; j < r; ++j) Rv[k * r + j] = Vc[(size_t)j * n + k];
    }
  }
  std::vector<double>().swap(Vc);

  // --- Z = U R_V^T (m x r, row j = z_j, contiguous) -----------------------------------------
  std::vector<double> Z((size_t)m * r);
  gemm_nt(m, r, r, U, r, Rv.data(), r, Z.data(), r);

  // --- greedy pivoted QR on the columns z_j of Z^T --------------------------------------------
  std::vector<double> norm2(m);
#pragma omp parallel for schedule(static)
  for (int64_t j = 0; j < m; ++j) {
    const double* z = &Z[(size_t)j * r];
    double s = 0.0;
    for (int64_t a = 0; a < r; ++a) s += z[a] * z[a];
    norm2[j] = s;
  }
  std::vector<unsigned char> chosen(m, 0);
  std::vector<int64_t> order;
  order.reserve(r);
  std::vector<double> rdiag(r), v(r);
  double min_gap = 1.0;
  const int nthreads = omp_get_max_threads();
  std::vector<double> tbest(nthreads), tsecond(nthreads);
  std::vector<int64_t> tidx(nthreads);
  for (int64_t k = 0; k < r; ++k) {
    // select: largest residual norm, lowest index among equals; also track the runner-up
#pragma omp parallel
    {
      const int t = omp_get_thread_num();
      double b = -1.0, s2 = -1.0;
      int64_t bi = -1;
#pragma omp for schedule(static)
      for (int64_t j = 0; j < m; ++j) {
        if (chosen[j]) continue;
        const double q = norm2[j];
        if (q > b) { s2 = b; b = q; bi = j; }
        else if (q > s2) { s2 = q; }
      }
      tbest[t] = b; tsecond[t] = s2; tidx[t] = bi;
    }
    double best = -1.0, second = -1.0;
    int64_t bj = -1;
    for (int t = 0; t < nthreads; ++t) {  // threads own ascending index ranges
      if (tidx[t] < 0) { second = std::max(second, tsecond[t]); continue; }
      if (tbest[t] > best) { second = std::max(second, best); best = tbest[t]; bj = tidx[t]; }
      else { second = std::max(second, tbest[t]); }
      second = std::max(second, tsecond[t]);
    }
    if (bj < 0) return pifa_fail(PIFA_ERR_RANK_DEFICIENT, "pifa_compress: ran out of rows");
    const double nb = std::sqrt(std::max(best, 0.0));
    const double ns = std::sqrt(std::max(second, 0.0));
    if (second >= 0.0 && nb > 0.0) min_gap = std::min(min_gap, (nb - ns) / nb);
    // reflect the pivot column onto e_k
    double* zp = &Z[(size_t)bj * r];
    const double alpha = make_reflector(zp + k, r - k, v.data());
    zp[k] = alpha;
    for (int64_t a = k + 1; a < r; ++a) zp[a] = 0.0;
    chosen[bj] = 1;
    order.push_back(bj);
    rdiag[k] = std::fabs(alpha);
    // apply to every unchosen column and recompute its residual norm over rows k+1..r-1
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < m; ++j) {
      if (chosen[j]) continue;
      double* z = &Z[(size_t)j * r + k];
      const int64_t len = r - k;
      double s = 0.0;
      for (int64_t a = 0; a < len; ++a) s += v[a] * z[a];
      s *= 2.0;
      double q = 0.0;
      z[0] -= s * v[0];
      for (int64_t a = 1; a < len; ++a) {
        z[a] -= s * v[a];
        q += z[a] * z[a];
      }
      norm2[j] = q;
    }
  }
  if (!(rdiag[0] > 0.0) || !(rdiag[r - 1] >= 1e-8 * rdiag[0]))
    return pifa_fail(PIFA_ERR_RANK_DEFICIENT,
                     "pifa_compress: |R_(r-1,r-1)| < 1e-8 |R_00| (W' has rank < r)");

  // --- I, I^c ascending --------------------------------------------------------------------
  std::vector<int64_t> sorted(order);
  std::sort(sorted.begin(), sorted.end());
  std::vector<int64_t> pos_of(m, -1);  // row -> position in ascending I
  for (int64_t a = 0; a < r; ++a) {
    pivot_idx[a] = (int32_t)sorted[a];
    pos_of[sorted[a]] = a;
  }
  std::vector<int64_t> nonp;
  nonp.reserve(m - r);
  for (int64_t j = 0; j < m; ++j)
    if (!chosen[j]) nonp.push_back(j);
  for (int64_t i = 0; i < m - r; ++i) nonpivot_idx[i] = (int32_t)nonp[i];

  // --- C = (R11^{-1} R12)^T, columns permuted from greedy order to ascending I -------------
  double max_abs_c = 0.0;
  if (m > r) {
    std::vector<double> R11((size_t)r * r, 0.0);  // row-major upper triangular
    for (int64_t q = 0; q < r; ++q) {
      const double* zc = &Z[(size_t)order[q] * r];
      for (int64_t p = 0; p <= q; ++p) R11[p * r + q] = zc[p];
    }
    const int64_t NB = 16;
    const int64_t nblk = (m - r + NB - 1) / NB;
    double mx = 0.0;
#pragma omp parallel for schedule(dynamic, 4) reduction(max : mx)
    for (int64_t blk = 0; blk < nblk; ++blk) {
      const int64_t i0 = blk * NB, i1 = std::min<int64_t>(m - r, i0 + NB), nb_ = i1 - i0;
      std::vector<double> t((size_t)r * NB, 0.0);  // t[p * NB + b]
      for (int64_t p = r - 1; p >= 0; --p) {
        double acc[NB];
        for (int64_t b = 0; b < NB; ++b) acc[b] = 0.0;
        const double* Rp = &R11[(size_t)p * r];
        for (int64_t q = p + 1; q < r; ++q) {
          const double rq = Rp[q];
          const double* tq = &t[(size_t)q * NB];
          for (int64_t b = 0; b < NB; ++b) acc[b] += rq * tq[b];
        }
        for (int64_t b = 0; b < nb_; ++b) {
          const double zb = Z[(size_t)nonp[i0 + b] * r + p];
          t[(size_t)p * NB + b] = (zb - acc[b]) / Rp[p];
        }
      }
      for (int64_t b = 0; b < nb_; ++b) {
        double* crow = C + (i0 + b) * ldc;
        for (int64_t p = 0; p < r; ++p) {
          const double c = t[(size_t)p * NB + b];
          crow[pos_of[order[p]]] = c;
          mx = std::max(mx, std::fabs(c));
        }
      }
    }
    max_abs_c = mx;
  }

  // --- W_p = U[I, :] V^T -------------------------------------------------------------------
  {
    std::vector<double> Up((size_t)r * r);
    for (int64_t a = 0; a < r; ++a) std::memcpy(&Up[(size_t)a * r], U + sorted[a] * r, sizeof(double) * r);
    gemm_nt(r, n, r, Up.data(), r, V, r, Wp, ldwp);
  }

  if (info) {
    info->min_pivot_gap = min_gap;
    info->r_ratio = rdiag[r - 1] / rdiag[0];
    info->max_abs_c = max_abs_c;
    info->threads = nthreads;
  }
  return PIFA_OK;
}
