// pifa_internal.h -- declarations shared by the host API (api.cpp) and the kernel files (*.cu).
// Not installed; the public interface is include/pifa.h.
#ifndef PIFA_INTERNAL_H_
#define PIFA_INTERNAL_H_

#include <stdint.h>

#include <cuda.h>
#include <cuda_runtime.h>

// ---- error reporting (api.cpp) ---------------------------------------------------------------
void pifa_clear_error();
int pifa_fail(int status, const char* msg);                       // records msg, returns status
int pifa_fail_cuda(const char* where, cudaError_t err);           // PIFA_ERR_CUDA with detail

// Device status word of the current device (api.cpp). Kernels latch the first error into it
// with atomicCAS(word, 0, code).
int* pifa_status_word(cudaError_t* err);

// Default bound of every device-side wait, nanoseconds (env PIFA_WAIT_TIMEOUT_NS overrides).
uint64_t pifa_wait_timeout_ns();

// Kernels this library has enqueued (status.cu): every launch site calls pifa_count_launch() once
// per successful launch; pifa_launch_count() reads the total.
void pifa_count_launch();

// Up to two side streams for independent work inside one call (status.cu): fork(i) makes side
// stream i wait for the work enqueued on the caller's stream so far and returns it; the destructor
// makes the caller's stream wait for every side stream that was forked. Per host thread and device.
class PifaSides {
 public:
  explicit PifaSides(cudaStream_t main) : main_(main) {}
  ~PifaSides();
  PifaSides(const PifaSides&) = delete;
  PifaSides& operator=(const PifaSides&) = delete;
  int fork(int i, cudaStream_t* side);  // PIFA_OK or PIFA_ERR_CUDA

 private:
  cudaStream_t main_;
  void* state_ = nullptr;
  bool forked_[2] = {false, false};
};

#ifdef __CUDACC__
#include <utility>
// cudaLaunchKernelEx, counted.
template <typename... K, typename... A>
inline cudaError_t pifa_launch_ex(const cudaLaunchConfig_t* cfg, void (*kernel)(K...), A&&... args) {
  const cudaError_t e = cudaLaunchKernelEx(cfg, kernel, std::forward<A>(args)...);
  if (e == cudaSuccess) pifa_count_launch();
  return e;
}
#endif

// Shape of one forward call after validation (element counts and pitches).
struct PifaShape {
  int64_t T, m, n, r;
  int64_t ldx, ldwp, ldc, ldy;
  int c_dtype;  // PIFA_DTYPE_BF16 or PIFA_DTYPE_FP16 (storage type of C)
  // G layers of one shape sharing X (pifa_forward_grouped): W_p holds G r rows, C G (m - r) rows,
  // Y G m columns (the pivot / non-pivot indices are absolute columns of Y), y_p G r columns; the
  // non-pivot rows of group g read y_p's columns [g r, (g + 1) r). G > 1 needs (m - r) % 128 == 0
  // and r % 8 == 0, so that no tile spans two groups and every group's y_p columns start 16-byte
  // aligned.
  int64_t groups = 1;
};

// The first kWorkspaceReserve bytes of every workspace are reserved for library state (no kernel
// of this version uses them); per-call scratch starts after them.
constexpr int64_t kWorkspaceReserve = 256;

struct PifaPointers {
  const void* X;
  const void* Wp;
  const void* C;
  const int32_t* piv;
  const int32_t* nonpiv;
  void* Y;
  void* ws;           // per-call scratch (workspace + kWorkspaceReserve)
  int64_t ws_bytes;   // bytes available at ws
};

// Byte span [lo, hi) of a row-major matrix (rows x cols used elements, pitch ld, elem bytes);
// empty for a null base or no rows/columns. Used to reject outputs that overlap inputs.
struct PifaSpan {
  uintptr_t lo, hi;
};
inline PifaSpan pifa_span(const void* base, int64_t rows, int64_t cols, int64_t ld, int64_t elem) {
  const uintptr_t b = reinterpret_cast<uintptr_t>(base);
  if (!base || rows <= 0 || cols <= 0) return {0, 0};
  return {b, b + (uintptr_t)(((rows - 1) * ld + cols) * elem)};
}
inline bool pifa_spans_overlap(PifaSpan a, PifaSpan b) {
  return a.lo < a.hi && b.lo < b.hi && a.lo < b.hi && b.lo < a.hi;
}

// ---- decode (decode.cu) ----------------------------------------------------------------------
int64_t decode_workspace_bytes(const PifaShape& s);
int launch_decode(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream);

// ---- decode on the tensor cores, split over K (decode_tc.cu) ------------------------------------
// One decode phase D = A B^T (A: R x K weight rows, B: T <= 128 token rows of K columns, NB =
// planes 1 or 2) as a split-K tcgen05 kernel: row blocks in clusters that add up their K-slices
// and write Y[t, cols[j]] (and, for phase 1, the y_p hi/lo planes) themselves, or, for phases of
// more row blocks than the grid holds, balanced ranges writing fp32 partial sums P and a reduction.
struct DecodeTcPhase {
  const void* A;
  int64_t lda, R, K;
  int dtype;            // storage type of A and B (PIFA_DTYPE_*)
  const void* B0;       // first (or only) B plane: T x bcols, pitch ldb
  const void* B1;       // second plane (planes == 2)
  int64_t ldb, bcols, T;
  int planes;
  int64_t gsz, goff;    // grouped layers: rows per group and B columns per group (0: one layer)
  bool mma_f16;         // A and B fp16 (else bf16)
  bool split_f16;       // phase 1: split y_p into fp16 hi/lo (else bf16)
  float* P;             // partial sums, decode_tc_partial_bytes(R, K, T, planes) bytes
  const int32_t* cols;  // output column of each weight row
  int64_t m;            // columns of Y (index bound)
  void* Y;
  int64_t ldy;
  uint16_t* yph;        // phase 1 with m > r: y_p planes (T x ldyp), else null
  uint16_t* ypl;
  int64_t ldyp;
};
int64_t decode_tc_partial_bytes(int64_t R, int64_t K, int64_t T, int NB);
int launch_decode_tc(const DecodeTcPhase& ph, int* status, uint64_t timeout_ns, cudaStream_t stream);

// ---- general tensor-core contraction (gemm_tc.cu) ------------------------------------------------
// D (M x N) = alpha A B^T (+ addend), bf16 operands, fp32 accumulation. A is M x K, B is N x K; each
// is K-major (a_mn = false: element (i, k) at [i * ld + k]) or MN-major (true: at [k * ld + i]).
// out_mode 0: D bf16; 1: D fp32; 2: D fp32 += result; 3: D = bf16 hi, D2 = bf16 lo of the result.
// A2 / B2 (optional, A's / B's layout and pitch): a second K pass with A2 for A and / or B2 for B,
// D = (A + A2) B^T or A (B + B2)^T. Optional addend:
// D[i][j] += add[i * ldadd + (add_idx ? add_idx[j] : j)] (bf16; add_idx values must lie in
// [0, add_bound)). Pointers 16-byte aligned, leading dimensions multiples of 8 elements (the caller
// checks).
struct GemmTc {
  int64_t M, N, K;
  const void* A;
  int64_t lda;
  bool a_mn;
  const void* B;
  int64_t ldb;
  bool b_mn;
  void* D;
  int64_t ldd;
  int out_mode;
  float alpha;
  const void* add;
  const int32_t* add_idx;
  int64_t ldadd;
  int64_t add_bound;
  const void* A2 = nullptr;
  const void* B2 = nullptr;
  void* D2 = nullptr;
  bool d_trans = false;  // store D^T: element (i, j) at D[j * ldd + i] (out_mode 0, 1 or 3 only)
  bool upper = false;    // M == N: skip tiles wholly below the diagonal (a symmetric product's upper triangle)
};
int gemm_tc(const GemmTc& g, int* status, uint64_t timeout_ns, cudaStream_t stream);

// ---- prefill (prefill.cu) --------------------------------------------------------------------
int64_t prefill_split_workspace_bytes(const PifaShape& s);
int launch_prefill_split(const PifaShape& s, const PifaPointers& p, int* status, uint64_t timeout_ns,
                         cudaStream_t stream);

// ---- TMA descriptors (api.cpp) ---------------------------------------------------------------
// 2-D tensor map over a row-major (rows x cols) matrix of 2-byte elements (bf16 or fp16, a
// PIFA_DTYPE_*) with row pitch `ld` elements; box of box_cols x box_rows elements, 128-byte
// swizzle, zero fill outside the matrix.
int make_tmap_2d(CUtensorMap* map, int dtype, const void* base, int64_t rows, int64_t cols, int64_t ld,
                 uint32_t box_cols, uint32_t box_rows);

#endif  // PIFA_INTERNAL_H_
