// api.cpp -- host side of the C ABI in include/pifa.h: argument checks, the variant selector,
// workspace sizing, dispatch to the kernel launchers, TMA descriptor encoding, error strings.
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <atomic>
#include <mutex>
#include <string>

#include <cuda.h>
#include <cuda_runtime.h>

#include "pifa.h"
#include "pifa_internal.h"

namespace {

thread_local std::string g_last_error;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Byte span [lo, hi) covered by a row-major matrix of `rows` rows, `cols` used columns, pitch ld.
struct Span {
  uintptr_t lo, hi;
};
Span span_of(const void* base, int64_t rows, int64_t cols, int64_t ld, int64_t elem) {
  const uintptr_t b = reinterpret_cast<uintptr_t>(base);
  if (!base || rows <= 0 || cols <= 0) return {0, 0};
  return {b, b + (uintptr_t)(((rows - 1) * ld + cols) * elem)};
}
bool overlaps(Span a, Span b) { return a.lo < a.hi && b.lo < b.hi && a.lo < b.hi && b.lo < a.hi; }

int validate_shape(int64_t T, int64_t m, int64_t n, int64_t r) {
  if (T < 0) return pifa_fail(PIFA_ERR_INVALID_ARG, "T must be >= 0");
  if (m < 1 || n < 1 || r < 1 || r > m || r > n)
    return pifa_fail(PIFA_ERR_INVALID_ARG, "need 1 <= r <= min(m, n)");
  const int64_t lim = (int64_t)1 << 30;
  if (T >= lim || m >= lim || n >= lim) return pifa_fail(PIFA_ERR_INVALID_ARG, "T, m or n too large (>= 2^30)");
  return PIFA_OK;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

}  // namespace

// ---- internal helpers used by the kernel files --------------------------------------------------
void pifa_clear_error() { g_last_error.clear(); }

int pifa_fail(int status, const char* msg) {
  g_last_error = msg ? msg : "";
  return status;
}

int pifa_fail_cuda(const char* where, cudaError_t err) {
  g_last_error = std::string(where) + ": " + cudaGetErrorName(err) + " (" + cudaGetErrorString(err) + ")";
  return PIFA_ERR_CUDA;
}

namespace {
uint64_t default_wait_timeout_ns() {
  const char* e = std::getenv("PIFA_WAIT_TIMEOUT_NS");
  if (e && *e) return (uint64_t)std::strtoull(e, nullptr, 10);
  return (uint64_t)1000000000ull;  // 1 s
}
std::atomic<uint64_t> g_wait_timeout_ns{default_wait_timeout_ns()};
}  // namespace

uint64_t pifa_wait_timeout_ns() { return g_wait_timeout_ns.load(std::memory_order_relaxed); }

int make_tmap_2d(CUtensorMap* map, int dtype, const void* base, int64_t rows, int64_t cols, int64_t ld,
                 uint32_t box_cols, uint32_t box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return pifa_fail(PIFA_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * 2)};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapDataType dt =
      dtype == PIFA_DTYPE_FP16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUresult r = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char buf[160];
    std::snprintf(buf, sizeof buf, "cuTensorMapEncodeTiled failed (CUresult %d) for %lld x %lld, ld %lld",
                  (int)r, (long long)rows, (long long)cols, (long long)ld);
    return pifa_fail(PIFA_ERR_CUDA, buf);
  }
  return PIFA_OK;
}

// ---- public API ---------------------------------------------------------------------------------
extern "C" {

const char* pifa_version(void) { return "libpifa 0.1 (sm_103a)"; }

int pifa_set_wait_timeout(int64_t ns) {
  if (ns < 0) return pifa_fail(PIFA_ERR_INVALID_ARG, "timeout must be >= 0");
  g_wait_timeout_ns.store(ns == 0 ? default_wait_timeout_ns() : (uint64_t)ns, std::memory_order_relaxed);
  return PIFA_OK;
}

const char* pifa_last_error(void) { return g_last_error.c_str(); }

const char* pifa_status_string(int status) {
  switch (status) {
    case PIFA_OK: return "PIFA_OK";
    case PIFA_ERR_INVALID_ARG: return "PIFA_ERR_INVALID_ARG";
    case PIFA_ERR_ALIGNMENT: return "PIFA_ERR_ALIGNMENT";
    case PIFA_ERR_UNSUPPORTED: return "PIFA_ERR_UNSUPPORTED";
    case PIFA_ERR_CUDA: return "PIFA_ERR_CUDA";
    case PIFA_ERR_TIMEOUT: return "PIFA_ERR_TIMEOUT";
    case PIFA_ERR_RANK_DEFICIENT: return "PIFA_ERR_RANK_DEFICIENT";
    case PIFA_ERR_WORKSPACE: return "PIFA_ERR_WORKSPACE";
    case PIFA_ERR_DEVICE_INDEX: return "PIFA_ERR_DEVICE_INDEX";
    case PIFA_ERR_RANGE: return "PIFA_ERR_RANGE";
    default: return "PIFA_ERR_UNKNOWN";
  }
}

const char* pifa_variant_name(int variant) {
  switch (variant) {
    case PIFA_VARIANT_AUTO: return "auto";
    case PIFA_VARIANT_DECODE: return "decode";
    case PIFA_VARIANT_PREFILL_SPLIT: return "prefill_split";
    case PIFA_VARIANT_PREFILL_FUSED: return "prefill_fused";
    default: return "?";
  }
}

}  // extern "C"

namespace {

// Whether the decode variant runs T tokens of G layers of this shape: any T <= 64; up to 128 when
// both phases (G r and G (m - r) rows) have at most kWideRowBlocks blocks of 128 rows, the limit of
// the row-block plan that 128-token tiles need on every sm_103a part (two CTAs on each of 148 SMs).
constexpr int64_t kWideRowBlocks = 296;
bool decode_takes(int64_t T, int64_t G, int64_t m, int64_t r) {
  if (T <= 64) return true;
  if (T > 128) return false;
  return (G * r + 127) / 128 <= kWideRowBlocks && (G * (m - r) + 127) / 128 <= kWideRowBlocks;
}

// The selector. Decode streams each weight once with every token's product per tile; against the
// split prefill (one process, interleaved, us) it measured 2.0-2.8x faster at T = 24 / 32 / 64 on
// the LLaMA-2 7B and 70B layers, whose prefill GEMMs hold one token tile at such T. From T = 65 the
// prefill's split-K clusters catch up on layers of few non-pivot rows (T = 128: 7B attention 26.9
// against 30.2, 7B MLP gate 36.2 against 39.3, 70B q/o 41.4 against 41.8; at T = 96 within 2-7%
// either way), while on a non-pivot phase of at least one 128-row block per SM decode keeps its
// lead (70B gate/up, 192 blocks: T = 128 83.7 against 124.4). So: decode for T <= 64, and up to 128
// where the non-pivot rows make at least kWideRowBlocks / 2 blocks.
int select_for(int64_t T, int64_t G, int64_t m, int64_t r) {
  if (T <= 64) return PIFA_VARIANT_DECODE;
  if (decode_takes(T, G, m, r) && (G * (m - r) + 127) / 128 >= kWideRowBlocks / 2) return PIFA_VARIANT_DECODE;
  return PIFA_VARIANT_PREFILL_SPLIT;
}
}  // namespace

extern "C" {

int pifa_select_variant(int64_t T, int64_t m, int64_t n, int64_t r, int c_dtype) {
  int st = validate_shape(T, m, n, r);
  if (st != PIFA_OK) return st;
  if (c_dtype != PIFA_DTYPE_BF16 && c_dtype != PIFA_DTYPE_FP16) return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown c_dtype");
  return select_for(T, 1, m, r);
}

int64_t pifa_workspace_size(int64_t T, int64_t m, int64_t n, int64_t r, int c_dtype, int variant) {
  int st = validate_shape(T, m, n, r);
  if (st != PIFA_OK) return st;
  if (c_dtype != PIFA_DTYPE_BF16 && c_dtype != PIFA_DTYPE_FP16) return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown c_dtype");
  if (variant == PIFA_VARIANT_AUTO) variant = pifa_select_variant(T, m, n, r, c_dtype);
  PifaShape s = {T, m, n, r, n, n, r, m, c_dtype};
  if (T == 0) return 0;
  switch (variant) {
    case PIFA_VARIANT_DECODE: return kWorkspaceReserve + decode_workspace_bytes(s);
    case PIFA_VARIANT_PREFILL_SPLIT: return kWorkspaceReserve + prefill_split_workspace_bytes(s);
    case PIFA_VARIANT_PREFILL_FUSED: return pifa_fail(PIFA_ERR_UNSUPPORTED, "variant not built in this version");
    default: return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown variant");
  }
}

}  // extern "C"

namespace {

// Extra conditions on G layers sharing X (groups > 1): each group's non-pivot rows a whole number
// of 128-row tiles and its y_p columns 16-byte aligned. PIFA_OK or the failure.
int validate_groups(int64_t groups, int64_t m, int64_t r) {
  if (groups < 1 || groups > 64) return pifa_fail(PIFA_ERR_INVALID_ARG, "groups must be in [1, 64]");
  if (groups == 1) return PIFA_OK;
  if (m == r) return pifa_fail(PIFA_ERR_UNSUPPORTED, "grouped layers need m > r");
  if ((m - r) % 128 != 0 || r % 8 != 0)
    return pifa_fail(PIFA_ERR_UNSUPPORTED, "grouped layers need (m - r) % 128 == 0 and r % 8 == 0");
  if (groups * m >= ((int64_t)1 << 30)) return pifa_fail(PIFA_ERR_INVALID_ARG, "groups * m too large (>= 2^30)");
  return PIFA_OK;
}

int64_t workspace_bytes_for(const PifaShape& s, int variant) {
  switch (variant) {
    case PIFA_VARIANT_DECODE: return kWorkspaceReserve + decode_workspace_bytes(s);
    case PIFA_VARIANT_PREFILL_SPLIT: return kWorkspaceReserve + prefill_split_workspace_bytes(s);
    case PIFA_VARIANT_PREFILL_FUSED: return pifa_fail(PIFA_ERR_UNSUPPORTED, "variant not built in this version");
    default: return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown variant");
  }
}

// Algorithm 2 for `groups` layers of one shape sharing X (groups == 1: one layer).
int forward_impl(int64_t groups, const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp, int64_t r,
                 int64_t ldwp, const void* C, int64_t m, int64_t ldc, int c_dtype, const int32_t* pivot_idx,
                 const int32_t* nonpivot_idx, void* Y, int64_t ldy, void* workspace, int64_t workspace_bytes,
                 int variant, void* cuda_stream) {
  pifa_clear_error();
  int st = validate_shape(T, m, n, r);
  if (st != PIFA_OK) return st;
  if ((st = validate_groups(groups, m, r)) != PIFA_OK) return st;
  const int64_t G = groups;
  const bool has_np = m > r;
  if (c_dtype != PIFA_DTYPE_BF16 && c_dtype != PIFA_DTYPE_FP16) return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown c_dtype");
  if (T == 0) return PIFA_OK;  // no-op: nothing is read or written (X and Y may be null)
  if (!X || !Wp || !pivot_idx || !Y) return pifa_fail(PIFA_ERR_INVALID_ARG, "null X, Wp, pivot_idx or Y");
  if (has_np && (!C || !nonpivot_idx)) return pifa_fail(PIFA_ERR_INVALID_ARG, "null C or nonpivot_idx with m > r");
  if (ldx < n || ldwp < n || ldy < G * m || (has_np && ldc < r))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row length");
  if (!aligned16(X) || !aligned16(Wp) || !aligned16(Y) || (has_np && !aligned16(C)))
    return pifa_fail(PIFA_ERR_ALIGNMENT, "X, Wp, C and Y must be 16-byte aligned");
  if ((ldx | ldwp | ldy | (has_np ? ldc : 0)) & 7)
    return pifa_fail(PIFA_ERR_ALIGNMENT, "ldx, ldwp, ldc and ldy must be multiples of 8 elements");
  if (variant < PIFA_VARIANT_AUTO || variant > PIFA_VARIANT_PREFILL_FUSED)
    return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown variant");
  {
    const Span y = span_of(Y, T, G * m, ldy, 2);
    if (overlaps(y, span_of(X, T, n, ldx, 2)) || overlaps(y, span_of(Wp, G * r, n, ldwp, 2)) ||
        (has_np && overlaps(y, span_of(C, G * (m - r), r, ldc, 2))))
      return pifa_fail(PIFA_ERR_INVALID_ARG, "Y overlaps an input");
  }
  if (variant == PIFA_VARIANT_AUTO) variant = select_for(T, G, m, r);

  PifaShape s = {T, m, n, r, ldx, ldwp, has_np ? ldc : r, ldy, c_dtype};
  s.groups = G;
  if (variant == PIFA_VARIANT_DECODE && !decode_takes(T, G, m, r))
    return pifa_fail(PIFA_ERR_UNSUPPORTED,
                     "decode variant needs T <= 64, or T <= 128 with at most 296 row blocks of 128 per phase");
  const int64_t need = workspace_bytes_for(s, variant);
  if (need < 0) return (int)need;
  if (!workspace || workspace_bytes < need)
    return pifa_fail(PIFA_ERR_WORKSPACE, "workspace missing or smaller than pifa_workspace_size()");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u)
    return pifa_fail(PIFA_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  {
    // the kernels write y_p into the workspace: it must not share a byte with Y or an input
    const Span w = {reinterpret_cast<uintptr_t>(workspace), reinterpret_cast<uintptr_t>(workspace) + (uintptr_t)need};
    if (overlaps(w, span_of(Y, T, G * m, ldy, 2)) || overlaps(w, span_of(X, T, n, ldx, 2)) ||
        overlaps(w, span_of(Wp, G * r, n, ldwp, 2)) || (has_np && overlaps(w, span_of(C, G * (m - r), r, ldc, 2))))
      return pifa_fail(PIFA_ERR_INVALID_ARG, "workspace overlaps Y or an input");
  }
  cudaError_t cerr = cudaSuccess;
  int* status = pifa_status_word(&cerr);
  if (!status) return pifa_fail_cuda("device status word", cerr);

  PifaPointers p = {X, Wp, has_np ? C : nullptr, pivot_idx, has_np ? nonpivot_idx : nullptr, Y,
                    static_cast<uint8_t*>(workspace) + kWorkspaceReserve, workspace_bytes - kWorkspaceReserve};
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(cuda_stream);
  switch (variant) {
    case PIFA_VARIANT_DECODE: return launch_decode(s, p, status, stream);
    case PIFA_VARIANT_PREFILL_SPLIT: return launch_prefill_split(s, p, status, pifa_wait_timeout_ns(), stream);
  }
  return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown variant");
}

}  // namespace

extern "C" {

int pifa_forward_variant(const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp, int64_t r, int64_t ldwp,
                         const void* C, int64_t m, int64_t ldc, int c_dtype, const int32_t* pivot_idx,
                         const int32_t* nonpivot_idx, void* Y, int64_t ldy, void* workspace,
                         int64_t workspace_bytes, int variant, void* cuda_stream) {
  return forward_impl(1, X, T, n, ldx, Wp, r, ldwp, C, m, ldc, c_dtype, pivot_idx, nonpivot_idx, Y, ldy, workspace,
                      workspace_bytes, variant, cuda_stream);
}

int pifa_forward_grouped(int64_t groups, const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp, int64_t r,
                         int64_t ldwp, const void* C, int64_t m, int64_t ldc, int c_dtype, const int32_t* pivot_idx,
                         const int32_t* nonpivot_idx, void* Y, int64_t ldy, void* workspace, int64_t workspace_bytes,
                         void* cuda_stream) {
  return forward_impl(groups, X, T, n, ldx, Wp, r, ldwp, C, m, ldc, c_dtype, pivot_idx, nonpivot_idx, Y, ldy,
                      workspace, workspace_bytes, PIFA_VARIANT_AUTO, cuda_stream);
}

int64_t pifa_workspace_size_grouped(int64_t groups, int64_t T, int64_t m, int64_t n, int64_t r, int c_dtype) {
  int st = validate_shape(T, m, n, r);
  if (st != PIFA_OK) return st;
  if ((st = validate_groups(groups, m, r)) != PIFA_OK) return st;
  if (c_dtype != PIFA_DTYPE_BF16 && c_dtype != PIFA_DTYPE_FP16) return pifa_fail(PIFA_ERR_INVALID_ARG, "unknown c_dtype");
  if (T == 0) return 0;
  PifaShape s = {T, m, n, r, n, n, r, groups * m, c_dtype};
  s.groups = groups;
  return workspace_bytes_for(s, select_for(T, groups, m, r));
}

int pifa_forward(const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp, int64_t r, int64_t ldwp,
                 const void* C, int64_t m, int64_t ldc, int c_dtype, const int32_t* pivot_idx,
                 const int32_t* nonpivot_idx, void* Y, int64_t ldy, void* workspace, int64_t workspace_bytes,
                 void* cuda_stream) {
  return pifa_forward_variant(X, T, n, ldx, Wp, r, ldwp, C, m, ldc, c_dtype, pivot_idx, nonpivot_idx, Y, ldy, workspace,
                              workspace_bytes, PIFA_VARIANT_AUTO, cuda_stream);
}

int pifa_validate_indices(const int32_t* pivot_idx, const int32_t* nonpivot_idx, int64_t m, int64_t r) {
  pifa_clear_error();
  if (m < 1 || r < 1 || r > m) return pifa_fail(PIFA_ERR_INVALID_ARG, "need 1 <= r <= m");
  if (!pivot_idx || (m > r && !nonpivot_idx)) return pifa_fail(PIFA_ERR_INVALID_ARG, "null index array");
  // strictly ascending and inside [0, m) each; disjoint by a merge walk (together they then
  // cover r + (m - r) = m distinct values of [0, m), i.e. a partition)
  for (int64_t a = 0; a < r; ++a) {
    if (pivot_idx[a] < 0 || pivot_idx[a] >= m) return pifa_fail(PIFA_ERR_INVALID_ARG, "pivot index out of range");
    if (a > 0 && pivot_idx[a] <= pivot_idx[a - 1]) return pifa_fail(PIFA_ERR_INVALID_ARG, "pivot_idx not ascending");
  }
  for (int64_t a = 0; a < m - r; ++a) {
    if (nonpivot_idx[a] < 0 || nonpivot_idx[a] >= m)
      return pifa_fail(PIFA_ERR_INVALID_ARG, "non-pivot index out of range");
    if (a > 0 && nonpivot_idx[a] <= nonpivot_idx[a - 1])
      return pifa_fail(PIFA_ERR_INVALID_ARG, "nonpivot_idx not ascending");
  }
  int64_t i = 0, j = 0;
  while (i < r && j < m - r) {
    if (pivot_idx[i] == nonpivot_idx[j]) return pifa_fail(PIFA_ERR_INVALID_ARG, "index in both sets");
    if (pivot_idx[i] < nonpivot_idx[j]) ++i; else ++j;
  }
  return PIFA_OK;
}

int pifa_device_status(void* cuda_stream) {
  pifa_clear_error();
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaStreamSynchronize", e);
  int* word = pifa_status_word(&e);
  if (!word) return pifa_fail_cuda("device status word", e);
  int v = 0;
  e = cudaMemcpy(&v, word, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return pifa_fail_cuda("read status word", e);
  e = cudaMemset(word, 0, sizeof(int));
  if (e != cudaSuccess) return pifa_fail_cuda("clear status word", e);
  return v;
}

}  // extern "C"
