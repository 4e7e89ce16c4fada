/*
 * pifa.h -- C ABI of libpifa: the forward pass of a Pivoting Factorization (PIFA) layer on
 * NVIDIA GB300 (sm_103a), plus a host-side reference compression.
 *
 * A rank-r weight W' (m x n) is stored as (Sec. 3.2, Eqs. 1-2):
 *   I    -- pivot-row indices, r of them (Algorithm 1, step 1);
 *   I^c  -- the other m - r row indices (Algorithm 1, step 2);
 *   W_p  -- the pivot rows W'[I, :], r x n (Eq. 1);
 *   C    -- coefficients with W'[I^c, :] = C W_p, (m - r) x r (Eq. 2).
 * The forward pass (Algorithm 2) maps activations to outputs:
 *   Y_p = W_p X,  Y_np = C Y_p,  Y[I, :] = Y_p,  Y[I^c, :] = Y_np.
 * The paper writes activations as columns (X is n x b). This library keeps tokens as ROWS:
 * X is T x n row-major and Y = X W'^T is T x m row-major, so Y_p = X W_p^T (T x r) and
 * Y_np = Y_p C^T (T x (m - r)); output column I[j] receives Y_p[:, j] and column I^c[i]
 * receives Y_np[:, i].
 *
 * Conventions for every call:
 *  - Status codes are returned (pifa_status); nothing aborts. pifa_status_string() names them
 *    and pifa_last_error() gives the calling thread's last detailed message.
 *  - Sizes and leading dimensions are counts of ELEMENTS, int64_t.
 *  - Matrices are row-major; a leading dimension is the distance between consecutive rows.
 *  - Device buffers are caller-owned. The library never keeps a pointer past the call and
 *    allocates no device memory in pifa_forward (scratch comes from the caller's workspace).
 *  - bf16 means IEEE-style bfloat16 (1 sign, 8 exponent, 7 mantissa bits); accumulation is fp32.
 */
#ifndef PIFA_H_
#define PIFA_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PIFA_OK = 0,
  PIFA_ERR_INVALID_ARG = -1,     /* null pointer, bad size or leading dimension, bad index set  */
  PIFA_ERR_ALIGNMENT = -2,       /* a base pointer or row pitch is not 16-byte aligned          */
  PIFA_ERR_UNSUPPORTED = -3,     /* shape/variant combination this build does not implement    */
  PIFA_ERR_CUDA = -4,            /* a CUDA runtime/driver call failed (see pifa_last_error)    */
  PIFA_ERR_TIMEOUT = -5,         /* a device-side bounded wait gave up (kernel returned early) */
  PIFA_ERR_RANK_DEFICIENT = -6,  /* W' = U V^T has fewer than r independent rows               */
  PIFA_ERR_WORKSPACE = -7,       /* workspace missing or smaller than pifa_workspace_size()    */
  PIFA_ERR_DEVICE_INDEX = -8,    /* a kernel met a pivot/non-pivot index outside [0, m)       */
  PIFA_ERR_RANGE = -9            /* a Y_p value exceeded the fp16 range (C stored as fp16)      */
} pifa_status;

/* Storage type of C. W_p, X and Y are always bf16. C may be bf16 or fp16 (both 2 bytes per
 * element). Y_p enters the second contraction as a hi + lo pair of C's type (bf16: 16
 * significant bits, fp16: 22). Y_p values beyond +-65504 cannot be represented in fp16: with
 * fp16 C they saturate and PIFA_ERR_RANGE is latched. */
typedef enum { PIFA_DTYPE_BF16 = 0, PIFA_DTYPE_FP16 = 1 } pifa_dtype;

/* Forward-pass implementations. PIFA_VARIANT_AUTO lets the selector choose (see
 * pifa_select_variant). The others force one implementation; a forced variant that cannot run
 * the given shape returns PIFA_ERR_UNSUPPORTED. */
typedef enum {
  PIFA_VARIANT_AUTO = 0,
  PIFA_VARIANT_DECODE = 1,        /* T <= 128: two HBM-streaming phases (mma.sync or tcgen05)    */
  PIFA_VARIANT_PREFILL_SPLIT = 2, /* tcgen05 GEMM 1 -> Y_p in workspace -> tcgen05 GEMM 2        */
  PIFA_VARIANT_PREFILL_FUSED = 3  /* reserved: not built in this version (PIFA_ERR_UNSUPPORTED)   */
} pifa_variant;

/* Diagnostics of pifa_compress (all optional to read). */
typedef struct {
  double min_pivot_gap;   /* min over greedy steps of (best - runner_up) / best residual norm  */
  double r_ratio;         /* |R_(r-1,r-1)| / |R_00| of the pivoted QR                          */
  double max_abs_c;       /* max |C_ij|                                                         */
  int32_t threads;        /* host threads used                                                  */
} pifa_compress_info;

/*
 * pifa_forward -- Algorithm 2 (Sec. 3.2) on the GPU, asynchronously on `cuda_stream`.
 *
 *   X            DEVICE, bf16, T x n, row pitch ldx >= n.
 *   Wp           DEVICE, bf16, r x n, row pitch ldwp >= n (row j is W'[I[j], :]).
 *   C            DEVICE, (m - r) x r, row pitch ldc >= r (row i gives W'[I^c[i], :]), stored as
 *                c_dtype (a pifa_dtype: bf16 or fp16). May be NULL when r == m.
 *   pivot_idx    DEVICE, int32[r], strictly ascending, values in [0, m).
 *   nonpivot_idx DEVICE, int32[m - r], strictly ascending; together with pivot_idx a partition
 *                of [0, m). May be NULL when r == m.
 *   Y            DEVICE, bf16, T x m, row pitch ldy >= m. Every element Y[t, 0..m-1] is written
 *                exactly once (round to nearest even from the fp32 accumulator); the padding
 *                columns m..ldy-1 are not touched. Y must not overlap any input.
 *   workspace    DEVICE scratch of at least pifa_workspace_size(T, m, n, r, c_dtype, variant) bytes,
 *                256-byte aligned; it needs no initialisation. Its first 256 bytes are reserved
 *                for library state (no kernel of this version reads or writes them); the rest
 *                holds Y_p between the two contractions and the split-K decode's fp32 partial sums. It must not overlap Y or an input
 *                (PIFA_ERR_INVALID_ARG; only the first pifa_workspace_size() bytes are checked),
 *                nor be used by another call that may run concurrently.
 *   cuda_stream  a cudaStream_t (NULL = legacy default stream).
 *
 *   Every matrix buffer spans rows x pitch elements: kernels may read a row's padding up to the
 *   next multiple of 8 columns (never write it) and ignore what it holds.
 *   Requirements: 1 <= r <= min(m, n); T >= 0 (T == 0 is a no-op: nothing is read or written and
 *   X and Y may be NULL); every base pointer of X, Wp,
 *   C, Y 16-byte aligned and ldx, ldwp, ldc, ldy multiples of 8 (16-byte row pitch), else
 *   PIFA_ERR_ALIGNMENT. Index sets are not validated on the host (that would need a copy back);
 *   kernels skip any write whose index is outside [0, m) and latch PIFA_ERR_DEVICE_INDEX, read
 *   with pifa_device_status(). pifa_validate_indices() checks host copies in full.
 *   Numerics: bf16 X and W_p, fp32 accumulation; Y_p enters the second contraction as a hi + lo
 *   pair of C's storage type, never as one bf16 or fp16 value.
 *   Returns PIFA_OK once the kernels are enqueued; launch errors give PIFA_ERR_CUDA.
 */
int pifa_forward(const void* X, int64_t T, int64_t n, int64_t ldx,
                 const void* Wp, int64_t r, int64_t ldwp,
                 const void* C, int64_t m, int64_t ldc, int c_dtype,
                 const int32_t* pivot_idx, const int32_t* nonpivot_idx,
                 void* Y, int64_t ldy,
                 void* workspace, int64_t workspace_bytes,
                 void* cuda_stream);

/* pifa_forward_variant -- pifa_forward with an explicit pifa_variant (tests and benchmarks). */
int pifa_forward_variant(const void* X, int64_t T, int64_t n, int64_t ldx,
                         const void* Wp, int64_t r, int64_t ldwp,
                         const void* C, int64_t m, int64_t ldc, int c_dtype,
                         const int32_t* pivot_idx, const int32_t* nonpivot_idx,
                         void* Y, int64_t ldy,
                         void* workspace, int64_t workspace_bytes,
                         int variant, void* cuda_stream);

/*
 * pifa_forward_grouped -- Algorithm 2 for `groups` (G) PIFA layers of one shape (m, n, r, c_dtype)
 * that share their input X, e.g. a transformer MLP's gate and up projections, as one computation:
 * their pivot rows are stacked into one first contraction Y_p = X [W_p^(0); ...; W_p^(G-1)]^T, and
 * the second runs over all groups' rows of C at once, group g's rows against y_p's columns
 * [g r, (g + 1) r) -- in matrix form the layers make one PIFA computation whose C is
 * block-diagonal. The paper treats one layer at a time (Sec. 3.2); stacking changes no result.
 *
 *   X            as pifa_forward (T x n, shared by the groups).
 *   Wp           G r x n, row-major, leading dimension ldwp >= n: group g's W_p in rows [g r, (g + 1) r).
 *   C            G (m - r) x r, leading dimension ldc >= r: group g's C in rows [g (m - r), (g + 1) (m - r)).
 *   pivot_idx    G r int32: group g's pivot indices I^(g) plus g m (columns of Y).
 *   nonpivot_idx G (m - r) int32: group g's non-pivot indices plus g m.
 *   Y            T x (G m), leading dimension ldy >= G m: group g's output in columns [g m, (g + 1) m).
 *   workspace    at least pifa_workspace_size_grouped(G, T, m, n, r, c_dtype) bytes, 256-byte aligned.
 *   Variant, alignment, aliasing, asynchrony and status codes as pifa_forward (the variant is the
 *   one pifa_select_variant picks for one layer).
 *   G in [1, 64]; G > 1 needs m > r, (m - r) % 128 == 0 and r % 8 == 0 (PIFA_ERR_UNSUPPORTED
 *   otherwise: call pifa_forward per layer), so that no tile spans two groups. G = 1 is
 *   pifa_forward.
 */
int pifa_forward_grouped(int64_t groups, const void* X, int64_t T, int64_t n, int64_t ldx,
                         const void* Wp, int64_t r, int64_t ldwp,
                         const void* C, int64_t m, int64_t ldc, int c_dtype,
                         const int32_t* pivot_idx, const int32_t* nonpivot_idx,
                         void* Y, int64_t ldy,
                         void* workspace, int64_t workspace_bytes,
                         void* cuda_stream);

/* pifa_workspace_size_grouped -- bytes of device scratch pifa_forward_grouped needs (y_p for all
 * groups); negative pifa_status on bad arguments. Pure host arithmetic. */
int64_t pifa_workspace_size_grouped(int64_t groups, int64_t T, int64_t m, int64_t n, int64_t r, int c_dtype);

/*
 * pifa_forward_decode_noalloc -- the decode variant of pifa_forward (T <= 16) for callers that
 * cannot allocate device memory, e.g. a runtime that plans all device memory up front and forbids
 * a library's cudaMalloc, or a decode loop where an allocation's implicit synchronization is not
 * acceptable. The paper has no counterpart; it is an interface convenience of this library.
 *
 *   Arguments, layouts and errors as pifa_forward with C in bf16, without the workspace: the
 *   call allocates nothing (no cudaMalloc, cudaFree or allocating library routine). Its scratch
 *   -- 256 reserved bytes, then y_p as bf16 hi and lo planes (T rows of pitch round_up(r, 8)
 *   each) -- lives in a 1 MiB array in this library's static device data, which every GPU that
 *   loads the library holds until the process exits. Shapes with
 *   256 + T * round_up(r, 8) * 4 > 1 MiB are rejected with PIFA_ERR_WORKSPACE; T > 16 with
 *   PIFA_ERR_UNSUPPORTED.
 *   The first call on a device looks up the array's device address (cudaGetSymbolAddress) with
 *   that device current; make that first call before any stream capture. The address is kept for
 *   the process, so only the device's primary context (the CUDA runtime's) is supported, and a
 *   cudaDeviceReset() ends this library's use on that device (so does the status word's). Every call on a device
 *   shares the one array and it keeps the last call's contents, which no call depends on: y_p is
 *   fully written before it is read. Calls that may overlap on the GPU, e.g. on different
 *   streams, race on the array.
 */
int pifa_forward_decode_noalloc(const void* X, int64_t T, int64_t n, int64_t ldx,
                                const void* Wp, int64_t r, int64_t ldwp,
                                const void* C, int64_t m, int64_t ldc,
                                const int32_t* pivot_idx, const int32_t* nonpivot_idx,
                                void* Y, int64_t ldy, void* cuda_stream);

/* pifa_workspace_size -- bytes of device scratch pifa_forward needs for this shape, C dtype and
 * variant (PIFA_VARIANT_AUTO: the variant the selector picks). Returns a negative pifa_status on
 * bad arguments. Pure host arithmetic; no GPU needed. */
int64_t pifa_workspace_size(int64_t T, int64_t m, int64_t n, int64_t r, int c_dtype, int variant);

/* pifa_select_variant -- the selector (host, < 1 us): the pifa_variant pifa_forward runs for
 * (T, m, n, r, c_dtype) on this build, never PIFA_VARIANT_AUTO; negative pifa_status on bad
 * arguments. Decode for T <= 64, and for T <= 128 when the m - r non-pivot rows make between 148
 * and 296 blocks of 128 rows and the r pivot rows at most 296; else the split prefill. The forced
 * decode variant takes T <= 64, and T <= 128 when both phases have at most 296 blocks
 * (PIFA_ERR_UNSUPPORTED otherwise). */
int pifa_select_variant(int64_t T, int64_t m, int64_t n, int64_t r, int c_dtype);

/* pifa_variant_name -- static string naming a pifa_variant ("decode", ...); "?" if unknown. */
const char* pifa_variant_name(int variant);

/*
 * pifa_compress -- Algorithm 1 (Sec. 3.2) on W' = U V^T, on the HOST in float64, synchronous.
 * A reference setup step (it is not part of the GPU hot path).
 *
 *   U            HOST, float64, m x r row-major (contiguous).
 *   V            HOST, float64, n x r row-major (contiguous); W' = U V^T.
 *   pivot_idx    HOST out, int32[r]: I, ascending.
 *   nonpivot_idx HOST out, int32[m - r]: I^c, ascending (may be NULL when r == m).
 *   Wp           HOST out, float64, r x n, row pitch ldwp >= n: W'[I, :] (Eq. 1).
 *   C            HOST out, float64, (m - r) x r, row pitch ldc >= r: W'[I^c, :] = C W_p (Eq. 2);
 *                column j of C multiplies row j of Wp (ascending-I order). May be NULL if r == m.
 *   info         HOST out, optional (NULL allowed).
 *
 *   Pivot rule: Businger-Golub QR with column pivoting on W'^T (greedy: the row of W' with the
 *   largest norm orthogonal to the rows already chosen, norms recomputed exactly every step,
 *   ties to the lowest index). Computed in the r-dimensional row space of U R_V^T, where
 *   V = Q_V R_V, which has the same row inner products as W'. Requires 1 <= r <= min(m, n);
 *   returns PIFA_ERR_RANK_DEFICIENT when |R_(r-1,r-1)| < 1e-8 |R_00|. Uses the host's cores
 *   (OpenMP); scratch is allocated on the host and freed before returning.
 */
int pifa_compress(const double* U, const double* V, int64_t m, int64_t n, int64_t r,
                  int32_t* pivot_idx, int32_t* nonpivot_idx,
                  double* Wp, int64_t ldwp, double* C, int64_t ldc,
                  pifa_compress_info* info);

/*
 * pifa_compress_device -- Algorithm 1 (Sec. 3.2) on W' = U V^T on the GPU in float64: the same
 * outputs as pifa_compress, for layers where the host route is slow (minutes at 28672 x 8192).
 *
 *   U, V         DEVICE, float64, m x r and n x r, row-major, contiguous (W' = U V^T).
 *   pivot_idx    DEVICE out, int32[r]: I, ascending.
 *   nonpivot_idx DEVICE out, int32[m - r]: I^c, ascending (may be NULL when r == m).
 *   Wp           DEVICE out, float64, r x n, row pitch ldwp >= n: W'[I, :] (Eq. 1).
 *   C            DEVICE out, float64, (m - r) x r, row pitch ldc >= r: W'[I^c, :] = C W_p (Eq. 2),
 *                columns in ascending-I order (may be NULL when r == m).
 *   workspace    DEVICE scratch of pifa_compress_device_workspace_size(m, n, r) bytes, 256-byte
 *                aligned, no initialisation needed (about 8 (m r + 4 r^2) bytes).
 *   info         HOST out, optional: min_pivot_gap, r_ratio and max_abs_c as pifa_compress
 *                (threads = 0).
 *   cuda_stream  the stream the work is enqueued on; the call synchronizes it before returning.
 *
 *   Pivot rule exactly as pifa_compress (greedy Businger-Golub on W'^T, residual norms recomputed
 *   every step, ties to the lowest index), computed in the r-dimensional row space Z = U L with
 *   L L^T = V^T V (Cholesky), which has the row inner products of W'. C = Z[I^c] R^{-T} from the
 *   triangular factor R of that pivoted QR; W_p = U[I] V^T. Requires 1 <= r <= min(m, n) and
 *   r <= 16384 (PIFA_ERR_UNSUPPORTED otherwise); PIFA_ERR_RANK_DEFICIENT when V^T V is not
 *   positive definite or |R_(r-1,r-1)| < 1e-8 |R_00|. Synchronous; no device memory is allocated.
 */
int pifa_compress_device(const double* U, const double* V, int64_t m, int64_t n, int64_t r,
                         int32_t* pivot_idx, int32_t* nonpivot_idx,
                         double* Wp, int64_t ldwp, double* C, int64_t ldc,
                         void* workspace, int64_t workspace_bytes,
                         pifa_compress_info* info, void* cuda_stream);

/* pifa_compress_device_workspace_size -- bytes of device scratch pifa_compress_device needs;
 * negative pifa_status on bad arguments. Pure host arithmetic. */
int64_t pifa_compress_device_workspace_size(int64_t m, int64_t n, int64_t r);

/*
 * pifa_backward -- the gradients of Algorithm 2 with respect to X, W_p and C, for fine-tuning a
 * compressed model (Sec. 5.1; the PIFA layer is differentiable, Sec. 6). With tokens as rows and
 * dY = dL/dY (T x m): dY_p = dY[:, I] + dY[:, I^c] C, dX = dY_p W_p, dW_p = dY_p^T X,
 * dC = dY[:, I^c]^T Y_p with Y_p = X W_p^T recomputed. The index sets are not trained.
 *
 *   X, Wp, C, pivot_idx, nonpivot_idx   as pifa_forward (DEVICE; C bf16).
 *   dY           DEVICE, bf16, T x m, row pitch lddy >= m.
 *   dX           DEVICE out, bf16, T x n, pitch lddx >= n (NULL: not computed).
 *   dWp          DEVICE out, fp32, r x n, pitch lddwp >= n (NULL: not computed).
 *   dC           DEVICE out, fp32, (m - r) x r, pitch lddc >= r (NULL: not computed).
 *   workspace    DEVICE scratch of pifa_backward_workspace_size(T, m, n, r) bytes, 256-byte
 *                aligned, no initialisation needed (dY[:, I], dY[:, I^c], Y_p and dY_p in bf16).
 *   Numerics: bf16 operands, fp32 accumulation; dY_p and Y_p pass between the contractions as
 *   hi + lo pairs of bf16. Alignment as pifa_forward (fp32 pitches multiples of 4 elements).
 *   T == 0 writes zero dW_p and dC. Asynchronous on cuda_stream; out-of-range indices latch
 *   PIFA_ERR_DEVICE_INDEX (read with pifa_device_status()).
 *   Concurrency: independent products run on two side streams that the library keeps per host
 *   thread and device, forked from cuda_stream and joined back into it inside the call (also on
 *   failure), so the call orders like one kernel sequence on cuda_stream and can be captured into a
 *   CUDA graph. The first call on a thread and device creates those streams: make it before a
 *   stream capture that contains the call.
 */
int pifa_backward(const void* X, int64_t T, int64_t n, int64_t ldx,
                  const void* Wp, int64_t r, int64_t ldwp,
                  const void* C, int64_t m, int64_t ldc,
                  const int32_t* pivot_idx, const int32_t* nonpivot_idx,
                  const void* dY, int64_t lddy,
                  void* dX, int64_t lddx, float* dWp, int64_t lddwp, float* dC, int64_t lddc,
                  void* workspace, int64_t workspace_bytes, void* cuda_stream);

/* pifa_backward_workspace_size -- bytes of device scratch pifa_backward needs; negative pifa_status
 * on bad arguments. Pure host arithmetic. */
int64_t pifa_backward_workspace_size(int64_t T, int64_t m, int64_t n, int64_t r);

/*
 * pifa_m_accumulate -- one calibration batch into the online accumulators of the M reconstruction
 * (Sec. 4, the accumulation steps of Algorithm 3): with the dense-flow inputs X_o and the
 * low-rank-flow inputs X_u of a layer W (m x n), tokens as rows,
 *   XXt  += X_u^T X_u                                      (n x n: the sum of x_u x_u^T)
 *   YtXt += Y_t^T X_u,  Y_t = (lambda X_o + (1 - lambda) X_u) W^T   (m x n: the sum of y_t x_u^T)
 * so that any number of batches can be folded in with constant memory.
 *
 *   Xo, Xu       DEVICE, bf16, T x n, common row pitch ldx >= n (Xo may be NULL when YtXt is).
 *   W            DEVICE, bf16, m x n, pitch ldw >= n (the dense weight; may be NULL when YtXt is).
 *   lambda       mix ratio in [0, 1] (Eq. 6; the paper uses 0.25).
 *   XXt          DEVICE in/out, fp32, n x n, pitch ldxx >= n. X X^T is symmetric: its upper
 *                triangle (column >= row) is accumulated; of the entries below it, those in tiles
 *                that straddle the diagonal are accumulated too and the rest are left as they were.
 *   YtXt         DEVICE in/out, fp32, m x n, pitch ldyx >= n (NULL: only XXt is accumulated).
 *   workspace    DEVICE scratch of pifa_m_accumulate_workspace_size(T, m, n) bytes, 256-byte
 *                aligned (X_u^T, the mixed input and Y_t^T in bf16).
 *   Numerics: bf16 operands, fp32 accumulation; the mixed input and Y_t pass as hi + lo bf16 pairs.
 *   T == 0 is a no-op. Asynchronous on cuda_stream; X X^T runs beside the Y_t chain on a side
 *   stream, as in pifa_backward (same ordering and capture rules).
 */
int pifa_m_accumulate(const void* Xo, const void* Xu, int64_t T, int64_t n, int64_t ldx,
                      const void* W, int64_t m, int64_t ldw, float lambda,
                      float* XXt, int64_t ldxx, float* YtXt, int64_t ldyx,
                      void* workspace, int64_t workspace_bytes, void* cuda_stream);

/* pifa_m_accumulate_workspace_size -- bytes of device scratch pifa_m_accumulate needs; negative
 * pifa_status on bad arguments. Pure host arithmetic. */
int64_t pifa_m_accumulate_workspace_size(int64_t T, int64_t m, int64_t n);

/*
 * pifa_m_reconstruct -- the two reconstruction steps of the M method (Sec. 4; Algorithm 3, part 1)
 * from the accumulators pifa_m_accumulate builds, in float64 on the GPU:
 *   U_r   = (Y_t X^T) V (V^T (X X^T) V)^{-1}                                       (Eq. 4)
 *   V_r^T = (U_r^T U_r)^{-1} U_r^T (Y_t X^T + alpha W) (X X^T + alpha I)^{-1}        (Eq. 8)
 * whose product U_r V_r^T is the low-rank weight that Algorithm 1 (pifa_compress_device) turns
 * into a PIFA layer.
 *
 *   XXt          DEVICE, fp32, n x n, pitch ldxx >= n (X X^T; only its upper triangle is read).
 *   YtXt         DEVICE, fp32, m x n, pitch ldyx >= n (Y_t X^T).
 *   V            DEVICE, float64, n x r, contiguous (the pruned layer's right factor).
 *   W            DEVICE, bf16, m x n, pitch ldw >= n (the dense weight; used when alpha > 0).
 *   alpha        the regulariser of Eq. 8 (>= 0; the paper uses 0.001; 0 gives Eq. 7).
 *   U_r, V_r     DEVICE out, float64, m x r and n x r, contiguous.
 *   workspace    DEVICE scratch of pifa_m_reconstruct_workspace_size(m, n, r) bytes, 256-byte
 *                aligned (about 8 (2 n^2 + m n + 4 r n + 4 r^2 + 2.25 p^2) bytes, p = n rounded up
 *                to 32 * 2^k).
 *   The symmetric positive definite matrices are inverted by Cholesky factorisation and the
 *   inverse of the triangular factor. Requires 1 <= r <= min(m, n) and n <= 16384;
 *   PIFA_ERR_RANK_DEFICIENT when a matrix to invert is not positive definite. Synchronous.
 */
int pifa_m_reconstruct(const float* XXt, int64_t ldxx, const float* YtXt, int64_t ldyx,
                       const double* V, const void* W, int64_t ldw,
                       int64_t m, int64_t n, int64_t r, double alpha,
                       double* U_r, double* V_r, void* workspace, int64_t workspace_bytes,
                       void* cuda_stream);

/* pifa_m_reconstruct_workspace_size -- bytes of device scratch pifa_m_reconstruct needs; negative
 * pifa_status on bad arguments. Pure host arithmetic. */
int64_t pifa_m_reconstruct_workspace_size(int64_t m, int64_t n, int64_t r);

/* pifa_validate_indices -- HOST copies: PIFA_OK iff pivot_idx (r entries) and nonpivot_idx
 * (m - r entries) are strictly ascending, inside [0, m) and disjoint (so together a partition
 * of [0, m), as Algorithm 1 step 2 defines I^c); else PIFA_ERR_INVALID_ARG. */
int pifa_validate_indices(const int32_t* pivot_idx, const int32_t* nonpivot_idx,
                          int64_t m, int64_t r);

/* pifa_device_status -- synchronizes `cuda_stream`, then returns and clears the error word the
 * kernels latch on the current device (PIFA_OK, PIFA_ERR_TIMEOUT or PIFA_ERR_DEVICE_INDEX). */
int pifa_device_status(void* cuda_stream);

/* pifa_set_wait_timeout -- bound, in nanoseconds, of every device-side wait of kernels launched
 * after this call (default 1 s, or the environment variable PIFA_WAIT_TIMEOUT_NS at load time;
 * ns == 0 restores that default). A wait that runs out makes its CTA latch PIFA_ERR_TIMEOUT, wait
 * (with a fixed bound) for its own copies in flight, and return; the outputs of that call are then
 * undefined. Process-wide; PIFA_ERR_INVALID_ARG for ns < 0. */
int pifa_set_wait_timeout(int64_t ns);

/* pifa_set_decode_grid -- how the decode variant with T <= 16 lays out each of its two phases for
 * calls made after this one (process-wide). Three forms compute a phase (R weight rows, K
 * columns): waves of one-tile clusters, every CTA staging its weight rows at launch; a persistent
 * grid of co-resident clusters that stream their tiles through a ring of TMA-filled stages; and
 * split-K on the tensor cores. The latter gives a phase of at most two 128-row blocks per SM 1, 2,
 * 4 or 8 CTAs per row block, each one K-slice of it, as a thread-block cluster that adds up its
 * slices in shared memory in rank order and writes the outputs itself (one kernel); a taller
 * phase deals equal ranges of 128 x 64 weight tiles to a persistent grid and a second kernel sums
 * the fp32 partial sums in a fixed order.
 * PIFA_DECODE_GRID_AUTO (0, the default) picks per phase from its shape and T: split-K when
 * T > 2 and R >= 4096, else waves while the phase takes at most two of them, else the persistent
 * grid. PIFA_DECODE_GRID_WAVES (1), PIFA_DECODE_GRID_PERSISTENT (2) and PIFA_DECODE_GRID_SPLITK
 * (3) force one form for both phases (a tuning and test knob: all compute the same result up to
 * the summation order of fp32 partial sums; forced split-K runs the persistent grid instead when the
 * workspace is too small for its partial sums). For 16 < T <= 128 only the split-K form exists
 * (token tiles of 32, 64 or 128 rows): both phases run it whatever the mode. PIFA_ERR_INVALID_ARG for
 * other values. */
#define PIFA_DECODE_GRID_AUTO 0
#define PIFA_DECODE_GRID_WAVES 1
#define PIFA_DECODE_GRID_PERSISTENT 2
#define PIFA_DECODE_GRID_SPLITK 3
int pifa_set_decode_grid(int mode);

/* pifa_launch_count -- how many kernels this library has enqueued since it was loaded, over all
 * threads, devices and entry points (a launch captured into a CUDA graph counts once, at capture;
 * its replays do not). The difference across one call is the number of kernels that call runs.
 * Not part of the paper. */
int64_t pifa_launch_count(void);

/* pifa_selftest_wait_timeout -- enqueues on `cuda_stream` a one-CTA kernel that waits, with the
 * current bound (pifa_set_wait_timeout), on an mbarrier that nothing arrives on, so the wait runs
 * out and PIFA_ERR_TIMEOUT is latched for pifa_device_status(). Checks the failure-detection path
 * of the bounded device waits without faulting or hanging the GPU. Not part of the paper. */
int pifa_selftest_wait_timeout(void* cuda_stream);

/* pifa_status_string -- static string for a pifa_status value. */
const char* pifa_status_string(int status);

/* pifa_last_error -- the calling thread's most recent detailed error message ("" if none). */
const char* pifa_last_error(void);

/* pifa_version -- static version string of this build. */
const char* pifa_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PIFA_H_ */
