// decode_tc.cu -- one decode phase (T <= 16 tokens) of Algorithm 2 on the 5th-generation tensor
// cores, split over K across a persistent grid: the form used for layers too large for one wave.
//
// A phase is a skinny product D = A B^T: A the weight rows (W_p for Y_p = X W_p^T, Algorithm 2
// step 2; C for Y_np = Y_p C^T, step 3), B the T token rows (x, or y_p as its hi and lo planes).
// The weight matrix is cut into units of 128 rows x one K-slice; units are numbered slice-major
// (u = s nrb + rb) and dealt to the CTAs in equal contiguous ranges, so every SM streams the same
// number of weight bytes and a CTA meets few distinct K-slices of B.
//
// Partial kernel (two CTAs per SM, 192 threads each):
//   warp 0     TMA producer: the weight tiles (128 rows x 64 columns, 16 KB, 128-byte swizzle)
//              through a ring of stages, the first ones before the dependency wait (the weights
//              do not depend on the previous kernel); the unit's K-slice of B into one of two
//              buffers (16 token rows x 64 columns per box; rows >= T zero-filled), after the wait.
//   warp 1     owns 256 TMEM columns (two units in flight) and issues tcgen05.mma.kind::f16
//              M = 128, K = 16, N = 16 (one B plane) or 32 (the y_p hi and lo planes as one
//              operand) from one thread, dealing a unit's MMAs round-robin over independent
//              accumulators so that consecutive MMAs do not wait for each other.
//   warps 2-5  sum a unit's accumulators (TMEM lane quarter each) while the next unit fills the
//              other set, and store its partial sums P[s][t][row] (fp32, coalesced over rows).
// Reduce kernel: Y[t, cols[j]] = bf16(sum_s P[s][t][j]) in slice order (deterministic); phase 1
// also writes y_p as the hi + lo planes of C's dtype that phase 2 reads.
// Every wait is bounded (globaltimer); on timeout the CTA latches PIFA_ERR_TIMEOUT, drains what
// it has in flight and returns.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

constexpr int TM = 128;                         // weight rows per unit (MMA M = TMEM lanes)
constexpr int TN = 16;                          // token rows of B, padded (MMA N)
constexpr int KB = 64;                          // K per chunk: one 128-byte swizzle row
constexpr uint32_t A_BYTES = TM * KB * 2;       // one weight tile
constexpr uint32_t BOX_BYTES = TN * KB * 2;     // one B box
constexpr int MAX_STAGES = 10;
constexpr int THREADS = 192;
// A unit's MMAs are dealt round-robin over NACC independent accumulators (summed in the
// epilogue), so that consecutive MMAs do not wait for each other. With two B planes (y_p hi and
// lo) one MMA of N = 32 covers both: the lo box follows the hi box in shared memory, making one
// 32-row operand, and accumulator columns t and 16 + t are added in the epilogue. Per unit
// NACC * 16 * NB columns; two units in flight: 256 TMEM columns either way.
template <int NB>
constexpr int kNacc = NB == 1 ? 8 : 4;
constexpr uint32_t TMEM_COLS = 256;
// Two CTAs per SM, each with its own producer and MMA-issuing thread: one issuing thread per SM
// measured as the limit (70B gate/up, T = 16: 73 us with one CTA of ten stages, 60 us with two of
// four, 73 us with three of two), so a CTA keeps to half an SM's shared memory and TMEM.
constexpr int CTAS_PER_SM = 2;
constexpr size_t SMEM_PER_CTA = 112 * 1024;

struct TcArgs {
  int R, K, T;
  int nrb, ns, KS;  // 128-row blocks, K-slices, slice width (a multiple of 64)
  int units;        // ns * nrb
  int gsz, goff;    // grouped layers: rows per group (a multiple of 128) and B columns per group
  int stages;
  uint32_t chunk_bytes;  // B bytes per 64-column chunk of a slice: NB boxes (hi, then lo)
  uint32_t idesc;
  float* P;              // partial sums [ns][T][R]
  int* status;
  uint64_t timeout_ns;
};

__device__ __forceinline__ int unit_key(const TcArgs& a, int u) {
  const int s = u / a.nrb, rb = u % a.nrb;
  const int g = a.gsz > 0 ? (rb * TM) / a.gsz : 0;
  return g * a.ns + s;
}
__device__ __forceinline__ int unit_chunks(const TcArgs& a, int u) {
  const int s = u / a.nrb;
  return (min(a.KS, a.K - s * a.KS) + KB - 1) / KB;
}

template <int NB>
__global__ void __launch_bounds__(THREADS, CTAS_PER_SM)
    decode_tc_partial(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                      const __grid_constant__ CUtensorMap tmB1, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t bbuf = (uint32_t)(a.KS / KB) * a.chunk_bytes;  // one B buffer (both planes)
  uint8_t* bsm = smem;                                  // two B buffers
  uint8_t* ring = smem + 2 * bbuf;                      // weight stages (1024-aligned: bbuf % 2048 == 0)
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + (size_t)a.stages * A_BYTES);
  uint64_t* empty = full + MAX_STAGES;
  uint64_t* bfull = empty + MAX_STAGES;
  uint64_t* bempty = bfull + 2;
  uint64_t* accf = bempty + 2;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int u0 = (int)(((int64_t)blockIdx.x * a.units) / gridDim.x);
  const int u1 = (int)(((int64_t)(blockIdx.x + 1) * a.units) / gridDim.x);

  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bfull[b], 1);
      mbar_init(&bempty[b], 1);
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB0);
    if (NB > 1) prefetch_tmap(&tmB1);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- producer ----------------
      int total = 0;
      for (int u = u0; u < u1; ++u) total += unit_chunks(a, u);
      const int pre = min(total, a.stages);
      {  // weight tiles of the first stages, before the dependency wait
        int it = 0;
        for (int u = u0; u < u1 && it < pre; ++u) {
          const int s = u / a.nrb, rb = u % a.nrb, nck = unit_chunks(a, u);
          for (int c = 0; c < nck && it < pre; ++c, ++it) {
            mbar_arrive_expect_tx(&full[it], A_BYTES);
            tma_load_2d(smem_u32(ring + (size_t)it * A_BYTES), &tmA, s * a.KS + c * KB, rb * TM, &full[it]);
          }
        }
      }
      pdl_wait_primary();
      int it = 0, kb = -1, cur = -1, issued = 0;
      bool dead = false;
      for (int u = u0; u < u1 && !dead; ++u) {
        const int s = u / a.nrb, rb = u % a.nrb, nck = unit_chunks(a, u);
        const int key = unit_key(a, u);
        if (key != cur) {  // the unit's K-slice of B into the next buffer
          ++kb;
          cur = key;
          const int b = kb & 1;
          if (kb >= 2 && !mbar_wait(&bempty[b], (uint32_t)((kb >> 1) - 1) & 1u, a.timeout_ns)) {
            latch_status(a.status, PIFA_ERR_TIMEOUT);
            *abort_flag = 1;
            dead = true;
            break;
          }
          const int x0 = (a.gsz > 0 ? ((rb * TM) / a.gsz) * a.goff : 0) + s * a.KS;
          mbar_arrive_expect_tx(&bfull[b], (uint32_t)(NB * nck) * BOX_BYTES);
          uint8_t* dst = bsm + b * bbuf;
          for (int c = 0; c < nck; ++c) {
            tma_load_2d(smem_u32(dst + c * a.chunk_bytes), &tmB0, x0 + c * KB, 0, &bfull[b]);
            if (NB > 1) tma_load_2d(smem_u32(dst + c * a.chunk_bytes + BOX_BYTES), &tmB1, x0 + c * KB, 0, &bfull[b]);
          }
        }
        for (int c = 0; c < nck; ++c, ++it) {
          if (it < pre) continue;  // issued before the wait
          const int st = it % a.stages;
          if (!mbar_wait(&empty[st], (uint32_t)((it / a.stages) - 1) & 1u, a.timeout_ns) || *abort_flag) {
            latch_status(a.status, PIFA_ERR_TIMEOUT);
            *abort_flag = 1;
            dead = true;
            break;
          }
          mbar_arrive_expect_tx(&full[st], A_BYTES);
          tma_load_2d(smem_u32(ring + (size_t)st * A_BYTES), &tmA, s * a.KS + c * KB, rb * TM, &full[st]);
        }
      }
      issued = dead ? it : total;
      if (issued < pre) issued = pre;
      // nothing may land in shared memory once the CTA has left: the last use of every stage and
      // of both B buffers
      for (int j = issued > a.stages ? issued - a.stages : 0; j < issued; ++j)
        if (!mbar_wait(&full[j % a.stages], (uint32_t)(j / a.stages) & 1u, 100000000ull))
          latch_status(a.status, PIFA_ERR_TIMEOUT);
      for (int k = kb > 1 ? kb - 1 : 0; k <= kb; ++k)
        if (k >= 0 && !mbar_wait(&bfull[k & 1], (uint32_t)(k >> 1) & 1u, 100000000ull))
          latch_status(a.status, PIFA_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int it = 0, kb = -1, cur = -1;
      bool dead = false;
      for (int u = u0; u < u1 && !dead; ++u) {
        const int j = u - u0, acc = j & 1, nck = unit_chunks(a, u);
        const int key = unit_key(a, u);
        if (key != cur) {
          ++kb;
          cur = key;
          if (!mbar_wait(&bfull[kb & 1], (uint32_t)(kb >> 1) & 1u, a.timeout_ns)) {
            dead = true;
            break;
          }
        }
        if (j >= 2 && !mbar_wait(&acce[acc], (uint32_t)((j >> 1) - 1) & 1u, a.timeout_ns)) {
          dead = true;
          break;
        }
        tc_fence_after();
        const uint32_t bbase = smem_u32(bsm + (kb & 1) * bbuf);
        constexpr int NACC = kNacc<NB>;
        const uint32_t dacc = tmem + (uint32_t)(acc * NACC * TN * NB);
        int e = 0;  // MMAs of this unit so far: accumulator e % NACC, first use overwrites
        for (int c = 0; c < nck; ++c, ++it) {
          const int st = it % a.stages;
          if (!mbar_wait(&full[st], (uint32_t)(it / a.stages) & 1u, a.timeout_ns) || *abort_flag) {
            dead = true;
            break;
          }
          tc_fence_after();
          const uint32_t at = smem_u32(ring + (size_t)st * A_BYTES);
#pragma unroll
          for (int kk = 0; kk < KB / 16; ++kk, ++e)
            mma_bf16_ss(dacc + (uint32_t)((e % NACC) * TN * NB), sw128_desc(at + kk * 32),
                        sw128_desc(bbase + c * a.chunk_bytes + kk * 32), a.idesc, e >= NACC ? 1u : 0u);
          mma_commit(&empty[st]);  // the stage is free once these MMAs have read it
        }
        if (dead) break;
        mma_commit(&accf[acc]);
        if (u + 1 == u1 || unit_key(a, u + 1) != cur) mma_commit(&bempty[kb & 1]);
      }
      if (dead) {
        latch_status(a.status, PIFA_ERR_TIMEOUT);
        *abort_flag = 1;
      }
      mma_commit(drain);  // every MMA issued above has completed before TMEM and SMEM are released
      if (!mbar_wait(drain, 0, 100000000ull)) latch_status(a.status, PIFA_ERR_TIMEOUT);
    }
  } else {
    // ---------------- epilogue: warps 2..5, TMEM lane quarter warp % 4 ----------------
    const int q = warp & 3;
    for (int u = u0; u < u1; ++u) {
      const int j = u - u0, acc = j & 1;
      const int s = u / a.nrb, rb = u % a.nrb;
      if (!mbar_wait(&accf[acc], (uint32_t)(j >> 1) & 1u, a.timeout_ns) || *abort_flag) {
        latch_status(a.status, PIFA_ERR_TIMEOUT);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      // the accumulators this unit wrote (fewer than NACC only when it has fewer MMAs), summed in
      // a fixed order
      constexpr int NACC = kNacc<NB>;
      const int used = min(NACC, unit_chunks(a, u) * (KB / 16));
      const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * NACC * TN * NB);
      float sum[TN];
#pragma unroll
      for (int t = 0; t < TN; ++t) sum[t] = 0.0f;
      // column groups of 16: accumulator a, plane nb at (a NB + nb) 16
      for (int g0 = 0; g0 < used * NB; g0 += 4) {
        uint32_t v[4][16];
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (g0 + k < used * NB) tmem_ld_32x32b_x16(base + (uint32_t)((g0 + k) * TN), v[k]);
        tmem_ld_wait();
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (g0 + k < used * NB)
#pragma unroll
            for (int t = 0; t < TN; ++t) sum[t] += __uint_as_float(v[k][t]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce[acc]);  // this quarter of the accumulators may be refilled
      const int row = rb * TM + q * 32 + lane;
      if (row < a.R) {
        float* dst = a.P + (size_t)s * a.T * a.R + row;
#pragma unroll
        for (int t = 0; t < TN; ++t)
          if (t < a.T) dst[(size_t)t * a.R] = sum[t];
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// hi + lo split of an fp32 value in bf16 (kF16 = false) or fp16 (kF16 = true); fp16 saturates at
// +-65504 and reports the overflow.
template <bool kF16>
__device__ __forceinline__ void split_hi_lo(float f, uint16_t& h, uint16_t& l, bool& range_err) {
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

struct ReduceArgs {
  const float* P;
  int ns, T, R;
  const int32_t* cols;  // output column of each row (I or I^c)
  int m;                // columns of Y (index bound)
  bf16* Y;
  int64_t ldy;
  uint16_t* yph;        // phase 1 with m > r: y_p hi and lo planes, else null
  uint16_t* ypl;
  int64_t ldyp;
  int* status;
};

// Y[t, cols[j]] = bf16(sum_s P[s][t][j]), slices summed in order; phase 1 also splits y_p.
template <bool kF16>
__global__ void __launch_bounds__(256) decode_tc_reduce(ReduceArgs a) {
  pdl_launch_dependents();
  pdl_wait_primary();
  const int64_t n = (int64_t)a.T * a.R;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int t = (int)(i / a.R), j = (int)(i % a.R);
  float sum = 0.0f;
  for (int s = 0; s < a.ns; ++s) sum += __ldcg(a.P + (size_t)s * n + i);
  bool range_err = false;
  if (a.yph) {
    uint16_t h, l;
    split_hi_lo<kF16>(sum, h, l, range_err);
    a.yph[(int64_t)t * a.ldyp + j] = h;
    a.ypl[(int64_t)t * a.ldyp + j] = l;
  }
  if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
  const int col = __ldg(a.cols + j);
  if ((unsigned)col >= (unsigned)a.m) {
    latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
    return;
  }
  a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(sum);
}

int sm_count_tc() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      n = 1;
  }
  return n;
}

int pick_ks(int R, int K, int NB) {
  // 256 columns: a K-slice of B (16 token rows, hi and lo) is 16 KB, so two buffers and a four-stage
  // ring of weight tiles fit half an SM; the partial sums are K / 256 fp32 values per output
  (void)R;
  (void)K;
  (void)NB;
  return 256;
}

}  // namespace

int64_t decode_tc_partial_bytes(int64_t R, int64_t K, int64_t T, int NB) {
  const int ks = pick_ks((int)R, (int)K, NB);
  return ((K + ks - 1) / ks) * T * R * 4;
}

int launch_decode_tc(const DecodeTcPhase& ph, int* status, uint64_t timeout_ns, cudaStream_t stream) {
  const int NB = ph.planes;
  TcArgs a = {};
  a.R = (int)ph.R;
  a.K = (int)ph.K;
  a.T = (int)ph.T;
  a.nrb = (a.R + TM - 1) / TM;
  a.KS = pick_ks(a.R, a.K, NB);
  a.ns = (a.K + a.KS - 1) / a.KS;
  a.units = a.ns * a.nrb;
  a.gsz = (int)ph.gsz;
  a.goff = (int)ph.goff;
  a.chunk_bytes = (uint32_t)NB * BOX_BYTES;
  const bool f16 = ph.mma_f16;
  a.idesc = f16 ? idesc_f16_f32(TM, TN * NB) : idesc_bf16_f32(TM, TN * NB);
  a.P = ph.P;
  a.status = status;
  a.timeout_ns = timeout_ns;
  const size_t fixed = 1024 + 2 * (size_t)(a.KS / KB) * a.chunk_bytes + 512;
  int stages = (int)((SMEM_PER_CTA - fixed) / A_BYTES);
  a.stages = stages > MAX_STAGES ? MAX_STAGES : stages;
  if (a.stages < 2) return pifa_fail(PIFA_ERR_UNSUPPORTED, "decode_tc: shared memory too small");
  const size_t smem = fixed + (size_t)a.stages * A_BYTES;

  CUtensorMap tA, tB0, tB1;
  int st;
  if ((st = make_tmap_2d(&tA, ph.dtype, ph.A, ph.R, ph.K, ph.lda, KB, TM)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tB0, ph.dtype, ph.B0, ph.T, ph.bcols, ph.ldb, KB, TN)) != PIFA_OK) return st;
  if (NB > 1 && (st = make_tmap_2d(&tB1, ph.dtype, ph.B1, ph.T, ph.bcols, ph.ldb, KB, TN)) != PIFA_OK) return st;
  if (NB == 1) tB1 = tB0;

  auto kern = NB == 1 ? decode_tc_partial<1> : decode_tc_partial<2>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaFuncSetAttribute(decode_tc)", e);
  cudaLaunchConfig_t cfg = {};
  const int nsm = sm_count_tc();
  cfg.gridDim = dim3((unsigned)(a.units < CTAS_PER_SM * nsm ? a.units : CTAS_PER_SM * nsm));
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, tA, tB0, tB1, a);
  if (e != cudaSuccess) return pifa_fail_cuda("decode_tc partial launch", e);

  ReduceArgs r = {};
  r.P = ph.P;
  r.ns = a.ns;
  r.T = a.T;
  r.R = a.R;
  r.cols = ph.cols;
  r.m = (int)ph.m;
  r.Y = reinterpret_cast<bf16*>(ph.Y);
  r.ldy = ph.ldy;
  r.yph = ph.yph;
  r.ypl = ph.ypl;
  r.ldyp = ph.ldyp;
  r.status = status;
  const int64_t n = (int64_t)a.T * a.R;
  cudaLaunchConfig_t rc = cfg;
  rc.gridDim = dim3((unsigned)((n + 255) / 256));
  rc.blockDim = dim3(256);
  rc.dynamicSmemBytes = 0;
  e = ph.split_f16 ? cudaLaunchKernelEx(&rc, decode_tc_reduce<true>, r) : cudaLaunchKernelEx(&rc, decode_tc_reduce<false>, r);
  if (e != cudaSuccess) return pifa_fail_cuda("decode_tc reduce launch", e);
  return PIFA_OK;
}
