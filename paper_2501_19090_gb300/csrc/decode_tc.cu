// decode_tc.cu -- one decode phase (T <= 128 tokens) of Algorithm 2 on the 5th-generation tensor
// cores, split over K: the decode form for large phases when T > 2, and the only one for
// 16 < T <= 128. Two cuts of a phase: the row-block plan (below) for phases of at most two 128-row
// blocks per SM, and balanced ranges with a reduce kernel for taller ones (described first).
//
// A phase is a skinny product D = A B^T: A the weight rows (W_p for Y_p = X W_p^T, Algorithm 2
// step 2; C for Y_np = Y_p C^T, step 3), B the T token rows (x, or y_p as its hi and lo planes).
// The weight matrix is cut into units of 128 rows x one K-slice, and a unit into chunks of 64
// columns (one 16 KB weight tile). Units are numbered slice-major (u = s nrb + rb) and the chunks
// of all units, in that order, are dealt to the CTAs in equal contiguous ranges: every CTA streams
// the same number of weight bytes to within one tile, whatever the unit count. The slice width is
// the largest multiple of 64 that keeps a unit no longer than a CTA's range, so a unit is split
// between at most two CTAs: its head (chunk 0 on) goes to P, its tail (if split) to P2.
//
// Partial kernel (two CTAs per SM, 192 threads each):
//   warp 0     TMA producer: per chunk, the weight tile (128 rows x 64 columns, 128-byte swizzle)
//              and the matching 64 columns of B (a token tile of TNT = 16, 32, 64 or 128 rows per
//              plane, the smallest that holds T; rows >= T zero-filled)
//              into one stage of a ring; the first weight tiles go out before the dependency wait
//              (the weights do not depend on the previous kernel), their B boxes after it.
//   warp 1     owns 256 TMEM columns (two segments in flight) and issues tcgen05.mma.kind::f16
//              M = 128, K = 16, N = TNT (one B plane) or 2 TNT (the y_p hi and lo planes as one
//              operand) from one thread, dealing a segment's MMAs round-robin over independent
//              accumulators (128 / N of them, at least one) so that consecutive MMAs do not wait
//              for each other. A 128-token tile's accumulator (N = 128 or 256) fills the 256
//              columns alone, so it is used only where a CTA has one segment (the row-block plan).
//   warps 2-5  sum a segment's accumulators (TMEM lane quarter each) while the next segment fills
//              the other set, and store its partial sums P[s][t][row] (fp32, coalesced over rows),
//              or, in the row-block plan, the outputs or the cluster's shared-memory sums.
// A unit's head CTA writes zeros to P2 when it holds the whole unit, so P2 is defined everywhere.
// Reduce kernel: Y[t, cols[j]] = bf16(sum_s (P[s][t][j] + P2[s][t][j])) in slice order
// (deterministic for a given grid); phase 1 also writes y_p as the hi + lo planes of C's dtype
// that phase 2 reads.
// Row-block plan, for every phase of at most two 128-row blocks per SM (all layers of LLaMA-2 7B
// and 70B): each row block gets cs CTAs (1, 2, 4 or 8), CTA k taking the block's K-slice k. With
// cs = 1 the epilogue's sums are the outputs. With cs > 1 the block's CTAs form a thread-block
// cluster: each stores its slice's sums in its own shared memory (the stage ring, free once its
// MMAs are done), and after a cluster barrier CTA k reads rows [k 128 / cs, (k + 1) 128 / cs) of
// every peer's sums through distributed shared memory, adds them in rank order and writes Y and
// y_p's planes. One kernel per phase: no partial sums in global memory and no reduce kernel.
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
constexpr int TN = 16;                          // token rows of B, padded (MMA N), for T <= 16
constexpr int kMaxTokensTc = 128;               // token tiles of 32, 64 and 128 rows serve T <= 128
constexpr int KB = 64;                          // K per chunk: one 128-byte swizzle row
constexpr uint32_t A_BYTES = TM * KB * 2;       // one weight tile
constexpr int MAX_STAGES = 10;
constexpr int THREADS = 192;
// A segment's MMAs are dealt round-robin over NACC independent accumulators (summed in the
// epilogue), so that consecutive MMAs do not wait for each other. With two B planes (y_p hi and
// lo) one MMA of N = 2 TNT covers both: the lo box follows the hi box in shared memory, making one
// 2 TNT-row operand, and accumulator columns t and TNT + t are added in the epilogue. Up to 64
// tokens, NACC * TNT * NB = 128 columns per segment and two segments in flight: 256 TMEM columns.
// A 128-token tile's one accumulator takes 128 or 256 columns: one segment (the row-block plan).
template <int NB, int TNT = TN>
constexpr int kNacc = TNT * NB >= 128 ? 1 : 128 / (TNT * NB);
constexpr uint32_t TMEM_COLS = 256;
// Two CTAs per SM, each with its own producer and MMA-issuing thread: one issuing thread per SM
// measured as the limit (70B gate/up, T = 16: 73 us with one CTA of ten stages, 60 us with two of
// four, 73 us with three of two), so a CTA keeps to half an SM's shared memory and TMEM.
constexpr int CTAS_PER_SM = 2;
constexpr size_t SMEM_PER_CTA = 112 * 1024;
// The grid never exceeds GRID_MAX CTAs: the slice plan made for GRID_MAX bounds the partial-sum
// bytes of every smaller grid (a smaller grid gives longer ranges, wider slices, fewer of them).
constexpr int GRID_MAX = 512;
constexpr int MIN_CHUNKS_PER_CTA = 4;
constexpr int MAX_CLUSTER_TC = 8;  // CTAs per row block in the row-block plan (portable cluster size)

// How one phase is cut: slice width, slice count and grid.
struct Plan {
  int nrb, nck;   // 128-row blocks; 64-column chunks over K
  int64_t total;  // chunks over all units (nrb * nck)
  int grid;       // CTAs
  int ncf;        // chunks per full slice
  int ns;         // slices
  int nclast;     // chunks in the last slice
};

// The cut for a given grid: the slice width is the largest that keeps a unit within the shortest
// CTA range (floor(total / grid) chunks), so a unit is split between at most two CTAs.
Plan make_plan_fixed(int64_t R, int64_t K, int grid) {
  Plan p;
  p.nrb = (int)((R + TM - 1) / TM);
  p.nck = (int)((K + KB - 1) / KB);
  p.total = (int64_t)p.nrb * p.nck;
  p.grid = grid;
  int64_t u = p.total / p.grid;
  if (u > p.nck) u = p.nck;
  if (u < 1) u = 1;
  p.ncf = (int)u;
  p.ns = (p.nck + p.ncf - 1) / p.ncf;
  p.nclast = p.nck - (p.ns - 1) * p.ncf;
  return p;
}

// The row-block plan: cs CTAs per 128-row block, CTA k of a block taking K-slice k (ncf chunks, the
// last slice nclast; slices beyond ns are empty).
Plan make_plan_rows(int64_t R, int64_t K, int cs) {
  Plan p;
  p.nrb = (int)((R + TM - 1) / TM);
  p.nck = (int)((K + KB - 1) / KB);
  p.total = (int64_t)p.nrb * p.nck;
  p.grid = p.nrb * cs;
  p.ncf = (p.nck + cs - 1) / cs;
  p.ns = (p.nck + p.ncf - 1) / p.ncf;
  p.nclast = p.nck - (p.ns - 1) * p.ncf;
  return p;
}

// The grid for one phase: at most grid_cap CTAs, each with at least MIN_CHUNKS_PER_CTA chunks.
Plan make_plan(int64_t R, int64_t K, int grid_cap) {
  const int64_t total = ((R + TM - 1) / TM) * ((K + KB - 1) / KB);
  int64_t g = total / MIN_CHUNKS_PER_CTA;
  if (g > grid_cap) g = grid_cap;
  if (g < 1) g = 1;
  return make_plan_fixed(R, K, (int)g);
}

struct TcArgs {
  int R, K, T;
  int nrb, ns, ncf, nclast;  // 128-row blocks, K-slices, chunks per full / last slice
  int64_t total;             // chunks over all units
  int grid;
  int gsz, goff;  // grouped layers: rows per group (a multiple of 128) and B columns per group
  int stages;
  uint32_t stage_bytes;  // one weight tile and NB B boxes (hi, then lo)
  uint32_t idesc;
  float* P;   // partial sums of unit heads [ns][T][R]
  float* P2;  // partial sums of the tails of split units [ns][T][R]
  // row-block plan (cs >= 1): CTA b takes slice b % cs of row block b / cs, one unit or none; the
  // cs CTAs of a row block form a cluster and sum their slices in shared memory (cs = 1: the CTA
  // holds the whole row block). 0: the balanced split-K plan with partial sums P, P2.
  int cs;
  const int32_t* cols;
  int m;  // columns of Y (index bound)
  bf16* Y;
  int64_t ldy;
  uint16_t* yph;  // row-block plan, phase 1 with m > r: y_p hi and lo planes, else null
  uint16_t* ypl;
  int64_t ldyp;
  int split_f16;  // the planes in fp16 (else bf16)
  int* status;
  uint64_t timeout_ns;
};

// A CTA's run of chunks inside one unit.
struct Seg {
  int s, rb;  // the unit
  int c0;     // its first chunk within the unit
  int nc;     // chunks
};

// The segment that starts at chunk g of the global order and ends at the unit's end or at e.
__host__ __device__ __forceinline__ Seg seg_at(int nrb, int ns, int ncf, int nclast, int64_t g, int64_t e) {
  const int64_t per = (int64_t)nrb * ncf;
  int s = (int)(g / per);
  if (s > ns - 1) s = ns - 1;
  const int64_t rem = g - (int64_t)s * per;
  const int n = s < ns - 1 ? ncf : nclast;
  Seg q;
  q.s = s;
  q.rb = (int)(rem / n);
  q.c0 = (int)(rem % n);
  const int64_t uend = g - q.c0 + n;
  q.nc = (int)((uend < e ? uend : e) - g);
  return q;
}

__device__ __forceinline__ Seg seg_at(const TcArgs& a, int64_t g, int64_t e) {
  return seg_at(a.nrb, a.ns, a.ncf, a.nclast, g, e);
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

// Column (within the unit's K-slice) of the c-th chunk a CTA loads for segment q.
__device__ __forceinline__ int seg_col(const Seg& q, int c) { return (q.c0 + c) * KB; }

// kCl: the row-block plan with cs > 1 (a cluster per row block); only these instantiations hold
// cluster barriers and distributed shared-memory loads.
template <int NB, int TNT, bool kCl>
__global__ void __launch_bounds__(THREADS, CTAS_PER_SM)
    decode_tc_partial(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                      const __grid_constant__ CUtensorMap tmB1, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + (size_t)a.stages * a.stage_bytes);
  uint64_t* empty = full + MAX_STAGES;
  uint64_t* accf = empty + MAX_STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int64_t g0, g1;
  if (a.cs > 0) {  // slice k of row block rb: the unit that starts at chunk k nrb ncf + rb len(k)
    const int rb = (int)blockIdx.x / a.cs, k = (int)blockIdx.x % a.cs;
    const int len = k < a.ns - 1 ? a.ncf : a.nclast;
    g0 = k < a.ns ? (int64_t)k * a.nrb * a.ncf + (int64_t)rb * len : 0;
    g1 = k < a.ns ? g0 + len : 0;
  } else {
    g0 = ((int64_t)blockIdx.x * a.total) / a.grid;
    g1 = ((int64_t)(blockIdx.x + 1) * a.total) / a.grid;
  }

  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
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
      const int total = (int)(g1 - g0);
      const int pre = min(total, a.stages);
      {  // weight tiles of the first stages, before the dependency wait; their B boxes follow it
        int it = 0;
        for (int64_t g = g0; it < pre;) {
          const Seg q = seg_at(a, g, g1);
          for (int c = 0; c < q.nc && it < pre; ++c, ++it) {
            mbar_arrive_expect_tx(&full[it], a.stage_bytes);
            tma_load_2d(smem_u32(ring + (size_t)it * a.stage_bytes), &tmA, q.s * a.ncf * KB + seg_col(q, c),
                        q.rb * TM, &full[it]);
          }
          g += q.nc;
        }
      }
      pdl_wait_primary();
      int it = 0;
      bool dead = false;
      for (int64_t g = g0; g < g1 && !dead;) {
        const Seg q = seg_at(a, g, g1);
        g += q.nc;
        const int x0 = (a.gsz > 0 ? ((q.rb * TM) / a.gsz) * a.goff : 0) + q.s * a.ncf * KB;
        for (int c = 0; c < q.nc; ++c, ++it) {
          const int st = it % a.stages;
          uint8_t* stage = ring + (size_t)st * a.stage_bytes;
          const int kx = seg_col(q, c);
          if (it >= pre) {
            if (!mbar_wait(&empty[st], (uint32_t)((it / a.stages) - 1) & 1u, a.timeout_ns) || *abort_flag) {
              latch_status(a.status, PIFA_ERR_TIMEOUT);
              *abort_flag = 1;
              dead = true;
              break;
            }
            mbar_arrive_expect_tx(&full[st], a.stage_bytes);
            tma_load_2d(smem_u32(stage), &tmA, q.s * a.ncf * KB + kx, q.rb * TM, &full[st]);
          }
          tma_load_2d(smem_u32(stage + A_BYTES), &tmB0, x0 + kx, 0, &full[st]);
          if (NB > 1) tma_load_2d(smem_u32(stage + A_BYTES + (uint32_t)TNT * KB * 2), &tmB1, x0 + kx, 0, &full[st]);
        }
      }
      int issued = dead ? it : total;
      if (issued < pre) issued = pre;
      // nothing may land in shared memory once the CTA has left: the last use of every stage
      for (int j = issued > a.stages ? issued - a.stages : 0; j < issued; ++j)
        if (!mbar_wait(&full[j % a.stages], (uint32_t)(j / a.stages) & 1u, 100000000ull))
          latch_status(a.status, PIFA_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int it = 0, j = 0;
      bool dead = false;
      for (int64_t g = g0; g < g1; ++j) {
        const Seg q = seg_at(a, g, g1);
        g += q.nc;
        const int acc = j & 1;
        if (j >= 2 && !mbar_wait(&acce[acc], (uint32_t)((j >> 1) - 1) & 1u, a.timeout_ns)) {
          dead = true;
          break;
        }
        tc_fence_after();
        constexpr int NACC = kNacc<NB, TNT>;
        const uint32_t dacc = tmem + (uint32_t)(acc * NACC * TNT * NB);
        int e = 0;  // MMAs of this segment so far: accumulator e % NACC, first use overwrites
        for (int c = 0; c < q.nc; ++c, ++it) {
          const int st = it % a.stages;
          if (!mbar_wait(&full[st], (uint32_t)(it / a.stages) & 1u, a.timeout_ns) || *abort_flag) {
            dead = true;
            break;
          }
          tc_fence_after();
          const uint32_t at = smem_u32(ring + (size_t)st * a.stage_bytes);
#pragma unroll
          for (int kk = 0; kk < KB / 16; ++kk, ++e)
            mma_bf16_ss(dacc + (uint32_t)((e % NACC) * TNT * NB), sw128_desc(at + kk * 32),
                        sw128_desc(at + A_BYTES + kk * 32), a.idesc, e >= NACC ? 1u : 0u);
          mma_commit(&empty[st]);  // the stage is free once these MMAs have read it
        }
        if (dead) break;
        mma_commit(&accf[acc]);
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
    const int q4 = warp & 3;
    int j = 0;
    for (int64_t g = g0; g < g1; ++j) {
      const Seg q = seg_at(a, g, g1);
      g += q.nc;
      const int acc = j & 1;
      if (!mbar_wait(&accf[acc], (uint32_t)(j >> 1) & 1u, a.timeout_ns) || *abort_flag) {
        latch_status(a.status, PIFA_ERR_TIMEOUT);
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      if constexpr (TNT > 64) {
        // 128-token tiles (row-block plan only: one segment per CTA, one accumulator of TNT NB
        // columns): tokens in groups of 16, the hi and lo columns 16 g and TNT + 16 g loaded,
        // added and written out at once
        const uint32_t base = tmem + ((uint32_t)(q4 * 32) << 16);
        const int row = q.rb * TM + q4 * 32 + lane;
        const bool in = row < a.R;
        int col = -1;
        if (!kCl && in) {
          col = __ldg(a.cols + row);
          if ((unsigned)col >= (unsigned)a.m) {
            latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
            col = -1;
          }
        }
        if (kCl) fence_proxy_async_smem();  // the ring's last operands were read by the MMAs
        float* red = reinterpret_cast<float*>(ring);
        bool range_err = false;
        for (int g16 = 0; g16 < TNT / 16 && 16 * g16 < a.T; ++g16) {
          uint32_t vh[16], vl[16];
          tmem_ld_32x32b_x16(base + (uint32_t)(16 * g16), vh);
          if (NB > 1) tmem_ld_32x32b_x16(base + (uint32_t)(TNT + 16 * g16), vl);
          tmem_ld_wait();
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const int t = 16 * g16 + u;
            const float v = __uint_as_float(vh[u]) + (NB > 1 ? __uint_as_float(vl[u]) : 0.0f);
            if (t >= a.T) continue;
            if (kCl) {
              red[t * TM + q4 * 32 + lane] = v;
            } else if (in) {
              if (a.yph) {
                uint16_t hi, lo;
                if (a.split_f16)
                  split_hi_lo<true>(v, hi, lo, range_err);
                else
                  split_hi_lo<false>(v, hi, lo, range_err);
                a.yph[(int64_t)t * a.ldyp + row] = hi;
                a.ypl[(int64_t)t * a.ldyp + row] = lo;
              }
              if (col >= 0) a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(v);
            }
          }
        }
        if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
        if (!kCl && a.cs != 1) latch_status(a.status, PIFA_ERR_UNSUPPORTED);  // host never launches this
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[acc]);
        continue;
      } else {
      // the accumulators this segment wrote (fewer than NACC only when it has fewer MMAs), summed
      // in a fixed order
      constexpr int NACC = kNacc<NB, TNT>;
      const int used = min(NACC, q.nc * (KB / 16));
      const uint32_t base = tmem + ((uint32_t)(q4 * 32) << 16) + (uint32_t)(acc * NACC * TNT * NB);
      float sum[TNT];
#pragma unroll
      for (int t = 0; t < TNT; ++t) sum[t] = 0.0f;
      if (TNT == TN) {
        // column groups of 16: accumulator a, plane nb at (a NB + nb) 16, four loads in flight
        for (int c0 = 0; c0 < used * NB; c0 += 4) {
          uint32_t v[4][16];
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (c0 + k < used * NB) tmem_ld_32x32b_x16(base + (uint32_t)((c0 + k) * TN), v[k]);
          tmem_ld_wait();
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (c0 + k < used * NB)
#pragma unroll
              for (int t = 0; t < TN; ++t) sum[t % TNT] += __uint_as_float(v[k][t]);
        }
      } else {
        // wider token tiles: accumulator a, plane nb, tokens 16 g .. 16 g + 15 at column
        // (a NB + nb) TNT + 16 g; one (a, nb) pair's TNT / 16 loads in flight at a time
        for (int a2 = 0; a2 < used; ++a2)
#pragma unroll
          for (int nb = 0; nb < NB; ++nb) {
            uint32_t v[TNT / 16][16];
#pragma unroll
            for (int g = 0; g < TNT / 16; ++g)
              tmem_ld_32x32b_x16(base + (uint32_t)((a2 * NB + nb) * TNT + 16 * g), v[g]);
            tmem_ld_wait();
#pragma unroll
            for (int g = 0; g < TNT / 16; ++g)
#pragma unroll
              for (int j = 0; j < 16; ++j) sum[16 * g + j] += __uint_as_float(v[g][j]);
          }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce[acc]);  // this quarter of the accumulators may be refilled
      // the head of a unit goes to P and, when the unit was not split, zeros to P2; a tail to P2
      const int row = q.rb * TM + q4 * 32 + lane;
      if (kCl) {  // this slice's sums, [t][row of the block], for the cluster to add up
        fence_proxy_async_smem();  // the ring's last operands were read by the MMAs (async proxy)
        float* red = reinterpret_cast<float*>(ring);
#pragma unroll
        for (int t = 0; t < TNT; ++t)
          if (t < a.T) red[t * TM + q4 * 32 + lane] = sum[t];
        continue;
      }
      if (a.cs == 1) {  // the unit is the row block over all of K: its sums are the outputs
        if (row < a.R) {
          bool range_err = false;
          if (a.yph) {
#pragma unroll
            for (int t = 0; t < TNT; ++t)
              if (t < a.T) {
                uint16_t hi, lo;
                if (a.split_f16)
                  split_hi_lo<true>(sum[t], hi, lo, range_err);
                else
                  split_hi_lo<false>(sum[t], hi, lo, range_err);
                a.yph[(int64_t)t * a.ldyp + row] = hi;
                a.ypl[(int64_t)t * a.ldyp + row] = lo;
              }
          }
          if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
          const int col = __ldg(a.cols + row);
          if ((unsigned)col >= (unsigned)a.m) {
            latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
          } else {
#pragma unroll
            for (int t = 0; t < TNT; ++t)
              if (t < a.T) a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(sum[t]);
          }
        }
        continue;
      }
      if (row < a.R) {
        const size_t off = (size_t)q.s * a.T * a.R + row;
        const bool whole = q.c0 == 0 && q.nc == (q.s < a.ns - 1 ? a.ncf : a.nclast);
        float* dst = (q.c0 == 0 ? a.P : a.P2) + off;
#pragma unroll
        for (int t = 0; t < TNT; ++t)
          if (t < a.T) {
            dst[(size_t)t * a.R] = sum[t];
            if (whole) a.P2[off + (size_t)t * a.R] = 0.0f;
          }
      }
      }  // TNT <= 64
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (kCl) {
    // Every CTA of the cluster has its slice's sums in its own shared memory once all arrive;
    // CTA k then finishes rows [k rpr, (k + 1) rpr) of the block, adding the slices in rank
    // order (deterministic). Every wait above is bounded, so each CTA reaches both barriers; the
    // second keeps each CTA resident until no peer reads its shared memory any more.
    cluster_sync_all();
    const int k = (int)blockIdx.x % a.cs, rb = (int)blockIdx.x / a.cs;
    const int rpr = TM / a.cs;
    const int nsrc = a.ns < a.cs ? a.ns : a.cs;
    const uint32_t red = smem_u32(ring);
    bool range_err = false;
    for (int idx = threadIdx.x; idx < rpr * a.T; idx += THREADS) {
      const int t = idx / rpr, rr = k * rpr + idx % rpr;
      const int row = rb * TM + rr;
      const uint32_t off = red + (uint32_t)(t * TM + rr) * 4u;
      float sum = 0.0f;
      for (int p = 0; p < nsrc; ++p) sum += ld_dsmem_f32(mapa_shared(off, (uint32_t)p));
      if (row >= a.R) continue;
      if (a.yph) {
        uint16_t hi, lo;
        if (a.split_f16)
          split_hi_lo<true>(sum, hi, lo, range_err);
        else
          split_hi_lo<false>(sum, hi, lo, range_err);
        a.yph[(int64_t)t * a.ldyp + row] = hi;
        a.ypl[(int64_t)t * a.ldyp + row] = lo;
      }
      const int col = __ldg(a.cols + row);
      if ((unsigned)col >= (unsigned)a.m)
        latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
      else
        a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(sum);
    }
    if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
    cluster_sync_all();
  }
}

struct ReduceArgs {
  const float* P;
  const float* P2;
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

// One row j of one token t per thread: Y[t, cols[j]] = bf16 of sum_s (P[s][t][j] + P2[s][t][j])
// in slice order. The loads of G slices (G >= ns up to 16) are all in flight at once (no load
// depends on another), so the kernel takes about one memory round trip; G is no larger than the
// slice count needs, which keeps registers low and the grid resident. Phase 1 also splits y_p.
template <bool kF16, int G>
__global__ void __launch_bounds__(256) decode_tc_reduce(ReduceArgs a) {
  pdl_launch_dependents();
  pdl_wait_primary();
  const int64_t n = (int64_t)a.T * a.R;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int t = (int)(i / a.R), j = (int)(i % a.R);
  float sum = 0.0f;
  for (int s0 = 0; s0 < a.ns; s0 += G) {
    float h[G], w[G];
#pragma unroll
    for (int k = 0; k < G; ++k)
      if (s0 + k < a.ns) {
        h[k] = __ldcg(a.P + (size_t)(s0 + k) * n + i);
        w[k] = __ldcg(a.P2 + (size_t)(s0 + k) * n + i);
      }
#pragma unroll
    for (int k = 0; k < G; ++k)
      if (s0 + k < a.ns) sum += h[k] + w[k];
  }
  bool range_err = false;
  if (a.yph) {
    uint16_t hi, lo;
    split_hi_lo<kF16>(sum, hi, lo, range_err);
    a.yph[(int64_t)t * a.ldyp + j] = hi;
    a.ypl[(int64_t)t * a.ldyp + j] = lo;
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

int grid_cap() {
  const int g = CTAS_PER_SM * sm_count_tc();
  return g < GRID_MAX ? g : GRID_MAX;
}

}  // namespace

int64_t decode_tc_partial_bytes(int64_t R, int64_t K, int64_t T, int NB) {
  (void)NB;
  const Plan p = make_plan(R, K, GRID_MAX);  // the most slices any grid can give
  return 2 * (int64_t)p.ns * T * R * 4;      // P and P2
}

int launch_decode_tc(const DecodeTcPhase& ph, int* status, uint64_t timeout_ns, cudaStream_t stream) {
  const int NB = ph.planes;
  if (ph.R < 1 || ph.K < 1 || ph.T < 1 || ph.T > kMaxTokensTc)
    return pifa_fail(PIFA_ERR_INVALID_ARG, "decode_tc: empty or oversized phase");
  // token tile (MMA N per plane): 16, 32, 64 or 128 rows of B, those beyond T zero-filled by TMA
  const int TNT = ph.T <= 16 ? 16 : ph.T <= 32 ? 32 : ph.T <= 64 ? 64 : 128;
  // Row-block plan: a phase of at most grid_cap() 128-row blocks gives each block cs CTAs (cs the
  // largest power of two up to 8 that keeps the grid within grid_cap() and every slice at least one
  // chunk), CTA k taking K-slice k; the block's cs CTAs form a cluster that adds up its slices in
  // shared memory and writes Y (and y_p's planes) itself. No partial sums in global memory and no
  // reduce kernel: one kernel and one kernel boundary fewer per phase (measured on the 70B gate/up
  // layer, whose phase 2 has 192 row blocks and takes cs = 1: T = 16 57.1 -> 53.0 us per call, T = 8
  // 54.3 -> 51.5 us; clusters where a phase has fewer blocks, against balanced ranges and a reduce
  // kernel: 70B q/o T = 16 28.9 -> 26.4 us, 70B gate/up T = 64 67.3 -> 60.8, 7B MLP down T = 64
  // 41.4 -> 27.0). Longer phases deal balanced chunk ranges and sum P + P2 in a second kernel.
  const int64_t nrb_all = (ph.R + TM - 1) / TM, nck_all = (ph.K + KB - 1) / KB;
  int cs = 0;
  if (nrb_all <= grid_cap()) {
    cs = 1;
    while (cs < MAX_CLUSTER_TC && nrb_all * cs * 2 <= grid_cap() && cs * 2 <= nck_all) cs *= 2;
  }
  // a 128-token tile fills all of a CTA's 256 TMEM columns with one accumulator (hi and lo as one
  // N = 256 operand), so only the row-block plan's one segment per CTA can use it
  if (TNT > 64 && cs == 0)
    return pifa_fail(PIFA_ERR_UNSUPPORTED, "decode with T > 64 needs phases of at most two row blocks per SM");
  const Plan p = cs > 0 ? make_plan_rows(ph.R, ph.K, cs) : make_plan(ph.R, ph.K, grid_cap());
  TcArgs a = {};
  a.R = (int)ph.R;
  a.K = (int)ph.K;
  a.T = (int)ph.T;
  a.nrb = p.nrb;
  a.ns = p.ns;
  a.ncf = p.ncf;
  a.nclast = p.nclast;
  a.total = p.total;
  a.grid = p.grid;
  a.gsz = (int)ph.gsz;
  a.goff = (int)ph.goff;
  a.stage_bytes = A_BYTES + (uint32_t)(NB * TNT) * KB * 2;
  const bool f16 = ph.mma_f16;
  a.idesc = f16 ? idesc_f16_f32(TM, (uint32_t)(TNT * NB)) : idesc_bf16_f32(TM, (uint32_t)(TNT * NB));
  a.P = ph.P;
  a.P2 = ph.P + (size_t)p.ns * ph.T * ph.R;
  a.cs = cs;
  a.cols = ph.cols;
  a.m = (int)ph.m;
  a.Y = reinterpret_cast<bf16*>(ph.Y);
  a.ldy = ph.ldy;
  a.yph = ph.yph;
  a.ypl = ph.ypl;
  a.ldyp = ph.ldyp;
  a.split_f16 = ph.split_f16 ? 1 : 0;
  a.status = status;
  a.timeout_ns = timeout_ns;
  const size_t fixed = 1024 + 512;  // alignment slack; barriers and the TMEM slot
  const int stages = (int)((SMEM_PER_CTA - fixed) / a.stage_bytes);
  a.stages = stages > MAX_STAGES ? MAX_STAGES : stages;
  const size_t smem = fixed + (size_t)a.stages * a.stage_bytes;
  // the row-block plan's cluster sums ([T][128] fp32) reuse the ring once its MMAs are done
  if (cs > 1 && (size_t)TM * TNT * 4 > (size_t)a.stages * a.stage_bytes)
    return pifa_fail(PIFA_ERR_UNSUPPORTED, "decode_tc: ring smaller than the cluster sums");

  CUtensorMap tA, tB0, tB1;
  int st;
  if ((st = make_tmap_2d(&tA, ph.dtype, ph.A, ph.R, ph.K, ph.lda, KB, TM)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tB0, ph.dtype, ph.B0, ph.T, ph.bcols, ph.ldb, KB, (uint32_t)TNT)) != PIFA_OK) return st;
  if (NB > 1 && (st = make_tmap_2d(&tB1, ph.dtype, ph.B1, ph.T, ph.bcols, ph.ldb, KB, (uint32_t)TNT)) != PIFA_OK)
    return st;
  if (NB == 1) tB1 = tB0;

  using Kern = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, TcArgs);
  static const Kern kerns[2][4][2] = {
      {{decode_tc_partial<1, 16, false>, decode_tc_partial<1, 16, true>},
       {decode_tc_partial<1, 32, false>, decode_tc_partial<1, 32, true>},
       {decode_tc_partial<1, 64, false>, decode_tc_partial<1, 64, true>},
       {decode_tc_partial<1, 128, false>, decode_tc_partial<1, 128, true>}},
      {{decode_tc_partial<2, 16, false>, decode_tc_partial<2, 16, true>},
       {decode_tc_partial<2, 32, false>, decode_tc_partial<2, 32, true>},
       {decode_tc_partial<2, 64, false>, decode_tc_partial<2, 64, true>},
       {decode_tc_partial<2, 128, false>, decode_tc_partial<2, 128, true>}}};
  const Kern kern = kerns[NB - 1][TNT == 16 ? 0 : TNT == 32 ? 1 : TNT == 64 ? 2 : 3][cs > 1 ? 1 : 0];
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaFuncSetAttribute(decode_tc)", e);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.grid);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)(cs > 1 ? cs : 1);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cs > 1 ? 2 : 1;
  e = pifa_launch_ex(&cfg, kern, tA, tB0, tB1, a);
  if (e != cudaSuccess) return pifa_fail_cuda("decode_tc partial launch", e);
  if (cs > 0) return PIFA_OK;

  ReduceArgs r = {};
  r.P = a.P;
  r.P2 = a.P2;
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
  rc.numAttrs = 1;  // programmatic serialization only, no cluster
  void (*red)(ReduceArgs);
  if (a.ns <= 2)
    red = ph.split_f16 ? decode_tc_reduce<true, 2> : decode_tc_reduce<false, 2>;
  else if (a.ns <= 4)
    red = ph.split_f16 ? decode_tc_reduce<true, 4> : decode_tc_reduce<false, 4>;
  else if (a.ns <= 8)
    red = ph.split_f16 ? decode_tc_reduce<true, 8> : decode_tc_reduce<false, 8>;
  else
    red = ph.split_f16 ? decode_tc_reduce<true, 16> : decode_tc_reduce<false, 16>;
  e = pifa_launch_ex(&rc, red, r);
  if (e != cudaSuccess) return pifa_fail_cuda("decode_tc reduce launch", e);
  return PIFA_OK;
}
