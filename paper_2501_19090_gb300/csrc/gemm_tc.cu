// gemm_tc.cu -- general bf16 contraction D = alpha A B^T (+ gathered addend) on the 5th-generation
// tensor cores, for the PIFA backward pass (fine-tuning, Sec. 5.1; Sec. 6) and the M online
// accumulators (Sec. 4): products whose operands are stored transposed (MN-major).
//
//   A is M x K, B is N x K (bf16). Each operand is either K-major (stored as rows of K contiguous
//   elements: A[m * lda + k]) or MN-major (stored as K rows of contiguous M or N: A[k * lda + m]);
//   the instruction descriptor's transpose bits tell the tensor core which, and TMA fetches
//   K-major tiles as 128 x 64 boxes and MN-major tiles as 64 (MN) x 64 (K) boxes, 128-byte swizzle.
//   D (M x N, fp32 accumulate) is written as bf16, as fp32, added into an fp32 matrix, or as a
//   hi + lo pair of bf16 matrices (hi = bf16(D), lo = bf16(D - hi)) for a later contraction that must
//   not lose D's low bits. A second K pass into the same accumulator with A2 in place of A and/or
//   B2 in place of B (same layouts) consumes such a pair: D = (A + A2) B^T or A (B + B2)^T.
//
// One CTA per 128 x bn tile (bn <= 256), 192 threads: warp 0 issues TMA loads into a 4-stage ring,
// warp 1 owns the TMEM accumulator (bn fp32 columns) and issues tcgen05.mma (M = 128, N = bn,
// K = 16) from one thread, warps 2-5 drain TMEM (a lane quarter each: one row of D per thread).
// Every wait is bounded (globaltimer); on timeout the CTA latches PIFA_ERR_TIMEOUT, drains what it
// has in flight and returns.
#include <cuda_bf16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

constexpr int BM = 128;
constexpr int BNMAX = 256;
constexpr int BK = 64;
constexpr int THREADS = 192;
// Two shapes of the kernel. Config 0: one CTA per SM, tiles up to 256 wide, a 4-stage ring, the
// values to add in (the old D, an addend) staged into shared memory while the MMAs run. Config 1:
// two CTAs per SM, tiles up to 128 wide, 3 stages, the values to add in (if any) loaded right
// before the stores: one CTA's epilogue runs under the other's MMAs. gemm_tc picks one per GEMM
// (measured, 4096 x 4096 r = 2048 layer, T = 2048: the backward 425.7 -> 353.3 us, bit for bit
// the same).
template <int CFG>
constexpr int kStages = CFG == 0 ? 4 : 3;
template <int CFG>
constexpr int kBnMax = CFG == 0 ? BNMAX : 128;
constexpr uint32_t A_BYTES = BM * BK * 2;     // 16 KB
constexpr uint32_t B_MAX = BNMAX * BK * 2;    // 32 KB
constexpr uint32_t MN_BOX = 64 * BK * 2;      // one MN-major box: 64 (MN) x 64 (K), 8 KB

struct GemmTcArgs {
  int M, N, K;
  int bn;             // N per tile
  int d_trans;        // 1: store D^T (element (i, j) at D[j * ldd + i]); no accumulation or addend
  int prefetch;       // 1: the epilogue adds values read from global memory (D itself or the addend),
                      //    staged into shared memory while the MMAs run
  uint32_t idesc;
  int passes;         // 1, or 2 (the second pass reads tmA2 and tmB2)
  void* D;            // M x N, pitch ldd: bf16 (out_mode 0) or fp32 (1: store, 2: add into), or
  void* D2;           // out_mode 3: D the hi and D2 the lo bf16 plane
  int64_t ldd;
  int out_mode;
  float alpha;
  const bf16* add;    // optional addend: D[i][j] += add[i * ldadd + (add_idx ? add_idx[j] : j)]
  const int32_t* add_idx;
  int64_t ldadd;
  int add_bound;      // columns of the addend (index bound)
  int late_add;       // 1 (config 1): the epilogue loads the old D and the addend itself
  int upper;          // 1: tiles wholly below the diagonal (rows all > columns) do nothing
  int* status;
  uint64_t timeout_ns;
};

// Shared-memory descriptor of an MN-major operand tile written by TMA as 64-element (128-byte)
// swizzled rows, one row per K index: 8-row groups 1024 bytes apart along K (stride byte offset),
// 64-element MN blocks `mn_stride` bytes apart (leading byte offset).
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t saddr, uint32_t mn_stride) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((mn_stride >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

template <bool AMN, bool BMN, int CFG>
__global__ void __launch_bounds__(THREADS, CFG == 0 ? 1 : 2)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                   const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmB2, GemmTcArgs p) {
  constexpr int STAGES = kStages<CFG>;
  constexpr uint32_t TMEM_ALLOC = (uint32_t)kBnMax<CFG>;
  // a symmetric product's tiles wholly below the diagonal are not computed
  if (p.upper && (int)blockIdx.y * BM >= (int)blockIdx.x * p.bn + p.bn) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t b_bytes = (uint32_t)p.bn * BK * 2;
  const uint32_t stage_bytes = A_BYTES + b_bytes;
  // the epilogue's staged addends: 4 warps x 32 rows x (bn + 1) fp32, after the stages
  float* ext_sm = reinterpret_cast<float*>(smem + STAGES * stage_bytes);
  const uint32_t ext_bytes = p.prefetch ? 4u * 32u * (uint32_t)(p.bn + 1) * 4u : 0u;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * stage_bytes + ((ext_bytes + 15) & ~15u));
  uint64_t* empty = full + STAGES;
  uint64_t* accf = empty + STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accf + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * p.bn, m0 = blockIdx.y * BM;
  const int kchunks = (p.K + BK - 1) / BK;
  const int total = kchunks * p.passes;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    if (p.passes > 1) {
      prefetch_tmap(&tmA2);
      prefetch_tmap(&tmB2);
    }
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_ALLOC);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      pdl_wait_primary();
      int issued = 0;
      for (int it = 0; it < total; ++it) {
        const int s = it % STAGES, kc = it % kchunks;
        const CUtensorMap* ma = it < kchunks ? &tmA : &tmA2;
        const CUtensorMap* mb = it < kchunks ? &tmB : &tmB2;
        if (it >= STAGES && !mbar_wait(&empty[s], (uint32_t)((it / STAGES) - 1) & 1u, p.timeout_ns)) {
          latch_status(p.status, PIFA_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        uint8_t* sa = smem + s * stage_bytes;
        uint8_t* sb = sa + A_BYTES;
        const int k0 = kc * BK;
        mbar_arrive_expect_tx(&full[s], A_BYTES + b_bytes);
        if (AMN) {
          tma_load_2d(smem_u32(sa), ma, m0, k0, &full[s]);
          tma_load_2d(smem_u32(sa + MN_BOX), ma, m0 + 64, k0, &full[s]);
        } else {
          tma_load_2d(smem_u32(sa), ma, k0, m0, &full[s]);
        }
        if (BMN) {
          for (int h = 0; h < p.bn / 64; ++h) tma_load_2d(smem_u32(sb + h * MN_BOX), mb, n0 + 64 * h, k0, &full[s]);
        } else {
          tma_load_2d(smem_u32(sb), mb, k0, n0, &full[s]);
        }
        issued = it + 1;
      }
      // nothing may land in shared memory after the CTA has left
      for (int i = issued > STAGES ? issued - STAGES : 0; i < issued; ++i)
        if (!mbar_wait(&full[i % STAGES], (uint32_t)(i / STAGES) & 1u, 100000000ull))
          latch_status(p.status, PIFA_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      for (int it = 0; it < total; ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&full[s], (uint32_t)(it / STAGES) & 1u, p.timeout_ns) || *abort_flag) {
          latch_status(p.status, PIFA_ERR_TIMEOUT);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t a = smem_u32(smem + s * stage_bytes);
        const uint32_t b = a + A_BYTES;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          // K-major tiles advance 32 bytes along a swizzled row per K = 16; MN-major tiles advance
          // 16 rows (2048 bytes)
          const uint64_t ad = AMN ? sw128_mn_desc(a + kk * 2048, MN_BOX) : sw128_desc(a + kk * 32);
          const uint64_t bd = BMN ? sw128_mn_desc(b + kk * 2048, MN_BOX) : sw128_desc(b + kk * 32);
          mma_bf16_ss(tmem, ad, bd, p.idesc, (it > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&empty[s]);
      }
      mma_commit(accf);
      if (!mbar_wait(accf, 0, 100000000ull)) latch_status(p.status, PIFA_ERR_TIMEOUT);
    }
  } else {
    // ---------------- epilogue: warps 2..5, TMEM lane quarter warp % 4 ----------------
    // Each 32 x 32 block (32 rows of this quarter, 32 columns) goes through this warp's 4 KB of the
    // stage memory (free once every MMA has completed): read from TMEM one row per lane, written to
    // global memory one row per store instruction, the lanes covering 32 consecutive columns.
    const int q = warp & 3;
    float* ext = ext_sm + (warp - 2) * 32 * (p.bn + 1);  // this warp's rows: [32][bn + 1]
    if (p.prefetch) {
      // while the MMAs run: the old D (accumulation) plus the addend. The lanes cover consecutive
      // columns (coalesced); each thread issues the loads of 8 rows x 4 columns before storing any
      // of them to shared memory, so that many loads are in flight at once.
      for (int r0 = 0; r0 < 32; r0 += 8) {
        float v[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int row = m0 + q * 32 + r0 + i, c = lane + 32 * j, col = n0 + c;
            float e = 0.0f;
            if (c < p.bn && row < p.M && col < p.N) {
              if (p.out_mode == 2) e = __ldcg(reinterpret_cast<const float*>(p.D) + (int64_t)row * p.ldd + col);
              if (p.add) {
                const int ac = p.add_idx ? __ldg(p.add_idx + col) : col;
                if ((unsigned)ac < (unsigned)p.add_bound)
                  e += __bfloat162float(p.add[(int64_t)row * p.ldadd + ac]);
                else
                  latch_status(p.status, PIFA_ERR_DEVICE_INDEX);
              }
            }
            v[i][j] = e;
          }
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (lane + 32 * j < p.bn) ext[(r0 + i) * (p.bn + 1) + lane + 32 * j] = v[i][j];
      }
      __syncwarp();
    }
    const bool ok = mbar_wait(accf, 0, p.timeout_ns) && !*abort_flag;
    if (!ok) latch_status(p.status, PIFA_ERR_TIMEOUT);
    tc_fence_after();
    if (ok) {
      float* tile = reinterpret_cast<float*>(smem) + (warp - 2) * (32 * 33);
      const int ncols = min(p.bn, p.N - n0);
      for (int c0 = 0; c0 < ncols; c0 += 32) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, v);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; ++j) tile[lane * 33 + j] = __uint_as_float(v[j]);
        __syncwarp();
        const int nrows = min(32, p.M - (m0 + q * 32));
        if (p.d_trans) {
          // D^T: one column of the block per step, the lanes covering consecutive rows (coalesced)
          const int row = m0 + q * 32 + lane;
          for (int cc = 0; cc < 32; ++cc) {
            const int col = n0 + c0 + cc;
            if (col >= p.N) break;
            if (lane >= nrows) continue;
            float f = p.alpha * tile[lane * 33 + cc];
            if (p.prefetch) f += ext[lane * (p.bn + 1) + c0 + cc];
            const int64_t o = (int64_t)col * p.ldd + row;
            if (p.out_mode == 3) {
              const bf16 h = __float2bfloat16_rn(f);
              reinterpret_cast<bf16*>(p.D)[o] = h;
              reinterpret_cast<bf16*>(p.D2)[o] = __float2bfloat16_rn(f - __bfloat162float(h));
            } else if (p.out_mode == 0) {
              reinterpret_cast<bf16*>(p.D)[o] = __float2bfloat16_rn(f);
            } else {
              reinterpret_cast<float*>(p.D)[o] = f;
            }
          }
        } else {
          // D: one row of the block per step, the lanes covering consecutive columns (coalesced)
          const int col = n0 + c0 + lane;
          auto put = [&](int rr, float f) {
            const int64_t o = (int64_t)(m0 + q * 32 + rr) * p.ldd + col;
            if (p.out_mode == 3) {
              const bf16 h = __float2bfloat16_rn(f);
              reinterpret_cast<bf16*>(p.D)[o] = h;
              reinterpret_cast<bf16*>(p.D2)[o] = __float2bfloat16_rn(f - __bfloat162float(h));
            } else if (p.out_mode == 0) {
              reinterpret_cast<bf16*>(p.D)[o] = __float2bfloat16_rn(f);
            } else {
              reinterpret_cast<float*>(p.D)[o] = f;
            }
          };
          if (CFG == 0) {
            for (int rr = 0; rr < nrows; ++rr) {
              if (col >= p.N) break;
              float f = p.alpha * tile[rr * 33 + lane];
              if (p.prefetch) f += ext[rr * (p.bn + 1) + c0 + lane];
              put(rr, f);
            }
          } else {
            float addv[32];
            if (p.late_add) {
              // the block's values to add in, all 32 loads in flight before the first store
              int ac = col;
              if (p.add && p.add_idx && col < p.N) {
                ac = __ldg(p.add_idx + col);
                if ((unsigned)ac >= (unsigned)p.add_bound) {
                  latch_status(p.status, PIFA_ERR_DEVICE_INDEX);
                  ac = -1;
                }
              }
#pragma unroll
              for (int rr = 0; rr < 32; ++rr) {
                const int row = m0 + q * 32 + rr;
                float e = 0.0f;
                if (rr < nrows && col < p.N) {
                  if (p.out_mode == 2) e = __ldcg(reinterpret_cast<const float*>(p.D) + (int64_t)row * p.ldd + col);
                  if (p.add && ac >= 0) e += __bfloat162float(p.add[(int64_t)row * p.ldadd + ac]);
                }
                addv[rr] = e;
              }
            }
#pragma unroll
            for (int rr = 0; rr < 32; ++rr) {
              if (rr >= nrows || col >= p.N) continue;
              float f = p.alpha * tile[rr * 33 + lane];
              if (p.late_add) f += addv[rr];
              put(rr, f);
            }
          }
        }
        __syncwarp();  // the next block reuses the tile
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_ALLOC);
  }
}

int sm_count_gemm() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      n = 1;
  }
  return n;
}

}  // namespace

int gemm_tc(const GemmTc& g, int* status, uint64_t timeout_ns, cudaStream_t stream) {
  if (g.M <= 0 || g.N <= 0) return PIFA_OK;
  if (g.K <= 0) return pifa_fail(PIFA_ERR_INVALID_ARG, "gemm_tc: K must be positive");
  const int64_t lim = (int64_t)1 << 30;
  if (g.M >= lim || g.N >= lim || g.K >= lim) return pifa_fail(PIFA_ERR_INVALID_ARG, "gemm_tc: size >= 2^30");
  GemmTcArgs a = {};
  a.M = (int)g.M;
  a.N = (int)g.N;
  a.K = (int)g.K;
  // tile width: MN-major B tiles come in 64-column boxes, K-major ones in multiples of 16
  const int64_t unit = g.b_mn ? 64 : 16;
  // with values to add in, a config-0 tile is at most 128 wide so that their staging fits beside
  // the ring
  const bool adds = g.out_mode == 2 || g.add;
  if (g.d_trans && adds) return pifa_fail(PIFA_ERR_UNSUPPORTED, "gemm_tc: transposed store with an addend");
  const int64_t bnmax0 = adds ? 128 : BNMAX;
  const int64_t bn0 = g.N >= bnmax0 ? bnmax0 : (g.N + unit - 1) / unit * unit;
  const int64_t tiles0 = ((g.N + bn0 - 1) / bn0) * ((g.M + BM - 1) / BM);
  // Config per GEMM, from timing each backward and M-accumulator product under both (4096 x 4096,
  // r = 2048 layer, T = 2048; us, config 0 -> 1):
  //   gathered addend, hi/lo out (dY_p)          78.8 -> 55.4   config 1
  //   bf16 or fp32 out, > 1 wave (dX, dW_p, dC)  81.5 -> 77.6, 82.9 -> 79.0, 42.3 -> 40.5   config 1
  //   fp32 read-modify-write (X X^T, Y_t X^T)    155.8 -> 344.0, 219.7 -> 391.6   config 0
  //   hi/lo out, no addend (Y_p, Y_t^T)          36.4 -> 41.0, 114.4 -> 128.4   config 0
  // Config 0 stages the old D while the MMAs run; config 1's 128-wide tiles read shared memory at
  // the MMA's limit, which only pays where the epilogue dominates.
  const bool multi = tiles0 > sm_count_gemm();
  const int cfg_id = g.out_mode == 2 ? 0 : g.add ? 1 : g.out_mode == 3 ? 0 : (multi ? 1 : 0);
  const int64_t bnmax = cfg_id == 0 ? bnmax0 : kBnMax<1>;
  a.bn = (int)(g.N >= bnmax ? bnmax : (g.N + unit - 1) / unit * unit);
  a.prefetch = (cfg_id == 0 && adds) ? 1 : 0;
  a.late_add = (cfg_id == 1 && adds) ? 1 : 0;
  a.d_trans = g.d_trans ? 1 : 0;
  if (g.upper && g.M != g.N) return pifa_fail(PIFA_ERR_INVALID_ARG, "gemm_tc: upper triangle of a non-square product");
  a.upper = g.upper ? 1 : 0;
  a.idesc = idesc_bf16_f32(BM, (uint32_t)a.bn) | (g.a_mn ? (1u << 15) : 0u) | (g.b_mn ? (1u << 16) : 0u);
  a.passes = (g.A2 || g.B2) ? 2 : 1;
  a.D = g.D;
  a.D2 = g.D2;
  a.ldd = g.ldd;
  a.out_mode = g.out_mode;
  a.alpha = g.alpha;
  a.add = reinterpret_cast<const bf16*>(g.add);
  a.add_idx = g.add_idx;
  a.ldadd = g.ldadd;
  a.add_bound = (int)g.add_bound;
  a.status = status;
  a.timeout_ns = timeout_ns;
  CUtensorMap tA, tA2, tB, tB2;
  int st;
  for (int k = 0; k < 2; ++k) {
    const void* base = k == 0 ? g.A : g.A2;
    CUtensorMap* map = k == 0 ? &tA : &tA2;
    if (!base) {
      tA2 = tA;
      continue;
    }
    if (g.a_mn)
      st = make_tmap_2d(map, PIFA_DTYPE_BF16, base, g.K, g.M, g.lda, 64, BK);
    else
      st = make_tmap_2d(map, PIFA_DTYPE_BF16, base, g.M, g.K, g.lda, BK, BM);
    if (st != PIFA_OK) return st;
  }
  for (int k = 0; k < 2; ++k) {
    const void* base = k == 0 ? g.B : g.B2;
    CUtensorMap* map = k == 0 ? &tB : &tB2;
    if (!base) {
      tB2 = tB;
      continue;
    }
    if (g.b_mn)
      st = make_tmap_2d(map, PIFA_DTYPE_BF16, base, g.K, g.N, g.ldb, 64, BK);
    else
      st = make_tmap_2d(map, PIFA_DTYPE_BF16, base, g.N, g.K, g.ldb, BK, (uint32_t)a.bn);
    if (st != PIFA_OK) return st;
  }
  auto kern = cfg_id == 0 ? (g.a_mn ? (g.b_mn ? gemm_tc_kernel<true, true, 0> : gemm_tc_kernel<true, false, 0>)
                                    : (g.b_mn ? gemm_tc_kernel<false, true, 0> : gemm_tc_kernel<false, false, 0>))
                          : (g.a_mn ? (g.b_mn ? gemm_tc_kernel<true, true, 1> : gemm_tc_kernel<true, false, 1>)
                                    : (g.b_mn ? gemm_tc_kernel<false, true, 1> : gemm_tc_kernel<false, false, 1>));
  const size_t ext_bytes = a.prefetch ? (size_t)4 * 32 * (a.bn + 1) * 4 : 0;
  const int stages = cfg_id == 0 ? kStages<0> : kStages<1>;
  const size_t smem = 1024 + (size_t)stages * (A_BYTES + (size_t)a.bn * BK * 2) + (ext_bytes + 15) / 16 * 16 + 256;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaFuncSetAttribute(gemm_tc)", e);
  const unsigned nt = (unsigned)((g.N + a.bn - 1) / a.bn), mt = (unsigned)((g.M + BM - 1) / BM);
  if (mt > 65535u) return pifa_fail(PIFA_ERR_UNSUPPORTED, "gemm_tc: more than 65535 row tiles");
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nt, mt);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  e = pifa_launch_ex(&cfg, kern, tA, tA2, tB, tB2, a);
  if (e != cudaSuccess) return pifa_fail_cuda("gemm_tc launch", e);
  return PIFA_OK;
}
