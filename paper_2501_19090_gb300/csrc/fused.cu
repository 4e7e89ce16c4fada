// fused.cu -- fused PIFA prefill: Algorithm 2 (Sec. 3.2) for one 256-token tile at a time in a
// single persistent kernel, one thread-block cluster of G CTAs (G <= 16) per token tile.
//
// For a token tile (256 rows of X):
//   GEMM 1 (steps 2, 4): the r rows of W_p are split in 128-row M-tiles over the G CTAs. Each CTA
//           accumulates its tiles of Y_p^T = W_p X^T in tensor memory (tcgen05, M = 128 weight
//           rows, N = 256 tokens, fp32), then writes bf16 Y_p into Y's pivot columns and Y_p as a
//           hi + lo pair (C's storage type) into L2-resident T x r staging matrices.
//   sync:   each CTA's epilogue releases its slice to every CTA of the cluster (remote mbarrier
//           arrive, cluster scope); producers acquire before loading Y_p.
//   GEMM 2 (steps 3, 5): the m - r rows of C are split the same way; K = r runs twice into one
//           accumulator, against hi and then lo, read back from L2; the epilogue writes bf16 Y_np
//           into Y's non-pivot columns.
// Y_p never leaves the chip (L2 and shared memory) between the two contractions, and there is
// no separate gather/scatter pass. A single fp16 Y_p (11 significant bits) is not enough: C's
// rows have norms near 8 and Y_np = C Y_p cancels, so the rounding error of Y_p is amplified
// past the 2e-2 elementwise bound on layers with large |Y_p|. fp16 values beyond +-65504
// saturate and latch PIFA_ERR_RANGE.
//
// The token operand of both GEMMs (X, then Y_p) is the same for every CTA of the cluster, so each
// CTA loads 256/G of its rows with TMA multicast into all G CTAs' shared memory: the cluster reads
// each token tile from L2 once per k-step instead of G times. Weight tiles are per CTA.
//
// Per CTA (192 threads): warp 0 = TMA producer, warp 1 = TMEM owner and MMA issuer (one
// thread), warps 2-5 = epilogue (TMEM lanes 0-127). Stages: up to two 128 x 64 weight tiles plus
// one 256 x 64 token tile, 128-byte swizzle; 4 stages with one weight tile, 3 with two. TMEM:
// two 256-column fp32 accumulators. Every wait is bounded (globaltimer); a CTA that times out
// latches PIFA_ERR_TIMEOUT, stops issuing work and unwinds to the closing cluster barrier.
#include <algorithm>
#include <cstdio>
#include <mutex>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;
constexpr uint32_t A_BYTES = BM * BK * 2;   // 16 KB
constexpr uint32_t B_BYTES = BN * BK * 2;   // 32 KB
constexpr uint32_t DATA_BYTES = 196608;     // 192 KB of stages
constexpr int MAX_STAGES = 4;
constexpr uint32_t TMEM_COLS = 512;         // two 256-column accumulators
constexpr size_t SMEM_BYTES = 1024 + DATA_BYTES + 256;

struct FusedArgs {
  int T, m, r;
  int mt1, mt2;          // 128-row M-tiles of W_p (r rows) and of C (m - r rows)
  int kc1, kc2;          // 64-wide k-chunks of GEMM 1 (K = n) and GEMM 2 (K = r)
  int passes1, passes2;  // passes per token tile, identical for every CTA of the cluster
  int a_slots;           // weight tiles per stage (1 or 2)
  int stages;
  int ntiles;            // 256-token tiles
  const int32_t* piv;
  const int32_t* nonpiv;
  bf16* Y;
  int64_t ldy;
  uint16_t* yp_hi;       // T x ldyp staging of Y_p's hi part (L2 resident), C's type
  uint16_t* yp_lo;       // the lo part
  int64_t ldyp;
  int c_f16;             // C (and the Y_p pair) in fp16 (1) or bf16 (0)
  int* status;
  uint64_t timeout_ns;
};

// M-tiles CTA `c` of a G-CTA cluster handles in pass q: c + G * (a_slots * q + i), i < a_slots.
__device__ __forceinline__ int pass_tiles(int mt, int G, int c, int a_slots, int q, int (&tiles)[2]) {
  int n = 0;
  for (int i = 0; i < a_slots; ++i) {
    const int t = c + G * (a_slots * q + i);
    if (t < mt) tiles[n++] = t;
  }
  return n;
}

__global__ void __launch_bounds__(192, 1)
    pifa_fused_prefill(const __grid_constant__ CUtensorMap tmWp, const __grid_constant__ CUtensorMap tmX,
                       const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmYp,
                       const __grid_constant__ CUtensorMap tmYl, FusedArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + DATA_BYTES);
  uint64_t* empty = full + MAX_STAGES;
  uint64_t* acc_full = empty + MAX_STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* yp_ready = acc_empty + 2;
  uint64_t* mma_drain = yp_ready + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = (int)cluster_nctarank();
  const int c = (int)cluster_ctarank();
  const uint16_t all_mask = (uint16_t)((1u << G) - 1u);
  const int rows_per = BN / G;  // token rows of the shared tile this CTA loads for everyone
  const uint32_t stage_bytes = p.a_slots * A_BYTES + B_BYTES;

  if (warp == 0 && lane == 0) {
    for (int s = 0; s < MAX_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], (uint32_t)G);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4);
    }
    mbar_init(yp_ready, (uint32_t)(4 * G));
    mbar_init(mma_drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmWp);
    prefetch_tmap(&tmX);
    prefetch_tmap(&tmC);
    prefetch_tmap(&tmYp);
    prefetch_tmap(&tmYl);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // every CTA's barriers exist before anyone multicasts or arrives remotely
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int cid = (int)cluster_id_x(), ncl = (int)nclusters_x();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      uint32_t it = 0, tile_iter = 0;
      bool dead = false;
      for (int tile = cid; tile < p.ntiles && !dead; tile += ncl, ++tile_iter) {
        const int tok0 = tile * BN;
        for (int phase = 1; phase <= 2 && !dead; ++phase) {
          if (phase == 2) {
            if (p.mt2 == 0) break;
            if (!mbar_wait_cluster(yp_ready, tile_iter & 1u, p.timeout_ns)) {
              latch_status(p.status, PIFA_ERR_TIMEOUT);
              *abort_flag = 1;
              dead = true;
              break;
            }
            fence_proxy_async_global();
          }
          const CUtensorMap* mA = phase == 1 ? &tmWp : &tmC;
          const int mt = phase == 1 ? p.mt1 : p.mt2;
          const int kc = phase == 1 ? p.kc1 : 2 * p.kc2;  // GEMM 2: K = r against hi, then lo
          const int passes = phase == 1 ? p.passes1 : p.passes2;
          for (int q = 0; q < passes && !dead; ++q) {
            int tiles[2];
            const int nA = pass_tiles(mt, G, c, p.a_slots, q, tiles);
            for (int kk2 = 0; kk2 < kc; ++kk2, ++it) {
              const bool lo_half = phase == 2 && kk2 >= p.kc2;
              const int k = lo_half ? kk2 - p.kc2 : kk2;
              const CUtensorMap* mB = phase == 1 ? &tmX : (lo_half ? &tmYl : &tmYp);
              const uint32_t s = it % (uint32_t)p.stages, u = it / (uint32_t)p.stages;
              if (u > 0 && !mbar_wait(&empty[s], (u - 1) & 1u, p.timeout_ns)) {
                latch_status(p.status, PIFA_ERR_TIMEOUT);
                *abort_flag = 1;
                dead = true;
                break;
              }
              uint8_t* st = smem + s * stage_bytes;
              mbar_arrive_expect_tx(&full[s], nA * A_BYTES + B_BYTES);
              for (int i = 0; i < nA; ++i) tma_load_2d(smem_u32(st + i * A_BYTES), mA, k * BK, tiles[i] * BM, &full[s]);
              tma_load_2d_multicast(smem_u32(st + p.a_slots * A_BYTES + c * rows_per * 128), mB, k * BK,
                                    tok0 + c * rows_per, &full[s], all_mask);
            }
          }
        }
      }
      // tail: every stage's last use must be released by all G consumers (their MMAs are done
      // reading this CTA's shared memory and their multicast arrivals have landed here)
      const uint32_t first = it > (uint32_t)p.stages ? it - (uint32_t)p.stages : 0u;
      for (uint32_t j = first; j < it; ++j) {
        const uint32_t s = j % (uint32_t)p.stages, u = j / (uint32_t)p.stages;
        if (!mbar_wait(&empty[s], u & 1u, dead ? 100000000ull : p.timeout_ns)) latch_status(p.status, PIFA_ERR_TIMEOUT);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      uint32_t it = 0, au[2] = {0u, 0u};
      bool dead = false;
      for (int tile = cid; tile < p.ntiles && !dead; tile += ncl) {
        for (int phase = 1; phase <= 2 && !dead; ++phase) {
          if (phase == 2 && p.mt2 == 0) break;
          const uint32_t idesc =
              (phase == 1 || !p.c_f16) ? idesc_bf16_f32(BM, BN) : idesc_f16_f32(BM, BN);
          const int mt = phase == 1 ? p.mt1 : p.mt2, kc = phase == 1 ? p.kc1 : 2 * p.kc2;
          const int passes = phase == 1 ? p.passes1 : p.passes2;
          for (int q = 0; q < passes && !dead; ++q) {
            int tiles[2];
            const int nA = pass_tiles(mt, G, c, p.a_slots, q, tiles);
            for (int i = 0; i < nA; ++i) {
              if (au[i] > 0 && !mbar_wait(&acc_empty[i], (au[i] - 1) & 1u, p.timeout_ns)) {
                latch_status(p.status, PIFA_ERR_TIMEOUT);
                *abort_flag = 1;
                dead = true;
              }
            }
            if (dead) break;
            tc_fence_after();
            for (int k = 0; k < kc; ++k, ++it) {
              const uint32_t s = it % (uint32_t)p.stages, u = it / (uint32_t)p.stages;
              if (!mbar_wait(&full[s], u & 1u, p.timeout_ns)) {
                latch_status(p.status, PIFA_ERR_TIMEOUT);
                *abort_flag = 1;
                dead = true;
                break;
              }
              tc_fence_after();
              const uint32_t st = smem_u32(smem + s * stage_bytes);
              const uint32_t b = st + p.a_slots * A_BYTES;
              for (int i = 0; i < nA; ++i) {
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                  mma_bf16_ss(tmem + (uint32_t)(i * 256), sw128_desc(st + i * A_BYTES + kk * 32),
                              sw128_desc(b + kk * 32), idesc, (k > 0 || kk > 0) ? 1u : 0u);
              }
              mma_commit_multicast(&empty[s], all_mask);  // this CTA is done reading stage s
            }
            if (dead) break;
            for (int i = 0; i < nA; ++i) {
              mma_commit(&acc_full[i]);
              ++au[i];
            }
          }
        }
      }
      if (dead) mma_commit(&acc_full[0]);  // harmless extra arrive; the epilogue sees the abort flag
      // TMEM is freed at the end only after every MMA this thread issued has completed
      mma_commit(mma_drain);
      if (!mbar_wait(mma_drain, 0, 100000000ull)) latch_status(p.status, PIFA_ERR_TIMEOUT);
    }
  } else {
    // ---------------- epilogue: warps 2..5 ----------------
    const int qd = warp & 3;  // TMEM lane quarter this warp may access
    uint32_t au[2] = {0u, 0u};
    bool dead = false;
    for (int tile = cid; tile < p.ntiles && !dead; tile += ncl) {
      const int tok0 = tile * BN;
      for (int phase = 1; phase <= 2 && !dead; ++phase) {
        if (phase == 2 && p.mt2 == 0) break;
        const int mt = phase == 1 ? p.mt1 : p.mt2;
        const int rows_total = phase == 1 ? p.r : p.m - p.r;
        const int32_t* cols = phase == 1 ? p.piv : p.nonpiv;
        const int passes = phase == 1 ? p.passes1 : p.passes2;
        for (int q = 0; q < passes && !dead; ++q) {
          int tiles[2];
          const int nA = pass_tiles(mt, G, c, p.a_slots, q, tiles);
          for (int i = 0; i < nA; ++i) {
            if (!mbar_wait(&acc_full[i], au[i] & 1u, p.timeout_ns) || *abort_flag) {
              latch_status(p.status, PIFA_ERR_TIMEOUT);
              dead = true;
              break;
            }
            tc_fence_after();
            const int row = tiles[i] * BM + qd * 32 + lane;  // weight row held by this thread
            int col = -1;
            if (row < rows_total) {
              col = cols[row];
              if ((unsigned)col >= (unsigned)p.m) {
                latch_status(p.status, PIFA_ERR_DEVICE_INDEX);
                col = -1;
              }
            }
            bool range_err = false;
#pragma unroll 1
            for (int cc = 0; cc < BN / 32; ++cc) {
              uint32_t v[32];
              tmem_ld_32x32b_x32(tmem + ((uint32_t)(qd * 32) << 16) + (uint32_t)(i * 256 + cc * 32), v);
              tmem_ld_wait();
              if (col >= 0) {
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                  const int t = tok0 + cc * 32 + j;
                  if (t < p.T) {
                    const float f = __uint_as_float(v[j]);
                    p.Y[(int64_t)t * p.ldy + col] = __float2bfloat16_rn(f);
                    if (phase == 1) {
                      uint16_t h, l;
                      if (p.c_f16) {
                        float fs = f;
                        if (fabsf(fs) > 65504.0f) {
                          range_err = true;
                          fs = copysignf(65504.0f, fs);
                        }
                        const __half hh = __float2half_rn(fs);
                        h = __half_as_ushort(hh);
                        l = __half_as_ushort(__float2half_rn(fs - __half2float(hh)));
                      } else {
                        const bf16 hb = __float2bfloat16_rn(f);
                        h = __bfloat16_as_ushort(hb);
                        l = __bfloat16_as_ushort(__float2bfloat16_rn(f - __bfloat162float(hb)));
                      }
                      p.yp_hi[(int64_t)t * p.ldyp + row] = h;
                      p.yp_lo[(int64_t)t * p.ldyp + row] = l;
                    }
                  }
                }
              }
            }
            if (range_err) latch_status(p.status, PIFA_ERR_RANGE);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[i]);
            ++au[i];
          }
        }
        if (phase == 1 && !dead) {
          // publish this warp's part of the tile's Y_p to every CTA of the cluster
          __threadfence();
          fence_proxy_async_global();
          __syncwarp();
          if (lane == 0) {
            const uint32_t local = smem_u32(yp_ready);
            for (int r2 = 0; r2 < G; ++r2) mbar_arrive_remote(mapa_shared(local, (uint32_t)r2));
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while another may still multicast into it or arrive on it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

inline int64_t pad8(int64_t v) { return (v + 7) / 8 * 8; }

struct ClusterPlan {
  int G = 0;
  int max_clusters = 0;
};

char g_plan_error[192] = "fused prefill: cluster plan not computed";

// Largest cluster size in {16, 8, 4, 2} the device can schedule with this kernel's shared memory,
// and how many such clusters fit at once. Queried once per device.
ClusterPlan query_plan() {
  static ClusterPlan plans[64];
  static bool done[64] = {};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return ClusterPlan{};
  std::lock_guard<std::mutex> lock(mu);
  if (done[dev]) return plans[dev];
  int major = 0;
  cudaError_t e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (e != cudaSuccess || major < 10) {
    std::snprintf(g_plan_error, sizeof g_plan_error, "fused prefill: compute capability query (%s, major %d)",
                  cudaGetErrorName(e), major);
    cudaGetLastError();
    return plans[dev];
  }
  e = cudaFuncSetAttribute(pifa_fused_prefill, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(pifa_fused_prefill, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) {
    std::snprintf(g_plan_error, sizeof g_plan_error, "fused prefill: cudaFuncSetAttribute failed (%s)",
                  cudaGetErrorName(e));
    cudaGetLastError();
    return plans[dev];
  }
  for (int G : {16, 8, 4, 2}) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(G);
    cfg.blockDim = dim3(192);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = G;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, pifa_fused_prefill, &cfg);
    if (e == cudaSuccess && n > 0) {
      plans[dev].G = G;
      plans[dev].max_clusters = n;
      done[dev] = true;  // only a successful plan is cached; a failure is retried next call
      break;
    }
    std::snprintf(g_plan_error, sizeof g_plan_error,
                  "fused prefill: cudaOccupancyMaxActiveClusters(G=%d) gave %d clusters (%s)", G, n,
                  cudaGetErrorName(e));
    cudaGetLastError();
  }
  return plans[dev];
}

}  // namespace

int64_t prefill_fused_workspace_bytes(const PifaShape& s) {
  return 2 * (((s.T * pad8(s.r) * 2 + 255) / 256) * 256);  // Y_p hi and lo staging, T x pad8(r) each
}

// (one layer only: grouped layers run the split GEMMs)
bool prefill_fused_supported(const PifaShape& s) { return s.groups == 1 && query_plan().G >= 2; }

int launch_prefill_fused(const PifaShape& s, const PifaPointers& p, int* status, uint64_t timeout_ns,
                         cudaStream_t stream) {
  const ClusterPlan plan = query_plan();
  if (plan.G < 2) return pifa_fail(PIFA_ERR_UNSUPPORTED, g_plan_error);
  const int G = plan.G;
  FusedArgs a = {};
  a.T = (int)s.T;
  a.m = (int)s.m;
  a.r = (int)s.r;
  a.mt1 = (int)((s.r + BM - 1) / BM);
  a.mt2 = (int)((s.m - s.r + BM - 1) / BM);
  a.kc1 = (int)((s.n + BK - 1) / BK);
  a.kc2 = (int)((s.r + BK - 1) / BK);
  const int per1 = (a.mt1 + G - 1) / G, per2 = (a.mt2 + G - 1) / G;
  a.a_slots = std::max(per1, per2) >= 2 ? 2 : 1;
  a.stages = a.a_slots == 2 ? 3 : 4;
  a.passes1 = (per1 + a.a_slots - 1) / a.a_slots;
  a.passes2 = (per2 + a.a_slots - 1) / a.a_slots;
  a.ntiles = (int)((s.T + BN - 1) / BN);
  a.piv = p.piv;
  a.nonpiv = p.nonpiv;
  a.Y = reinterpret_cast<bf16*>(p.Y);
  a.ldy = s.ldy;
  const int64_t one = ((s.T * pad8(s.r) * 2 + 255) / 256) * 256;
  a.yp_hi = reinterpret_cast<uint16_t*>(p.ws);
  a.yp_lo = reinterpret_cast<uint16_t*>(reinterpret_cast<uint8_t*>(p.ws) + one);
  a.ldyp = pad8(s.r);
  a.c_f16 = s.c_dtype == PIFA_DTYPE_FP16 ? 1 : 0;
  a.status = status;
  a.timeout_ns = timeout_ns;

  const uint32_t rows_per = (uint32_t)(BN / G);
  CUtensorMap tWp, tX, tC, tYp, tYl;
  int st;
  if ((st = make_tmap_2d(&tWp, PIFA_DTYPE_BF16, p.Wp, s.r, s.n, s.ldwp, BK, BM)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tX, PIFA_DTYPE_BF16, p.X, s.T, s.n, s.ldx, BK, rows_per)) != PIFA_OK) return st;
  if (s.m > s.r) {
    if ((st = make_tmap_2d(&tC, s.c_dtype, p.C, s.m - s.r, s.r, s.ldc, BK, BM)) != PIFA_OK) return st;
  } else {
    tC = tWp;  // never read when m == r
  }
  if ((st = make_tmap_2d(&tYp, s.c_dtype, a.yp_hi, s.T, s.r, a.ldyp, BK, rows_per)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tYl, s.c_dtype, a.yp_lo, s.T, s.r, a.ldyp, BK, rows_per)) != PIFA_OK) return st;

  const int nclusters = std::max(1, std::min(a.ntiles, plan.max_clusters));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(nclusters * G));
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = G;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, pifa_fused_prefill, tWp, tX, tC, tYp, tYl, a);
  if (e != cudaSuccess) return pifa_fail_cuda("fused prefill launch", e);
  return PIFA_OK;
}
