// prefill.cu -- PIFA forward for many tokens on the 5th-generation tensor cores (tcgen05).
//
// Split variant: two launches of one warp-specialised tcgen05 GEMM.
//   GEMM 1 (Algorithm 2, steps 2 and 4): D1 = W_p X^T, tile 128 weight rows x 256 tokens.
//           Epilogue writes bf16(Y_p) into the pivot columns Y[:, I[j]] and the pair
//           hi = rnd(Y_p), lo = rnd(Y_p - hi) into two T x r scratch matrices, rnd rounding to
//           C's storage type (bf16 or fp16).
//   GEMM 2 (Algorithm 2, steps 3 and 5): D2 = C [hi | lo]^T accumulated over K = r twice (hi pass
//           then lo pass), epilogue writes bf16(Y_np) into Y[:, I^c[i]].
// Weight rows are the MMA M dimension and tokens the N dimension, so the accumulator in tensor
// memory holds one weight row per TMEM lane: an epilogue warp's 32 lanes are 32 consecutive
// weight rows, which for a fixed token land in 32 ascending output columns of one row of Y.
//
// Per CTA (576 threads): warp 0 issues TMA loads into a 4-stage shared-memory ring (A tile
// 128 x 64, B tile 256 x 64, bf16, 128-byte swizzle), warp 1 owns the TMEM allocation and issues
// tcgen05.mma (M=128, N=256, K=16) from one thread, warps 2-17 drain the fp32 accumulator
// (128 lanes x 256 columns of TMEM) through tcgen05.ld. The epilogue, not the tensor cores, was
// the largest cost of this kernel (16 of 66 us at 4096 x 4096, r = 2048, T = 2048): its output is
// a column scatter into Y of 2-byte stores. Sixteen warps issue them, and Y_p's hi/lo planes go
// out as 16-byte stores after a transpose through shared memory. Every wait is bounded
// (globaltimer); on timeout the CTA latches PIFA_ERR_TIMEOUT, drains what it has in flight and
// returns.
//
// GEMMs whose full-width tiles leave most SMs idle (GEMM 1 of the 70B layers has 32 row blocks;
// T of a few hundred gives one token tile) split K instead: a tile's 2 or 4 CTAs form a cluster,
// each accumulates its K-slice, stores the fp32 partial tile in its own freed stage ring, and the
// cluster adds the slices through distributed shared memory in rank order before the epilogue.
#include <utility>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

constexpr int BM = 128;  // weight rows per tile (MMA M)
constexpr int BK = 64;   // K per stage: one 128-byte swizzle row of bf16
constexpr uint32_t A_BYTES = BM * BK * 2;

// Two shapes of the same kernel. Config 0: one CTA per SM, up to 256 tokens per tile, a 4-stage
// ring and 16 epilogue warps (the fastest when a GEMM fits one or two waves). Config 1: two CTAs
// per SM, up to 160 tokens per tile, 3 stages and 8 epilogue warps: one CTA's epilogue runs while
// the other's MMAs keep the tensor core busy, which pays on GEMMs of many waves (measured, same
// outputs bit for bit: T = 8192 on the 4096 x 4096, r = 2048 layer 241.1 -> 226.2 us; 70B q/o
// T = 4096 427.3 -> 390.1 us). A GEMM of one or two waves leaves little to overlap, and there the
// one-CTA shape's wider tiles and deeper ring are kept.
template <int CFG>
struct PCfg;
template <>
struct PCfg<0> {
  static constexpr int BN = 256, STAGES = 4, EPI_WARPS = 16, CTAS = 1;
};
template <>
struct PCfg<1> {
  static constexpr int BN = 160, STAGES = 3, EPI_WARPS = 8, CTAS = 2;
};
template <int CFG>
struct PC : PCfg<CFG> {
  using B = PCfg<CFG>;
  static constexpr int THREADS = 64 + 32 * B::EPI_WARPS;  // + the TMA producer and the MMA warp
  static constexpr uint32_t B_BYTES = B::BN * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t TMEM_COLS = 256;  // fp32 accumulator, one column per token (a power of two)
  static constexpr size_t SMEM_BYTES = 1024 /*alignment slack*/ + B::STAGES * STAGE_BYTES + 256 /*barriers*/;
};

// Epilogue modes: what GEMM 1 also writes besides Y (GEMM 2 writes Y only).
enum { EPI_Y_ONLY = 0, EPI_SPLIT_BF16 = 1, EPI_SPLIT_F16 = 2 };

struct GemmArgs {
  uint32_t idesc;        // tcgen05 instruction descriptor (bf16 or fp16 operands)
  int M;                 // weight rows (r for GEMM 1, m - r for GEMM 2)
  int N;                 // tokens T
  int bn;                // tokens per tile (MMA N, TMA box rows of B): a multiple of 16, <= BN
  int tok_fast;          // 1: blockIdx.x walks token tiles (CTAs of one weight-row block together), else row tiles
  int kchunks;           // ceil(K / 64) per pass
  int passes;            // 1, or 2 for the hi + lo passes of GEMM 2
  int gsz;               // grouped layers (GEMM 2): weight rows per group (whole tiles), else 0
  int goff;              // B columns between consecutive groups' K ranges (r), when gsz > 0
  const int32_t* cols;   // output column of each weight row (I or I^c)
  int m;                 // columns of Y (index bound)
  bf16* Y;
  int64_t ldy;
  void* yp_hi;           // GEMM 1 only: T x ldyp scratch, hi part (bf16 or fp16)
  void* yp_lo;           // lo part
  int64_t ldyp;
  int* status;
  uint64_t timeout_ns;
  int ks;                // K-slices per tile (kCl): the CTAs blockIdx.z = 0 .. ks - 1 of a tile form a cluster
};

// kCl: split-K over a cluster of ks CTAs per tile (grids with too few tiles to fill the GPU). CTA z
// accumulates the K-steps [z total / ks, (z + 1) total / ks) of both passes, stores its fp32
// partial tile in its own shared memory (the stage ring, free once its MMAs are done) and, after a
// cluster barrier, adds rows [z 128 / ks, (z + 1) 128 / ks) of every peer's partial tile in rank
// order (distributed shared memory) and writes them out as the epilogue would. Only these
// instantiations hold cluster barriers and distributed shared-memory loads.
template <int kEpi, int CFG, bool kCl>
__global__ void __launch_bounds__(PC<CFG>::THREADS, PC<CFG>::CTAS)
    pifa_umma_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                   const __grid_constant__ CUtensorMap tmB1, GemmArgs p) {
  constexpr int STAGES = PC<CFG>::STAGES, EPI_WARPS = PC<CFG>::EPI_WARPS, BN = PC<CFG>::BN;
  constexpr uint32_t STAGE_BYTES = PC<CFG>::STAGE_BYTES, TMEM_COLS = PC<CFG>::TMEM_COLS;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  pdl_launch_dependents();  // the next kernel may launch now (its CTAs take SMs this grid leaves idle)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // launch order: along the shorter of M and T (see run_gemm), so that one wave's operand tiles
  // stay in L2
  const int m0 = (p.tok_fast ? blockIdx.y : blockIdx.x) * BM;
  const int n0 = (p.tok_fast ? blockIdx.x : blockIdx.y) * p.bn;
  const uint32_t b_bytes = (uint32_t)p.bn * BK * 2;  // one B box
  const int bx0 = p.gsz > 0 ? (m0 / p.gsz) * p.goff : 0;  // the tile's group's first B column
  const int ksteps = p.kchunks * p.passes;
  const int z = kCl ? (int)blockIdx.z : 0;
  const int i0 = kCl ? (int)(((int64_t)z * ksteps) / p.ks) : 0;  // this CTA's K-steps [i0, i0 + total)
  const int total = kCl ? (int)(((int64_t)(z + 1) * ksteps) / p.ks) - i0 : ksteps;

  if (warp == 0 && lane == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB0);
    if (p.passes > 1) prefetch_tmap(&tmB1);
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
      // ---------------- TMA producer ----------------
      // The weight tiles (A) do not depend on the previous kernel: those of the first stages go out
      // before the dependency wait, raising the expected bytes without arriving; the activation
      // tiles (B: X, or the y_p planes GEMM 1 wrote) follow the wait and bring the arrival.
      const int pre = total < STAGES ? total : STAGES;
      for (int i = 0; i < pre; ++i) {
        mbar_expect_tx(&full[i], A_BYTES);
        tma_load_2d(smem_u32(smem + i * STAGE_BYTES), &tmA, ((i0 + i) % p.kchunks) * BK, m0, &full[i]);
      }
      pdl_wait_primary();
      for (int i = 0; i < pre; ++i) {
        const int pass = (i0 + i) / p.kchunks, kc = (i0 + i) % p.kchunks;
        mbar_arrive_expect_tx(&full[i], b_bytes);
        tma_load_2d(smem_u32(smem + i * STAGE_BYTES + A_BYTES), pass ? &tmB1 : &tmB0, bx0 + kc * BK, n0, &full[i]);
      }
      int issued = pre;
      for (int i = pre; i < total; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (uint32_t)(i / STAGES) & 1u;
        if (!mbar_wait(&empty[s], ph ^ 1u, p.timeout_ns)) {
          *abort_flag = 1;
          latch_status(p.status, PIFA_ERR_TIMEOUT);
          break;
        }
        if (*abort_flag) break;
        const int pass = (i0 + i) / p.kchunks, kc = (i0 + i) % p.kchunks;
        uint8_t* sa = smem + s * STAGE_BYTES;
        mbar_arrive_expect_tx(&full[s], A_BYTES + b_bytes);
        tma_load_2d(smem_u32(sa), &tmA, kc * BK, m0, &full[s]);
        tma_load_2d(smem_u32(sa + A_BYTES), pass ? &tmB1 : &tmB0, bx0 + kc * BK, n0, &full[s]);
        issued = i + 1;
      }
      // drain: the last use of every stage must have landed before the CTA may exit
      const uint64_t drain_ns = 100000000ull;
      for (int i = (issued > STAGES ? issued - STAGES : 0); i < issued; ++i) {
        const int s = i % STAGES;
        if (!mbar_wait(&full[s], (uint32_t)(i / STAGES) & 1u, drain_ns)) latch_status(p.status, PIFA_ERR_TIMEOUT);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      for (int i = 0; i < total; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (uint32_t)(i / STAGES) & 1u;
        if (!mbar_wait(&full[s], ph, p.timeout_ns)) {
          *abort_flag = 1;
          latch_status(p.status, PIFA_ERR_TIMEOUT);
          break;
        }
        tc_fence_after();
        const uint32_t a = smem_u32(smem + s * STAGE_BYTES);
        const uint32_t b = a + A_BYTES;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          mma_bf16_ss(tmem, sw128_desc(a + kk * 32), sw128_desc(b + kk * 32), p.idesc, (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit(&empty[s]);
      }
      mma_commit(acc_full);  // arrives once every MMA issued above has completed
      // the CTA frees TMEM only after its MMAs are done, even if the epilogue gave up waiting
      if (!mbar_wait(acc_full, 0, 100000000ull)) latch_status(p.status, PIFA_ERR_TIMEOUT);
    }
  } else {
    // ---------------- epilogue: warps 2 .. 2 + EPI_WARPS - 1 ----------------
    // Warp w may access TMEM lanes 32 (w % 4) .. + 31, one quarter of the tile's weight rows; the
    // EPI_WARPS / 4 warps of a quarter split the tile's tokens. Many warps keep the store issue
    // rate up: the scattered 2-byte stores into Y's columns are instruction-bound.
    constexpr int kSlices = EPI_WARPS / 4;
    constexpr int kChunks = (BN / 32 + kSlices - 1) / kSlices;  // 32-token chunks per warp (the last ones may lie beyond bn)
    const int tend = min(n0 + p.bn, p.N);       // this tile's tokens end here
    const int q = warp & 3;
    const int slice = (warp - 2) >> 2;
    const int row = m0 + q * 32 + lane;
    // Y_p's hi and lo planes are written transposed through this warp's 4 KB of the stage memory
    // (free once every MMA has completed) as 16-byte stores of 8 consecutive weight rows.
    uint16_t* st_hi = reinterpret_cast<uint16_t*>(smem) + (warp - 2) * 2048;
    uint16_t* st_lo = st_hi + 1024;
    const bool ok = mbar_wait(acc_full, 0, p.timeout_ns);
    if (!ok) latch_status(p.status, PIFA_ERR_TIMEOUT);
    tc_fence_after();
    if (kCl) {
      // this K-slice's partial tile into the ring as [token][128 rows] fp32 (the lanes of a
      // warp on consecutive rows): the cluster adds the slices below
      if (ok && !*abort_flag) {
        fence_proxy_async_smem();  // the ring's last operands were read by the MMAs (async proxy)
        float* red = reinterpret_cast<float*>(smem);
        const int tend = min(n0 + p.bn, p.N);
#pragma unroll 1
        for (int ci = 0; ci < kChunks; ++ci) {
          const int tb = n0 + (slice * kChunks + ci) * 32;
          if (tb >= tend) break;  // warp-uniform
          uint32_t v[32];
          tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(tb - n0), v);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; ++j) red[(tb - n0 + j) * BM + q * 32 + lane] = __uint_as_float(v[j]);
        }
      }
    } else if (ok && !*abort_flag) {
      int col = -1;
      if (row < p.M) {
        col = p.cols[row];
        if ((unsigned)col >= (unsigned)p.m) {
          latch_status(p.status, PIFA_ERR_DEVICE_INDEX);
          col = -1;
        }
      }
      bool range_err = false;
#pragma unroll 1
      for (int ci = 0; ci < kChunks; ++ci) {
        const int tb = n0 + (slice * kChunks + ci) * 32;  // first token of the chunk
        if (tb >= tend) break;  // warp-uniform; TMEM columns beyond bn hold no result
        uint32_t v[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(tb - n0), v);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float f = __uint_as_float(v[j]);
          if (col >= 0 && tb + j < tend) p.Y[(int64_t)(tb + j) * p.ldy + col] = __float2bfloat16_rn(f);
          if (kEpi == EPI_SPLIT_BF16) {
            const bf16 h = __float2bfloat16_rn(f);
            st_hi[j * 32 + lane] = __bfloat16_as_ushort(h);
            st_lo[j * 32 + lane] = __bfloat16_as_ushort(__float2bfloat16_rn(f - __bfloat162float(h)));
          } else if (kEpi == EPI_SPLIT_F16) {
            float fs = f;
            if (fabsf(fs) > 65504.0f) {
              range_err = true;
              fs = copysignf(65504.0f, fs);
            }
            const __half hh = __float2half_rn(fs);
            st_hi[j * 32 + lane] = __half_as_ushort(hh);
            st_lo[j * 32 + lane] = __half_as_ushort(__float2half_rn(fs - __half2float(hh)));
          }
        }
        if (kEpi != EPI_Y_ONLY) {
          __syncwarp();
          // 128 chunks of 16 bytes per plane: token j = c / 4, weight rows 8 (c % 4) .. + 7
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int c = lane + 32 * k;
            const int t = tb + (c >> 2);
            const int rr = m0 + q * 32 + (c & 3) * 8;  // rows beyond M hold zeros (padding columns)
            if (t < tend && rr < p.ldyp) {
              *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(p.yp_hi) + (int64_t)t * p.ldyp + rr) =
                  *reinterpret_cast<const uint4*>(st_hi + c * 8);
              *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(p.yp_lo) + (int64_t)t * p.ldyp + rr) =
                  *reinterpret_cast<const uint4*>(st_lo + c * 8);
            }
          }
          __syncwarp();  // the next chunk reuses the staging
        }
      }
      if (range_err) latch_status(p.status, PIFA_ERR_RANGE);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (kCl) {
    // Every CTA of the cluster has its partial tile in its own shared memory once all arrive (every
    // wait above is bounded, so each CTA gets here); CTA z then finishes rows [z rpc, (z + 1) rpc)
    // of the tile for all its tokens, adding the slices in rank order (deterministic), and a
    // second barrier keeps each CTA resident until no peer reads its shared memory any more.
    cluster_sync_all();
    const int rpc = BM / p.ks;
    const int ntok = min(p.bn, p.N - n0);
    const uint32_t red = smem_u32(smem);
    bool range_err = false;
    for (int idx = threadIdx.x; idx < rpc * ntok; idx += PC<CFG>::THREADS) {
      const int t = idx / rpc, rr = z * rpc + idx % rpc;
      const int row = m0 + rr;
      const uint32_t off = red + (uint32_t)(t * BM + rr) * 4u;
      float f = 0.0f;
      for (int k = 0; k < p.ks; ++k) f += ld_dsmem_f32(mapa_shared(off, (uint32_t)k));
      if (row >= p.M) continue;
      const int tok = n0 + t;
      const int col = __ldg(p.cols + row);
      if ((unsigned)col >= (unsigned)p.m)
        latch_status(p.status, PIFA_ERR_DEVICE_INDEX);
      else
        p.Y[(int64_t)tok * p.ldy + col] = __float2bfloat16_rn(f);
      if (kEpi == EPI_SPLIT_BF16) {
        const bf16 h = __float2bfloat16_rn(f);
        reinterpret_cast<uint16_t*>(p.yp_hi)[(int64_t)tok * p.ldyp + row] = __bfloat16_as_ushort(h);
        reinterpret_cast<uint16_t*>(p.yp_lo)[(int64_t)tok * p.ldyp + row] =
            __bfloat16_as_ushort(__float2bfloat16_rn(f - __bfloat162float(h)));
      } else if (kEpi == EPI_SPLIT_F16) {
        float fs = f;
        if (fabsf(fs) > 65504.0f) {
          range_err = true;
          fs = copysignf(65504.0f, fs);
        }
        const __half hh = __float2half_rn(fs);
        reinterpret_cast<uint16_t*>(p.yp_hi)[(int64_t)tok * p.ldyp + row] = __half_as_ushort(hh);
        reinterpret_cast<uint16_t*>(p.yp_lo)[(int64_t)tok * p.ldyp + row] =
            __half_as_ushort(__float2half_rn(fs - __half2float(hh)));
      }
    }
    if (range_err) latch_status(p.status, PIFA_ERR_RANGE);
    cluster_sync_all();
  }
}

template <int CFG>
int run_gemm(int epi, const CUtensorMap& a, const CUtensorMap& b0, const CUtensorMap& b1, const GemmArgs& args,
             cudaStream_t stream) {
  const bool cl = CFG == 0 && args.ks > 1;  // split-K clusters: config 0 only (one CTA per SM)
  auto kern = cl ? (epi == EPI_SPLIT_BF16 ? pifa_umma_gemm<EPI_SPLIT_BF16, CFG, CFG == 0>
                    : epi == EPI_SPLIT_F16 ? pifa_umma_gemm<EPI_SPLIT_F16, CFG, CFG == 0>
                                          : pifa_umma_gemm<EPI_Y_ONLY, CFG, CFG == 0>)
                 : (epi == EPI_SPLIT_BF16 ? pifa_umma_gemm<EPI_SPLIT_BF16, CFG, false>
                    : epi == EPI_SPLIT_F16 ? pifa_umma_gemm<EPI_SPLIT_F16, CFG, false>
                                          : pifa_umma_gemm<EPI_Y_ONLY, CFG, false>);
  if (args.ks > 1 && !cl) return pifa_fail(PIFA_ERR_UNSUPPORTED, "prefill: split-K needs the one-CTA shape");
  if (cl && (size_t)args.bn * BM * 4 > (size_t)PC<CFG>::B::STAGES * PC<CFG>::STAGE_BYTES)
    return pifa_fail(PIFA_ERR_UNSUPPORTED, "prefill: partial tile larger than the stage ring");
  constexpr size_t SMEM_BYTES = PC<CFG>::SMEM_BYTES;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaFuncSetAttribute(prefill gemm)", e);
  // programmatic dependent launch: each GEMM may start (weight tiles in flight) while the previous
  // kernel of the stream drains; its dependent loads follow griddepcontrol.wait
  cudaLaunchConfig_t cfg = {};
  // CTAs launch x-fastest. Walking token tiles first (when M > T) runs a weight-row block's tiles
  // together, sharing its A tile, with all of B (T x K) the wave's other operand; walking row tiles
  // first shares B tiles with all of A (M x K): the wave's working set is the smaller way round.
  // Measured: grouped 7B MLP gate+up T = 2048 (GEMM 2 M = 17920) 377 -> 356 us token-first;
  // attention T = 8192 (M = 2048) 239 us row-first against 259.
  const unsigned mt = (unsigned)((args.M + BM - 1) / BM), nt = (unsigned)((args.N + args.bn - 1) / args.bn);
  GemmArgs g = args;
  g.tok_fast = args.M > args.N ? 1 : 0;
  if ((g.tok_fast ? mt : nt) > 65535u) g.tok_fast ^= 1;  // gridDim.y is at most 65535
  if ((g.tok_fast ? mt : nt) > 65535u) return pifa_fail(PIFA_ERR_UNSUPPORTED, "more than 65535 tiles along both M and T");
  g.ks = cl ? args.ks : 1;
  cfg.gridDim = g.tok_fast ? dim3(nt, mt, (unsigned)g.ks) : dim3(mt, nt, (unsigned)g.ks);
  cfg.blockDim = dim3(PC<CFG>::THREADS);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;  // a tile's K-slices: consecutive along z
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = (unsigned)g.ks;
  cfg.attrs = attr;
  cfg.numAttrs = cl ? 2 : 1;
  e = pifa_launch_ex(&cfg, kern, a, b0, b1, g);
  if (e != cudaSuccess) return pifa_fail_cuda("prefill gemm launch", e);
  return PIFA_OK;
}

inline int64_t pad8(int64_t v) { return (v + 7) / 8 * 8; }

// Tokens per tile for an M x T GEMM: the multiple of 16 (16..256) minimising the slowest SM's time,
// waves x (tile time); ties to the larger bn. The tile time is the measured fit on the 4096 x 4096,
// r = 2048 layer (T = 8192: 4 waves of 256-token tiles 254 us, 6 waves of 144-token tiles 320 us):
// t(bn) ~ t0 (432 + bn), most of a tile's time not shrinking with its width. There T = 2048 takes
// 240 (144 tiles, one wave of 152 SMs, where 256 leaves 24 SMs idle: 58.3 -> 57.3 us) and
// T = 8192 224 (254.4 -> 242.8 us).
int sm_count_prefill() {
  int sms = 0, dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      sms < 1)
    sms = 1;
  return sms;
}

// The kernel shape and token-tile width of one GEMM: config 0 with pick_bn's width unless that
// takes three or more waves, then config 1 (CTA slots = 2 per SM) with its own width.
struct GemmShape {
  int cfg, bn, ks;  // kernel shape, tokens per tile, K-slices per tile (a cluster when > 1)
};
int pick_bn_slots(int64_t M, int64_t T, int bnmax, int64_t slots) {
  const int64_t mt = (M + BM - 1) / BM;
  int best = bnmax;
  int64_t best_cost = -1;
  for (int bn = bnmax; bn >= 16; bn -= 16) {
    const int64_t tiles = mt * ((T + bn - 1) / bn);
    const int64_t cost = (tiles + slots - 1) / slots * (432 + bn);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}
// Split-K: when the GEMM's full-width tiles (256 tokens, or all of T) fill at most half the SMs and
// the one-wave plan would otherwise fall back to tiles of 64 tokens or fewer, each full-width tile
// gets ks CTAs (2 or 4, keeping one CTA per SM, every K-slice at least 16 steps of 64) as a
// cluster that adds its partial tiles in shared memory. Measured against the narrow-tile plan (us,
// one process, interleaved): 7B attention T = 256 44.5 -> 34.8, T = 512 47.3 -> 37.0; 7B MLP down
// T = 256 76.7 -> 43.5, T = 512 80.4 -> 46.7; 7B MLP gate T = 256 46.6 -> 42.7; 70B q/o T = 256
// 88.9 -> 53.0; 70B gate/up T = 256 159.4 -> 142.8; 4096 x 4096, r = 1024, T = 512 36.4 -> 32.3.
// Splitting also where the plan keeps tiles of 96-128 tokens lost (r = 1024, T = 2048: 55.4 ->
// 59.0), as did clusters of 8 (8 K-steps per slice: 7B attention T = 256 44.5 -> 49.2).
GemmShape pick_shape(int64_t M, int64_t T, int64_t ksteps) {
  const int64_t sms = sm_count_prefill();
  const int64_t mt = (M + BM - 1) / BM;
  const int bnw = (int)(T >= PC<0>::BN ? PC<0>::BN : (T + 15) / 16 * 16);
  const int64_t tiles_w = mt * ((T + bnw - 1) / bnw);
  const int bn0 = pick_bn_slots(M, T, PC<0>::BN, sms);
  if (tiles_w * 2 <= sms && bn0 <= 64) {
    int ks = 1;
    while (ks < 4 && tiles_w * ks * 2 <= sms && ksteps / (ks * 2) >= 16) ks *= 2;
    if (ks > 1) return {0, bnw, ks};
  }
  const int64_t waves0 = (mt * ((T + bn0 - 1) / bn0) + sms - 1) / sms;
  if (waves0 < 3) return {0, bn0, 1};
  return {1, pick_bn_slots(M, T, PC<1>::BN, 2 * sms), 1};
}

template <typename... A>
int run_gemm_cfg(int cfg, A&&... args) {
  return cfg == 0 ? run_gemm<0>(std::forward<A>(args)...) : run_gemm<1>(std::forward<A>(args)...);
}

}  // namespace

int64_t prefill_split_workspace_bytes(const PifaShape& s) {
  const int64_t one = ((s.T * pad8(s.groups * s.r) * 2 + 255) / 256) * 256;  // 2-byte T x pad8(G r)
  return 2 * one;  // hi and lo
}

int launch_prefill_split(const PifaShape& s, const PifaPointers& p, int* status, uint64_t timeout_ns,
                         cudaStream_t stream) {
  const bool f16 = s.c_dtype == PIFA_DTYPE_FP16;
  const int64_t G = s.groups;  // layers sharing X: GEMM 1 over their stacked pivot rows
  const int64_t ldyp = pad8(G * s.r);
  const int64_t one = ((s.T * ldyp * 2 + 255) / 256) * 256;
  void* hi = p.ws;
  void* lo = reinterpret_cast<uint8_t*>(p.ws) + one;

  CUtensorMap tWp, tX, tC, tHi, tLo;
  int st;
  const GemmShape sh1 = pick_shape(G * s.r, s.T, (s.n + BK - 1) / BK);
  const int bn1 = sh1.bn;
  if ((st = make_tmap_2d(&tWp, PIFA_DTYPE_BF16, p.Wp, G * s.r, s.n, s.ldwp, BK, BM)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tX, PIFA_DTYPE_BF16, p.X, s.T, s.n, s.ldx, BK, bn1)) != PIFA_OK) return st;

  GemmArgs g1 = {};
  g1.idesc = idesc_bf16_f32(BM, bn1);
  g1.M = (int)(G * s.r);
  g1.N = (int)s.T;
  g1.bn = bn1;
  g1.kchunks = (int)((s.n + BK - 1) / BK);
  g1.passes = 1;
  g1.cols = p.piv;
  g1.m = (int)(G * s.m);
  g1.Y = reinterpret_cast<bf16*>(p.Y);
  g1.ldy = s.ldy;
  g1.yp_hi = hi;
  g1.yp_lo = lo;
  g1.ldyp = ldyp;
  g1.status = status;
  g1.timeout_ns = timeout_ns;
  g1.ks = sh1.ks;
  if ((st = run_gemm_cfg(sh1.cfg, f16 ? EPI_SPLIT_F16 : EPI_SPLIT_BF16, tWp, tX, tX, g1, stream)) != PIFA_OK) return st;
  if (s.m == s.r) return PIFA_OK;

  const GemmShape sh2 = pick_shape(G * (s.m - s.r), s.T, 2 * ((s.r + BK - 1) / BK));
  const int bn2 = sh2.bn;
  if ((st = make_tmap_2d(&tC, s.c_dtype, p.C, G * (s.m - s.r), s.r, s.ldc, BK, BM)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tHi, s.c_dtype, hi, s.T, G * s.r, ldyp, BK, bn2)) != PIFA_OK) return st;
  if ((st = make_tmap_2d(&tLo, s.c_dtype, lo, s.T, G * s.r, ldyp, BK, bn2)) != PIFA_OK) return st;
  GemmArgs g2 = g1;
  g2.bn = bn2;
  g2.idesc = f16 ? idesc_f16_f32(BM, bn2) : idesc_bf16_f32(BM, bn2);
  g2.M = (int)(G * (s.m - s.r));
  if (G > 1) {  // group g's non-pivot rows (whole tiles) read the hi/lo columns [g r, (g + 1) r)
    g2.gsz = (int)(s.m - s.r);
    g2.goff = (int)s.r;
  }
  g2.kchunks = (int)((s.r + BK - 1) / BK);
  g2.passes = 2;
  g2.ks = sh2.ks;
  g2.cols = p.nonpiv;
  g2.yp_hi = nullptr;
  g2.yp_lo = nullptr;
  return run_gemm_cfg(sh2.cfg, EPI_Y_ONLY, tC, tHi, tLo, g2, stream);
}

