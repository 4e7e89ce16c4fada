// decode.cu -- PIFA forward for small token counts (T <= 128): Algorithm 2 as two HBM-streaming
// phases. Up to T = 16 each phase runs one of the forms below or the split-K tensor-core form of
// decode_tc.cu; for 16 < T <= 128 both phases run the latter.
//
//   phase 1: Y_p = X W_p^T  (the r rows of W_p, each read once)  -> Y[:, I[j]] = bf16(Y_p[:, j]),
//            and y_p to the workspace as a hi + lo pair of C's dtype  (Algorithm 2, steps 2 and 4)
//   phase 2: Y_np = Y_p C^T (the m - r rows of C, each read once) -> Y[:, I^c[i]] = bf16(Y_np[:, i])
//                                                                     (Algorithm 2, steps 3 and 5)
//
// Both phases have one shape. A CTA owns a tile of 16 RG consecutive weight rows (RG m16 MMA row
// groups; RG = 1 or 4 by token count) and a K range; a thread-block cluster of up to 8 CTAs
// splits K when a tile's rows do not fit one stage, so each CTA reads only
// its slice of the broadcast operand (x or y_p). Every CTA of the grid reads the whole broadcast
// slice of its K range once, so taller tiles mean proportionally less of that L2 traffic, which
// otherwise competes with the weight streams and delays the dependent step. At launch -- before
// the CTA waits on its predecessor (programmatic dependent launch, PDL) -- warp 0 bulk-copies the
// CTA's weight rows into shared memory: the whole K range when it fits, else K-chunks through two
// stages refilled as they are used. The weights do not depend on the previous kernel, so their
// HBM traffic overlaps its compute: phase 2 stages its rows of C while phase 1 computes, and the
// next call's phase 1 stages its W_p while this call's phase 2 computes. The stage budgets let a
// phase-1 CTA and a phase-2 CTA share one SM.
//
// Once the predecessor has completed, each warp loads the B fragments of its K steps from L2
// into registers and runs mma.sync.m16n8k16 over its steps and all RG row groups with A from
// shared memory. For a 32-wide K step, lane (g = lane/4, c = lane%4) takes 8 consecutive elements
// of rows g and g+8 of a row group at offset 8c as the A fragments of two k16 MMAs and the
// matching 8 elements of token g as its B fragment: K is permuted identically in both operands,
// which a dot product does not notice. The warps' partial tiles are summed through shared memory,
// then the cluster's K slices: each CTA stores its sums of a peer's rows into that peer's shared
// memory and finishes 16 RG / ks rows itself. Both sums run in a fixed order, so the result is
// deterministic.
//
// Layers with more row tiles than one wave of clusters holds run a second kernel, decode_stream:
// a persistent grid (as many clusters as are co-resident) in which every cluster streams the
// K-chunks of its tiles through a ring of shared-memory stages filled by 2-D TMA boxes (few large
// copies: per-row bulk copies of 1-2 KB stream well below the HBM rate), with the CTA's K range
// of the broadcast operand resident in shared memory for all its tiles (per-chunk L2 loads of it
// wait behind the weight stream).
//
// y_p enters the second contraction as a hi + lo pair of C's storage type (bf16 or fp16): C has
// large entries and Y_np = C Y_p cancels, so rounding y_p to one bf16 alone would amplify its
// rounding error several-fold. Phase 1 splits each value once; phase 2 runs one MMA per plane.
#include <atomic>
#include <map>
#include <mutex>
#include <tuple>
#include <utility>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pifa.h"
#include "pifa_internal.h"
#include "ptx.cuh"

namespace {

using namespace pifa;
using bf16 = __nv_bfloat16;

// Weight rows per CTA: RG MMA row groups of 16. Taller tiles read less of the broadcast operand
// per weight byte (RG = 4 reads 4x less than RG = 1) but split K over larger clusters whose
// partial tiles must be summed; RG = 1 (no cluster) wins at T <= 2, RG = 4 up to T = 8, RG = 2
// with two token tiles.
template <int RG>
constexpr int kRowsOf = 16 * RG;
constexpr int kChunk = 32;          // K elements per warp step (two k16 MMAs)
constexpr int kWarps = 8;           // warps per CTA, both phases
constexpr int kMaxCluster = 8;      // CTAs per cluster splitting K (portable cluster size)
// Shared-memory budgets of one CTA's weight stages. 144 KB (phase 1) + 76 KB (phase 2) and the
// small rest fit in one SM's 228 KB, so a phase-2 CTA can stage its rows of C beside a computing
// phase-1 CTA (and a phase-1 CTA its rows of W_p beside a phase-2 CTA).
constexpr uint32_t kStageBudget1 = 144u * 1024u;
constexpr uint32_t kStageBudget2 = 76u * 1024u;
// decode_stream: shared memory of one CTA (two fit an SM), and its largest ring
constexpr uint32_t kStreamBudget = 108u * 1024u;
constexpr int kMaxStages = 8;

__device__ __forceinline__ uint32_t pack2(uint16_t a, uint16_t b) { return (uint32_t)a | ((uint32_t)b << 16); }

// 8 consecutive 16-bit elements of row `row` starting at column k; zero beyond column K or when
// !ok. Read through L2 only (ld.global.cg): the data may have been written by the previous kernel
// and a stale L1 line must never be used.
__device__ __forceinline__ uint4 ldg8_cg(const uint16_t* __restrict__ base, int64_t ld, int row, bool ok, int k,
                                         int K) {
  if (!ok || k >= K) return make_uint4(0u, 0u, 0u, 0u);
  const uint16_t* p = base + (int64_t)row * ld + k;
  if (k + 8 <= K) return __ldcg(reinterpret_cast<const uint4*>(p));
  uint16_t e[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) e[i] = (k + i < K) ? __ldcg(p + i) : (uint16_t)0;
  return make_uint4(pack2(e[0], e[1]), pack2(e[2], e[3]), pack2(e[4], e[5]), pack2(e[6], e[7]));
}

// 8 weights of one staged row at local column kl; elements at or beyond `len` are zeroed (the
// stage may hold stale bytes there, which must not reach the MMA even as NaN * 0).
__device__ __forceinline__ uint4 lds8_masked(const uint8_t* rowp, int kl, int len, bool row_ok) {
  if (!row_ok || kl >= len) return make_uint4(0u, 0u, 0u, 0u);
  uint4 v = *reinterpret_cast<const uint4*>(rowp + kl * 2);
  if (kl + 8 > len) {
    const int keep = len - kl;  // 1..7 valid elements
    uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t m0 = 2 * i < keep ? 0x0000FFFFu : 0u, m1 = 2 * i + 1 < keep ? 0xFFFF0000u : 0u;
      w[i] &= (m0 | m1);
    }
    v = make_uint4(w[0], w[1], w[2], w[3]);
  }
  return v;
}

// hi + lo split of an fp32 value in bf16 (kF16 = false) or fp16 (kF16 = true). fp16 saturates at
// +-65504 and reports the overflow through `range_err`.
template <bool kF16>
__device__ __forceinline__ void split2(float f, uint16_t& h, uint16_t& l, bool& range_err) {
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

template <bool kF16>
__device__ __forceinline__ void mma16816(float (&d)[4], const uint4& wa, const uint4& wb, uint32_t b0, uint32_t b1,
                                         bool upper) {
  const uint32_t a0 = upper ? wa.z : wa.x, a1 = upper ? wb.z : wb.x;
  const uint32_t a2 = upper ? wa.w : wa.y, a3 = upper ? wb.w : wb.y;
  if (kF16)
    mma_m16n8k16_f16(d, a0, a1, a2, a3, b0, b1);
  else
    mma_m16n8k16_bf16(d, a0, a1, a2, a3, b0, b1);
}

struct DecodeArgs {
  const uint16_t* A;    // weight rows: W_p (phase 1) or C (phase 2), 2-byte elements
  int64_t lda;
  int R, K;             // rows and columns of A
  const uint16_t* B0;   // B operand, T rows of K: X (phase 1) or the y_p hi plane (phase 2)
  const uint16_t* B1;   // phase 2: the y_p lo plane
  int64_t ldb;
  uint16_t* yph;        // phase 1 with m > r: y_p as hi and lo planes, T rows of pitch ldyp each
  uint16_t* ypl;
  int64_t ldyp;
  const int32_t* cols;  // output column of each weight row (I or I^c)
  int m;
  bf16* Y;
  int64_t ldy;
  int T;
  int ks;               // CTAs of a cluster, splitting K (1, 2, 4 or 8)
  int kcta;             // K columns per CTA (multiple of 32)
  int kc;               // K columns per shared-memory stage (multiple of 32, at most kcta)
  int stages;           // 1 (the CTA's whole K range resident) or 2
  uint32_t recv_off;    // ks > 1: byte offset in dynamic shared memory of the receive buffer(s)
  // decode_stream only
  int ntiles;           // row tiles of kRows rows
  int ncl;              // clusters in the grid: cluster c owns tiles c, c + ncl, c + 2 ncl, ...
  uint32_t bres_off;    // byte offset of the resident B rows (NB planes x T, pitch row_pitch(kcta))
  uint32_t red_off;     // byte offset of the warps' partial tiles
  int bstaged;          // 1: the chunk's B rows ride in each stage (TMA boxes of tb rows), else resident
  int gsz;              // grouped layers: weight rows per group (a tile never spans two), else 0
  int goff;             // B columns between consecutive groups' K ranges (r), when gsz > 0
  int bcols;            // columns of the B operand (K, or G r when grouped)
  int ngrp;             // groups whose K range of B a persistent CTA keeps resident (1 when not grouped)
  int tb;               // B box rows: T rounded up to 8
  int* status;
  uint64_t timeout_ns;
};

// Bytes between staged rows: the row's bytes, plus 64 when they are a multiple of 128, so that
// rows g and g + 1 start 64 bytes apart and a quarter warp's 16-byte fragment loads (two rows,
// four 16-byte columns each) cover all 32 banks.
__host__ __device__ constexpr uint32_t row_pitch(int kc) {
  return (uint32_t)kc * 2u + (((uint32_t)kc * 2u) % 128u == 0u ? 64u : 0u);
}

// One CTA: 16 RG weight rows x its K range [q kcta, (q + 1) kcta) against the T tokens, q = its
// rank in the cluster. The cluster's CTAs sum their partial tiles through distributed shared
// memory, each finishing kRows / ks of the rows. PHASE 1: bf16 MMAs against x, and y_p split in
// C's dtype (kF16C). PHASE 2: MMAs in C's dtype against the y_p hi and lo planes.
template <int PHASE, int NT, bool kF16C, int RG>
__global__ void __launch_bounds__(kWarps * 32, 2) decode_rows(DecodeArgs a) {
  constexpr int kRows = kRowsOf<RG>;
  constexpr int NB = PHASE == 1 ? 1 : 2;  // B planes (both accumulate into one tile)
  constexpr bool kF16Mma = PHASE == 2 && kF16C;
  // K steps whose B fragments a warp loads at once (about 64 registers of B and accumulators)
  constexpr int NBATCH = 16 / (RG * NB * NT) > 0 ? 16 / (RG * NB * NT) : 1;
  constexpr int NU = RG == 1 ? 2 : 1;     // accumulator sets (even / odd steps): shorter MMA chains
  constexpr int RP = 8 * NT + 1;          // floats per row of the reduction tiles
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ uint64_t full[2];
  __shared__ int s_cols[kRows];
  pdl_launch_dependents();  // the next kernel may launch now and start staging its weights
  const uint32_t pitch = row_pitch(a.kc);
  const uint32_t stage_bytes = (uint32_t)kRows * pitch;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
  const int q = (int)cluster_ctarank();
  const int64_t row0 = (int64_t)(blockIdx.x / a.ks) * kRows;
  const int nrows = (int)((int64_t)a.R - row0 < kRows ? (int64_t)a.R - row0 : kRows);
  const int k0 = q * a.kcta;
  const int klen = max(0, min(a.kcta, a.K - k0));
  const int nchunks = (klen + a.kc - 1) / a.kc;
  // Warp 0 stages K-chunk j: lane 0 arms the stage barrier, then each lane copies every 32nd row.
  auto issue = [&](int j) {
    const int s = j % a.stages;
    const int len = min(a.kc, klen - j * a.kc);
    const uint32_t bytes = (uint32_t)((len + 7) & ~7) * 2u;  // 16-byte multiple within the row pitch
    if (lane == 0) mbar_arrive_expect_tx(&full[s], bytes * (uint32_t)nrows);
    __syncwarp();
    uint8_t* st = smem + s * stage_bytes;
    for (int rr = lane; rr < nrows; rr += 32)
      bulk_copy_g2s(smem_u32(st + rr * pitch), a.A + (row0 + rr) * a.lda + k0 + (int64_t)j * a.kc, bytes, &full[s]);
  };
  if (warp == 0) {
    if (lane == 0) {
      for (int s = 0; s < a.stages; ++s) mbar_init(&full[s], 1);
      fence_mbar_init();
    }
    __syncwarp();
    for (int j = 0; j < a.stages && j < nchunks; ++j) issue(j);
  }
  // the output columns of this CTA's rows are layer constants: read them before waiting
  for (int i = threadIdx.x; i < kRows; i += kWarps * 32) s_cols[i] = i < nrows ? a.cols[row0 + i] : 0;
  // One thread waits for the previous kernel (its outputs visible, ours free to overwrite) while
  // the other warps park in the CTA barrier instead of taking issue slots from co-resident CTAs.
  if (threadIdx.x == 0) pdl_wait_primary();
  __syncthreads();  // also: barriers initialised before anyone waits on them

  float acc[NU][RG][NT][4];
#pragma unroll
  for (int u = 0; u < NU; ++u)
#pragma unroll
    for (int gq = 0; gq < RG; ++gq)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) acc[u][gq][nt][0] = acc[u][gq][nt][1] = acc[u][gq][nt][2] = acc[u][gq][nt][3] = 0.0f;
  // This lane's B rows: token t = 8 nt + g, clamped to T - 1. The output columns of tokens >= T
  // are computed from a duplicate row and never stored, and so are the output rows of weight
  // rows >= nrows (their stage rows hold stale bytes): an MMA row or column only ever affects
  // itself. Only a K tail beyond the last full step needs masking, and it gets its own step.
  // grouped layers: this tile's group reads its own K range of B
  const uint16_t* bp0 = a.B0 + (a.gsz > 0 ? (row0 / a.gsz) * a.goff : 0);
  const uint16_t* bp1 = NB > 1 ? a.B1 + (a.gsz > 0 ? (row0 / a.gsz) * a.goff : 0) : nullptr;
  const uint16_t* brow[NB][NT];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int t = nt * 8 + g < a.T ? nt * 8 + g : a.T - 1;
      brow[nb][nt] = (nb == 0 ? bp0 : bp1) + (int64_t)t * a.ldb + 8 * c;
    }
  bool dead = false;
  for (int j = 0; j < nchunks; ++j) {
    const int s = j % a.stages;
    const int kb = k0 + j * a.kc;  // first K column of the chunk
    const int len = min(a.kc, klen - j * a.kc);
    if (!dead && !mbar_wait(&full[s], (uint32_t)(j / a.stages) & 1u, a.timeout_ns)) {
      latch_status(a.status, PIFA_ERR_TIMEOUT);
      dead = true;
    }
    dead = __any_sync(0xffffffffu, dead);  // the MMAs below are warp-collective
    if (!dead) {
      // The hot loop is kept short: it runs once per launch, and its instruction fetch (not its
      // arithmetic) would otherwise dominate the kernel.
      const uint32_t wbase = smem_u32(smem + s * stage_bytes) + g * pitch + 16 * c;
      const int nfull = len / kChunk;
      for (int s0 = warp; s0 < nfull; s0 += kWarps * NBATCH) {
        const int nmine = min(NBATCH, (nfull - s0 + kWarps - 1) / kWarps);  // this batch's steps
        uint4 bv[NBATCH][NB][NT];  // the batch's B loads in flight together
#pragma unroll
        for (int i = 0; i < NBATCH; ++i)
          if (i < nmine)
#pragma unroll
            for (int nb = 0; nb < NB; ++nb)
#pragma unroll
              for (int nt = 0; nt < NT; ++nt)
                bv[i][nb][nt] = __ldcg(reinterpret_cast<const uint4*>(brow[nb][nt] + kb + (s0 + i * kWarps) * kChunk));
#pragma unroll
        for (int i = 0; i < NBATCH; ++i)
          if (i < nmine) {
            const uint32_t at = wbase + (uint32_t)((s0 + i * kWarps) * kChunk * 2);
#pragma unroll
            for (int gq = 0; gq < RG; ++gq) {
              const uint4 wa = lds128(at + (uint32_t)(16 * gq) * pitch);      // row 16 gq + g
              const uint4 wb = lds128(at + (uint32_t)(16 * gq + 8) * pitch);  // row 16 gq + g + 8
#pragma unroll
              for (int nb = 0; nb < NB; ++nb)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                  mma16816<kF16Mma>(acc[i % NU][gq][nt], wa, wb, bv[i][nb][nt].x, bv[i][nb][nt].y, false);
                  mma16816<kF16Mma>(acc[i % NU][gq][nt], wa, wb, bv[i][nb][nt].z, bv[i][nb][nt].w, true);
                }
            }
          }
      }
      if (nfull * kChunk < len && warp == nfull % kWarps) {  // ragged K tail, masked
        const int kl = nfull * kChunk + 8 * c;
        const uint8_t* st = smem + s * stage_bytes;
        uint4 bt[NB][NT];
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int t = nt * 8 + g < a.T ? nt * 8 + g : a.T - 1;
            bt[nb][nt] = ldg8_cg(nb == 0 ? bp0 : bp1, a.ldb, t, true, kb + kl, a.K);
          }
#pragma unroll
        for (int gq = 0; gq < RG; ++gq) {
          const uint4 wa = lds8_masked(st + (16 * gq + g) * pitch, kl, len, true);
          const uint4 wb = lds8_masked(st + (16 * gq + g + 8) * pitch, kl, len, true);
#pragma unroll
          for (int nb = 0; nb < NB; ++nb)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              mma16816<kF16Mma>(acc[0][gq][nt], wa, wb, bt[nb][nt].x, bt[nb][nt].y, false);
              mma16816<kF16Mma>(acc[0][gq][nt], wa, wb, bt[nb][nt].z, bt[nb][nt].w, true);
            }
        }
      }
    }
    if (j + a.stages < nchunks) {  // refill stage s once every warp is done with it
      dead = __syncthreads_or(dead);
      if (warp == 0 && !dead) issue(j + a.stages);
    }
  }
  if (threadIdx.x == 0) {
    // nothing may still be landing in shared memory when it is reused or the CTA exits
    for (int j = nchunks > a.stages ? nchunks - a.stages : 0; j < nchunks; ++j)
      if (!mbar_wait(&full[j % a.stages], (uint32_t)(j / a.stages) & 1u, 100000000ull))
        latch_status(a.status, PIFA_ERR_TIMEOUT);
  }
  __syncthreads();  // every warp is done with the stages: they hold the reduction tiles now

  // 1. the warps' partial tiles, red[warp][row][t]; 2. their sum, in place in warp 0's tile
  float* red = reinterpret_cast<float*>(smem);
  // ks > 1: the cluster's partial sums of the rows this CTA finishes, [source rank][token][row],
  // beyond the stages and partial tiles (peers write it while this CTA may still be computing)
  float* recv = reinterpret_cast<float*>(smem + a.recv_off);
#pragma unroll
  for (int gq = 0; gq < RG; ++gq)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      float v[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[e] = acc[0][gq][nt][e];
#pragma unroll
        for (int u = 1; u < NU; ++u) v[e] += acc[u][gq][nt][e];
      }
      float* r0p = red + (warp * kRows + 16 * gq + g) * RP + nt * 8 + 2 * c;
      r0p[0] = v[0];
      r0p[1] = v[1];
      r0p[8 * RP] = v[2];
      r0p[8 * RP + 1] = v[3];
    }
  __syncthreads();
  // CTA q of the cluster finishes rows [q rpr, (q + 1) rpr): every CTA stores its sums of those
  // rows straight into q's receive buffer (remote stores before the cluster barrier, so no CTA
  // reads another's shared memory after it and none has to wait for its peers before exiting)
  const int rpr = kRows / a.ks;
  for (int idx = threadIdx.x; idx < kRows * 8 * NT; idx += kWarps * 32) {
    const int row = idx % kRows, t = idx / kRows;  // each (row, t) belongs to one thread
    float sum = 0.0f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) sum += red[(w * kRows + row) * RP + t];
    if (a.ks == 1)
      red[row * RP + t] = sum;
    else if (t < a.T)  // consecutive threads store consecutive words of the owner's buffer
      st_dsmem_f32(mapa_shared(smem_u32(recv + (q * 8 * NT + t) * rpr + row % rpr), (uint32_t)(row / rpr)), sum);
  }
  // 3. the cluster's K-slices, summed in rank order
  if (a.ks > 1) cluster_sync_all();
  else __syncthreads();
  bool range_err = false;
  for (int idx = threadIdx.x; idx < rpr * 8 * NT; idx += kWarps * 32) {
    const int row = q * rpr + idx % rpr, t = idx / rpr;
    if (t >= a.T || row >= nrows) continue;
    float sum = 0.0f;
    if (a.ks == 1)
      sum = red[row * RP + t];
    else
      for (int rk = 0; rk < a.ks; ++rk) sum += recv[(rk * 8 * NT + t) * rpr + idx % rpr];
    if (PHASE == 1 && a.yph != nullptr) {
      uint16_t h, l;
      split2<kF16C>(sum, h, l, range_err);
      a.yph[(int64_t)t * a.ldyp + row0 + row] = h;
      a.ypl[(int64_t)t * a.ldyp + row0 + row] = l;
    }
    const int col = s_cols[row];
    if ((unsigned)col >= (unsigned)a.m) {
      latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
      continue;
    }
    a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(sum);
  }
  if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
}

// MMA row g of a 16-row group reads shared-memory row rho(g) = (g >> 1) | ((g & 1) << 2) of that
// group in decode_stream's TMA blocks. A quarter warp's fragment loads (MMA rows 2i and 2i + 1,
// four 16-byte columns each) then hit rows i and i + 4 of a 128-byte-swizzled block, whose chunks
// the swizzle places in opposite halves of the 128-byte bank window: no bank conflicts.
__device__ __forceinline__ int rho8(int g) { return (g >> 1) | ((g & 1) << 2); }

// Persistent form of decode_rows, warp-specialised. Cluster cid (of ncl) owns the row tiles cid,
// cid + ncl, ...; CTA q of the cluster covers the K range [q kcta, (q + 1) kcta) of each. A producer
// warp streams the weights through `stages` stages of kc / 64 TMA boxes each (64 columns x kRows
// rows, 128-byte swizzle, zero-filled beyond the layer), the first stages before the dependency
// wait, each later one as soon as all eight consumer warps have released the stage (an "empty"
// mbarrier): issuing never stalls the MMAs. The consumers hold their K range of the B operand
// (NB planes x T rows) in shared memory, copied once after the dependency wait and zero-padded to
// whole 32-column steps. Per tile the warps' partial tiles are summed through a region of their
// own, and the cluster's partials are pushed into the owners' receive buffers (two, alternating
// by tile) with mbarrier hand-offs in both directions -- "ready" when a source's pushes are
// visible, "released" when an owner has read them -- instead of cluster barriers, which the
// producer, running ahead, could not join.
template <int PHASE, int NT, bool kF16C, int RG>
__global__ void __launch_bounds__((kWarps + 1) * 32, 2)
    decode_stream(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                  const __grid_constant__ CUtensorMap tmB1, DecodeArgs a) {
  constexpr int kRows = kRowsOf<RG>;
  constexpr int NB = PHASE == 1 ? 1 : 2;
  constexpr bool kF16Mma = PHASE == 2 && kF16C;
  constexpr int NU = RG == 1 ? 2 : 1;     // accumulator sets (alternate steps): shorter MMA chains
  constexpr int RP = 8 * NT + 1;
  constexpr uint32_t kBlk = kRows * 128;  // one TMA box: 64 columns x kRows rows
  constexpr uint32_t kCons = kWarps * 32; // consumer threads (named barrier 1)
  extern __shared__ __align__(128) uint8_t smem_raw[];
  __shared__ uint64_t full[kMaxStages], empty[kMaxStages];
  __shared__ uint64_t bbar, rready[2], rfree[2];
  __shared__ int s_cols[kRows];
  pdl_launch_dependents();  // the next kernel may launch now and start staging its weights
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int nblkmax = a.kc / 64;  // 64-column blocks of a stage
  const uint32_t bblk = (uint32_t)a.tb * 128u;  // one staged B box: 64 columns x tb token rows
  const uint32_t bplane = a.bstaged ? (uint32_t)nblkmax * bblk : 0u;
  const uint32_t stage_bytes = (uint32_t)nblkmax * kBlk + (uint32_t)NB * bplane;
  const uint32_t bpitch = row_pitch(a.kcta);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
  const int q = (int)cluster_ctarank();
  const int cid = (int)blockIdx.x / a.ks;
  const int ntile = cid < a.ntiles ? (a.ntiles - 1 - cid) / a.ncl + 1 : 0;
  const int k0 = q * a.kcta;
  const int klen = max(0, min(a.kcta, a.K - k0));
  const int nchunks = (klen + a.kc - 1) / a.kc;
  const int nitems = ntile * nchunks;
  auto tile_row0 = [&](int t) { return (int64_t)(cid + t * a.ncl) * kRows; };
  auto tile_rows = [&](int64_t r0) { return (int)((int64_t)a.R - r0 < kRows ? (int64_t)a.R - r0 : kRows); };
  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kWarps);
    }
    mbar_init(&bbar, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&rready[b], (uint32_t)a.ks);  // one arrival per source CTA
      mbar_init(&rfree[b], (uint32_t)a.ks);   // one arrival per owner CTA
    }
    fence_mbar_init();
  }
  // the peers' barriers are initialised before anyone arrives on them remotely
  if (a.ks > 1) cluster_sync_all();
  else __syncthreads();

  if (warp == kWarps) {  // ---- producer ----
    if (lane == 0) {
      prefetch_tmap(&tmA);
      if (a.bstaged) {
        prefetch_tmap(&tmB0);
        if (NB > 1) prefetch_tmap(&tmB1);
      }
      // item `it` into stage it % stages: its weight boxes (wa) and/or B boxes (wb); the barrier's
      // one arrival comes with the last part (zero-filled parts of a box count too)
      auto issue = [&](int it, bool wa, bool wb) {
        const int s = it % a.stages, j = it % nchunks;
        const int nblk = (min(a.kc, klen - j * a.kc) + 63) / 64;
        const uint32_t tx = (wa ? (uint32_t)nblk * kBlk : 0u) + (wb ? (uint32_t)(NB * nblk) * bblk : 0u);
        if (wb || !a.bstaged)
          mbar_arrive_expect_tx(&full[s], tx);
        else
          mbar_expect_tx(&full[s], tx);
        uint8_t* st = smem + s * stage_bytes;
        const int x0 = k0 + j * a.kc;
        if (wa)
          for (int b = 0; b < nblk; ++b)
            tma_load_2d(smem_u32(st + b * kBlk), &tmA, x0 + 64 * b, (int)tile_row0(it / nchunks), &full[s]);
        if (wb) {
          const int64_t r0 = tile_row0(it / nchunks);
          const int xb = x0 + (a.gsz > 0 ? (int)(r0 / a.gsz) * a.goff : 0);  // the tile's group's B columns
          for (int nb = 0; nb < NB; ++nb)
            for (int b = 0; b < nblk; ++b)
              tma_load_2d(smem_u32(st + nblkmax * kBlk + nb * bplane + b * bblk), nb ? &tmB1 : &tmB0, xb + 64 * b, 0,
                          &full[s]);
        }
      };
      const int pre = min(a.stages, nitems);
      for (int it = 0; it < pre; ++it) issue(it, true, false);  // weights: before the dependency wait
      if (a.bstaged) {  // B depends on the previous kernel
        pdl_wait_primary();
        for (int it = 0; it < pre; ++it) issue(it, false, true);
      }
      int issued = pre;
      for (int it = pre; it < nitems; ++it) {
        const int s = it % a.stages;
        if (!mbar_wait(&empty[s], (uint32_t)((it / a.stages) - 1) & 1u, a.timeout_ns)) {
          latch_status(a.status, PIFA_ERR_TIMEOUT);
          break;
        }
        issue(it, true, a.bstaged != 0);
        issued = it + 1;
      }
      // nothing may land in shared memory after the CTA retires: wait for the last copies
      for (int it = issued > a.stages ? issued - a.stages : 0; it < issued; ++it)
        if (!mbar_wait(&full[it % a.stages], (uint32_t)(it / a.stages) & 1u, 100000000ull))
          latch_status(a.status, PIFA_ERR_TIMEOUT);
    }
    __syncwarp();
    // the producer warp's share of the closing cluster barrier (see the end of the consumers)
    if (a.ks > 1) cluster_sync_all();
    return;  // from here on the consumers synchronise on named barrier 1 only
  }

  // ---- consumers ----
  if (ntile > 0)
    for (int i = threadIdx.x; i < kRows; i += kCons) s_cols[i] = i < tile_rows(tile_row0(0)) ? a.cols[tile_row0(0) + i] : 0;
  if (threadIdx.x == 0) pdl_wait_primary();
  named_barrier_sync(1, kCons);

  // B rows, resident: [0, klen rounded down to 8) by bulk copies, the rest up to whole steps by
  // plain loads and zeros (the steps read up to kpad; the TMA boxes are zero beyond K as well)
  uint8_t* bres = smem + a.bres_off;
  const int kbulk = a.bstaged ? 0 : klen & ~7, kpad = a.bstaged ? 0 : (klen + kChunk - 1) / kChunk * kChunk;
  if (warp == 0 && !a.bstaged) {
    const uint32_t bytes = (uint32_t)kbulk * 2u;
    if (lane == 0) mbar_arrive_expect_tx(&bbar, bytes * (uint32_t)(a.ngrp * NB * a.T));
    __syncwarp();
    // row i: group i / (NB T), plane (i / T) % NB, token i % T
    if (bytes)
      for (int i = lane; i < a.ngrp * NB * a.T; i += 32)
        bulk_copy_g2s(smem_u32(bres + i * bpitch),
                      ((i / a.T) % NB ? a.B1 : a.B0) + (int64_t)(i % a.T) * a.ldb + (int64_t)(i / (NB * a.T)) * a.goff + k0,
                      bytes, &bbar);
  }
  const int wtail = kpad - kbulk;
  if (wtail > 0)
    for (int idx = threadIdx.x; idx < a.ngrp * NB * a.T * wtail; idx += kCons) {
      const int i = idx / wtail, col = kbulk + idx % wtail;
      const uint16_t* src = ((i / a.T) % NB ? a.B1 : a.B0) + (int64_t)(i % a.T) * a.ldb + (int64_t)(i / (NB * a.T)) * a.goff;
      reinterpret_cast<uint16_t*>(bres + i * bpitch)[col] = col < klen ? __ldcg(src + k0 + col) : (uint16_t)0;
    }
  bool dead = false;
  if (threadIdx.x == 0 && !a.bstaged && !mbar_wait(&bbar, 0, a.timeout_ns)) {
    latch_status(a.status, PIFA_ERR_TIMEOUT);
    dead = true;
  }
  dead = named_barrier_or(1, kCons, dead);

  const int arow = rho8(g);
  const uint32_t lane_off = (uint32_t)arow * 128u + (uint32_t)((c ^ arow) << 4);
  // this lane's B row (token t = 8 nt + g, clamped to T - 1) and column 8 c:
  //   resident: bres + (nb T + t) bpitch + 16 c  (+ 2 column)
  //   staged:   stage + nblkmax kBlk + nb bplane + (st / 2) bblk + t 128 + ((4 (st & 1) + c) ^ (t & 7)) 16
  uint32_t boff[NB][NT];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int t = nt * 8 + g < a.T ? nt * 8 + g : a.T - 1;
      boff[nb][nt] = a.bstaged ? (uint32_t)nblkmax * kBlk + (uint32_t)nb * bplane + (uint32_t)t * 128u +
                                     (uint32_t)((c ^ (t & 7)) << 4)
                               : smem_u32(bres) + (uint32_t)(nb * a.T + t) * bpitch + 16u * c;
    }
  float* red = reinterpret_cast<float*>(smem + a.red_off);
  bool range_err = false;
  const int rpr = kRows / a.ks;
  for (int tt = 0; tt < ntile; ++tt) {
    const int64_t row0 = tile_row0(tt);
    const int nrows = tile_rows(row0);
    // grouped layers, resident B: this tile's group's rows of it
    const uint32_t bgrp = a.gsz > 0 && !a.bstaged ? (uint32_t)((row0 / a.gsz) * NB * a.T) * bpitch : 0u;
    if (tt > 0)  // the columns of this tile's rows, in flight while it computes
      for (int i = threadIdx.x; i < kRows; i += kCons)
        if (i < nrows) cp_async4(smem_u32(&s_cols[i]), a.cols + row0 + i);
    float acc[NU][RG][NT][4];
#pragma unroll
    for (int u = 0; u < NU; ++u)
#pragma unroll
      for (int gq = 0; gq < RG; ++gq)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) acc[u][gq][nt][0] = acc[u][gq][nt][1] = acc[u][gq][nt][2] = acc[u][gq][nt][3] = 0.0f;
    for (int j = 0; j < nchunks; ++j) {
      const int it = tt * nchunks + j;
      const int s = it % a.stages;
      const int nst = (min(a.kc, klen - j * a.kc) + kChunk - 1) / kChunk;
      // every warp waits for the stage, steps or not: a warp that released stages it had not
      // waited for could run ahead and count its release of a later item toward this one's
      if (!dead && !mbar_wait(&full[s], (uint32_t)(it / a.stages) & 1u, a.timeout_ns)) {
        latch_status(a.status, PIFA_ERR_TIMEOUT);
        dead = true;
      }
      dead = __any_sync(0xffffffffu, dead);
      if (warp < nst) {
        if (!dead) {
          const uint32_t sbase = smem_u32(smem + s * stage_bytes);
          const uint32_t sb = sbase + lane_off;
          const uint32_t bj = (uint32_t)(j * a.kc) * 2u;
          // one 32-column step: the stage base is 1024-byte aligned and kBlk a multiple of 1024,
          // so the odd step's chunk flip (bit 6) acts on lane_off alone
          auto step = [&](int st, float (&ac)[RG][NT][4]) {
            const uint32_t at = (sb + (uint32_t)(st >> 1) * kBlk) ^ ((uint32_t)(st & 1) << 6);
            uint4 bv[NB][NT];
#pragma unroll
            for (int nb = 0; nb < NB; ++nb)
#pragma unroll
              for (int nt = 0; nt < NT; ++nt)
                bv[nb][nt] = lds128(a.bstaged ? sbase + (uint32_t)(st >> 1) * bblk + (boff[nb][nt] ^ ((uint32_t)(st & 1) << 6))
                                              : boff[nb][nt] + bgrp + bj + (uint32_t)st * 64u);
#pragma unroll
            for (int gq = 0; gq < RG; ++gq) {
              const uint4 wa = lds128(at + (uint32_t)(16 * gq) * 128u);      // MMA row g
              const uint4 wb = lds128(at + (uint32_t)(16 * gq + 8) * 128u);  // MMA row g + 8
#pragma unroll
              for (int nb = 0; nb < NB; ++nb)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                  mma16816<kF16Mma>(ac[gq][nt], wa, wb, bv[nb][nt].x, bv[nb][nt].y, false);
                  mma16816<kF16Mma>(ac[gq][nt], wa, wb, bv[nb][nt].z, bv[nb][nt].w, true);
                }
            }
          };
#pragma unroll 1
          for (int st = warp; st < nst; st += kWarps * NU) {
            step(st, acc[0]);
            if (NU > 1 && st + kWarps < nst) step(st + kWarps, acc[NU - 1]);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[s]);  // this warp is done with stage s
    }
    named_barrier_sync(1, kCons);  // every warp is done with the previous tile's partials and columns

    // the warps' partial tiles, red[warp][row][t] in weight-row order
#pragma unroll
    for (int gq = 0; gq < RG; ++gq)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        float v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          v[e] = acc[0][gq][nt][e];
#pragma unroll
          for (int u = 1; u < NU; ++u) v[e] += acc[u][gq][nt][e];
        }
        float* r0p = red + (warp * kRows + 16 * gq + arow) * RP + nt * 8 + 2 * c;
        r0p[0] = v[0];
        r0p[1] = v[1];
        r0p[8 * RP] = v[2];
        r0p[8 * RP + 1] = v[3];
      }
    const int b = tt & 1;
    float* recv = reinterpret_cast<float*>(smem + a.recv_off) + b * (kRows * 8 * NT);
    if (a.ks > 1 && tt >= 2 && threadIdx.x == 0 && !dead &&
        !mbar_wait_cluster(&rfree[b], (uint32_t)((tt - 2) >> 1) & 1u, a.timeout_ns)) {
      latch_status(a.status, PIFA_ERR_TIMEOUT);  // every owner has read this buffer's last pushes
      dead = true;
    }
    dead = named_barrier_or(1, kCons, dead);
    // the sum over the warps; with a cluster, pushed into the owner's receive buffer
    for (int idx = threadIdx.x; idx < kRows * 8 * NT; idx += kCons) {
      const int row = idx % kRows, t = idx / kRows;
      float sum = 0.0f;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) sum += red[(w * kRows + row) * RP + t];
      if (a.ks == 1)
        red[row * RP + t] = sum;
      else if (t < a.T)
        st_dsmem_f32(mapa_shared(smem_u32(recv + (q * 8 * NT + t) * rpr + row % rpr), (uint32_t)(row / rpr)), sum);
    }
    cp_async_wait_all();  // this thread's column loads (if any) have landed
    named_barrier_sync(1, kCons);
    if (a.ks > 1) {
      if (threadIdx.x == 0) {
        // this CTA's pushes (ordered before by the barrier) are released with one arrival at
        // every owner; then wait until every source's pushes to this CTA are visible
        asm volatile("fence.acq_rel.cluster;" ::: "memory");
        for (int o = 0; o < a.ks; ++o) mbar_arrive_remote(mapa_shared(smem_u32(&rready[b]), (uint32_t)o));
        if (!dead && !mbar_wait_cluster(&rready[b], (uint32_t)(tt >> 1) & 1u, a.timeout_ns)) {
          latch_status(a.status, PIFA_ERR_TIMEOUT);
          dead = true;
        }
      }
      dead = named_barrier_or(1, kCons, dead);
    }
    for (int idx = threadIdx.x; idx < rpr * 8 * NT; idx += kCons) {
      const int row = q * rpr + idx % rpr, t = idx / rpr;
      if (t >= a.T || row >= nrows) continue;
      float sum = 0.0f;
      if (a.ks == 1)
        sum = red[row * RP + t];
      else
        for (int rk = 0; rk < a.ks; ++rk) sum += recv[(rk * 8 * NT + t) * rpr + idx % rpr];
      if (PHASE == 1 && a.yph != nullptr) {
        uint16_t h, l;
        split2<kF16C>(sum, h, l, range_err);
        a.yph[(int64_t)t * a.ldyp + row0 + row] = h;
        a.ypl[(int64_t)t * a.ldyp + row0 + row] = l;
      }
      const int col = s_cols[row];
      if ((unsigned)col >= (unsigned)a.m) {
        latch_status(a.status, PIFA_ERR_DEVICE_INDEX);
        continue;
      }
      a.Y[(int64_t)t * a.ldy + col] = __float2bfloat16_rn(sum);
    }
    if (tt + 1 < ntile) {
      named_barrier_sync(1, kCons);  // the partials, the columns and buffer b have been read
      // release buffer b to every source that will push into it again (tile tt + 2); a source
      // with no such tile may have retired, and gets no arrival
      if (a.ks > 1 && tt + 2 < ntile && threadIdx.x == 0)
        for (int o = 0; o < a.ks; ++o) mbar_arrive_remote(mapa_shared(smem_u32(&rfree[b]), (uint32_t)o));
    }
  }
  if (range_err) latch_status(a.status, PIFA_ERR_RANGE);
  // No CTA retires before every CTA of its cluster has made its last remote access to it: every
  // thread of every CTA of the cluster (the producer warps included) arrives on the hardware
  // cluster barrier after its last push or remote arrival, and leaves only once all have arrived.
  // That barrier has no time limit, but every wait before it is bounded (after a timeout the CTA
  // skips its waits and runs to here), so each CTA reaches it: a CTA whose wait ran out cannot
  // retire while a late peer may still write into its shared memory.
  if (a.ks > 1) cluster_sync_all();
}

// Once per kernel, device and size: the dynamic shared-memory limit, and the largest shared-memory
// carveout, so that a phase-1 CTA and a phase-2 CTA fit on one SM together.
int prepare_kernel(const void* fn, size_t smem, const char* what) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, size_t> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return pifa_fail_cuda(what, e);
  std::lock_guard<std::mutex> lock(mu);
  auto it = done.find({fn, dev});
  if (it != done.end() && it->second >= smem) return PIFA_OK;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, (int)cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return pifa_fail_cuda(what, e);
  done[{fn, dev}] = smem;
  return PIFA_OK;
}

// Launch with programmatic dependent launch and a (ks, 1, 1) cluster.
template <typename Kern>
int launch_phase(Kern kernel, int rows, const DecodeArgs& args, size_t smem, cudaStream_t stream, const char* what) {
  const int st = prepare_kernel(reinterpret_cast<const void*>(kernel), smem, what);
  if (st != PIFA_OK) return st;
  const unsigned tiles = (unsigned)((args.R + rows - 1) / rows);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles * (unsigned)args.ks);
  cfg.blockDim = dim3(kWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)args.ks;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaError_t e = pifa_launch_ex(&cfg, kernel, args);
  if (e != cudaSuccess) return pifa_fail_cuda(what, e);
  return PIFA_OK;
}

// The K split and the stages of one phase: the fewest CTAs per cluster (1, 2, 4, 8) whose K range
// fits one stage within `budget`; else 8 CTAs, each streaming its range through two stages.
void plan_phase(int kRows, uint32_t budget, DecodeArgs& a) {
  for (int ks = 1; ks <= kMaxCluster; ks *= 2) {
    const int kcta = ((a.K + ks - 1) / ks + kChunk - 1) / kChunk * kChunk;
    if ((uint64_t)kRows * row_pitch(kcta) <= budget) {
      a.ks = ks;
      a.kcta = a.kc = kcta;
      a.stages = 1;
      return;
    }
  }
  a.ks = kMaxCluster;
  a.kcta = ((a.K + kMaxCluster - 1) / kMaxCluster + kChunk - 1) / kChunk * kChunk;
  a.stages = 2;
  int kc = kChunk;
  while (kc + kChunk <= a.kcta && 2ull * kRows * row_pitch(kc + kChunk) <= budget) kc += kChunk;
  a.kc = kc;
}

// Dynamic shared memory of one CTA: the stages, overlaid by the warps' partial tiles, then (ks > 1)
// the receive buffer at a.recv_off, which this sets.
size_t smem_bytes(int kRows, DecodeArgs& a, int NT) {
  const size_t stages = (size_t)a.stages * kRows * row_pitch(a.kc);
  const size_t red = (size_t)kWarps * kRows * (8 * NT + 1) * 4;
  const size_t body = ((stages > red ? stages : red) + 15) / 16 * 16;
  a.recv_off = (uint32_t)body;
  return a.ks > 1 ? body + (size_t)kRows * 8 * NT * 4 : body;
}

// Co-resident clusters of ks CTAs of `fn` with `smem` bytes of dynamic shared memory each, on the
// current device (cached per kernel, device, cluster size and size). 0 if unknown.
int max_clusters(const void* fn, int ks, size_t smem, int threads = kWarps * 32) {
  static std::mutex mu;
  static std::map<std::tuple<const void*, int, int, size_t>, int> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(fn, dev, ks, smem);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  int n = 0;
  if (ks == 1) {
    int per_sm = 0, sms = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, smem) == cudaSuccess &&
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
      n = per_sm * sms;
  } else {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)ks);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = (unsigned)ks;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();  // a failed query leaves no sticky error behind
  cache[key] = n;
  return n;
}

std::atomic<int> g_decode_grid{PIFA_DECODE_GRID_AUTO};  // pifa_set_decode_grid

int kcta_of(int K, int ks) { return ((K + ks - 1) / ks + kChunk - 1) / kChunk * kChunk; }

int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      n = 1;
  }
  return n;
}

// decode_stream's split of one phase into (ks, kcta, kc, stages, ntiles, ncl) and its shared memory
// (returned, with 1 KB of alignment slack): the fewest CTAs per cluster giving at least one
// (tile, K-range) unit per SM (measured: two per SM, through larger clusters, cost more in per-tile
// reductions than they gain), with resident B rows of at most a third of the budget; then chunks
// of whole 64-column blocks, four stages where they fit.
size_t plan_stream(const void* fn, int kRows, int NT, int NB, DecodeArgs& a, const char* what, int* st) {
  auto round16 = [](size_t b) { return (b + 15) / 16 * 16; };
  a.ntiles = (a.R + kRows - 1) / kRows;
  const size_t red = round16((size_t)kWarps * kRows * (8 * NT + 1) * 4);
  const size_t recv1 = (size_t)kRows * 8 * NT * 4;
  // B rows: resident for T <= 2 (a few KB per CTA, no per-chunk traffic), else staged with the
  // weights in every stage, which frees the cluster split from the resident rows' size
  a.bstaged = a.T > 2 ? 1 : 0;
  a.tb = (a.T + 7) / 8 * 8;
  int ks = 1;
  while (ks < kMaxCluster && ((int64_t)a.ntiles * ks < sm_count() ||
                              (!a.bstaged && (size_t)a.ngrp * NB * a.T * row_pitch(kcta_of(a.K, ks)) > kStreamBudget / 3)))
    ks *= 2;
  a.ks = ks;
  a.kcta = kcta_of(a.K, ks);
  const size_t bres = a.bstaged ? 0 : round16((size_t)a.ngrp * NB * a.T * row_pitch(a.kcta));
  const size_t side = bres + red + (ks > 1 ? 2 * recv1 : 0);
  const size_t blk = (size_t)kRows * 128 + (a.bstaged ? (size_t)NB * a.tb * 128 : 0);  // one 64-column block
  const size_t ring = kStreamBudget > side + 2 * blk ? kStreamBudget - side : 2 * blk;
  const int kblocks = (a.kcta + 63) / 64;
  int nblk = (int)(ring / (4 * blk));
  if (nblk < 1) nblk = 1;
  if (nblk > kblocks) nblk = kblocks;
  a.kc = 64 * nblk;
  const size_t stage = (size_t)nblk * blk;
  a.stages = (int)(ring / stage);
  if (a.stages > kMaxStages) a.stages = kMaxStages;
  if (a.stages < 2) a.stages = 2;
  a.bres_off = (uint32_t)(a.stages * stage);
  a.red_off = a.bres_off + (uint32_t)bres;
  a.recv_off = a.red_off + (uint32_t)red;
  const size_t smem = 1024 + a.recv_off + (ks > 1 ? 2 * recv1 : 0);
  *st = prepare_kernel(fn, smem, what);
  if (*st != PIFA_OK) return 0;
  // as many clusters as are co-resident, but the tiles dealt evenly: rounds = ceil(ntiles / cap)
  // tiles for every cluster (a last round on a few clusters would run at their share of HBM alone)
  const int nclu = max_clusters(fn, ks, smem, (kWarps + 1) * 32);
  const int cap = nclu > 0 ? nclu : 1;
  const int rounds = (a.ntiles + cap - 1) / cap;
  a.ncl = (a.ntiles + rounds - 1) / rounds;
  return smem;
}

template <typename Kern>
int launch_stream(Kern kernel, const CUtensorMap& tm, const CUtensorMap& tb0, const CUtensorMap& tb1,
                  const DecodeArgs& args, size_t smem, cudaStream_t stream, const char* what) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(args.ncl * args.ks));
  cfg.blockDim = dim3((kWarps + 1) * 32);  // eight consumer warps and the producer warp
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)args.ks;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaError_t e = pifa_launch_ex(&cfg, kernel, tm, tb0, tb1, args);
  if (e != cudaSuccess) return pifa_fail_cuda(what, e);
  return PIFA_OK;
}

// One phase: decode_rows (16 RG-row tiles) or decode_stream (16 RGS-row tiles, over a TMA map of
// the weights in their storage type `dtype`). The stream reads its B operand once per CTA, so its
// tiles can be taller than decode_rows': 32 rows make 4 KB TMA boxes (2 KB boxes of 16 rows
// issue too many copies per byte).
// Scratch of the split-K tensor-core form (decode_tc.cu): where its partial sums go, and how many
// bytes are available there.
struct SplitKScratch {
  float* P;
  int64_t bytes;
};

// The split-K tensor-core form of one phase (decode_tc.cu) on the same operands.
template <int PHASE, bool kF16C>
int launch_phase_tc(const DecodeArgs& a, int dtype, const SplitKScratch& sk, cudaStream_t stream) {
  DecodeTcPhase ph = {};
  ph.A = a.A;
  ph.lda = a.lda;
  ph.R = a.R;
  ph.K = a.K;
  ph.dtype = dtype;
  ph.B0 = a.B0;
  ph.B1 = a.B1;
  ph.ldb = a.ldb;
  ph.bcols = a.bcols;
  ph.T = a.T;
  ph.planes = PHASE == 1 ? 1 : 2;
  ph.gsz = a.gsz;
  ph.goff = a.goff;
  ph.mma_f16 = PHASE == 2 && kF16C;
  ph.split_f16 = kF16C;
  ph.P = sk.P;
  ph.cols = a.cols;
  ph.m = a.m;
  ph.Y = a.Y;
  ph.ldy = a.ldy;
  ph.yph = a.yph;
  ph.ypl = a.ypl;
  ph.ldyp = a.ldyp;
  return launch_decode_tc(ph, a.status, a.timeout_ns, stream);
}

template <int PHASE, int NT, bool kF16C, int RG, int RGS>
int launch_one_phase(DecodeArgs& a, uint32_t budget, int dtype, const SplitKScratch& sk, cudaStream_t stream) {
  constexpr int kRows = kRowsOf<RG>;
  const char* what = PHASE == 1 ? "decode phase 1 launch" : "decode phase 2 launch";
  const int mode = g_decode_grid.load(std::memory_order_relaxed);
  const bool tc_fits = sk.P != nullptr && decode_tc_partial_bytes(a.R, a.K, a.T, PHASE == 1 ? 1 : 2) <= sk.bytes;
  if (a.T > 16) {  // token tiles of 32 and 64 rows exist only in the split-K tensor-core form
    if (!tc_fits) return pifa_fail(PIFA_ERR_INVALID_ARG, "decode with T > 16 needs the split-K workspace");
    return launch_phase_tc<PHASE, kF16C>(a, dtype, sk, stream);
  }
  if (mode == PIFA_DECODE_GRID_SPLITK && tc_fits) return launch_phase_tc<PHASE, kF16C>(a, dtype, sk, stream);
  // Auto, keyed on the phase's shape and T (phase 1: r rows of K = n; phase 2: m - r rows of
  // K = r): for T > 2 a phase of at least 32 blocks of 128 rows runs split-K on the tensor cores
  // (decode_tc.cu); a shorter one gives the grid too few row blocks, so that each CTA's range
  // spans many K-slices and the partial sums grow with them. Measured per phase, every
  // combination of the three forms (us, T = 4 / 8 / 16):
  //   70B gate/up 28672x8192 r4096 (4096 and 24576 rows): tc+tc 51.5 / 54.1 / 56.9, best of all
  //   70B q/o     8192x8192 r4096  (4096 and 4096 rows):  tc+tc 27.6 / 27.1 / 28.9, best within 1%
  //   7B gate     11008x4096 r2048 (2048 and 8960 rows):  waves+tc 16.1 / 17.5 / 20.8 (was 19.0 /
  //                                                       19.5 / 21.1 in waves+waves)
  //   7B down     4096x11008 r2048 (2048 and 2048 rows):  stream+waves 18.9 / 19.1 / 22.6 (was
  //                                                       21.4 / 22.3 / 22.3 with phase 1 on tc)
  //   7B attn     4096x4096 r2048  (2048 and 2048 rows):  waves+waves 8.6 / 8.7 / 13.0
  // For T <= 2 decode_stream's resident x / y_p and short loop win (70B gate/up, T = 1: 46.9
  // against 51.7 us on the tensor cores).
  if (mode == PIFA_DECODE_GRID_AUTO && a.T > 2 && a.R >= 32 * 128 && tc_fits)
    return launch_phase_tc<PHASE, kF16C>(a, dtype, sk, stream);
  const auto kr = decode_rows<PHASE, NT, kF16C, RG>;
  plan_phase(kRows, budget, a);
  const size_t smem = smem_bytes(kRows, a, NT);
  int st = prepare_kernel(reinterpret_cast<const void*>(kr), smem, what);
  if (st != PIFA_OK) return st;
  // decode_rows in waves while a phase takes at most two of them (its weights staged at launch,
  // before the dependency wait, outweigh the persistent grid's streaming); else decode_stream
  const int tiles = (a.R + kRows - 1) / kRows;
  if (mode == PIFA_DECODE_GRID_WAVES ||
      (mode == PIFA_DECODE_GRID_AUTO && tiles <= 2 * max_clusters(reinterpret_cast<const void*>(kr), a.ks, smem)))
    return launch_phase(kr, kRows, a, smem, stream, what);
  const auto ks = decode_stream<PHASE, NT, kF16C, RGS>;
  const size_t smem_s =
      plan_stream(reinterpret_cast<const void*>(ks), kRowsOf<RGS>, NT, PHASE == 1 ? 1 : 2, a, what, &st);
  if (st != PIFA_OK) return st;
  CUtensorMap tm, tb0 = {}, tb1 = {};  // B maps (x, or the y_p planes in C's type): staged B only
  if ((st = make_tmap_2d(&tm, dtype, a.A, a.R, a.K, a.lda, 64, kRowsOf<RGS>)) != PIFA_OK) return st;
  if (a.bstaged && (st = make_tmap_2d(&tb0, dtype, a.B0, a.T, a.bcols, a.ldb, 64, a.tb)) != PIFA_OK) return st;
  if (a.bstaged && PHASE == 2 && (st = make_tmap_2d(&tb1, dtype, a.B1, a.T, a.bcols, a.ldb, 64, a.tb)) != PIFA_OK)
    return st;
  return launch_stream(ks, tm, tb0, tb1, a, smem_s, stream, what);
}

int64_t decode_planes_bytes(const PifaShape& s) {
  // y_p as hi and lo planes of 2-byte elements, T rows of pitch round_up(G r, 8) each, rounded up
  // to 256 bytes
  return ((s.T * ((s.groups * s.r + 7) / 8 * 8) * 4 + 255) / 256) * 256;
}

template <int NT, bool kF16C, int RG, int RGS>
int launch_decode_t(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream) {
  const int64_t G = s.groups;                      // layers sharing X (1: one layer)
  const int64_t ldyp = (G * s.r + 7) / 8 * 8;  // 16-byte rows keep the fragment loads aligned
  uint16_t* yph = reinterpret_cast<uint16_t*>(p.ws);
  uint16_t* ypl = yph + s.T * ldyp;
  // the split-K form's partial sums follow the planes (phase 2 reuses phase 1's: the reduction of
  // phase 1 has completed before phase 2 writes)
  const int64_t planes = decode_planes_bytes(s);
  const SplitKScratch sk = {p.ws_bytes > planes ? reinterpret_cast<float*>(static_cast<uint8_t*>(p.ws) + planes) : nullptr,
                            p.ws_bytes - planes};
  DecodeArgs a = {};
  a.A = reinterpret_cast<const uint16_t*>(p.Wp);
  a.lda = s.ldwp;
  a.R = (int)(G * s.r);  // the groups' pivot rows, stacked: phase 1 is one contraction against x
  a.K = (int)s.n;
  a.B0 = reinterpret_cast<const uint16_t*>(p.X);
  a.ldb = s.ldx;
  a.bcols = (int)s.n;
  a.ngrp = 1;
  a.yph = s.m > s.r ? yph : nullptr;
  a.ypl = s.m > s.r ? ypl : nullptr;
  a.ldyp = ldyp;
  a.cols = p.piv;
  a.m = (int)(G * s.m);
  a.Y = reinterpret_cast<bf16*>(p.Y);
  a.ldy = s.ldy;
  a.T = (int)s.T;
  a.status = status;
  a.timeout_ns = pifa_wait_timeout_ns();
  int st = launch_one_phase<1, NT, kF16C, RG, RGS>(a, kStageBudget1, PIFA_DTYPE_BF16, sk, stream);
  if (st != PIFA_OK || s.m == s.r) return st;
  DecodeArgs b = a;
  b.A = reinterpret_cast<const uint16_t*>(p.C);
  b.lda = s.ldc;
  b.R = (int)(G * (s.m - s.r));
  b.K = (int)s.r;
  b.B0 = yph;
  b.B1 = ypl;
  b.ldb = ldyp;
  b.bcols = (int)(G * s.r);
  if (G > 1) {  // group g's non-pivot rows (a whole number of tiles) read y_p's columns [g r, (g + 1) r)
    b.gsz = (int)(s.m - s.r);
    b.goff = (int)s.r;
    b.ngrp = (int)G;
  }
  b.yph = b.ypl = nullptr;
  b.cols = p.nonpiv;
  return launch_one_phase<2, NT, kF16C, RG, RGS>(b, kStageBudget2, (int)s.c_dtype, sk, stream);
}

}  // namespace

extern "C" int pifa_set_decode_grid(int mode) {
  if (mode != PIFA_DECODE_GRID_AUTO && mode != PIFA_DECODE_GRID_WAVES && mode != PIFA_DECODE_GRID_PERSISTENT &&
      mode != PIFA_DECODE_GRID_SPLITK)
    return pifa_fail(PIFA_ERR_INVALID_ARG,
                     "decode grid mode must be 0 (auto), 1 (waves), 2 (persistent) or 3 (split-K tensor cores)");
  g_decode_grid.store(mode, std::memory_order_relaxed);
  return PIFA_OK;
}

int64_t decode_workspace_bytes(const PifaShape& s) {
  // the y_p planes, then room for the split-K form's partial sums of either phase
  const int64_t G = s.groups;
  int64_t part = decode_tc_partial_bytes(G * s.r, s.n, s.T, 1);
  if (s.m > s.r) {
    const int64_t p2 = decode_tc_partial_bytes(G * (s.m - s.r), s.r, s.T, 2);
    part = p2 > part ? p2 : part;
  }
  return decode_planes_bytes(s) + (part + 255) / 256 * 256;
}

int launch_decode(const PifaShape& s, const PifaPointers& p, int* status, cudaStream_t stream) {
  const bool f16 = s.c_dtype == PIFA_DTYPE_FP16;
  // Tile height by token count (measured on the 4096 x 4096, r = 2048 layer): 16 rows for T <= 2,
  // 64 rows for T <= 8, 32 rows for T <= 16 (two token tiles).
  // Persistent-grid tiles (layers beyond two waves): 32 rows (4 KB TMA boxes) at any T.
  if (s.T <= 2)
    return f16 ? launch_decode_t<1, true, 1, 2>(s, p, status, stream) : launch_decode_t<1, false, 1, 2>(s, p, status, stream);
  if (s.T <= 8)
    return f16 ? launch_decode_t<1, true, 4, 2>(s, p, status, stream) : launch_decode_t<1, false, 4, 2>(s, p, status, stream);
  return f16 ? launch_decode_t<2, true, 2, 2>(s, p, status, stream) : launch_decode_t<2, false, 2, 2>(s, p, status, stream);
}

// ---- allocation-free decode entry point -------------------------------------------------------
// For callers that cannot allocate device memory at all: for example an inference runtime that
// plans every device byte ahead of time and forbids libraries from calling cudaMalloc, or code
// running where an allocation would synchronize the device in the middle of a latency-critical
// decode loop. Such callers cannot provide the workspace pifa_forward asks for, so this entry
// point keeps the decode scratch (y_p as hi and lo planes of 2-byte elements, T rows of pitch
// round_up(r, 8) each) in a fixed array in
// the library's static device data instead. The array exists once per GPU that loads the
// library and stays allocated until the process exits.
namespace {

constexpr int64_t kNoAllocScratchBytes = int64_t(1) << 20;  // 1 MiB: 256 + T * round_up(r, 8) * 4 bytes
__device__ __align__(256) unsigned char g_decode_scratch[kNoAllocScratchBytes];

constexpr int kNoAllocMaxDevices = 64;
void* g_decode_scratch_addr[kNoAllocMaxDevices] = {};
std::mutex g_decode_scratch_mu;

bool noalloc_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" int pifa_forward_decode_noalloc(const void* X, int64_t T, int64_t n, int64_t ldx, const void* Wp,
                                           int64_t r, int64_t ldwp, const void* C, int64_t m, int64_t ldc,
                                           const int32_t* pivot_idx, const int32_t* nonpivot_idx, void* Y,
                                           int64_t ldy, void* cuda_stream) {
  pifa_clear_error();
  if (T < 0 || m < 1 || n < 1 || r < 1 || r > m || r > n || m >= (int64_t(1) << 30) || n >= (int64_t(1) << 30))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "need T >= 0 and 1 <= r <= min(m, n) < 2^30");
  if (T == 0) return PIFA_OK;
  if (T > 16) return pifa_fail(PIFA_ERR_UNSUPPORTED, "pifa_forward_decode_noalloc needs T <= 16");
  const bool has_np = m > r;
  if (!X || !Wp || !pivot_idx || !Y || (has_np && (!C || !nonpivot_idx)))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "null X, Wp, C, pivot_idx, nonpivot_idx or Y");
  if (ldx < n || ldwp < n || ldy < m || (has_np && ldc < r))
    return pifa_fail(PIFA_ERR_INVALID_ARG, "leading dimension smaller than the row length");
  if (!noalloc_aligned16(X) || !noalloc_aligned16(Wp) || !noalloc_aligned16(Y) || (has_np && !noalloc_aligned16(C)))
    return pifa_fail(PIFA_ERR_ALIGNMENT, "X, Wp, C and Y must be 16-byte aligned");
  if ((ldx | ldwp | ldy | (has_np ? ldc : 0)) & 7)
    return pifa_fail(PIFA_ERR_ALIGNMENT, "ldx, ldwp, ldc and ldy must be multiples of 8 elements");
  {
    // as pifa_forward: Y must not share a byte with an input
    const PifaSpan y = pifa_span(Y, T, m, ldy, 2);
    if (pifa_spans_overlap(y, pifa_span(X, T, n, ldx, 2)) || pifa_spans_overlap(y, pifa_span(Wp, r, n, ldwp, 2)) ||
        (has_np && pifa_spans_overlap(y, pifa_span(C, m - r, r, ldc, 2))))
      return pifa_fail(PIFA_ERR_INVALID_ARG, "Y overlaps an input");
  }
  const PifaShape s = {T, m, n, r, ldx, ldwp, has_np ? ldc : r, ldy, PIFA_DTYPE_BF16};
  const int64_t need = kWorkspaceReserve + decode_planes_bytes(s);
  if (need > kNoAllocScratchBytes)
    return pifa_fail(PIFA_ERR_WORKSPACE,
                     "256 + T * round_up(r, 8) * 4 bytes exceeds the 1 MiB static scratch of "
                     "pifa_forward_decode_noalloc");

  // Set-up, once per device, with that device current: the device address of the static array.
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return pifa_fail_cuda("cudaGetDevice", e);
  if (dev < 0 || dev >= kNoAllocMaxDevices) return pifa_fail(PIFA_ERR_UNSUPPORTED, "device ordinal >= 64");
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_decode_scratch_mu);
    if (!g_decode_scratch_addr[dev]) {
      void* ptr = nullptr;
      e = cudaGetSymbolAddress(&ptr, g_decode_scratch);
      if (e != cudaSuccess) return pifa_fail_cuda("cudaGetSymbolAddress(decode scratch)", e);
      g_decode_scratch_addr[dev] = ptr;
    }
    scratch = g_decode_scratch_addr[dev];
  }
  int* status = pifa_status_word(&e);
  if (!status) return pifa_fail_cuda("device status word", e);
  // The first kWorkspaceReserve bytes of the array are reserved like those of a workspace; y_p
  // after them is written in full before it is read.
  const PifaPointers p = {X,
                          Wp,
                          has_np ? C : nullptr,
                          pivot_idx,
                          has_np ? nonpivot_idx : nullptr,
                          Y,
                          static_cast<uint8_t*>(scratch) + kWorkspaceReserve,
                          kNoAllocScratchBytes - kWorkspaceReserve};
  return launch_decode(s, p, status, reinterpret_cast<cudaStream_t>(cuda_stream));
}
