// Device code of the dense path of libframefb: frames outside the structured
// kernels (the paper's rho = 2 regime, where Phi is a dense realified DFT of
// size d/2, and redundant frames with T blocks, k*rho > d).  Phi is treated
// as a dense d x K matrix (K = k*rho frame columns), so one pass of the
// adapter is three contractions around the coefficient SpMM (Sec. 3.1
// update, Lemma 1 gradient of Appendix A):
//   analysis    V = X Phi_in,  U = dY Phi_out              dense_gemm_kernel<BF16_HILO>
//   SpMM        Z = V C^T,  G = U C,  dC_q = s sum_t U[t,a_q] V[t,b_q]
//                                                           dense_spmm_kernel
//   synthesis   Y += s Z Phi_out^T,  dX += s G Phi_in^T    dense_gemm_kernel<TF32>
// Included by framefb_dense.cu only.
//
// The contraction kernel is a persistent tcgen05 GEMM, D[M x N] = A[M x K]
// B[N x K]^T with both operands K-major: M = tokens (128-row tiles, one TMEM
// lane per token), N = output columns (BN per tile, fp32 accumulators in
// TMEM, double-buffered so that the epilogue of one tile overlaps the MMAs
// of the next), K in stages of 128 bytes per row landed by TMA tensor copies
// with 128-byte swizzle (the canonical SWIZZLE_128B K-major operand).
// Warp roles: warp 0 issues the copies, warp 1 owns TMEM and issues the
// MMAs (one thread), warps 2-5 read the accumulators back (warp w reads TMEM
// lanes 32 (w mod 4) ..) and run the epilogue.
//   BF16_HILO: A bf16 (X or dY, exact), B = Phi split into bf16 hi and lo
//              parts: two kind::f16 MMAs per K step into one accumulator, so
//              V carries Phi to about 2^-16 instead of bf16's 2^-9.
//   TF32:      A fp32 (Z or G, stored rounded to tf32 by the SpMM), B = Phi
//              rounded to tf32, kind::tf32.
// Every wait is bounded (about 2^31 cycles) and also gives up once another
// role of the CTA has given up; a CTA that gives up counts it in
// g_dense_timeouts, lets its copies and MMAs land, frees TMEM and exits.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "framefb_ptx.cuh"
#include "plan_layout.h"

namespace ffb {
namespace dense {

// Bounded waits of the dense kernels that gave up (see framefb_wait_timeouts).
__device__ unsigned int g_dense_timeouts;

constexpr int kGemmThreads = 192;  // warp 0 copies, warp 1 MMAs, warps 2-5 epilogue
constexpr int kStages = 4;
constexpr int kBM = 128;           // tokens per tile (TMEM lanes)
constexpr int kRowBytes = 128;     // K bytes per operand row and stage (the swizzle span)
constexpr long long kWaitCycles = 1ll << 31;

enum { KIND_BF16_HILO = 0, KIND_TF32 = 1 };
enum { EPI_STORE_F32 = 0, EPI_ACCUM_BF16 = 1 };

// One contraction of a launch.  Tensor maps: a = A [M][K] (box {128 B of K,
// 128 rows}), b0 / b1 = B parts [N][K] (box {128 B of K, BN rows}).
struct GemmProblem {
  CUtensorMap a, b0, b1;
  void* out;      // EPI_STORE_F32: fp32 [M][ldo]; EPI_ACCUM_BF16: bf16 [M][ldo], accumulated
  int64_t ldo;    // elements
  int32_t M, N, K;
  int32_t nt;     // tiles along N
  int32_t tile0;  // first tile of this problem in the launch's tile order
  float alpha;    // EPI_ACCUM_BF16: out += alpha * D
};

struct GemmLaunch {
  GemmProblem p[2];
  int32_t nprob, total_tiles;
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int32_t x, int32_t y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// Wait for phase `parity`; false when the time limit passes (the CTA gives
// up: counted once, flagged for the other roles) or another role gave up.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_test_wait(bar, parity)) return true;
  const long long start = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort_flag) return false;
    if (clock64() - start > kWaitCycles) {
      if (atomicExch(const_cast<int*>(abort_flag), 1) == 0) atomicAdd(&g_dense_timeouts, 1u);
      return false;
    }
  }
  return true;
}

// Tile t of the launch -> problem, token-tile and column-tile (columns
// fastest, so that concurrent CTAs share their A rows through L2).
__device__ __forceinline__ void tile_of(const GemmLaunch& L, int t, int& pi, int& mt, int& nt) {
  pi = (L.nprob > 1 && t >= L.p[1].tile0) ? 1 : 0;
  const int local = t - L.p[pi].tile0;
  mt = local / L.p[pi].nt;
  nt = local - mt * L.p[pi].nt;
}

template <int KIND, int BN>
struct GemmShape {
  static constexpr int NB = KIND == KIND_BF16_HILO ? 2 : 1;  // B parts per stage
  static constexpr int ELEM = KIND == KIND_BF16_HILO ? 2 : 4;
  static constexpr int BK = kRowBytes / ELEM;                // K elements per stage
  static constexpr uint32_t A_BYTES = kBM * kRowBytes;
  static constexpr uint32_t B_BYTES = BN * kRowBytes;
  static constexpr uint32_t STAGE = A_BYTES + NB * B_BYTES;
  static constexpr uint32_t SMEM = kStages * STAGE + 1024;   // + alignment slack
  static constexpr uint32_t TMEM_COLS = 2 * BN;              // two accumulators
  static_assert(BN % 32 == 0 && BN >= 32 && BN <= 256, "UMMA N for M = 128");
  static_assert(TMEM_COLS == 64 || TMEM_COLS == 128 || TMEM_COLS == 256 || TMEM_COLS == 512, "TMEM allocation");
};

// y (8 bf16 of one 16-byte chunk) += alpha * d[0..7]
__device__ __forceinline__ uint4 axpy_bf16x8(uint4 y, const float* d, float alpha) {
  uint32_t w[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float lo = fmaf(alpha, d[2 * i], __uint_as_float(w[i] << 16));
    const float hi = fmaf(alpha, d[2 * i + 1], __uint_as_float(w[i] & 0xFFFF0000u));
    w[i] = pack_bf16(lo, hi);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Epilogue of 32 accumulator columns [col, col + 32) of token row r.
template <int EPI>
__device__ __forceinline__ void epilogue32(const GemmProblem& P, int r, int col, const float (&v)[32]) {
  if (r >= P.M || col >= P.N) return;
  if constexpr (EPI == EPI_STORE_F32) {
    // rows are padded to whole float4 chunks (ldo >= N rounded up to 4)
    float* o = static_cast<float*>(P.out) + static_cast<int64_t>(r) * P.ldo + col;
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (col + 4 * i < P.N) reinterpret_cast<float4*>(o)[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
  } else {
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(P.out) + static_cast<int64_t>(r) * P.ldo + col;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = col + 8 * i;
      if (c + 8 <= P.N) {
        uint4* q = reinterpret_cast<uint4*>(o + 8 * i);
        *q = axpy_bf16x8(*q, v + 8 * i, P.alpha);
      } else if (c < P.N) {  // ragged last chunk of a row
        for (int e = 0; e < P.N - c; ++e)
          o[8 * i + e] = __float2bfloat16_rn(fmaf(P.alpha, v[8 * i + e], __bfloat162float(o[8 * i + e])));
      }
    }
  }
}

template <int KIND, int EPI, int BN>
__global__ void __launch_bounds__(kGemmThreads, 1) dense_gemm_kernel(const __grid_constant__ GemmLaunch L) {
  using S = GemmShape<KIND, BN>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[kStages], empty[kStages], tfull[2], tempty[2];
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // 1024-byte aligned stage ring (SWIZZLE_128B atoms)
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);   // the producer's expect_tx arrival (+ the copies' bytes)
      mbar_init(&empty[s], 1);  // the MMA thread's commit
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);   // commit after a tile's last MMA
      mbar_init(&tempty[b], 4);  // one arrival per epilogue warp
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(S::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  volatile int* abort_p = &abort_flag;

  if (warp == 0) {
    // ---------------------------------------------------------------- copies
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < L.total_tiles && ok; t += gridDim.x) {
        int pi, mt, nt;
        tile_of(L, t, pi, mt, nt);
        const GemmProblem& P = L.p[pi];
        const int kb_n = (P.K + S::BK - 1) / S::BK;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const uint32_t s = it % kStages, use = it / kStages;
          if (use > 0 && !wait_or_abort(&empty[s], (use - 1) & 1u, abort_p)) {
            ok = false;
            break;
          }
          const uint32_t st = base + s * S::STAGE;
          mbar_arrive_expect_tx(&full[s], S::STAGE);  // whole boxes: out-of-range parts land as zeros
          tma_load_2d(st, &P.a, kb * S::BK, mt * kBM, &full[s]);
          tma_load_2d(st + S::A_BYTES, &P.b0, kb * S::BK, nt * BN, &full[s]);
          if constexpr (S::NB == 2) tma_load_2d(st + S::A_BYTES + S::B_BYTES, &P.b1, kb * S::BK, nt * BN, &full[s]);
        }
      }
      if (!ok) {
        // let the copies in flight land before the CTA's shared memory goes away
        for (uint32_t i = it > kStages ? it - kStages : 0; i < it; ++i)
          mbar_wait_bounded(&full[i % kStages], (i / kStages) & 1u);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMAs
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc(KIND == KIND_BF16_HILO ? 1u : 2u, kBM, BN);
      uint32_t it = 0, tl = 0;
      bool ok = true, pending = false;
      uint64_t* last = nullptr;
      uint32_t last_par = 0;
      for (int t = blockIdx.x; t < L.total_tiles && ok; t += gridDim.x, ++tl) {
        int pi, mt, nt;
        tile_of(L, t, pi, mt, nt);
        const GemmProblem& P = L.p[pi];
        const int kb_n = (P.K + S::BK - 1) / S::BK;
        const uint32_t buf = tl & 1u, use = tl >> 1;
        if (use > 0 && !wait_or_abort(&tempty[buf], (use - 1) & 1u, abort_p)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * BN;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const uint32_t s = it % kStages;
          if (!wait_or_abort(&full[s], (it / kStages) & 1u, abort_p)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = base + s * S::STAGE;
#pragma unroll
          for (int ks = 0; ks < kRowBytes / 32; ++ks) {  // 32 bytes of K per MMA: 16 bf16 or 8 tf32
            const uint64_t a = umma_sdesc_sw128(st + 32 * ks);
            const uint64_t b0 = umma_sdesc_sw128(st + S::A_BYTES + 32 * ks);
            const uint32_t acc = (kb > 0 || ks > 0) ? 1u : 0u;
            if constexpr (KIND == KIND_BF16_HILO) {
              umma_f16(d, a, b0, idesc, acc);
              umma_f16(d, a, umma_sdesc_sw128(st + S::A_BYTES + S::B_BYTES + 32 * ks), idesc, 1u);
            } else {
              umma_tf32(d, a, b0, idesc, acc);
            }
          }
          umma_commit(&empty[s]);  // the stage is free once these MMAs have read it
          last = &empty[s];
          last_par = (it / kStages) & 1u;
          pending = true;
        }
        if (!ok) break;
        umma_commit(&tfull[buf]);
      }
      if (!ok && pending) mbar_wait_bounded(last, last_par);  // MMAs in flight
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quarter this warp may read
    const int row = 32 * q + lane;
    uint32_t tl = 0;
    for (int t = blockIdx.x; t < L.total_tiles; t += gridDim.x, ++tl) {
      int pi, mt, nt;
      tile_of(L, t, pi, mt, nt);
      const GemmProblem& P = L.p[pi];
      const uint32_t buf = tl & 1u, use = tl >> 1;
      const bool ok = wait_or_abort(&tfull[buf], use & 1u, abort_p);
      if (__any_sync(0xffffffffu, !ok)) break;
      tc_fence_after();
      const uint32_t taddr = tmem + (static_cast<uint32_t>(32 * q) << 16) + buf * BN;
      const int r = mt * kBM + row;
      const int cend = min(BN, P.N - nt * BN);  // columns of this tile inside the output
#pragma unroll 1
      for (int c0 = 0; c0 < cend; c0 += 32) {
        float v[32];
        tmem_ld32(taddr + c0, v);
        epilogue32<EPI>(P, r, nt * BN + c0, v);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(S::TMEM_COLS) : "memory");
  }
}

// ---------------------------------------------------------------------------
// Coefficient SpMM of the dense path over one token chunk of one matrix.
// Units are TT consecutive tokens; a CTA takes a contiguous range of units.
// Per unit the rows of V (and U) are staged token-minor in shared memory
// (TT values per coefficient, one vector access per gather), thread p walks
// plan column p of the row path (run sums of c V[b] into RZ) and of the
// column path (c U[a] into RG, U[a] . V[b] into its dC accumulators), the
// fix-up list adds the pieces of runs split between columns, and the rows
// of Z = V C^T and G = U C are written out rounded to tf32 for the
// synthesis.
// MODE bits: 1 row path (Z), 2 column path (G), 4 dC.
// ---------------------------------------------------------------------------
constexpr int kSpmmThreads = 256;  // = plan columns (FRAMEFB_THREADS)

struct SpmmLaunch {
  const uint8_t* plan;  // device plan image (either layout: the tables index V / U / Z / G rows)
  const float* c_val;   // [nnz]
  const float* V;       // [N][ldv] analysis of X (K_n columns)
  const float* U;       // [N][ldu] analysis of dY (K_m columns)
  float* Z;             // [N][ldz] row sums for Y (K_m columns)
  float* G;             // [N][ldg] column sums for dX (K_n columns)
  float* partial;       // dC partial sums: slot (slot0 + CTA) of stride floats
  int64_t ldv, ldu, ldz, ldg;  // floats per row (multiples of 4)
  int32_t N;            // tokens of the chunk
  int32_t stride, slot0;
  // shared-memory map (floats): V, U, RZ, RG token-minor regions, dC accumulators
  int32_t oV, oU, oRZ, oRG, oDC;
};

template <int TT>
struct TokVec {
  float v[TT];
};

template <int TT>
__device__ __forceinline__ TokVec<TT> tv_load(const float* base, int slot) {
  TokVec<TT> r;
  if constexpr (TT == 2) {
    const float2 x = reinterpret_cast<const float2*>(base)[slot];
    r.v[0] = x.x;
    r.v[1] = x.y;
  } else {
#pragma unroll
    for (int k = 0; k < TT; ++k) r.v[k] = base[slot * TT + k];
  }
  return r;
}

template <int TT>
__device__ __forceinline__ void tv_store(float* base, int slot, const TokVec<TT>& x) {
  if constexpr (TT == 2) {
    reinterpret_cast<float2*>(base)[slot] = make_float2(x.v[0], x.v[1]);
  } else {
#pragma unroll
    for (int k = 0; k < TT; ++k) base[slot * TT + k] = x.v[k];
  }
}

// rows t0 .. t0 + tc - 1 of a [N][ld] fp32 buffer, K columns, into a
// token-minor shared region (missing tokens as zeros)
template <int TT>
__device__ __forceinline__ void stage_rows(float* dst, const float* src, int64_t ld, int64_t t0, int tc, int K) {
  const int K4 = (K + 3) >> 2;
  for (int c4 = threadIdx.x; c4 < K4; c4 += kSpmmThreads) {
    float4 x[TT];
#pragma unroll
    for (int k = 0; k < TT; ++k)
      x[k] = k < tc ? __ldcs(reinterpret_cast<const float4*>(src + (t0 + k) * ld) + c4) : make_float4(0.f, 0.f, 0.f, 0.f);
    float* d = dst + 4 * c4 * TT;
#pragma unroll
    for (int k = 0; k < TT; ++k) {
      d[0 * TT + k] = x[k].x;
      d[1 * TT + k] = x[k].y;
      d[2 * TT + k] = x[k].z;
      d[3 * TT + k] = x[k].w;
    }
  }
}

// the K columns of a token-minor shared region back to rows of a [N][ld]
// buffer, rounded to tf32 (whole float4 chunks: padding columns get zeros)
template <int TT>
__device__ __forceinline__ void write_rows(float* dst, const float* src, int64_t ld, int64_t t0, int tc, int K) {
  const int K4 = (K + 3) >> 2;
  for (int c4 = threadIdx.x; c4 < K4; c4 += kSpmmThreads) {
    const float* s = src + 4 * c4 * TT;
#pragma unroll
    for (int k = 0; k < TT; ++k) {
      if (k >= tc) break;
      float4 y;
      y.x = 4 * c4 + 0 < K ? __uint_as_float(to_tf32(s[0 * TT + k])) : 0.f;
      y.y = 4 * c4 + 1 < K ? __uint_as_float(to_tf32(s[1 * TT + k])) : 0.f;
      y.z = 4 * c4 + 2 < K ? __uint_as_float(to_tf32(s[2 * TT + k])) : 0.f;
      y.w = 4 * c4 + 3 < K ? __uint_as_float(to_tf32(s[3 * TT + k])) : 0.f;
      reinterpret_cast<float4*>(dst + (t0 + k) * ld)[c4] = y;
    }
  }
}

// E: entries per plan column held in registers (the plan's EZ and EG are at
// most E): the entry words and the coefficient values are loaded once per
// CTA, so that the loop over a unit's entries only gathers from shared
// memory; the dC sums live in registers as well.
template <int MODE, int TT, int E>
__global__ void __launch_bounds__(kSpmmThreads, 1) dense_spmm_kernel(const __grid_constant__ SpmmLaunch a) {
  constexpr bool F = MODE & 1, D = MODE & 2, C = MODE & 4;
  extern __shared__ float4 smem4[];
  float* sm = reinterpret_cast<float*>(smem4);
  const FfbPlanHeader& h = *reinterpret_cast<const FfbPlanHeader*>(a.plan);
  const int p = threadIdx.x;
  const int64_t units = (a.N + TT - 1) / TT;
  const int64_t u0 = blockIdx.x * units / gridDim.x, u1 = (blockIdx.x + 1) * units / gridDim.x;
  const int32_t* tzb = reinterpret_cast<const int32_t*>(a.plan + h.off_zb);
  const int32_t* tzq = reinterpret_cast<const int32_t*>(a.plan + h.off_zq);
  const int32_t* tga = reinterpret_cast<const int32_t*>(a.plan + h.off_ga);
  const int32_t* tgb = reinterpret_cast<const int32_t*>(a.plan + h.off_gb);
  const int32_t* tgq = reinterpret_cast<const int32_t*>(a.plan + h.off_gq);
  const int4* fixZ = reinterpret_cast<const int4*>(a.plan + h.off_fixZ);
  const int4* fixG = reinterpret_cast<const int4*>(a.plan + h.off_fixG);
  float* V = sm + a.oV;
  float* U = sm + a.oU;
  float* RZ = sm + a.oRZ;
  float* RG = sm + a.oRG;
  // this thread's plan column: padding entries gather slot 0, add 0, store nowhere
  uint32_t zb[E], ga[E], gb[E];
  float zc[E], gc[E], dc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    zb[e] = ga[e] = FFB_NO_STORE << 16;
    gb[e] = 0;
    zc[e] = gc[e] = dc[e] = 0.f;
    if (F && e < h.EZ) {
      zb[e] = static_cast<uint32_t>(__ldg(tzb + e * kSpmmThreads + p)) & ~0x8000u;  // drop the parity bit
      const int32_t qi = __ldg(tzq + e * kSpmmThreads + p);
      zc[e] = qi >= 0 ? __ldg(a.c_val + qi) : 0.f;
    }
    if ((D || C) && e < h.EG) {
      ga[e] = static_cast<uint32_t>(__ldg(tga + e * kSpmmThreads + p)) & ~0x8000u;
      gb[e] = static_cast<uint32_t>(__ldg(tgb + e * kSpmmThreads + p));
      const int32_t qi = __ldg(tgq + e * kSpmmThreads + p);
      gc[e] = (D && qi >= 0) ? __ldg(a.c_val + qi) : 0.f;
    }
  }
  // run-sum slots that no run writes stay zero for every unit
  if constexpr (F)
    for (int i = p; i < (h.m + h.ovfZ) * TT; i += kSpmmThreads) RZ[i] = 0.f;
  if constexpr (D)
    for (int i = p; i < (h.n + h.ovfG) * TT; i += kSpmmThreads) RG[i] = 0.f;
  for (int64_t u = u0; u < u1; ++u) {
    const int64_t t0 = u * TT;
    const int tc = static_cast<int>(min(static_cast<int64_t>(TT), a.N - t0));
    __syncthreads();  // the previous unit's rows are written out
    if constexpr (F || C) stage_rows<TT>(V, a.V, a.ldv, t0, tc, h.n);
    if constexpr (D || C) stage_rows<TT>(U, a.U, a.ldu, t0, tc, h.m);
    __syncthreads();
    if constexpr (F) {  // row path: Z[a] = sum over the run of c V[b]
      TokVec<TT> acc{};
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const TokVec<TT> x = tv_load<TT>(V, zb[e] & 0xFFFFu);
#pragma unroll
        for (int k = 0; k < TT; ++k) acc.v[k] = fmaf(zc[e], x.v[k], acc.v[k]);
        if ((zb[e] >> 16) != FFB_NO_STORE) {
          tv_store<TT>(RZ, zb[e] >> 16, acc);
          acc = TokVec<TT>{};
        }
      }
    }
    if constexpr (D || C) {  // column path: G[b] = sum over the run of c U[a]; dC += U[a] . V[b]
      TokVec<TT> acc{};
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const TokVec<TT> x = tv_load<TT>(U, ga[e] & 0xFFFFu);
        if constexpr (C) {
          const TokVec<TT> y = tv_load<TT>(V, gb[e]);
#pragma unroll
          for (int k = 0; k < TT; ++k) dc[e] = fmaf(x.v[k], y.v[k], dc[e]);
        }
        if constexpr (D) {
#pragma unroll
          for (int k = 0; k < TT; ++k) acc.v[k] = fmaf(gc[e], x.v[k], acc.v[k]);
          if ((ga[e] >> 16) != FFB_NO_STORE) {
            tv_store<TT>(RG, ga[e] >> 16, acc);
            acc = TokVec<TT>{};
          }
        }
      }
    }
    if constexpr (F || D) {
      const int nfz = F ? h.nfixZ : 0, nfg = D ? h.nfixG : 0;
      if (nfz + nfg > 0) {  // runs split between columns: add the overflow pieces
        __syncthreads();
        for (int i = p; i < nfz + nfg; i += kSpmmThreads) {
          const bool z = i < nfz;
          const int4 it = z ? __ldg(fixZ + i) : __ldg(fixG + (i - nfz));
          float* R = z ? RZ : RG;
#pragma unroll
          for (int k = 0; k < TT; ++k) {
            float s = R[it.x * TT + k];
            for (int c2 = 0; c2 < it.z; ++c2) s += R[(it.y + c2) * TT + k];
            R[it.x * TT + k] = s;
          }
        }
      }
      __syncthreads();
      if constexpr (F) write_rows<TT>(a.Z, RZ, a.ldz, t0, tc, h.m);
      if constexpr (D) write_rows<TT>(a.G, RG, a.ldg, t0, tc, h.n);
    }
  }
  if constexpr (C) {
    float* dst = a.partial + static_cast<int64_t>(a.slot0 + blockIdx.x) * a.stride;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (e < h.EG) {
        const int32_t qi = __ldg(tgq + e * kSpmmThreads + p);
        if (qi >= 0) dst[qi] = dc[e];
      }
    }
  }
}

// Operands of the 32 x 32 group block D of a k = 16, k*rho = d frame (every
// group of coordinates [32r, 32r + 32) carries the same block, Sec. 3.2
// construction): D[w][x] = Phi[w][column of x], x = 2i + s <-> column
// i*rho + s, read from the frame's fp32 CSC values (32 per column).
//   out_hi / out_lo [x][w] bf16:  analysis B (rows = coefficients)
//   out_sy          [w][x] fp32:  synthesis B (rows = coordinates), tf32
// One CTA of 1024 threads per frame (blockIdx.x), one entry per thread.
struct GroupBlockArgs {
  const float* val[8];
  int32_t rho[8];
  uint8_t* out[8];  // 2 KB hi, 2 KB lo, 4 KB sy
};

__global__ void __launch_bounds__(1024) group_block_kernel(const __grid_constant__ GroupBlockArgs a) {
  const int f = blockIdx.x, w = threadIdx.x >> 5, x = threadIdx.x & 31;
  const float v = __ldg(a.val[f] + 32 * ((x >> 1) * a.rho[f] + (x & 1)) + w);
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
  __nv_bfloat16* bh = reinterpret_cast<__nv_bfloat16*>(a.out[f]);
  bh[32 * x + w] = hi;
  bh[1024 + 32 * x + w] = lo;
  reinterpret_cast<float*>(a.out[f] + 4096)[32 * w + x] = __uint_as_float(to_tf32(v));
}

// dC_q = alpha * sum over partial slots [0, nslots) in slot order.
__global__ void __launch_bounds__(256) dense_dc_reduce_kernel(const float* partial, int32_t nslots, int32_t stride,
                                                              int32_t nnz, float alpha, float* dC) {
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= nnz) return;
  float s = 0.f;
  for (int i = 0; i < nslots; ++i) s += partial[static_cast<int64_t>(i) * stride + q];
  dC[q] = alpha * s;
}

}  // namespace dense
}  // namespace ffb
