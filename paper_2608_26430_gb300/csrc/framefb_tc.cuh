// Pipelined bf16 tile kernel on 5th-generation tensor cores (tcgen05, TMEM).
// Included by framefb_cuda.cu after framefb_mma.cuh.
//
// The work per one-token tile is that of mma_tile_kernel (Sec. 3.1 update and
// the Lemma 1 gradient of Appendix A), pipelined over one-token tiles: in
// step s the tensor side runs the analysis of tile s and the synthesis of
// tile s-2, the SpMM warps the coefficient SpMM of tile s-1, and one barrier
// ends the step.  Compared with the warp-MMA kernel:
//   * the group contractions are UMMA instructions, issued by four threads
//     in parallel (one per operand side; a single issuing thread spends about
//     150 cycles per instruction at these small shapes):
//       analysis   [V D_hi | V D_lo] (M = 128 groups x N = 64) = X_rows (K = 32
//                  coordinates, bf16) x [D_hi | D_lo], D split into bf16 hi +
//                  lo parts side by side (kind::f16, fp32 accumulate in TMEM),
//                  the two halves added when read back;
//       synthesis  dY_rows (M = 128 groups x N = 32 coordinates) = Z (K = 32
//                  coefficients, fp32 read as tf32) x D^T (kind::tf32);
//     the results are read back with tcgen05.ld, one TMEM lane per group;
//   * X / dY token rows land by tensor copies (TMA) directly as the
//     SWIZZLE_64B K-major bf16 operand (one 64-byte row per group);
//   * the fp32 coefficient buffers V, U, RZ, RG use the canonical K-major
//     core-matrix layout of a tf32 operand (8 groups x 4 coefficients per
//     128-byte core matrix), so RZ / RG feed the tensor core directly and a
//     warp's row writes are bank-conflict free;
//   * 4 tensor warps (one per TMEM lane quarter) and 8 SpMM warps: SpMM
//     thread t owns plan column t, its entries and dC sums in registers.
// Shapes: every group count a multiple of 8 and at most 256 (n, m <= 8192).
//
// All waits (copies, MMA completion) are bounded; a wait that gives up
// increments g_wait_timeouts, the CTA stops at the end of the step, lets its
// copies and MMAs finish, frees its TMEM and exits.
#pragma once
#include <cuda.h>

#include "framefb_mma.cuh"

namespace ffb {

constexpr int kTcThreads = 384;            // 4 tensor warps + 8 SpMM warps
constexpr int kTcSpmm = kTcThreads - 128;  // SpMM threads (= plan columns)
constexpr int kTcMaxTiles = 2;             // 128-group tiles per side
// TMEM columns: analysis (X, dY) x 2 tiles x 64 (hi | lo), then synthesis
// (Y, dX) x 2 tiles x 32
constexpr uint32_t kTcTmemCols = 512;
constexpr uint32_t kTcColSyn = 256;

static_assert(kTcSpmm == kThreads, "one SpMM thread per plan column");

// Canonical K-major, no-swizzle operand layouts (core matrix = 8 rows x 16 B,
// rows 16 B apart; K-adjacent core matrices LBO = 128 B apart; 8-row blocks
// SBO apart).  bf16 rows of 32 elements: SBO = 512 B.  fp32 rows of 32
// elements: SBO = 1024 B.
__host__ __device__ __forceinline__ int can_bf16_off(int row, int k) {  // bytes
  return ((row >> 3) * 4 + (k >> 3)) * 128 + (row & 7) * 16 + (k & 7) * 2;
}
__host__ __device__ __forceinline__ int can_f32_off(int row, int k) {  // floats
  return ((row >> 3) * 8 + (k >> 2)) * 32 + (row & 7) * 4 + (k & 3);
}
// Slot of group-major index x (x < K) in a canonical fp32 buffer; overflow
// slots (x >= K) as they are.
__host__ __device__ __forceinline__ int32_t tc_slot(int32_t x, int32_t K) {
  return x >= K ? x : can_f32_off(x >> 5, x & 31);
}

// dC partial sums of one plan column (held in registers) to the CTA's
// workspace slot of the matrix.
template <int KE = kEreg>
__device__ __forceinline__ void dc_flush(const uint8_t* plan, float* dst, const float (&dc)[kEreg], int col) {
  const FfbPlanHeader& h = hdr(plan);
  const int32_t* gq = table<int32_t>(plan, h.off_gq);
#pragma unroll
  for (int e = 0; e < KE; ++e) {
    if (e < h.EG) {
      const int32_t q = __ldg(gq + e * kThreads + col);
      if (q >= 0) dst[q] = dc[e];
    }
  }
}

__device__ __forceinline__ void tensor_bar() { asm volatile("bar.sync 2, 128;" ::: "memory"); }
// barrier of the 128 tensor threads that also ORs a flag over them
__device__ __forceinline__ bool tensor_bar_or(bool f) {
  uint32_t out;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 2, 128, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(out)
      : "r"(static_cast<uint32_t>(f))
      : "memory");
  return out != 0;
}
__device__ __forceinline__ void tc_spmm_bar() { asm volatile("bar.sync 1, %0;" ::"n"(kTcSpmm) : "memory"); }

// Bounded wait with a non-suspending first test (the common case here: the
// phase completed long ago).
__device__ __forceinline__ bool tc_wait_bounded(uint64_t* bar, uint32_t parity) {
  return mbar_test_wait(bar, parity) || mbar_wait_bounded(bar, parity);
}
// Two blocks of 32 columns of this thread's TMEM lane, one wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta, uint32_t tb, float (&v)[32], float (&w)[32]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
      "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(ta), "r"(tb));
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    v[i] = __uint_as_float(r[i]);
    w[i] = __uint_as_float(r[32 + i]);
  }
}

// 16 consecutive fp32 columns at each of two TMEM addresses of this lane, one wait.
__device__ __forceinline__ void tmem_ld16x2(uint32_t ta, uint32_t tb, float (&v)[16], float (&w)[16]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%32];\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, "
      "[%33];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(ta), "r"(tb));
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    v[i] = __uint_as_float(r[i]);
    w[i] = __uint_as_float(r[16 + i]);
  }
}

// y (8 bf16 of one 16-byte chunk) += seff * d[0..7]
// 32 contiguous bytes of global memory (one sector) in one access: a warp whose
// lanes stride 64 bytes apart (one 32-coordinate bf16 group per lane) then
// touches each 128-byte line once per instruction instead of twice.
__device__ __forceinline__ void ld_global_256(const void* p, uint4& a, uint4& b) {
  asm volatile("ld.global.v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
               : "l"(p));
}
__device__ __forceinline__ void st_global_256(void* p, const uint4& a, const uint4& b) {
  asm volatile("st.global.v8.u32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w),
               "r"(b.x), "r"(b.y), "r"(b.z), "r"(b.w)
               : "memory");
}

__device__ __forceinline__ uint4 axpy8(uint4 y, const float* d, float seff) {
  uint32_t w[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float lo = fmaf(seff, d[2 * i], __uint_as_float(w[i] << 16));
    const float hi = fmaf(seff, d[2 * i + 1], __uint_as_float(w[i] & 0xFFFF0000u));
    w[i] = pack_bf16(lo, hi);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Coefficient SpMM of one register chunk for one token (canonical fp32 slots,
// no sign folding): run sums of c V[b] into RZ, of c U[a] into RG; dc += U V.
// Gathers go out in blocks of FFB_ENTRY_BLOCK entries: more in flight per
// thread only lengthens the shared-memory request queue that every warp of
// the SM waits in.
template <int MODE>
__device__ __forceinline__ void tc_spmm(const Chunk<MODE, true, false>& ch, float (&dc)[kEreg], float* fs,
                                        const FfbTileLayout& L) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  constexpr int B = FFB_ENTRY_BLOCK;
  const float* __restrict__ V = fs + L.oV;
  const float* __restrict__ U = fs + L.oU;
  float* __restrict__ RZ = fs + L.oRZ;
  float* __restrict__ RG = fs + L.oRG;
  if constexpr (F) {
    float acc = 0.f;
#pragma unroll
    for (int e0 = 0; e0 < kEreg; e0 += B) {
      if (e0 < ch.EZ) {
        float v[B];
#pragma unroll
        for (int e = 0; e < B; ++e) v[e] = V[ch.zb[e0 + e] & 0xFFFFu];
#pragma unroll
        for (int e = 0; e < B; ++e) {
          acc = fmaf(ch.zc[e0 + e], v[e], acc);
          const uint32_t st = ch.zb[e0 + e] >> 16;
          if (st != FFB_NO_STORE) {
            RZ[st] = acc;
            acc = 0.f;
          }
        }
      }
    }
  }
  if constexpr (D || C) {
    float acc = 0.f, vlast = 0.f;
#pragma unroll
    for (int e0 = 0; e0 < kEreg; e0 += B) {
      if (e0 < ch.EG) {
        float u[B], v[B];
#pragma unroll
        for (int e = 0; e < B; ++e) {
          u[e] = U[ch.ga[e0 + e] & 0xFFFFu];
          if constexpr (C) {
            const int ep = e0 + e - 1;
            if (ep < 0 || ch.gb[e0 + e] != ch.gb[ep])
              v[e] = V[ch.gb[e0 + e]];
            else
              v[e] = e > 0 ? v[e - 1] : vlast;
          }
        }
        if constexpr (C) vlast = v[B - 1];
#pragma unroll
        for (int e = 0; e < B; ++e) {
          if constexpr (C) dc[e0 + e] = fmaf(u[e], v[e], dc[e0 + e]);
          if constexpr (D) {
            acc = fmaf(ch.gc[e0 + e], u[e], acc);
            const uint32_t st = ch.ga[e0 + e] >> 16;
            if (st != FFB_NO_STORE) {
              RG[st] = acc;
              acc = 0.f;
            }
          }
        }
      }
    }
  }
}

// Register chunk of plan column `col` with canonical slots (the plan words
// hold group-major indices, mapped here with tc_slot; no sign folding).
template <int MODE>
__device__ __forceinline__ void tc_load_chunk(Chunk<MODE, true, false>& ch, const uint8_t* plan, const float* c_val,
                                              int col) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  const FfbPlanHeader& h = hdr(plan);
  ch.EZ = h.EZ;
  ch.EG = h.EG;
  ch.n = h.n;
  ch.m = h.m;
  const int32_t* tzb = table<int32_t>(plan, h.off_zb);
  const int32_t* tzq = table<int32_t>(plan, h.off_zq);
  const int32_t* tga = table<int32_t>(plan, h.off_ga);
  const int32_t* tgb = table<int32_t>(plan, h.off_gb);
  const int32_t* tgq = table<int32_t>(plan, h.off_gq);
  auto slots = [](uint32_t w, int Klo, int Khi) {
    const uint32_t lo = w & 0x7FFFu, hi = w >> 16;
    const uint32_t slo = static_cast<uint32_t>(tc_slot(static_cast<int32_t>(lo), Klo));
    const uint32_t shi =
        hi == FFB_NO_STORE ? FFB_NO_STORE : static_cast<uint32_t>(tc_slot(static_cast<int32_t>(hi), Khi));
    return slo | (shi << 16);
  };
#pragma unroll
  for (int e = 0; e < kEreg; ++e) {
    ch.zb[e] = FFB_NO_STORE << 16;
    ch.ga[e] = FFB_NO_STORE << 16;
    ch.gb[e] = 0;
    ch.zc[e] = ch.gc[e] = 0.f;
    if (F && e < ch.EZ) {
      const uint32_t w = static_cast<uint32_t>(__ldg(tzb + e * kThreads + col));
      ch.zb[e] = slots(w, ch.n, ch.m);
      const int32_t q = __ldg(tzq + e * kThreads + col);
      ch.zc[e] = q >= 0 ? __ldg(c_val + q) : 0.f;
    }
    if ((D || C) && e < ch.EG) {
      const uint32_t w = static_cast<uint32_t>(__ldg(tga + e * kThreads + col));
      ch.ga[e] = slots(w, ch.m, ch.n);
      ch.gb[e] = static_cast<uint32_t>(tc_slot(__ldg(tgb + e * kThreads + col), ch.n));
      const int32_t q = __ldg(tgq + e * kThreads + col);
      ch.gc[e] = (D && q >= 0) ? __ldg(c_val + q) : 0.f;
    }
  }
}

// Launch parameters of the tensor-core kernel: the fields of LaunchK it
// uses, at most kTcMaxMats matrices, and one TMA tensor map per activation
// tensor (X of matrix j at 2j, dY at 2j + 1): a 3-D view {32 coordinates,
// groups, tokens} of the row-major bf16 rows, box {32, G, 1}, 64-byte
// swizzle, which lands one token row as the canonical SWIZZLE_64B K-major
// UMMA operand (8-row atoms of 512 bytes).
constexpr int kTcMaxMats = 64;
constexpr int kTcMaxSeg = 256;  // segments of a mixed-tenant launch
struct TcLaunchK {
  int32_t nmats, total_units, stride, S;
  float* partial;
  int32_t stage, xbox_u, fbase, mbar;  // staging ring: stage stride, dY box offset (bytes)
  int32_t set_oU, set_oRZ, set_oRG, set_total;
  int32_t fixc, fixc_items, bops, pad;
  // two-token kernel: stage token strides (bytes), V/U and RZ/RG regions
  // (bytes offsets), floats of one token's RZ/RG region
  int32_t tok_x, tok_u, vu, rzg, rzg_tok, pad2;
  MatK m[kTcMaxMats];
  alignas(64) CUtensorMap maps[2 * kTcMaxMats];
  // mixed-tenant forward (two-token kernels): the tokens of every matrix
  // fall in nseg segments, segment s = tokens [seg_tok[s], seg_tok[s + 1])
  // of tenant seg_tenant[s], and a matrix's units are its segments' runs of
  // units, unit seg_u0[s] + i holding tokens seg_tok[s] + T i .. of segment
  // s only (nseg = 0: one run over all N tokens)
  int32_t nseg, pad3;
  int32_t seg_tok[kTcMaxSeg + 1], seg_u0[kTcMaxSeg + 1], seg_tenant[kTcMaxSeg];
};

__device__ __forceinline__ void tma_row3d(void* dst, const CUtensorMap* map, int32_t token, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::
          "r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(0), "r"(token), "r"(smem_u32(bar))
      : "memory");
}

// Matrix of the units a role walks through in increasing order: the
// descriptors live in the kernel parameters (constant cache, off the
// shared-memory request path); j advances when u passes its last unit.
struct TileTrack {
  int j;
  int64_t end;
  template <typename Args>
  __device__ __forceinline__ void start(const Args& args, int64_t u) {
    j = matrix_of(args, 0, u);
    end = args.m[j].ubeg + args.m[j].ntiles;
  }
  // returns true when the matrix changed
  template <typename Args>
  __device__ __forceinline__ bool advance(const Args& args, int64_t u) {
    bool moved = false;
    while (u >= end) {
      ++j;
      end = args.m[j].ubeg + args.m[j].ntiles;
      moved = true;
    }
    return moved;
  }
};

template <int MODE>
__global__ void __launch_bounds__(kTcThreads, 1) tc_tile_kernel(const __grid_constant__ TcLaunchK args) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  constexpr bool NEED_V = F || C, NEED_U = D || C, SYN = F || D;
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ uint32_t tmem_slot;
  const int S = args.S;
  uint8_t* stg0 = smem;              // stage b at b * stage: X box, dY box at xbox_u
  float* fset0 = reinterpret_cast<float*>(smem + args.fbase);
  uint8_t* bops = smem + args.bops;  // B operands: [D hi | D lo] (bf16), D^T (tf32)
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + args.mbar);
  uint64_t* mma_bar = bar + S;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  FfbTileLayout PL{};
  PL.oV = 0;
  PL.oU = args.set_oU;
  PL.oRZ = args.set_oRZ;
  PL.oRG = args.set_oRG;
  PL.total = args.set_total;

  const int64_t units = args.total_units;
  const int64_t u_begin = (static_cast<int64_t>(blockIdx.x) * units) / gridDim.x;
  const int64_t u_end = (static_cast<int64_t>(blockIdx.x + 1) * units) / gridDim.x;
  const int count = static_cast<int>(u_end - u_begin);
  if (count <= 0) return;

  if (tid == 0) {
    for (int b = 0; b < S; ++b) mbar_init(bar + b, 1);
    mbar_init(mma_bar, 4);  // the four MMA issuers
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(kTcTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();  // barriers initialised before the first copy names them

  // ---- copy issue (the first SpMM thread): tensor copies of tile `issued`
  // into its stage
  constexpr int kIssuer = 128;
  TileTrack ti{};
  int issued = 0;
  auto issue = [&]() {
    const int64_t u = u_begin + issued;
    ti.advance(args, u);
    const int jn = ti.j;
    const int32_t t = static_cast<int32_t>(u - args.m[jn].ubeg);
    uint8_t* dst = stg0 + (issued % S) * args.stage;
    uint64_t* b = bar + (issued % S);
    mbar_arrive_expect_tx(b, (NEED_V ? 2u * args.m[jn].n : 0u) + (NEED_U ? 2u * args.m[jn].m : 0u));
    if (NEED_V) tma_row3d(dst, &args.maps[2 * jn], t, b);
    if (NEED_U) tma_row3d(dst + args.xbox_u, &args.maps[2 * jn + 1], t, b);
    ++issued;
  };
  if (tid == kIssuer) {
    ti.start(args, u_begin);
    while (issued < S - 1 && issued < count) issue();
  }
  tc_fence_before();
  __syncthreads();  // TMEM address ready
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  if (warp < 4) {
    // ------------------------------------------------------------ tensor warps
    TileTrack ta{}, ts{};  // matrices of the analysis (s) and synthesis (s - 2) tiles
    ta.start(args, u_begin);
    ts.start(args, u_begin);
    {
      // B operands from the k = 16 group block (the same for every matrix):
      // analysis B[n][k = coordinate], n < 32: D4[k][n] rounded to bf16 (hi),
      // n >= 32: the bf16 remainder D4[k][n - 32] - hi (lo), so that one
      // N = 64 MMA gives both partial products; synthesis B[n = coordinate]
      // [k = coefficient] = D4[n][k] as tf32
      const float* fv = args.m[ta.j].fval_in;
      const int rho = args.m[ta.j].rho_in;
      __nv_bfloat16* ban = reinterpret_cast<__nv_bfloat16*>(bops);
      float* bsy = reinterpret_cast<float*>(bops + 4096);
      for (int i = tid; i < 1024; i += 128) {
        const int r = i >> 5, k = i & 31;
        const float dk = d4(fv, rho, k, r);  // D4[k][r]
        const __nv_bfloat16 hi = __float2bfloat16_rn(dk);
        const __nv_bfloat16 lo = __float2bfloat16_rn(dk - __bfloat162float(hi));
        ban[can_bf16_off(r, k) / 2] = hi;
        ban[can_bf16_off(32 + r, k) / 2] = lo;
        bsy[can_f32_off(r, k)] = __uint_as_float(to_tf32(d4(fv, rho, r, k)));  // D4[r][k]
      }
      fence_async_smem();
      tensor_bar();
    }
    const uint32_t id_an = umma_idesc(1, 128, 64), id_sy = umma_idesc(2, 128, 32);
    const uint64_t d_ban = umma_sdesc(smem_u32(bops), 128, 512);
    const uint64_t d_bsy = umma_sdesc(smem_u32(bops + 4096), 128, 1024);
    uint32_t mma_phase = 0;
    bool failed = false, mma_pending = false;
    const uint32_t lane_base = static_cast<uint32_t>(32 * warp) << 16;
    // synthesis matrix, in registers: output rows, sizes, scale, and for this
    // thread's groups r = 32 warp + lane (+ 128) whether they have entries
    const int r0 = 32 * warp + lane;
    bool on_y[kTcMaxTiles] = {}, on_x[kTcMaxTiles] = {};
    int js = -1;
    auto load_syn = [&](int j) {
      js = j;
      const uint8_t* plan = args.m[j].plan;
      const FfbPlanHeader& h = hdr(plan);
      const uint32_t* zm = table<uint32_t>(plan, h.off_zmask);
      const uint32_t* gm = table<uint32_t>(plan, h.off_gmask);
#pragma unroll
      for (int mt = 0; mt < kTcMaxTiles; ++mt) {
        const int r = r0 + 128 * mt;
        on_y[mt] = F && r < h.Gm && __ldg(zm + r) != 0u;
        on_x[mt] = D && r < h.Gn && __ldg(gm + r) != 0u;
      }
    };
    for (int s = 0; s < count + 2; ++s) {
      const int i2 = s - 2;
      const bool syn = SYN && i2 >= 0;
      const bool ana = s < count;
      // synthesis of tile s-2: its operands (RZ / RG written last step) are
      // ready now, so its MMAs go first (threads 64: Y, 96: dX)
      __nv_bfloat16* yrow = nullptr;
      __nv_bfloat16* xrow = nullptr;
      int Gm2 = 0, Gn2 = 0;
      float seff2 = 0.f;
      if (syn) {
        const int64_t u2 = u_begin + i2;
        ts.advance(args, u2);
        if (ts.j != js) load_syn(ts.j);
        const MatK& M2 = args.m[ts.j];
        const int64_t t2 = u2 - M2.ubeg;
        yrow = static_cast<__nv_bfloat16*>(M2.Y) + t2 * M2.ldy;
        xrow = static_cast<__nv_bfloat16*>(M2.dX) + t2 * M2.ldx;
        Gm2 = M2.m / FFB_GROUP;
        Gn2 = M2.n / FFB_GROUP;
        seff2 = M2.seff;
      }
      const bool any = (ana || syn) && !failed;  // failed is uniform here (end of the last step)
      if (lane == 0 && warp >= 2 && any) {
        const int side = warp & 1;
        if (syn && (side == 0 ? F : D)) {
          tc_fence_after();
          float* fs2 = fset0 + (i2 & 1) * PL.total;
          const int G = side == 0 ? Gm2 : Gn2;
          const uint64_t abase = umma_sdesc(smem_u32(fs2 + (side == 0 ? PL.oRZ : PL.oRG)), 128, 1024);
          for (int mt = 0; mt * 128 < G; ++mt) {
            const uint32_t d = tmem + kTcColSyn + (side * kTcMaxTiles + mt) * 32;
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
              umma_tf32(d, abase + ((mt * 16 * 1024 + ks * 256) >> 4), d_bsy + ((ks * 256) >> 4), id_sy, ks > 0);
          }
          umma_commit(mma_bar);
        } else {
          mbar_arrive(mma_bar);
        }
      }
      // output rows of tile s-2 for this thread's group of the first tile of
      // each side (read now, used after the MMAs)
      uint4 yp[2][4];
      if (syn) {
        if (F && on_y[0]) {
          const uint4* p = reinterpret_cast<const uint4*>(yrow + 32 * r0);
#pragma unroll
          for (int j = 0; j < 4; ++j) yp[0][j] = p[j];
        }
        if (D && on_x[0]) {
          const uint4* p = reinterpret_cast<const uint4*>(xrow + 32 * r0);
#pragma unroll
          for (int j = 0; j < 4; ++j) yp[1][j] = p[j];
        }
      }
      // analysis of tile s once its rows have landed (threads 0: X, 32: dY)
      if (any && lane == 0 && warp < 2) {
        const int side = warp;
        bool issued_mma = false;
        if (ana) {
          ta.advance(args, u_begin + s);
          const bool landed = tc_wait_bounded(bar + (s % S), static_cast<uint32_t>((s / S) & 1));
          if (!landed) failed = true;
          if (landed && (side == 0 ? NEED_V : NEED_U)) {
            tc_fence_after();
            const int G = (side == 0 ? args.m[ta.j].n : args.m[ta.j].m) / FFB_GROUP;
            const uint32_t abase = smem_u32(stg0 + (s % S) * args.stage) + (side == 0 ? 0 : args.xbox_u);
            for (int mt = 0; mt * 128 < G; ++mt) {
              const uint32_t d = tmem + (side * kTcMaxTiles + mt) * 64;
#pragma unroll
              for (int ks = 0; ks < 2; ++ks)
                umma_f16(d, umma_sdesc_sw64(abase + mt * 8192 + ks * 32), d_ban + ((ks * 256) >> 4), id_an, ks > 0);
            }
            umma_commit(mma_bar);
            issued_mma = true;
          }
        }
        if (!issued_mma) mbar_arrive(mma_bar);  // keeps the phase count; a failure is seen below
      }
      if (any) {
        const bool ok = tc_wait_bounded(mma_bar, mma_phase);
        if (ok)
          mma_phase ^= 1u;
        else
          mma_pending = true;
        failed = tensor_bar_or(failed || !ok);
        tc_fence_after();
      }
      if (!failed) {
        // synthesis results: y += seff * delta for groups with support entries
        if (syn) {
#pragma unroll
          for (int side = 0; side < 2; ++side) {
            const bool on = side == 0 ? F : D;
            const int G = side == 0 ? Gm2 : Gn2;
            if (on) {
#pragma unroll
              for (int mt = 0; mt < kTcMaxTiles; ++mt) {
                if (mt * 128 >= G) break;
                float v[32];
                tmem_ld32(tmem + lane_base + kTcColSyn + (side * kTcMaxTiles + mt) * 32, v);
                const bool has = side == 0 ? on_y[mt] : on_x[mt];
                if (has) {
                  uint4* p = reinterpret_cast<uint4*>((side == 0 ? yrow : xrow) + 32 * (r0 + 128 * mt));
#pragma unroll
                  for (int j = 0; j < 4; ++j) {
                    const uint4 y = mt == 0 ? yp[side][j] : p[j];
                    p[j] = axpy8(y, v + 8 * j, seff2);
                  }
                }
              }
            }
          }
        }
      }
      tc_fence_before();
      if (__syncthreads_or(failed)) break;
    }
    if (failed && tid == 0) {
      atomicAdd(&g_wait_timeouts, 1u);
      if (mma_pending) mbar_wait_bounded(mma_bar, mma_phase);  // MMAs still in flight (bounded)
    }
  } else {
    // ------------------------------------------------------------ SpMM warps
    const int st = tid - 128;
    Chunk<MODE, true, false> ch;
    float dc[kEreg];
#pragma unroll
    for (int e = 0; e < kEreg; ++e) dc[e] = 0.f;
    TileTrack tp{}, tq{};  // matrices of the SpMM tile (s - 1) and the analysis tile (s)
    tp.start(args, u_begin);
    tq.start(args, u_begin);
    uint32_t mph = 0;  // phase of the MMA barrier
    const int aside = (warp - 4) >> 2;  // analysis results written: warps 4-7 V (X), 8-11 U (dY)
    const uint32_t alane = static_cast<uint32_t>(32 * (warp & 3)) << 16;
    const int ar0 = 32 * (warp & 3) + lane;
    int cur = -1;
    const uint8_t* splan = nullptr;
    int4* fixc = reinterpret_cast<int4*>(smem + args.fixc);
    int nfZ = 0, nfix = 0, mcur = 0, ncur = 0;
    uint32_t zero_pending = 3u;
    bool failed = false;
    for (int s = 0; s < count + 2; ++s) {
      if (tid == kIssuer && issued < count) issue();  // tile s + S - 1 into the stage tile s - 1 used
      const int i1 = s - 1;
      if (i1 >= 0 && i1 < count) {
        tp.advance(args, u_begin + i1);
        if (tp.j != cur) {
          if constexpr (C) {
            if (cur >= 0) {
              float* dst = args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride;
              dc_flush(splan, dst, dc, st);
            }
          }
          cur = tp.j;
          splan = args.m[cur].plan;
          mcur = args.m[cur].m;
          ncur = args.m[cur].n;
          tc_load_chunk<MODE>(ch, splan, args.m[cur].c_val, st);
#pragma unroll
          for (int e = 0; e < kEreg; ++e) dc[e] = 0.f;
          zero_pending = 3u;
          if constexpr (SYN) {
            const FfbPlanHeader& h = hdr(splan);
            nfZ = F ? h.nfixZ : 0;
            nfix = nfZ + (D ? h.nfixG : 0);
            for (int i = st; i < nfix; i += kTcSpmm)
              fixc[i] = i < nfZ ? __ldg(table<int4>(splan, h.off_fixZ) + i)
                                : __ldg(table<int4>(splan, h.off_fixG) + (i - nfZ));
            tc_spmm_bar();
          }
        }
        float* fs1 = fset0 + (i1 & 1) * PL.total;
        if constexpr (SYN) {
          if ((zero_pending >> (i1 & 1)) & 1u) {
            for (int x = PL.oRZ + st; x < PL.total; x += kTcSpmm) fs1[x] = 0.f;
            zero_pending &= ~(1u << (i1 & 1));
            tc_spmm_bar();
          }
        }
        tc_spmm<MODE>(ch, dc, fs1, PL);
        if constexpr (SYN) {
          if (nfix > 0) {
            tc_spmm_bar();
            for (int i = st; i < nfix; i += kTcSpmm) {
              const int4 it = fixc[i];
              const bool z = i < nfZ;
              float* R = fs1 + (z ? PL.oRZ : PL.oRG);
              const int dst = tc_slot(it.x, z ? mcur : ncur);
              float sacc = R[dst];
              for (int c2 = 0; c2 < it.z; ++c2) sacc += R[it.y + c2];
              R[dst] = sacc;
            }
          }
          fence_async_smem();  // RZ / RG are read by the tensor cores next step
        }
      }
      // analysis results of tile s (TMEM, [X D_hi | X D_lo] per group) -> V / U
      // of set s & 1, one group per thread, once the step's MMAs completed
      const bool ana = s < count;
      if (ana || (SYN && s >= 2)) {
        bool ok = tc_wait_bounded(mma_bar, mph);
        if (ok) mph ^= 1u;
        failed = !ok;
        tc_fence_after();
        const bool on = aside == 0 ? NEED_V : NEED_U;
        if (ok && ana && on) {
          tq.advance(args, u_begin + s);
          const int G = (aside == 0 ? args.m[tq.j].n : args.m[tq.j].m) / FFB_GROUP;
          float* dst = fset0 + (s & 1) * PL.total + (aside == 0 ? PL.oV : PL.oU);
#pragma unroll
          for (int mt = 0; mt < kTcMaxTiles; ++mt) {
            if (mt * 128 >= G) break;
            const int r = mt * 128 + ar0;
#pragma unroll
            for (int hlf = 0; hlf < 2; ++hlf) {
              float v[16], w[16];
              const uint32_t col = tmem + alane + (aside * kTcMaxTiles + mt) * 64 + 16 * hlf;
              tmem_ld16x2(col, col + 32, v, w);  // coefficients 16 hlf .. +15: hi and lo parts
              if (r < G) {
#pragma unroll
                for (int c = 0; c < 4; ++c)
                  *reinterpret_cast<float4*>(dst + can_f32_off(r, 16 * hlf + 4 * c)) =
                      make_float4(v[4 * c] + w[4 * c], v[4 * c + 1] + w[4 * c + 1], v[4 * c + 2] + w[4 * c + 2],
                                  v[4 * c + 3] + w[4 * c + 3]);
              }
            }
          }
        }
      }
      tc_fence_before();
      if (__syncthreads_or(failed)) {
        failed = true;
        break;
      }
    }
    if (failed && tid == kIssuer) {
      // the last tile issued into each stage: let its copy land (bounded)
      for (int i = issued > S ? issued - S : 0; i < issued; ++i)
        mbar_wait_bounded(bar + (i % S), static_cast<uint32_t>((i / S) & 1));
    }
    if (!failed) {
      if constexpr (C) {
        if (cur >= 0) {
          float* dst = args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride;
          dc_flush(splan, dst, dc, st);
        }
      }
    }
  }
  // every thread is past its last TMEM access
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcTmemCols) : "memory");
  }
}

}  // namespace ffb
