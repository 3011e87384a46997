// Pipelined bf16 tile kernel on tcgen05 tensor cores, two tokens per tile.
// Included by framefb_cuda.cu after framefb_tc.cuh.
//
// Same work as tc_tile_kernel (Sec. 3.1 update, Lemma 1 gradient of
// Appendix A), with units of two tokens of one matrix, so that every
// coefficient SpMM instruction serves both tokens:
//   * V and U are held token-minor (a float2 per coefficient), so one 64-bit
//     gather feeds both tokens; they are not tensor-core operands, their
//     layout is free: group r's sixteen 16-byte chunks (two coefficients x
//     two tokens) are permuted by r mod 8 (vu_slot), which makes the
//     write-back of one group per lane conflict-free;
//   * RZ and RG stay per token in the canonical tf32 K-major layout (they are
//     the synthesis A operands);
//   * shared memory holds one V/U set and one RZ/RG set (two tokens each).
//     Step s: the SpMM warps wait until the synthesis MMAs of unit s-2 have
//     read RZ/RG, run unit s-1 (one pass over the column path gives dC and
//     G, one over the row path gives Z) and signal RZ/RG complete; the four
//     tensor warps then issue the synthesis of unit s-1 at once (one
//     (token, side) each), into the TMEM half of its parity, while the SpMM
//     warps write the analysis results of unit s into V/U;
//   * analysis (token x side) of unit s is issued by threads 0 (X) and 32
//     (dY) at the start of the step; the tensor warps apply the synthesis of
//     unit s-2 to the output rows.
// Shapes: every group count a multiple of 8 and at most 128 (n, m <= 4096).
// Waits are bounded as in tc_tile_kernel.
#pragma once
#include <type_traits>

#include "framefb_tc.cuh"

namespace ffb {

// float2 (two-token) slot of group-major index x in the V / U buffers.
__host__ __device__ __forceinline__ int32_t vu_slot(int32_t x) {
  const int32_t r = x >> 5, c = x & 31;
  return 32 * r + 2 * ((c >> 1) ^ (r & 7)) + (c & 1);
}

// barrier of the 256 SpMM threads that also ORs a flag over them
__device__ __forceinline__ bool spmm_bar_or(bool f) {
  uint32_t out;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, 256, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(out)
      : "r"(static_cast<uint32_t>(f))
      : "memory");
  return out != 0;
}

// Matrix and segment of the units a role walks through in increasing order,
// in a launch with a segment table (TcLaunchK::nseg > 0): every matrix's
// units are its segments' runs of units, so a unit's tokens lie in one
// segment and have one tenant.
struct SegTrack {
  int j, s;
  int64_t end;       // first unit past matrix j
  int64_t ubeg;      // first unit of matrix j
  int32_t T;         // tokens per unit of matrix j
  int32_t u1;        // end of segment s in matrix-local units
  int64_t base;      // first token of unit u = base + T u
  int32_t tk1;       // end of segment s in tokens
  bool seg_moved;    // the last advance entered another segment
  __device__ __forceinline__ void load_mat(const TcLaunchK& a) {
    ubeg = a.m[j].ubeg;
    end = ubeg + a.m[j].ntiles;
    T = a.m[j].T;
  }
  __device__ __forceinline__ void load_seg(const TcLaunchK& a) {
    u1 = a.seg_u0[s + 1];
    tk1 = a.seg_tok[s + 1];
    base = a.seg_tok[s] - static_cast<int64_t>(T) * (ubeg + a.seg_u0[s]);
  }
  // segment of unit u of matrix j, from segment s on (empty segments have
  // no units); the bounds of the current segment stay in registers
  __device__ __forceinline__ void seek(const TcLaunchK& a, int64_t u) {
    seg_moved = false;
    if (u - ubeg < u1) return;
    do ++s;
    while (u - ubeg >= a.seg_u0[s + 1]);
    load_seg(a);
    seg_moved = true;
  }
  __device__ __forceinline__ void start(const TcLaunchK& a, int64_t u) {
    j = matrix_of(a, 0, u);
    load_mat(a);
    s = 0;
    load_seg(a);
    seek(a, u);
    seg_moved = true;
  }
  // returns true when the matrix changed
  __device__ __forceinline__ bool advance(const TcLaunchK& a, int64_t u) {
    bool moved = false;
    if (u >= end) {
      do {
        ++j;
        load_mat(a);
      } while (u >= end);
      s = 0;
      load_seg(a);
      moved = true;
    }
    seek(a, u);
    seg_moved = seg_moved || moved;
    return moved;
  }
  // first token of unit u (u in matrix j, segment s) and the end of its segment
  __device__ __forceinline__ int64_t tok0(const TcLaunchK&, int64_t u) const { return base + T * u; }
  __device__ __forceinline__ int32_t tend(const TcLaunchK&) const { return tk1; }
};

// Register chunk of plan column `col` (its first KE entries): gather slots
// in the float2 V / U layout, store targets in the canonical RZ / RG layout.
template <int MODE, int KE = kEreg>
__device__ __forceinline__ void tc2_load_chunk(Chunk<MODE, true, false>& ch, const uint8_t* plan, const float* c_val,
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
  auto slots = [](uint32_t w, int Khi) {
    const uint32_t lo = w & 0x7FFFu, hi = w >> 16;
    const uint32_t slo = static_cast<uint32_t>(vu_slot(static_cast<int32_t>(lo)));
    const uint32_t shi =
        hi == FFB_NO_STORE ? FFB_NO_STORE : static_cast<uint32_t>(tc_slot(static_cast<int32_t>(hi), Khi));
    return slo | (shi << 16);
  };
#pragma unroll
  for (int e = 0; e < KE; ++e) {
    ch.zb[e] = FFB_NO_STORE << 16;
    ch.ga[e] = FFB_NO_STORE << 16;
    ch.gb[e] = 0;
    ch.zc[e] = ch.gc[e] = 0.f;
    if (F && e < ch.EZ) {
      const uint32_t w = static_cast<uint32_t>(__ldg(tzb + e * kThreads + col));
      ch.zb[e] = slots(w, ch.m);
      const int32_t q = __ldg(tzq + e * kThreads + col);
      ch.zc[e] = q >= 0 ? __ldg(c_val + q) : 0.f;
    }
    if ((D || C) && e < ch.EG) {
      const uint32_t w = static_cast<uint32_t>(__ldg(tga + e * kThreads + col));
      ch.ga[e] = slots(w, ch.n);
      ch.gb[e] = static_cast<uint32_t>(vu_slot(__ldg(tgb + e * kThreads + col)));
      const int32_t q = __ldg(tgq + e * kThreads + col);
      ch.gc[e] = (D && q >= 0) ? __ldg(c_val + q) : 0.f;
    }
  }
}

// SEG: the launch carries a segment table (mixed-tenant forward): units
// follow the segments and the coefficient values are the unit's tenant's.
template <int MODE, bool SEG = false>
__global__ void __launch_bounds__(kTcThreads, 1) tc2_tile_kernel(const __grid_constant__ TcLaunchK args) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  static_assert(!SEG || MODE == MODE_F, "segment tables serve the forward pass");
  using Track = std::conditional_t<SEG, SegTrack, TileTrack>;
  // first token of unit u (tracked by t), end of its tokens
  auto tok0 = [&](const Track& t, int64_t u) -> int64_t {
    if constexpr (SEG)
      return t.tok0(args, u);
    else
      return 2 * (u - args.m[t.j].ubeg);
  };
  auto tend = [&](const Track& t) -> int64_t {
    if constexpr (SEG)
      return t.tend(args);
    else
      return args.m[t.j].N;
  };
  constexpr bool NEED_V = F || C, NEED_U = D || C, SYN = F || D;
  constexpr int B = FFB_ENTRY_BLOCK;
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ uint32_t tmem_slot;
  const int S = args.S;
  uint8_t* stg0 = smem;  // stage b at b * stage: X tokens at k * tok_x, dY tokens at xbox_u + k * tok_u
  float2* V2 = reinterpret_cast<float2*>(smem + args.vu);
  float2* U2 = V2 + args.set_oU;
  float* rzg = reinterpret_cast<float*>(smem + args.rzg);  // token k at k * rzg_tok: RZ at set_oRZ, RG at set_oRG
  uint8_t* bops = smem + args.bops;
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + args.mbar);
  uint64_t* ana_bar = bar + S;
  uint64_t* syn_bar = bar + S + 1;
  uint64_t* rzg_bar = bar + S + 2;  // RZ / RG of the step's SpMM unit written
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  const int64_t units = args.total_units;
  const int64_t u_begin = (static_cast<int64_t>(blockIdx.x) * units) / gridDim.x;
  const int64_t u_end = (static_cast<int64_t>(blockIdx.x + 1) * units) / gridDim.x;
  const int count = static_cast<int>(u_end - u_begin);
  if (count <= 0) return;

  if (tid == 0) {
    for (int b = 0; b < S; ++b) mbar_init(bar + b, 1);
    mbar_init(ana_bar, 2);  // threads 0 and 32
    mbar_init(syn_bar, 4);  // lane 0 of each tensor warp
    mbar_init(rzg_bar, 1);  // SpMM thread 0
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(kTcTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();  // barriers initialised before the first copy names them

  // ---- copy issue (thread 32, at the start of its step, before it waits for
  // its own rows): both token rows of unit `issued`
  constexpr int kIssuer = 32;
  Track ti{};
  int issued = 0;
  auto issue = [&]() {
    const int64_t u = u_begin + issued;
    ti.advance(args, u);
    const int jn = ti.j;
    const int32_t t0 = static_cast<int32_t>(tok0(ti, u));
    const int Tc = min(2, static_cast<int>(tend(ti) - t0));
    uint8_t* dst = stg0 + (issued % S) * args.stage;
    uint64_t* b = bar + (issued % S);
    mbar_arrive_expect_tx(b, static_cast<uint32_t>(Tc) * ((NEED_V ? 2u * args.m[jn].n : 0u) +
                                                         (NEED_U ? 2u * args.m[jn].m : 0u)));
    for (int k = 0; k < Tc; ++k) {
      if (NEED_V) tma_row3d(dst + k * args.tok_x, &args.maps[2 * jn], t0 + k, b);
      if (NEED_U) tma_row3d(dst + args.xbox_u + k * args.tok_u, &args.maps[2 * jn + 1], t0 + k, b);
    }
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
    Track ta{}, ts{}, tr{};  // units of the analysis (s), the output rows (s-2), the synthesis issue (s-1)
    ta.start(args, u_begin);
    ts.start(args, u_begin);
    tr.start(args, u_begin);
    {
      const float* fv = args.m[ta.j].fval_in;
      const int rho = args.m[ta.j].rho_in;
      __nv_bfloat16* ban = reinterpret_cast<__nv_bfloat16*>(bops);
      float* bsy = reinterpret_cast<float*>(bops + 4096);
      for (int i = tid; i < 1024; i += 128) {
        const int r = i >> 5, k = i & 31;
        const float dk = d4(fv, rho, k, r);  // D4[k][r]
        const __nv_bfloat16 hi = __float2bfloat16_rn(dk);
        const __nv_bfloat16 lo = __float2bfloat16_rn(dk - __bfloat162float(hi));
        ban[can_bf16_off(16 * (r >> 3) + (r & 7), k) / 2] = hi;      // output column 16 (c / 8) + c % 8
        ban[can_bf16_off(16 * (r >> 3) + 8 + (r & 7), k) / 2] = lo;  // output column 16 (c / 8) + 8 + c % 8
        bsy[can_f32_off(r, k)] = __uint_as_float(to_tf32(d4(fv, rho, r, k)));  // D4[r][k]
      }
      fence_async_smem();
      tensor_bar();
    }
    const uint32_t id_an = umma_idesc(1, 128, 64), id_sy = umma_idesc(2, 128, 32);
    const uint64_t d_ban = umma_sdesc(smem_u32(bops), 128, 512);
    const uint64_t d_bsy = umma_sdesc(smem_u32(bops + 4096), 128, 1024);
    uint32_t syn_ph = 0, rzg_ph = 0;
    bool failed = false, syn_open = false;  // syn_open: a synthesis issued and not yet waited for
    const uint32_t lane_base = static_cast<uint32_t>(32 * warp) << 16;
    const int r0 = 32 * warp + lane;  // this thread's group (one 128-group tile)
    // synthesis matrix, in registers
    int js = -1, Gm2 = 0, Gn2 = 0;
    bool on_y = false, on_x = false, wide_y = false, wide_x = false;
    __nv_bfloat16 *Y2 = nullptr, *X2 = nullptr;
    int64_t ldy2 = 0, ldx2 = 0;
    float seff2 = 0.f;
    auto load_syn = [&](int j) {
      js = j;
      Y2 = static_cast<__nv_bfloat16*>(args.m[j].Y);
      X2 = static_cast<__nv_bfloat16*>(args.m[j].dX);
      ldy2 = args.m[j].ldy;
      ldx2 = args.m[j].ldx;
      Gm2 = args.m[j].m / FFB_GROUP;
      Gn2 = args.m[j].n / FFB_GROUP;
      seff2 = args.m[j].seff;
      // 256-bit row accesses need 32-byte aligned rows (the interface promises 16)
      wide_y = (reinterpret_cast<uintptr_t>(Y2) & 31u) == 0 && (ldy2 & 15) == 0;
      wide_x = (reinterpret_cast<uintptr_t>(X2) & 31u) == 0 && (ldx2 & 15) == 0;
      const uint8_t* plan = args.m[j].plan;
      const FfbPlanHeader& h = hdr(plan);
      on_y = F && r0 < Gm2 && __ldg(table<uint32_t>(plan, h.off_zmask) + r0) != 0u;
      on_x = D && r0 < Gn2 && __ldg(table<uint32_t>(plan, h.off_gmask) + r0) != 0u;
    };
    for (int s = 0; s < count + 2; ++s) {
      const int i2 = s - 2, i1 = s - 1;
      const bool epi = SYN && i2 >= 0;                // output rows of unit s-2
      const bool iss = SYN && i1 >= 0 && i1 < count;  // synthesis of unit s-1, after its SpMM
      const bool ana = s < count;
      // both rows of unit s + S - 1 into the stage unit s - 1 used (its MMAs completed last step)
      if (tid == kIssuer && issued < count) issue();
      int64_t t2 = 0;
      int Tc2 = 0;
      if (epi) {
        ts.advance(args, u_begin + i2);
        if (ts.j != js) load_syn(ts.j);
        t2 = tok0(ts, u_begin + i2);
        Tc2 = min(2, static_cast<int>(tend(ts) - t2));
      }
      // output rows of unit s-2 for this thread's group (read now, used after the wait)
      uint4 yp[2][2][4];
      if (epi) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          if (k < Tc2) {
#pragma unroll
            for (int side = 0; side < 2; ++side) {
              if (!(side == 0 ? on_y : on_x)) continue;
              const __nv_bfloat16* p = side == 0 ? Y2 + (t2 + k) * ldy2 + 32 * r0 : X2 + (t2 + k) * ldx2 + 32 * r0;
              if (side == 0 ? wide_y : wide_x) {
                ld_global_256(p, yp[k][side][0], yp[k][side][1]);
                ld_global_256(p + 16, yp[k][side][2], yp[k][side][3]);
              } else {
#pragma unroll
                for (int j = 0; j < 4; ++j) yp[k][side][j] = reinterpret_cast<const uint4*>(p)[j];
              }
            }
          }
        }
      }
      // analysis of unit s once its rows have landed: threads 0 (X) and 32 (dY)
      if (ana && lane == 0 && warp < 2) {
        const int side = warp;
        ta.advance(args, u_begin + s);
        const int64_t t0 = tok0(ta, u_begin + s);
        const int Tc0 = min(2, static_cast<int>(tend(ta) - t0));
        const bool landed = tc_wait_bounded(bar + (s % S), static_cast<uint32_t>((s / S) & 1));
        if (!landed) failed = true;
        if (landed && (side == 0 ? NEED_V : NEED_U)) {
          tc_fence_after();
          const uint32_t st0 = smem_u32(stg0 + (s % S) * args.stage);
          for (int k = 0; k < Tc0; ++k) {
            const uint32_t abase = st0 + (side == 0 ? k * args.tok_x : args.xbox_u + k * args.tok_u);
            const uint32_t d = tmem + (2 * k + side) * 64;
#pragma unroll
            for (int ks = 0; ks < 2; ++ks)
              umma_f16(d, umma_sdesc_sw64(abase + ks * 32), d_ban + ((ks * 256) >> 4), id_an, ks > 0);
          }
          umma_commit(ana_bar);
        } else {
          mbar_arrive(ana_bar);  // keeps the phase count; a failure is seen below
        }
      }
      failed = tensor_bar_or(failed);
      // synthesis results of unit s-2: y += seff * delta for groups with support entries
      if (epi && !failed) {
        const bool ok = tc_wait_bounded(syn_bar, syn_ph);
        if (ok) {
          syn_ph ^= 1u;
          syn_open = false;
        }
        failed = tensor_bar_or(!ok);
        tc_fence_after();
        if (!failed) {
          const uint32_t col0 = tmem + lane_base + kTcColSyn + 128 * static_cast<uint32_t>(i2 & 1);
#pragma unroll
          for (int k = 0; k < 2; ++k) {
            if (k >= Tc2) break;
#pragma unroll
            for (int side = 0; side < 2; ++side) {
              if (!(side == 0 ? F : D)) continue;
              float v[32];
              tmem_ld32(col0 + (2 * k + side) * 32, v);
              if (side == 0 ? on_y : on_x) {
                __nv_bfloat16* p = side == 0 ? Y2 + (t2 + k) * ldy2 + 32 * r0 : X2 + (t2 + k) * ldx2 + 32 * r0;
                if (side == 0 ? wide_y : wide_x) {
#pragma unroll
                  for (int j = 0; j < 2; ++j)
                    st_global_256(p + 16 * j, axpy8(yp[k][side][2 * j], v + 16 * j, seff2),
                                  axpy8(yp[k][side][2 * j + 1], v + 16 * j + 8, seff2));
                } else {
#pragma unroll
                  for (int j = 0; j < 4; ++j)
                    reinterpret_cast<uint4*>(p)[j] = axpy8(yp[k][side][j], v + 8 * j, seff2);
                }
              }
            }
          }
        }
      }
      // synthesis of unit s-1 once the SpMM warps have written its RZ / RG:
      // lane 0 of tensor warp w issues (token w / 2, side w % 2) into the TMEM
      // half of the unit's parity
      if (iss && !failed && lane == 0) {
        tr.advance(args, u_begin + i1);
        const int64_t t1 = tok0(tr, u_begin + i1);
        const int Tc1 = min(2, static_cast<int>(tend(tr) - t1));
        const int k = warp >> 1, side = warp & 1;
        const bool ok = tc_wait_bounded(rzg_bar, rzg_ph);
        if (ok)
          rzg_ph ^= 1u;
        else
          failed = true;
        if (ok && k < Tc1 && (side == 0 ? F : D)) {
          tc_fence_after();
          const float* A = rzg + k * args.rzg_tok + (side == 0 ? args.set_oRZ : args.set_oRG);
          const uint64_t abase = umma_sdesc(smem_u32(A), 128, 1024);
          const uint32_t d = tmem + kTcColSyn + 128 * static_cast<uint32_t>(i1 & 1) + (2 * k + side) * 32;
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_tf32(d, abase + ((ks * 256) >> 4), d_bsy + ((ks * 256) >> 4), id_sy, ks > 0);
          umma_commit(syn_bar);
        } else {
          mbar_arrive(syn_bar);  // keeps the phase count
        }
        syn_open = true;
      }
      tc_fence_before();
      if (__syncthreads_or(failed)) break;
    }
    if (failed) {
      if (tid == 0) {
        atomicAdd(&g_wait_timeouts, 1u);
        if (syn_open) mbar_wait_bounded(syn_bar, syn_ph);  // synthesis MMAs in flight (bounded)
      }
      if (tid == kIssuer) {
        for (int i = issued > S ? issued - S : 0; i < issued; ++i)
          mbar_wait_bounded(bar + (i % S), static_cast<uint32_t>((i / S) & 1));
      }
    }
  } else {
    // ------------------------------------------------------------ SpMM warps
    const int st = tid - 128;
    Chunk<MODE, true, false> ch;
    float dc[kEreg];
#pragma unroll
    for (int e = 0; e < kEreg; ++e) dc[e] = 0.f;
    Track tp{}, tq{};
    tp.start(args, u_begin);
    tq.start(args, u_begin);
    int tenant = -1;  // SEG: tenant of the loaded coefficient values
    uint32_t ana_ph = 0, syn_ph = 0;
    const int aside = (warp - 4) >> 2;  // analysis results written: warps 4-7 V (X), 8-11 U (dY)
    const uint32_t alane = static_cast<uint32_t>(32 * (warp & 3)) << 16;
    const int ar = 32 * (warp & 3) + lane;
    int cur = -1, mcur = 0, ncur = 0;
    const uint8_t* splan = nullptr;
    int4* fixc = reinterpret_cast<int4*>(smem + args.fixc);
    int nfZ = 0, nfix = 0;
    bool zero_pending = true;
    bool failed = false, ana_open = false;  // analysis MMAs of this step not yet waited for
    for (int s = 0; s < count + 2; ++s) {
      const int i1 = s - 1;
      const bool work = i1 >= 0 && i1 < count;
      const bool ana = s < count;
      ana_open = ana;
      if (work) {
        tp.advance(args, u_begin + i1);
        if constexpr (SEG) {
          // another tenant of the same matrix: its coefficient values
          if (tp.seg_moved && tp.j == cur && args.seg_tenant[tp.s] != tenant) {
            tenant = args.seg_tenant[tp.s];
            tc2_load_chunk<MODE>(ch, splan, args.m[cur].c_val + static_cast<int64_t>(tenant) * hdr(splan).nnz, st);
          }
        }
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
          if constexpr (SEG) {
            tenant = args.seg_tenant[tp.s];
            tc2_load_chunk<MODE>(ch, splan, args.m[cur].c_val + static_cast<int64_t>(tenant) * hdr(splan).nnz, st);
          } else {
            tc2_load_chunk<MODE>(ch, splan, args.m[cur].c_val, st);
          }
#pragma unroll
          for (int e = 0; e < kEreg; ++e) dc[e] = 0.f;
          zero_pending = true;
          if constexpr (SYN) {
            const FfbPlanHeader& h = hdr(splan);
            nfZ = F ? h.nfixZ : 0;
            nfix = nfZ + (D ? h.nfixG : 0);
            for (int i = st; i < nfix; i += kTcSpmm)
              fixc[i] = i < nfZ ? __ldg(table<int4>(splan, h.off_fixZ) + i)
                                : __ldg(table<int4>(splan, h.off_fixG) + (i - nfZ));
          }
        }
      }
      // RZ / RG are free once the synthesis MMAs of unit s-2 have read them
      if (SYN && work && i1 >= 1) {
        const bool ok = tc_wait_bounded(syn_bar, syn_ph);
        if (ok) syn_ph ^= 1u;
        failed = spmm_bar_or(failed || !ok);  // uniform before the barriers below
      }
      if (work && !failed) {
        if constexpr (SYN) {
          if (zero_pending) {
            for (int x = st; x < 2 * args.rzg_tok; x += kTcSpmm) rzg[x] = 0.f;
            zero_pending = false;
            tc_spmm_bar();
          }
        }
        float* RZ0 = rzg + args.set_oRZ;
        float* RZ1 = RZ0 + args.rzg_tok;
        float* RG0 = rzg + args.set_oRG;
        float* RG1 = RG0 + args.rzg_tok;
        // column path: one gather of U[a] per entry serves dC (with V[b],
        // reloaded where b changes) and the run sums of G
        if constexpr (NEED_U) {
          float2 vk = make_float2(0.f, 0.f), acc = make_float2(0.f, 0.f);
#pragma unroll
          for (int e0 = 0; e0 < kEreg; e0 += B) {
            if (e0 < ch.EG) {
              float2 ub[B], vb[B];
#pragma unroll
              for (int e = 0; e < B; ++e) {
                ub[e] = U2[ch.ga[e0 + e] & 0xFFFFu];
                if constexpr (C) {
                  const int ep = e0 + e - 1;
                  vb[e] = (ep < 0 || ch.gb[e0 + e] != ch.gb[ep]) ? V2[ch.gb[e0 + e]] : make_float2(0.f, 0.f);
                }
              }
#pragma unroll
              for (int e = 0; e < B; ++e) {
                if constexpr (C) {
                  const int ep = e0 + e - 1;
                  if (ep < 0 || ch.gb[e0 + e] != ch.gb[ep]) vk = vb[e];
                  dc[e0 + e] = fmaf(ub[e].x, vk.x, fmaf(ub[e].y, vk.y, dc[e0 + e]));
                }
                if constexpr (D) {
                  acc.x = fmaf(ch.gc[e0 + e], ub[e].x, acc.x);
                  acc.y = fmaf(ch.gc[e0 + e], ub[e].y, acc.y);
                  const uint32_t sg = ch.ga[e0 + e] >> 16;
                  if (sg != FFB_NO_STORE) {
                    RG0[sg] = acc.x;
                    RG1[sg] = acc.y;
                    acc = make_float2(0.f, 0.f);
                  }
                }
              }
            }
          }
        }
        // row path: run sums of Z
        if constexpr (F) {
          float2 acc = make_float2(0.f, 0.f);
#pragma unroll
          for (int e0 = 0; e0 < kEreg; e0 += B) {
            if (e0 < ch.EZ) {
              float2 v[B];
#pragma unroll
              for (int e = 0; e < B; ++e) v[e] = V2[ch.zb[e0 + e] & 0xFFFFu];
#pragma unroll
              for (int e = 0; e < B; ++e) {
                acc.x = fmaf(ch.zc[e0 + e], v[e].x, acc.x);
                acc.y = fmaf(ch.zc[e0 + e], v[e].y, acc.y);
                const uint32_t sz = ch.zb[e0 + e] >> 16;
                if (sz != FFB_NO_STORE) {
                  RZ0[sz] = acc.x;
                  RZ1[sz] = acc.y;
                  acc = make_float2(0.f, 0.f);
                }
              }
            }
          }
        }
        if constexpr (SYN) {
          if (nfix > 0) {
            // rows (columns) split between chunks: add the overflow pieces
            tc_spmm_bar();
            for (int i = st; i < nfix; i += kTcSpmm) {
              const int4 it = fixc[i];
              const bool z = i < nfZ;
              const int dst = tc_slot(it.x, z ? mcur : ncur);
#pragma unroll
              for (int k = 0; k < 2; ++k) {
                float* R = rzg + k * args.rzg_tok + (z ? args.set_oRZ : args.set_oRG);
                float sacc = R[dst];
                for (int c2 = 0; c2 < it.z; ++c2) sacc += R[it.y + c2];
                R[dst] = sacc;
              }
            }
          }
          fence_async_smem();  // RZ / RG are read by the tensor cores next
        }
      }
      // RZ / RG of unit s-1 complete (also on a failure: the tensor warps'
      // wait keeps its phase count)
      if (SYN && work) {
        tc_spmm_bar();
        if (st == 0) mbar_arrive(rzg_bar);
      }
      // analysis results of unit s -> V / U (float2: both tokens), once every
      // SpMM warp finished gathering from them and the MMAs completed
      if (ana && !failed) {
        if (!(SYN && work)) tc_spmm_bar();  // (else the barrier above): all gathers done
        const bool ok = tc_wait_bounded(ana_bar, ana_ph);
        if (ok) {
          ana_ph ^= 1u;
          ana_open = false;
        }
        failed = !ok;
        tc_fence_after();
        const bool on = aside == 0 ? NEED_V : NEED_U;
        if (ok && on) {
          tq.advance(args, u_begin + s);
          const int G = (aside == 0 ? args.m[tq.j].n : args.m[tq.j].m) / FFB_GROUP;
          const int64_t t0 = tok0(tq, u_begin + s);
          const bool two = tend(tq) - t0 >= 2;
          float2* dst = aside == 0 ? V2 : U2;
#pragma unroll
          for (int q8 = 0; q8 < 4; ++q8) {  // coefficients 8 q8 .. 8 q8 + 7: hi and lo in 16 columns
            float x0[16], x1[16];
            const uint32_t c0 = tmem + alane + (0 * 2 + aside) * 64 + 16 * q8;
            const uint32_t c1 = tmem + alane + (1 * 2 + aside) * 64 + 16 * q8;
            tmem_ld16x2(c0, c1, x0, x1);
            if (ar < G) {
#pragma unroll
              for (int j = 0; j < 4; ++j) {  // chunk q = 4 q8 + j: coefficients 2q, 2q + 1
                const int q = 4 * q8 + j;
                const float a0 = x0[2 * j] + x0[8 + 2 * j], a1 = x0[2 * j + 1] + x0[8 + 2 * j + 1];
                const float b0 = two ? x1[2 * j] + x1[8 + 2 * j] : 0.f, b1 = two ? x1[2 * j + 1] + x1[8 + 2 * j + 1] : 0.f;
                *reinterpret_cast<float4*>(dst + 32 * ar + 2 * (q ^ (ar & 7))) = make_float4(a0, b0, a1, b1);
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
    if (failed) {
      // analysis MMAs of the failing step may still be in flight (bounded)
      if (st == 0 && ana_open) mbar_wait_bounded(ana_bar, ana_ph);
    } else {
      if constexpr (C) {
        if (cur >= 0) {
          float* dst = args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride;
          dc_flush(splan, dst, dc, st);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcTmemCols) : "memory");
  }
}

}  // namespace ffb
