// Packed bf16 tile kernel on tcgen05 tensor cores: the two-token kernel's
// pipeline for small dimensions (at most 64 groups a side), with P token
// pairs per unit.  Included by framefb_cuda.cu after framefb_tc2.cuh.
//
// Same work as tc2_tile_kernel (Sec. 3.1 update, Lemma 1 gradient of
// Appendix A).  The M = 128 lanes of a tile carry P tokens of each slot,
// lane p G + g holding group g of token p (P G <= 128 on both sides), so a
// unit is 2P tokens and the step's fixed costs (MMA issue and completion,
// TMEM loads, barriers, and the tensor core's shared-memory reads of whole
// 128-row operands) are shared by P token pairs:
//   * slot k (k = 0, 1) holds tokens t0 + kP .. t0 + kP + P - 1, landed by
//     one tensor copy of P rows (box {32, G, P}; tokens past N land as zeros
//     and count toward the copy's bytes);
//   * the SpMM warps run pair p = (t0 + p, t0 + P + p) from its own V/U set
//     (stride n + m float2), both paths of a block of entries in one
//     shared-memory round trip, storing into rows p G .. p G + G - 1 of RZ /
//     RG (offset p m resp. p n floats in the canonical layout); overflow
//     slots of pair p sit after the P canonical blocks; the fix-ups run one
//     (item, pair) per thread;
//   * plan chunks of at most kEregPack entries are held in registers.
// Waits are bounded as in tc_tile_kernel.
#pragma once
#include "framefb_tc2.cuh"

namespace ffb {

// Chunk entries the packed kernel holds in registers (plans with more take
// the unpacked kernel).
constexpr int kEregPack = 8;

// SEG: the launch carries a segment table (mixed-tenant forward): units
// follow the segments and the coefficient values are the unit's tenant's.
template <int MODE, bool SEG = false>
__global__ void __launch_bounds__(kTcThreads, 1) tc2p_tile_kernel(const __grid_constant__ TcLaunchK args) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  static_assert(!SEG || MODE == MODE_F, "segment tables serve the forward pass");
  using Track = std::conditional_t<SEG, SegTrack, TileTrack>;
  constexpr bool NEED_V = F || C, NEED_U = D || C, SYN = F || D;
  constexpr int B = FFB_ENTRY_BLOCK;
  constexpr int KE = kEregPack;  // register chunk entries
  static_assert(KE % B == 0 && KE <= kEreg, "register chunk must hold whole blocks");
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ uint32_t tmem_slot;
  const int S = args.S;
  uint8_t* stg0 = smem;  // stage b at b * stage: X tokens at k * tok_x, dY tokens at xbox_u + k * tok_u
  float2* V2 = reinterpret_cast<float2*>(smem + args.vu);  // pair p: V at p (n + m), U after it
  float* rzg = reinterpret_cast<float*>(smem + args.rzg);  // token k at k * rzg_tok: RZ at set_oRZ, RG at set_oRG
  uint8_t* bops = smem + args.bops;
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + args.mbar);
  uint64_t* ana_bar = bar + S;
  uint64_t* syn_bar = bar + S + 1;
  uint64_t* rzg_bar = bar + S + 2;  // RZ / RG of the step's SpMM unit written
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // token pairs per slot of matrix j (a unit is 2P tokens)
  auto pairs = [&](int j) { return args.m[j].T >> 1; };
  // slots of a unit starting at token t0 that hold tokens (1 or 2)
  auto slots = [](int64_t N, int64_t t0, int P) { return N - t0 > P ? 2 : 1; };
  // first token of unit u (tracked by t), end of its tokens
  auto tok0 = [&](const Track& t, int64_t u) -> int64_t {
    if constexpr (SEG)
      return t.tok0(args, u);
    else
      return 2 * static_cast<int64_t>(pairs(t.j)) * (u - args.m[t.j].ubeg);
  };
  auto tend = [&](const Track& t) -> int64_t {
    if constexpr (SEG)
      return t.tend(args);
    else
      return args.m[t.j].N;
  };

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
    const int P = pairs(jn);
    const int32_t t0 = static_cast<int32_t>(tok0(ti, u));
    const int ns = slots(tend(ti), t0, P);
    uint8_t* dst = stg0 + (issued % S) * args.stage;
    uint64_t* b = bar + (issued % S);
    // whole boxes of P token rows: rows past N land as zeros and count;
    // rows past the segment's end (of the next segment) are not used
    mbar_arrive_expect_tx(b, static_cast<uint32_t>(ns * P) * ((NEED_V ? 2u * args.m[jn].n : 0u) +
                                                             (NEED_U ? 2u * args.m[jn].m : 0u)));
    for (int k = 0; k < ns; ++k) {
      if (NEED_V) tma_row3d(dst + k * args.tok_x, &args.maps[2 * jn], t0 + k * P, b);
      if (NEED_U) tma_row3d(dst + args.xbox_u + k * args.tok_u, &args.maps[2 * jn + 1], t0 + k * P, b);
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
    const int r0 = 32 * warp + lane;  // this thread's TMEM lane: (pair, group) p G + g
    // synthesis matrix, in registers: pairs, and this lane's pair and group
    // per side (Y: out groups, dX: in groups)
    int js = -1, P2 = 1, py = 0, gy = 0, px = 0, gx = 0;
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
      P2 = pairs(j);
      const int Gm2 = args.m[j].m / FFB_GROUP, Gn2 = args.m[j].n / FFB_GROUP;
      py = r0 / Gm2;
      gy = r0 - py * Gm2;
      px = r0 / Gn2;
      gx = r0 - px * Gn2;
      seff2 = args.m[j].seff;
      // 256-bit row accesses need 32-byte aligned rows (the interface promises 16)
      wide_y = (reinterpret_cast<uintptr_t>(Y2) & 31u) == 0 && (ldy2 & 15) == 0;
      wide_x = (reinterpret_cast<uintptr_t>(X2) & 31u) == 0 && (ldx2 & 15) == 0;
      const uint8_t* plan = args.m[j].plan;
      const FfbPlanHeader& h = hdr(plan);
      on_y = F && py < P2 && __ldg(table<uint32_t>(plan, h.off_zmask) + gy) != 0u;
      on_x = D && px < P2 && __ldg(table<uint32_t>(plan, h.off_gmask) + gx) != 0u;
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
      int64_t N2 = 0;  // end of the unit's tokens
      if (epi) {
        ts.advance(args, u_begin + i2);
        if (ts.j != js) load_syn(ts.j);
        t2 = tok0(ts, u_begin + i2);
        N2 = tend(ts);
        Tc2 = slots(N2, t2, P2);
      }
      // token of slot k on this lane's side, and whether it is one
      auto tok = [&](int k, int side) { return t2 + k * P2 + (side == 0 ? py : px); };
      auto live = [&](int k, int side) { return (side == 0 ? on_y : on_x) && tok(k, side) < N2; };
      // output rows of unit s-2 for this thread's group (read now, used after the wait)
      uint4 yp[2][2][4];
      if (epi) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          if (k < Tc2) {
#pragma unroll
            for (int side = 0; side < 2; ++side) {
              if (!live(k, side)) continue;
              const __nv_bfloat16* p =
                  side == 0 ? Y2 + tok(k, 0) * ldy2 + 32 * gy : X2 + tok(k, 1) * ldx2 + 32 * gx;
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
        const int P0 = pairs(ta.j);
        const int64_t t0 = tok0(ta, u_begin + s);
        const int Tc0 = slots(tend(ta), t0, P0);
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
              if (live(k, side)) {
                __nv_bfloat16* p = side == 0 ? Y2 + tok(k, 0) * ldy2 + 32 * gy : X2 + tok(k, 1) * ldx2 + 32 * gx;
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
        const int P1 = pairs(tr.j);
        const int64_t t1 = tok0(tr, u_begin + i1);
        const int Tc1 = slots(tend(tr), t1, P1);
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
    for (int e = 0; e < KE; ++e) dc[e] = 0.f;
    Track tp{}, tq{};
    tp.start(args, u_begin);
    tq.start(args, u_begin);
    int tenant = -1;  // SEG: tenant of the loaded coefficient values
    uint32_t ana_ph = 0, syn_ph = 0;
    const int aside = (warp - 4) >> 2;  // analysis results written: warps 4-7 V (X), 8-11 U (dY)
    const uint32_t alane = static_cast<uint32_t>(32 * (warp & 3)) << 16;
    const int ar = 32 * (warp & 3) + lane;
    // matrix of the SpMM unit: features, pairs, overflow slots per pair
    int cur = -1, mcur = 0, ncur = 0, Pc = 1, ovz = 0, ovg = 0;
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
            tc2_load_chunk<MODE, KE>(ch, splan, args.m[cur].c_val + static_cast<int64_t>(tenant) * hdr(splan).nnz, st);
          }
        }
        if (tp.j != cur) {
          if constexpr (C) {
            if (cur >= 0) {
              float* dst = args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride;
              dc_flush<KE>(splan, dst, dc, st);
            }
          }
          cur = tp.j;
          splan = args.m[cur].plan;
          mcur = args.m[cur].m;
          ncur = args.m[cur].n;
          Pc = pairs(cur);
          if constexpr (SEG) {
            tenant = args.seg_tenant[tp.s];
            tc2_load_chunk<MODE, KE>(ch, splan, args.m[cur].c_val + static_cast<int64_t>(tenant) * hdr(splan).nnz, st);
          } else {
            tc2_load_chunk<MODE, KE>(ch, splan, args.m[cur].c_val, st);
          }
#pragma unroll
          for (int e = 0; e < KE; ++e) dc[e] = 0.f;
          zero_pending = true;
          const FfbPlanHeader& h = hdr(splan);
          ovz = h.ovfZ;
          ovg = h.ovfG;
          if constexpr (SYN) {
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
        // pairs of the unit that hold tokens
        const int64_t t0s = tok0(tp, u_begin + i1);
        const int np = static_cast<int>(min(static_cast<int64_t>(Pc), tend(tp) - t0s));
        for (int p = 0; p < np; ++p) {
          const float2* V2p = V2 + p * (ncur + mcur);
          const float2* U2p = V2p + ncur;
          // store bases of pair p: canonical rows p G .., overflow slots
          // (index >= the side's features) after the P canonical blocks
          float* RZ0 = rzg + args.set_oRZ;
          float* RZ1 = RZ0 + args.rzg_tok;
          float* RG0 = rzg + args.set_oRG;
          float* RG1 = RG0 + args.rzg_tok;
          const int zc = p * mcur, zo = Pc * mcur + p * ovz - mcur;
          const int gc = p * ncur, go = Pc * ncur + p * ovg - ncur;
          // both paths per block of entries: the gathers of the column path
          // (U[a], V[b] where b changes) and of the row path (V[b]) go out
          // together, one shared-memory round trip per block
          float2 vk = make_float2(0.f, 0.f), accg = make_float2(0.f, 0.f), accz = make_float2(0.f, 0.f);
#pragma unroll
          for (int e0 = 0; e0 < KE; e0 += B) {
            const bool cg = NEED_U && e0 < ch.EG, cz = F && e0 < ch.EZ;
            if (!cg && !cz) continue;
            float2 ub[B], vb[B], vz[B];
            if (cg) {
#pragma unroll
              for (int e = 0; e < B; ++e) {
                ub[e] = U2p[ch.ga[e0 + e] & 0xFFFFu];
                if constexpr (C) {
                  const int ep = e0 + e - 1;
                  vb[e] = (ep < 0 || ch.gb[e0 + e] != ch.gb[ep]) ? V2p[ch.gb[e0 + e]] : make_float2(0.f, 0.f);
                }
              }
            }
            if (cz) {
#pragma unroll
              for (int e = 0; e < B; ++e) vz[e] = V2p[ch.zb[e0 + e] & 0xFFFFu];
            }
            if (cg) {
#pragma unroll
              for (int e = 0; e < B; ++e) {
                if constexpr (C) {
                  const int ep = e0 + e - 1;
                  if (ep < 0 || ch.gb[e0 + e] != ch.gb[ep]) vk = vb[e];
                  dc[e0 + e] = fmaf(ub[e].x, vk.x, fmaf(ub[e].y, vk.y, dc[e0 + e]));
                }
                if constexpr (D) {
                  accg.x = fmaf(ch.gc[e0 + e], ub[e].x, accg.x);
                  accg.y = fmaf(ch.gc[e0 + e], ub[e].y, accg.y);
                  const uint32_t sg = ch.ga[e0 + e] >> 16;
                  if (sg != FFB_NO_STORE) {
                    const int o = static_cast<int>(sg) + (static_cast<int>(sg) < ncur ? gc : go);
                    RG0[o] = accg.x;
                    RG1[o] = accg.y;
                    accg = make_float2(0.f, 0.f);
                  }
                }
              }
            }
            if (cz) {
#pragma unroll
              for (int e = 0; e < B; ++e) {
                accz.x = fmaf(ch.zc[e0 + e], vz[e].x, accz.x);
                accz.y = fmaf(ch.zc[e0 + e], vz[e].y, accz.y);
                const uint32_t sz = ch.zb[e0 + e] >> 16;
                if (sz != FFB_NO_STORE) {
                  const int o = static_cast<int>(sz) + (static_cast<int>(sz) < mcur ? zc : zo);
                  RZ0[o] = accz.x;
                  RZ1[o] = accz.y;
                  accz = make_float2(0.f, 0.f);
                }
              }
            }
          }
        }
        if constexpr (SYN) {
          if (nfix > 0) {
            // rows (columns) split between chunks: add the overflow pieces
            tc_spmm_bar();
            // one (item, pair) per thread
            const int tot = nfix * np;
            for (int w = st; w < tot; w += kTcSpmm) {
              const int p = w / nfix;
              const int i = w - p * nfix;
              const int4 it = fixc[i];
              const bool z = i < nfZ;
              const int M = z ? mcur : ncur, ov = z ? ovz : ovg;
              const int dst = p * M + tc_slot(it.x, M);
              const int src = Pc * M + p * ov - M + it.y;
#pragma unroll
              for (int k = 0; k < 2; ++k) {
                float* R = rzg + k * args.rzg_tok + (z ? args.set_oRZ : args.set_oRG);
                float sacc = R[dst];
                for (int c2 = 0; c2 < it.z; ++c2) sacc += R[src + c2];
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
      // analysis results of unit s -> V / U (float2: both tokens of a pair),
      // once every SpMM warp finished gathering from them and the MMAs
      // completed
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
          const int nq = args.m[tq.j].n, mq = args.m[tq.j].m;
          const int G = (aside == 0 ? nq : mq) / FFB_GROUP;
          const int P = pairs(tq.j);
          // this lane's pair and group
          const int pp = ar / G;
          const int g = ar - pp * G;
          const int64_t t0 = tok0(tq, u_begin + s);
          const bool two = tend(tq) - t0 > P + pp;  // token t0 + P + pp (slot 1) exists
          float2* dst = V2 + pp * (nq + mq) + (aside == 0 ? 0 : nq);
#pragma unroll
          for (int q8 = 0; q8 < 4; ++q8) {  // coefficients 8 q8 .. 8 q8 + 7: hi and lo in 16 columns
            float x0[16], x1[16];
            const uint32_t c0 = tmem + alane + (0 * 2 + aside) * 64 + 16 * q8;
            const uint32_t c1 = tmem + alane + (1 * 2 + aside) * 64 + 16 * q8;
            tmem_ld16x2(c0, c1, x0, x1);
            if (pp < P) {
#pragma unroll
              for (int j = 0; j < 4; ++j) {  // chunk q = 4 q8 + j: coefficients 2q, 2q + 1
                const int q = 4 * q8 + j;
                const float a0 = x0[2 * j] + x0[8 + 2 * j], a1 = x0[2 * j + 1] + x0[8 + 2 * j + 1];
                const float b0 = two ? x1[2 * j] + x1[8 + 2 * j] : 0.f, b1 = two ? x1[2 * j + 1] + x1[8 + 2 * j + 1] : 0.f;
                *reinterpret_cast<float4*>(dst + 32 * g + 2 * (q ^ (g & 7))) = make_float4(a0, b0, a1, b1);
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
          dc_flush<KE>(splan, dst, dc, st);
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
