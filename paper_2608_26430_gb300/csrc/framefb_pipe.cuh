// Pipelined bf16 tile kernel of libframefb: warp-specialised, one token per
// tile, three tiles in flight per CTA.  Included by framefb_cuda.cu after
// framefb_mma.cuh.
//
// Per tile the work is the same as in mma_tile_kernel (analysis V = X Phi_in,
// U = dY Phi_out on tensor cores; the coefficient SpMM Z = V C^T, G = U C and
// the dC products; synthesis Y += s Z Phi_out^T, dX += s G Phi_in^T, Sec. 3.1
// and the Lemma 1 gradient of Appendix A), but the three phases of
// consecutive tiles overlap.  In step s of the CTA's loop:
//   warps 0-3 (tensor warps)  analysis of tile s, then synthesis of tile s-2;
//   warps 4-7 (SpMM warps)    coefficient SpMM, dC and fix-up of tile s-1;
//   one SpMM thread           issues the bulk copies of tile s + S - 1.
// One CTA-wide barrier ends each step.  The fp32 coefficient buffers are
// double-buffered by tile parity: analysis of tile s writes V/U of set s&1
// while the SpMM reads V/U and writes RZ/RG of set (s-1)&1 and synthesis
// reads RZ/RG of set (s-2)&1 = s&1.  X/dY rows land in a ring of S staging
// buffers (one bulk copy per row, an mbarrier per buffer); Y/dX rows are
// read from global memory by the tensor warps at the start of the step and
// written after the synthesis of the same step.
//
// The plan is the one of the 256-thread kernels: SpMM thread t (0..127) owns
// the entry chunks of plan columns t and t + 128, held in registers, with
// its dC partial sums in registers too.  The two roles run separate loops
// so that their register working sets do not add up.
//
// Every wait on a bulk copy is bounded; a wait that gives up increments
// g_wait_timeouts, the CTA stops at the end of the step and lets the copies
// already issued land before it exits.
#pragma once
#include "framefb_mma.cuh"

namespace ffb {

constexpr int kPipeMmaWarps = 4;
constexpr int kPipeSpmm = kThreads - 32 * kPipeMmaWarps;  // SpMM threads
constexpr int kDescRing = 8;                              // tiles / matrices with a live descriptor
constexpr int kGroupWords = 32;                           // group bitmap words: d <= 32768

// Shared-memory map of the pipelined kernel (bytes, in LaunchK): staging
// ring at stg_in with stage stride stg_out and depth stage_out, two fp32
// sets at fbase (set_total floats each, layout set_o*), mbarriers at mbar;
// pad = the issuing thread.

__device__ __forceinline__ void spmm_bar() { asm volatile("bar.sync 1, %0;" ::"n"(kPipeSpmm) : "memory"); }

// Bulk copies of tile u (one token) of matrix M: the X row, then the dY row.
__device__ __forceinline__ void pipe_stage(const MatK& M, uint8_t* dst, uint64_t* bar, int64_t u, bool has_x,
                                           bool has_y) {
  const int64_t t0 = u - M.ubeg;
  const uint32_t bytes = (has_x ? 2u * M.n : 0u) + (has_y ? 2u * M.m : 0u);
  mbar_arrive_expect_tx(bar, bytes);
  if (has_x) bulk_load(dst, static_cast<const char*>(M.X) + t0 * M.ldx * 2, 2u * M.n, bar);
  if (has_y)
    bulk_load(dst + (has_x ? stage_rx(M) : 0), static_cast<const char*>(M.dY) + t0 * M.ldy * 2, 2u * M.m, bar);
}

// Coefficient SpMM of one register chunk for one token (fp32 slots):
//   RZ[run target] = sum over a run of equal rows of c V[b]      (forward)
//   RG[run target] = sum over a run of equal columns of c U[a]   (dX)
//   dc[e] += U[a] V[b]                                           (dC)
template <int MODE>
__device__ __forceinline__ void pipe_spmm(const Chunk<MODE, true, true>& ch, float (&dc)[kEreg], float* fs,
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
    float acc = 0.f;
    float vlast = 0.f;  // V[b] of the previous entry: reloaded only when the column changes
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

// dC partial sums of one plan column to the CTA's workspace slot.
__device__ __forceinline__ void pipe_flush(const uint8_t* plan, float* dst, const float (&dc)[kEreg], int col) {
  const FfbPlanHeader& h = hdr(plan);
  const int32_t* gq = table<int32_t>(plan, h.off_gq);
#pragma unroll
  for (int e = 0; e < kEreg; ++e) {
    if (e < h.EG) {
      const int32_t q = __ldg(gq + e * kThreads + col);
      if (q >= 0) dst[q] = dc[e];
    }
  }
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1) pipe_tile_kernel(const __grid_constant__ LaunchK args) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  constexpr bool NEED_V = F || C, NEED_U = D || C, SYN = F || D;
  constexpr int GB = 16;  // groups per 16-row MMA block (one token)
  constexpr int MW = kPipeMmaWarps;
  extern __shared__ __align__(128) uint8_t smem[];
  // descriptors of the matrices with a tile in flight: the q-th distinct
  // matrix of the CTA at q % kDescRing (index in mat_idx); tile i's q at
  // tile_mat[i % kDescRing].  At most S + 2 <= 6 tiles are live.
  __shared__ MatK mats_sm[kDescRing];
  __shared__ int32_t mat_idx[kDescRing];
  __shared__ int32_t tile_mat[kDescRing];
  // groups of each live matrix with support entries (bit per group), out side
  // [0] and in side [1]: the synthesis skips the others
  __shared__ uint32_t mat_bits[kDescRing][2][kGroupWords];
  const int S = args.stage_out;
  uint8_t* stg0 = smem + args.stg_in;
  float* fset0 = reinterpret_cast<float*>(smem + args.fbase);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + args.mbar);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  FfbTileLayout PL{};  // set layout (token-minor with one token: only the offsets matter)
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
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp < MW) {
    // ---------------- tensor warps: analysis of tile s, synthesis of tile s-2
    DFrags Df;
    {
      // both frames of every matrix are k = 16 DFT-group frames, whose group
      // block depends on k alone: one set of fragments serves the launch
      __syncthreads();  // descriptors of the first tiles written (prologue)
      const MatK& M0 = mats_sm[tile_mat[0] % kDescRing];
      Df.load(M0.fval_in, M0.rho_in, lane);
    }
    bool failed = false;
    for (int s = 0; s < count + 2; ++s) {
      // output rows of tile s-2, read now and used after the analysis
      const int i2 = s - 2;
      const bool syn = SYN && i2 >= 0;
      uint4 y0[2][2], y1[2][2];
      const MatK* M2 = nullptr;
      const uint32_t* bits2 = nullptr;
      float* fs2 = nullptr;
      int64_t t2 = 0;
      int bY = 0, nb2 = 0;
      auto sblk = [&](int b) {
        Blk k{};
        if (b < bY) {
          k.buf = fs2 + PL.oRZ, k.out = static_cast<__nv_bfloat16*>(M2->Y), k.ld = M2->ldy;
          k.mbits = bits2, k.G = M2->m / FFB_GROUP, k.b = b;
        } else if (b < nb2) {
          k.buf = fs2 + PL.oRG, k.out = static_cast<__nv_bfloat16*>(M2->dX), k.ld = M2->ldx;
          k.mbits = bits2 + kGroupWords, k.G = M2->n / FFB_GROUP, k.b = b - bY;
        }  // else: empty block (G = 0), nothing read or written
        return k;
      };
      if (syn) {
        const int q2 = tile_mat[i2 % kDescRing] % kDescRing;
        M2 = &mats_sm[q2];
        bits2 = mat_bits[q2][0];
        fs2 = fset0 + (i2 & 1) * PL.total;
        t2 = u_begin + i2 - M2->ubeg;
        bY = F ? (M2->m / FFB_GROUP + GB - 1) / GB : 0;
        nb2 = bY + (D ? (M2->n / FFB_GROUP + GB - 1) / GB : 0);
        if (warp < nb2) {
          const Blk k[2] = {sblk(warp), sblk(warp + MW)};
          syn_load<1, 2>(k, t2, 1, lane, y0);
        }
        if (warp + 2 * MW < nb2) {
          const Blk k[2] = {sblk(warp + 2 * MW), sblk(warp + 3 * MW)};
          syn_load<1, 2>(k, t2, 1, lane, y1);
        }
      }
      // analysis of tile s into set s & 1
      if (s < count) {
        if (!mbar_wait_bounded(bar + (s % S), static_cast<uint32_t>((s / S) & 1))) {
          failed = true;
        } else {
          const MatK& M0 = mats_sm[tile_mat[s % kDescRing] % kDescRing];
          const int Gn0 = M0.n / FFB_GROUP, Gm0 = M0.m / FFB_GROUP;
          float* fs0 = fset0 + (s & 1) * PL.total;
          const uint8_t* xs = stg0 + (s % S) * args.stg_out;
          const int rx = stage_rx(M0), ry = stage_ry(M0);
          const uint8_t* dys = xs + (NEED_V ? rx : 0);
          const int bV = NEED_V ? (Gn0 + GB - 1) / GB : 0;
          const int nb0 = bV + (NEED_U ? (Gm0 + GB - 1) / GB : 0);
          auto ablk = [&](int b) {
            Blk k{};
            if (b < bV) {
              k.stg = xs, k.rs = rx, k.buf = fs0 + PL.oV, k.G = Gn0, k.b = b;
            } else if (b < nb0) {
              k.stg = dys, k.rs = ry, k.buf = fs0 + PL.oU, k.G = Gm0, k.b = b - bV;
            }
            return k;
          };
          for (int b = warp; b < nb0; b += 2 * MW) {
            const Blk k[2] = {ablk(b), ablk(b + MW)};
            analysis_blocks<1, 2>(Df, k, 1, lane);
          }
        }
      }
      // synthesis of tile s-2 from set (s-2) & 1
      if (syn && !failed) {
        if (warp < nb2) {
          const Blk k[2] = {sblk(warp), sblk(warp + MW)};
          syn_compute<1, 2>(Df, k, t2, 1, M2->seff, lane, y0);
        }
        if (warp + 2 * MW < nb2) {
          const Blk k[2] = {sblk(warp + 2 * MW), sblk(warp + 3 * MW)};
          syn_compute<1, 2>(Df, k, t2, 1, M2->seff, lane, y1);
        }
        for (int b = warp + 4 * MW; b < nb2; b += 2 * MW) {
          const Blk k[2] = {sblk(b), sblk(b + MW)};
          synthesis_blocks<1, 2>(Df, k, t2, 1, M2->seff, lane);
        }
      }
      if (__syncthreads_or(failed)) break;
    }
  } else {
    // ---------------- SpMM warps: SpMM, dC and fix-up of tile s-1; copies
    const int st = tid - 32 * MW;
    const bool issuer = tid == args.pad;
    int jn = 0, jn_end = 0, jn_loaded = -1, nq = -1, issued = 0;
    auto issue = [&]() {
      const int64_t u = u_begin + issued;
      while (u >= jn_end) {
        ++jn;
        jn_end = args.m[jn].ubeg + args.m[jn].ntiles;
      }
      if (jn != jn_loaded) {
        ++nq;
        const int q = nq % kDescRing;
        mats_sm[q] = args.m[jn];
        mat_idx[q] = jn;
        jn_loaded = jn;
        if constexpr (SYN) {
          const uint8_t* plan = args.m[jn].plan;
          const FfbPlanHeader& h = hdr(plan);
          for (int side = 0; side < 2; ++side) {
            const uint32_t* mask = table<uint32_t>(plan, side ? h.off_gmask : h.off_zmask);
            const int G = side ? h.Gn : h.Gm;
            for (int w = 0; w < (G + 31) / 32; ++w) {
              uint32_t bits = 0;
#pragma unroll 8
              for (int i = 0; i < 32; ++i)
                if (32 * w + i < G && __ldg(mask + 32 * w + i) != 0u) bits |= 1u << i;
              mat_bits[q][side][w] = bits;
            }
          }
        }
      }
      tile_mat[issued % kDescRing] = nq;
      pipe_stage(mats_sm[nq % kDescRing], stg0 + (issued % S) * args.stg_out, bar + (issued % S), u, NEED_V,
                 NEED_U);
      ++issued;
    };
    if (issuer) {
      jn = matrix_of(args, 0, u_begin);
      jn_end = args.m[jn].ubeg + args.m[jn].ntiles;
      while (issued < S - 1 && issued < count) issue();
    }
    __syncthreads();  // descriptors of the first tiles written

    Chunk<MODE, true, true> ch0, ch1;
    float dc0[kEreg], dc1[kEreg];
#pragma unroll
    for (int e = 0; e < kEreg; ++e) dc0[e] = dc1[e] = 0.f;
    int cur = -1, cur_j = -1;  // descriptor sequence number and matrix index
    const uint8_t* splan = nullptr;
    int4* fixc = reinterpret_cast<int4*>(smem + args.fixc);  // fix-up items of the current matrix
    int nfZ = 0, nfix = 0;
    uint32_t zero_pending = 3u;  // fp32 sets still holding another matrix's row sums
    bool failed = false;
    int s = 0;
    for (; s < count + 2; ++s) {
      if (issuer && issued < count) issue();  // tile s + S - 1 into the buffer tile s - 1 used
      const int i1 = s - 1;
      if (i1 >= 0 && i1 < count) {
        const int q = tile_mat[i1 % kDescRing];
        const MatK& M1 = mats_sm[q % kDescRing];
        if (q != cur) {
          if constexpr (C) {
            if (cur >= 0) {
              float* dst = args.partial + static_cast<size_t>(blockIdx.x + cur_j) * args.stride;
              pipe_flush(splan, dst, dc0, st);
              pipe_flush(splan, dst, dc1, st + kPipeSpmm);
            }
          }
          cur = q;
          cur_j = mat_idx[q % kDescRing];
          splan = M1.plan;
          ch0.load(splan, M1.c_val, st);
          ch1.load(splan, M1.c_val, st + kPipeSpmm);
          if constexpr (SYN) {
            const FfbPlanHeader& h = hdr(splan);
            nfZ = F ? h.nfixZ : 0;
            nfix = nfZ + (D ? h.nfixG : 0);
            if (nfix > args.fixc_items) nfix = -nfix;  // over the cache: read from the plan
            for (int i = st; i < nfix; i += kPipeSpmm)
              fixc[i] = i < nfZ ? __ldg(table<int4>(splan, h.off_fixZ) + i)
                                : __ldg(table<int4>(splan, h.off_fixG) + (i - nfZ));
            spmm_bar();
          }
#pragma unroll
          for (int e = 0; e < kEreg; ++e) dc0[e] = dc1[e] = 0.f;
          zero_pending = 3u;
        }
        float* fs1 = fset0 + (i1 & 1) * PL.total;
        if constexpr (SYN) {
          if ((zero_pending >> (i1 & 1)) & 1u) {
            for (int x = PL.oRZ + st; x < PL.total; x += kPipeSpmm) fs1[x] = 0.f;
            zero_pending &= ~(1u << (i1 & 1));
            spmm_bar();
          }
        }
        pipe_spmm<MODE>(ch0, dc0, fs1, PL);
        pipe_spmm<MODE>(ch1, dc1, fs1, PL);
        if constexpr (SYN) {
          if (nfix > 0) {
            // rows (columns) split between chunks: add the overflow pieces
            spmm_bar();
            for (int i = st; i < nfix; i += kPipeSpmm) {
              const int4 it = fixc[i];
              const bool z = i < nfZ;
              float* R = fs1 + (z ? PL.oRZ : PL.oRG);
              const int dst = ffb_slot(it.x, z ? M1.m : M1.n);
              float sacc = R[dst];
              for (int c2 = 0; c2 < it.z; ++c2) sacc += R[it.y + c2];
              R[dst] = sacc;
            }
          } else if (nfix < 0) {
            spmm_bar();
            fixup<MODE, true, kPipeSpmm>(splan, PL, fs1, 1, 1, st);
          }
        }
      }
      if (__syncthreads_or(false)) {
        failed = true;
        break;
      }
    }
    if (failed) {
      // tiles [s, issued) were issued and not consumed: let them land
      if (issuer) {
        atomicAdd(&g_wait_timeouts, 1u);
        for (int i = s; i < issued; ++i) mbar_wait_bounded(bar + (i % S), static_cast<uint32_t>((i / S) & 1));
      }
      return;
    }
    if constexpr (C) {
      if (cur >= 0) {
        float* dst = args.partial + static_cast<size_t>(blockIdx.x + cur_j) * args.stride;
        pipe_flush(splan, dst, dc0, st);
        pipe_flush(splan, dst, dc1, st + kPipeSpmm);
      }
    }
  }
}

}  // namespace ffb
