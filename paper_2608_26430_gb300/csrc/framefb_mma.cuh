// bf16 tile kernel of libframefb: the group transforms on tensor cores, the
// activation rows staged in shared memory by bulk asynchronous copies (TMA).
// Included by framefb_cuda.cu after framefb_kernels.cuh.
//
// For a k = 16, k*rho = d frame the projection of a 32-coordinate group onto
// its 32 frame coefficients is one dense 32 x 32 block D (the realified
// DFT_16 / 4, Sec. 3.2 construction) applied to every (token, group) row:
//     analysis   V_row = X_row D          (per group of Phi_in, U likewise with Phi_out)
//     synthesis  dY_row = Z_row D^T       (Z = coefficient-SpMM row sums)
// Each is a [rows x 32] x [32 x 32] contraction, run with warp-level tf32
// MMA: data rows are the M side (16 rows per instruction group), D the N
// side, held as per-lane fragments for the whole matrix.  The DFT_16 matrix
// is symmetric, so its realified block satisfies D^T = S D S exactly, with
// S = diag(+1, -1, +1, -1, ...): synthesis runs on the same fragments as
// analysis, from S Z (the sign folded into the coefficient values) and with
// S applied to the result (the sign folded into the output scale).  bf16
// inputs are exact in tf32; D and the fp32 row sums are rounded to tf32.
// Index slots are permuted so that every lane reads or writes 16 contiguous
// bytes of a row: 8 consecutive indices 8t..8t+7 (t = lane % 4) for rows g
// and g + 8 (g = lane / 4) of the 16-row block.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "framefb_kernels.cuh"
#include "framefb_ptx.cuh"

namespace ffb {

// Counts bounded waits that gave up (a bulk copy never completed).
__device__ unsigned int g_wait_timeouts;

// One contiguous global -> shared bulk copy completing on `bar`.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void mma_tf32(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 4 x the group-0 block of a k = 16 frame: D4[w][x], coordinate w of the
// group, coefficient x = 2i + s <-> frame column i*rho + s.
__device__ __forceinline__ float d4(const float* val, int rho, int w, int x) {
  return 4.f * __ldg(val + 32 * ((x >> 1) * rho + (x & 1)) + w);
}

// Slot permutations (see file comment).  Analysis: K slot k = 16s + 8h + 2t + e
// reads coordinate 8t + 4s + 2h + e; N slot n = 8j + 2t + e writes
// coefficient 8t + 2j + e.  Synthesis: K slot k = 8s + 4h + t reads
// coefficient 8t + 2s + h; N slot n = 8j + 2t + e writes coordinate 8t + 2j + e.
__device__ __forceinline__ int an_coord(int k) { return 8 * ((k & 7) >> 1) + 4 * (k >> 4) + 2 * ((k >> 3) & 1) + (k & 1); }
__device__ __forceinline__ int nslot_pos(int n) { return 8 * ((n & 7) >> 1) + 2 * (n >> 3) + (n & 1); }
__device__ __forceinline__ int sy_coef(int k) { return 8 * (k & 3) + 2 * (k >> 3) + ((k >> 2) & 1); }

// B fragments of D (tf32) for m16n8k8: N-tile j, k-step s.  K slot
// 8s + 4h + t <-> row index 8t + 2s + h of D (sy_coef); N slot 8j + 2t + e
// <-> column index 8t + 2j + e (nslot_pos).
struct DFrags {
  uint32_t b[4][4][2];

  __device__ __forceinline__ void load(const float* val, int rho, int lane) {
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int x = nslot_pos(8 * j + g);
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        b[j][s][0] = to_tf32(d4(val, rho, sy_coef(8 * s + t), x));
        b[j][s][1] = to_tf32(d4(val, rho, sy_coef(8 * s + t + 4), x));
      }
    }
  }
};

// Pair p (0..15) of group r in a tile buffer: see ffb_slot.
__device__ __forceinline__ int pair_slot(int p, int r) { return p ^ (((p >> 3) & 1) << 1) ^ (r & 1) ^ ((r & 1) << 3); }

// One token per slot: 16-byte chunk position of chunk q (pairs 2q, 2q + 1;
// stored swapped in odd groups) of group r, see ffb_slot.
__device__ __forceinline__ int chunk_slot(int q, int r) { return q ^ ((q >> 2) & 1) ^ ((r & 1) << 2); }

__device__ __forceinline__ uint4 lds128(const uint8_t* p) { return *reinterpret_cast<const uint4*>(p); }

// y += seff * S d for 8 bf16 values (one 16-byte chunk of 8 consecutive
// coordinates starting at an even one), returns the new chunk.
__device__ __forceinline__ uint4 axpy_sd_bf16x8(uint4 y, const float (&d)[8], float seff) {
  uint32_t w[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float lo = fmaf(seff, d[2 * i], __uint_as_float(w[i] << 16));
    const float hi = fmaf(-seff, d[2 * i + 1], __uint_as_float(w[i] & 0xFFFF0000u));
    w[i] = pack_bf16(lo, hi);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ uint32_t word_of(const uint4& w, int s) {
  return s == 0 ? w.x : s == 1 ? w.y : s == 2 ? w.z : w.w;
}

// One 16-row MMA block.  T = 2: rows g and g + 8 of block b are tokens 0 and
// 1 of group 8b + g, and the fp32 buffer is token-minor (float2 per slot);
// T = 1: rows g and g + 8 are groups 16b + g and 16b + g + 8 of the single
// token.
struct Blk {
  const uint8_t* stg;  // staged bf16 token rows (stride rs bytes), or NULL
  float* buf;          // fp32 slot buffer (V / U written, RZ / RG read)
  __nv_bfloat16* out;  // synthesis: global output rows
  const uint32_t* mask;   // group masks of the plan (a group is skipped when its word is 0)
  const uint32_t* mbits;  // or, when set: one bit per group (0: skipped)
  int64_t ld;
  int rs, G, b;
};

__device__ __forceinline__ bool blk_group_on(const Blk& k, int grp) {
  return k.mbits ? ((k.mbits[grp >> 5] >> (grp & 31)) & 1u) != 0u : k.mask[grp] != 0u;
}

template <int T>
__device__ __forceinline__ void blk_rows(const Blk& k, int Tc, int lane, int& grp0, int& grp1, bool& v0, bool& v1,
                                         bool masked) {
  const int g = lane >> 2;
  grp0 = T == 2 ? 8 * k.b + g : 16 * k.b + g;
  grp1 = T == 2 ? grp0 : grp0 + 8;
  v0 = grp0 < k.G && (!masked || blk_group_on(k, grp0));
  v1 = T == 2 ? (v0 && Tc > 1) : (grp1 < k.G && (!masked || blk_group_on(k, grp1)));
}

// Analysis of NB blocks into V (or U): K slot 8s + 4h + t reads coordinate
// 8t + 2s + h, i.e. half h of bf16 word s of the lane's 16-byte chunk (a bf16
// value is exact as tf32); N slot 8j + 2t + e writes coefficient 8t + 2j + e.
// Tc = tokens present.
template <int T, int NB>
__device__ __forceinline__ void analysis_blocks(const DFrags& Df, const Blk (&k)[NB], int Tc, int lane) {
  const int t = lane & 3;
  int grp0[NB], grp1[NB];
  bool v0[NB], v1[NB];
  uint4 w0[NB], w1[NB];
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    blk_rows<T>(k[i], Tc, lane, grp0[i], grp1[i], v0[i], v1[i], false);
    w0[i] = v0[i] ? lds128(k[i].stg + grp0[i] * 64 + t * 16) : make_uint4(0, 0, 0, 0);
    w1[i] = v1[i] ? lds128(k[i].stg + (T == 2 ? k[i].rs : 0) + grp1[i] * 64 + t * 16) : make_uint4(0, 0, 0, 0);
  }
  float c[NB][4][4];
#pragma unroll
  for (int i = 0; i < NB; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) c[i][j][0] = c[i][j][1] = c[i][j][2] = c[i][j][3] = 0.f;
#pragma unroll
  for (int s = 0; s < 4; ++s) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int i = 0; i < NB; ++i) {
        const uint32_t x0 = word_of(w0[i], s), x1 = word_of(w1[i], s);
        mma_tf32(c[i][j], x0 << 16, x1 << 16, x0 & 0xFFFF0000u, x1 & 0xFFFF0000u, Df.b[j][s][0], Df.b[j][s][1]);
      }
  }
  // row g holds coefficients 8t + 2j + e in c[j][e], row g + 8 in c[j][2 + e]
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    if constexpr (T == 2) {
      if (v0[i]) {
        float* grow = k[i].buf + 64 * grp0[i];
#pragma unroll
        for (int j = 0; j < 4; ++j)  // pair 4t + j: (x, tok0), (x, tok1), (x + 1, tok0), (x + 1, tok1)
          *reinterpret_cast<float4*>(grow + 4 * pair_slot(4 * t + j, grp0[i])) =
              make_float4(c[i][j][0], c[i][j][2], c[i][j][1], c[i][j][3]);
      }
    } else {
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int grp = r ? grp1[i] : grp0[i];
        if (r ? v1[i] : v0[i]) {
          float* grow = k[i].buf + 32 * grp;
          const int o = 2 * r;
#pragma unroll
          for (int h = 0; h < 2; ++h) {  // float4 chunk q = 2t + h holds pairs 2q, 2q + 1
            const int q = 2 * t + h;
            const float4 lo =
                make_float4(c[i][2 * h][o], c[i][2 * h][o + 1], c[i][2 * h + 1][o], c[i][2 * h + 1][o + 1]);
            const float4 v = (grp & 1) ? make_float4(lo.z, lo.w, lo.x, lo.y) : lo;
            *reinterpret_cast<float4*>(grow + 4 * chunk_slot(q, grp)) = v;
          }
        }
      }
    }
  }
}

// Output rows of NB synthesis blocks (the two rows of each lane's 16-byte
// chunk), from staging or, when stg is NULL, from global memory.  Rows of
// groups outside the matrix or with an empty mask are not read.
template <int T, int NB>
__device__ __forceinline__ void syn_load(const Blk (&k)[NB], int64_t t0, int Tc, int lane, uint4 (&y)[NB][2]) {
  const int t = lane & 3;
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    int grp0, grp1;
    bool v0, v1;
    blk_rows<T>(k[i], Tc, lane, grp0, grp1, v0, v1, true);
    const int64_t row0 = t0, row1 = T == 2 ? t0 + 1 : t0;
    y[i][0] = y[i][1] = make_uint4(0, 0, 0, 0);
    if (v0)
      y[i][0] = k[i].stg ? lds128(k[i].stg + grp0 * 64 + t * 16)
                         : *reinterpret_cast<const uint4*>(k[i].out + row0 * k[i].ld + 32 * grp0 + 8 * t);
    if (v1)
      y[i][1] = k[i].stg ? lds128(k[i].stg + (T == 2 ? k[i].rs : 0) + grp1 * 64 + t * 16)
                         : *reinterpret_cast<const uint4*>(k[i].out + row1 * k[i].ld + 32 * grp1 + 8 * t);
  }
}

// Synthesis of NB blocks: S Z (the row sums, with the sign pattern S folded
// into the coefficient values) from the fp32 buffer in the analysis layout;
// y += seff * S (S Z) D^T-fragments = seff * Z D^T, with y the output rows
// read by syn_load, written to the global rows out + (t0 + token) * ld.
// K slot 8s + 4h + t reads coefficient 8t + 2s + h; N slot 8j + 2t + e writes
// coordinate 8t + 2j + e.  Groups whose mask is zero have no support entries
// and are left untouched.
template <int T, int NB>
__device__ __forceinline__ void syn_compute(const DFrags& Df, const Blk (&k)[NB], int64_t t0, int Tc, float seff,
                                            int lane, const uint4 (&y)[NB][2]) {
  const int t = lane & 3;
  int grp0[NB], grp1[NB];
  bool v0[NB], v1[NB];
  // A fragment of k-step s: (row g, coef 8t + 2s), (row g + 8, same), (row g, +1), (row g + 8, +1)
  float4 a[NB][4];
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    blk_rows<T>(k[i], Tc, lane, grp0[i], grp1[i], v0[i], v1[i], true);
    if constexpr (T == 2) {
      const float* grow = k[i].buf + 64 * grp0[i];
#pragma unroll
      for (int s = 0; s < 4; ++s)
        a[i][s] = v0[i] ? *reinterpret_cast<const float4*>(grow + 4 * pair_slot(4 * t + s, grp0[i]))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
    } else {
      float z[2][8];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int grp = r ? grp1[i] : grp0[i];
        const bool v = r ? v1[i] : v0[i];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int q = 2 * t + h;
          float4 f = v ? *reinterpret_cast<const float4*>(k[i].buf + 32 * grp + 4 * chunk_slot(q, grp))
                       : make_float4(0.f, 0.f, 0.f, 0.f);
          if (grp & 1) f = make_float4(f.z, f.w, f.x, f.y);
          z[r][4 * h] = f.x;
          z[r][4 * h + 1] = f.y;
          z[r][4 * h + 2] = f.z;
          z[r][4 * h + 3] = f.w;
        }
      }
#pragma unroll
      for (int s = 0; s < 4; ++s) a[i][s] = make_float4(z[0][2 * s], z[1][2 * s], z[0][2 * s + 1], z[1][2 * s + 1]);
    }
  }
  float c[NB][4][4];
#pragma unroll
  for (int i = 0; i < NB; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) c[i][j][0] = c[i][j][1] = c[i][j][2] = c[i][j][3] = 0.f;
#pragma unroll
  for (int s = 0; s < 4; ++s) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int i = 0; i < NB; ++i)
        mma_tf32(c[i][j], __float_as_uint(a[i][s].x), __float_as_uint(a[i][s].y), __float_as_uint(a[i][s].z),
                 __float_as_uint(a[i][s].w), Df.b[j][s][0], Df.b[j][s][1]);
  }
  // N slot 8j + 2t + e holds coordinate 8t + 2j + e
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    const int64_t row0 = t0, row1 = T == 2 ? t0 + 1 : t0;
    if (v0[i]) {
      const float d[8] = {c[i][0][0], c[i][0][1], c[i][1][0], c[i][1][1], c[i][2][0], c[i][2][1], c[i][3][0], c[i][3][1]};
      *reinterpret_cast<uint4*>(k[i].out + row0 * k[i].ld + 32 * grp0[i] + 8 * t) = axpy_sd_bf16x8(y[i][0], d, seff);
    }
    if (v1[i]) {
      const float d[8] = {c[i][0][2], c[i][0][3], c[i][1][2], c[i][1][3], c[i][2][2], c[i][2][3], c[i][3][2], c[i][3][3]};
      *reinterpret_cast<uint4*>(k[i].out + row1 * k[i].ld + 32 * grp1[i] + 8 * t) = axpy_sd_bf16x8(y[i][1], d, seff);
    }
  }
}

template <int T, int NB>
__device__ __forceinline__ void synthesis_blocks(const DFrags& Df, const Blk (&k)[NB], int64_t t0, int Tc, float seff,
                                                 int lane) {
  uint4 y[NB][2];
  syn_load<T, NB>(k, t0, Tc, lane, y);
  syn_compute<T, NB>(Df, k, t0, Tc, seff, lane, y);
}

// Staged row strides (bytes) of a matrix: n-wide rows and m-wide rows.
__device__ __forceinline__ int stage_rx(const MatK& M) { return ((2 * M.n + 127) / 128) * 128; }
__device__ __forceinline__ int stage_ry(const MatK& M) { return ((2 * M.m + 127) / 128) * 128; }

// Issue the bulk copies of the rows of unit u (tokens [t0, t0 + Tc) of
// matrix M): the analysis inputs (X then dY, at stg_in) or the synthesis
// outputs (Y then dX, at stg_out).  Called by the 32 lanes of one warp: lane
// 0 posts the byte count, then each lane issues at most one row copy.
template <int MODE, bool OUTPUTS>
__device__ __forceinline__ void stage_rows(const MatK& M, const LaunchK& args, uint8_t* smem, uint64_t* bar,
                                           int64_t u, int lane) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  const int64_t t0 = static_cast<int64_t>(u - M.ubeg) * M.T;
  const int64_t left = static_cast<int64_t>(M.N) - t0;
  const int Tc = static_cast<int>(left < M.T ? left : M.T);
  const int n = M.n, m = M.m;
  const int rx = stage_rx(M), ry = stage_ry(M);
  const bool first_x = OUTPUTS ? false : (F || C);  // X (inputs) comes first
  const bool has_x = OUTPUTS ? D : (F || C);        // n-wide rows: X or dX
  const bool has_y = OUTPUTS ? F : (D || C);        // m-wide rows: dY or Y
  uint8_t* base = smem + (OUTPUTS ? args.stg_out : args.stg_in);
  // inputs: X at 0, dY after T rows of X; outputs: Y at 0, dX after T rows of Y
  uint8_t* xs = base + (first_x ? 0 : (has_y ? M.T * ry : 0));
  uint8_t* ys = base + (first_x ? M.T * rx : 0);
  if (lane == 0) {
    const uint32_t bytes = static_cast<uint32_t>(Tc) * ((has_x ? 2u * n : 0u) + (has_y ? 2u * m : 0u));
    mbar_arrive_expect_tx(bar, bytes);
  }
  __syncwarp();
  const int nx = has_x ? Tc : 0, ny = has_y ? Tc : 0;
  if (lane < nx) {
    const char* src = static_cast<const char*>(OUTPUTS ? M.dX : M.X) + (t0 + lane) * M.ldx * 2;
    bulk_load(xs + lane * rx, src, 2u * n, bar);
  } else if (lane < nx + ny) {
    const int t = lane - nx;
    const char* src = static_cast<const char*>(OUTPUTS ? M.Y : M.dY) + (t0 + t) * M.ldy * 2;
    bulk_load(ys + t * ry, src, 2u * m, bar);
  }
}

template <typename Args>
__device__ __forceinline__ int matrix_of(const Args& args, int j, int64_t u) {
  while (u >= args.m[j].ubeg + args.m[j].ntiles) ++j;
  return j;
}

// ---------------------------------------------------------------------------
// bf16 tile kernel.  Persistent CTAs walk a contiguous range of units
// (matrix, tile of T tokens, T = 1 or 2), matrix-major.  Per tile:
//   A  analysis on tensor cores from the staged X / dY rows into V / U;
//      then the X / dY rows of the next tile start streaming in;
//   B1 sparse phase (token-minor buffers: both tokens per access);
//   B2 fix-up;
//   B3 synthesis on tensor cores; Y / dX rows (staged one phase earlier)
//      read-modify-written to global memory; then the next tile's Y / dX
//      rows start streaming in.
// All waits on bulk copies are bounded; a wait that gives up increments
// g_wait_timeouts and the CTA stops after letting its copies land.
// ---------------------------------------------------------------------------
template <int MODE, bool REG, int T>
__global__ void __launch_bounds__(kThreads, 1) mma_tile_kernel(const __grid_constant__ LaunchK args) {
  static_assert(T == 1 || T == 2, "tile of one or two tokens");
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  constexpr bool NEED_V = F || C, NEED_U = D || C, SYN = F || D;
  constexpr int GB = T == 2 ? 8 : 16;  // groups per 16-row MMA block
  extern __shared__ __align__(128) uint8_t smem[];
  // descriptors of the current matrix [0] and of the matrix being staged [1]:
  // kernel-parameter reads with a runtime index miss the constant cache
  __shared__ MatK mat_sm[2];
  float* fsm = reinterpret_cast<float*>(smem + args.fbase);
  uint64_t* bar_in = reinterpret_cast<uint64_t*>(smem + args.mbar);
  uint64_t* bar_out = bar_in + 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  const int64_t units = args.total_units;
  const int64_t u_begin = (static_cast<int64_t>(blockIdx.x) * units) / gridDim.x;
  const int64_t u_end = (static_cast<int64_t>(blockIdx.x + 1) * units) / gridDim.x;
  if (u_begin >= u_end) return;

  if (tid == 0) {
    mbar_init(bar_in, 1);
    mbar_init(bar_out, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  int j = matrix_of(args, 0, u_begin);
  if (warp == 0) {
    if (lane == 0) mat_sm[1] = args.m[j];
    __syncwarp();
    stage_rows<MODE, false>(mat_sm[1], args, smem, bar_in, u_begin, lane);
    if constexpr (SYN)
      if (args.stage_out) stage_rows<MODE, true>(mat_sm[1], args, smem, bar_out, u_begin, lane);
  }
  uint32_t ph_in = 0, ph_out = 0;
  int jn = j;  // matrix of the next unit to stage (warp 0)

  Chunk<MODE, REG, true> ch;
  DFrags Df;
  int cur = -1;
  const uint8_t* plan = nullptr;
  FfbTileLayout L{};
  int Gn = 0, Gm = 0;
  bool failed = false;

  for (int64_t u = u_begin; u < u_end; ++u) {
    if (cur < 0 || u >= mat_sm[0].ubeg + mat_sm[0].ntiles) j = matrix_of(args, j, u);
    const MatK& M = mat_sm[0];
    if (j != cur) {
      __syncthreads();  // every thread is done with the previous matrix's descriptor and buffers
      if (cur >= 0) ch.flush(plan, args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride, L, fsm, tid);
      if (tid == 0) mat_sm[0] = args.m[j];
      __syncthreads();
      cur = j;
      plan = M.plan;
      const FfbPlanHeader& h = hdr(plan);
      Gn = h.Gn;
      Gm = h.Gm;
      FfbPlanHeader hc = h;
      L = ffb_tile_layout(hc, MODE, T, C);
      // both frames of a matrix are k = 16 DFT-group frames, whose group block
      // depends on k alone: one set of fragments (from Phi_in) serves both sides
      Df.load(M.fval_in, M.rho_in, lane);
      for (int i = tid; i < L.total - L.oRZ; i += kThreads) fsm[L.oRZ + i] = 0.f;
      ch.load(plan, M.c_val, tid);
      __syncthreads();
    }
    const int64_t t0 = static_cast<int64_t>(u - M.ubeg) * T;
    const int64_t left = static_cast<int64_t>(M.N) - t0;
    const int Tc = static_cast<int>(left < T ? left : T);

    // ---- A: analysis ------------------------------------------------------
    failed = !mbar_wait_bounded(bar_in, ph_in);
    if (__syncthreads_or(failed)) break;
    ph_in ^= 1u;
    {
      const int rx = stage_rx(M), ry = stage_ry(M);
      const uint8_t* xs = smem + args.stg_in;
      const uint8_t* dys = smem + args.stg_in + (NEED_V ? T * rx : 0);
      const int bV = NEED_V ? (Gn + GB - 1) / GB : 0, bU = NEED_U ? (Gm + GB - 1) / GB : 0;
      auto blk = [&](int b) {
        Blk k{};
        if (b < bV) {
          k.stg = xs, k.rs = rx, k.buf = fsm + L.oV, k.G = Gn, k.b = b;
        } else {
          k.stg = dys, k.rs = ry, k.buf = fsm + L.oU, k.G = Gm, k.b = b - bV;
        }
        return k;
      };
      constexpr int W = kThreads / 32;
      int b = warp;
      for (; b + W < bV + bU; b += 2 * W) {
        const Blk k[2] = {blk(b), blk(b + W)};
        analysis_blocks<T, 2>(Df, k, Tc, lane);
      }
      if (b < bV + bU) {
        const Blk k[1] = {blk(b)};
        analysis_blocks<T, 1>(Df, k, Tc, lane);
      }
    }
    __syncthreads();
    if (warp == 0 && u + 1 < u_end) {
      const int jprev = jn;
      jn = matrix_of(args, jn, u + 1);
      if (jn != jprev) {
        if (lane == 0) mat_sm[1] = args.m[jn];
        __syncwarp();
      }
      stage_rows<MODE, false>(mat_sm[1], args, smem, bar_in, u + 1, lane);
    }

    // ---- B1 / B2: sparse phase and fix-up -----------------------------------
    // tokens absent from a ragged tile have zero V / U (analysis wrote zeros),
    // so the whole T-token layout is processed
    ch.template sparse_tt<T, true>(plan, M.c_val, tid, L, fsm);
    if constexpr (SYN) {
      if (fix_count(plan, MODE) > 0) {
        __syncthreads();
        fixup<MODE, true>(plan, L, fsm, T, Tc, tid);
      }
    }
    __syncthreads();

    // ---- B3: synthesis --------------------------------------------------------
    if constexpr (SYN) {
      if (args.stage_out) {
        failed = !mbar_wait_bounded(bar_out, ph_out);
        if (__syncthreads_or(failed)) break;
        ph_out ^= 1u;
      }
      const int rx = stage_rx(M), ry = stage_ry(M);
      const uint8_t* ys = args.stage_out ? smem + args.stg_out : nullptr;
      const uint8_t* dxs = args.stage_out ? smem + args.stg_out + (F ? T * ry : 0) : nullptr;
      const uint32_t* zmask = table<uint32_t>(plan, hdr(plan).off_zmask);
      const uint32_t* gmask = table<uint32_t>(plan, hdr(plan).off_gmask);
      const int bY = F ? (Gm + GB - 1) / GB : 0, bX = D ? (Gn + GB - 1) / GB : 0;
      auto blk = [&](int b) {
        Blk k{};
        if (b < bY) {
          k.stg = ys, k.rs = ry, k.buf = fsm + L.oRZ, k.out = static_cast<__nv_bfloat16*>(M.Y), k.ld = M.ldy;
          k.mask = zmask, k.G = Gm, k.b = b;
        } else {
          k.stg = dxs, k.rs = rx, k.buf = fsm + L.oRG, k.out = static_cast<__nv_bfloat16*>(M.dX), k.ld = M.ldx;
          k.mask = gmask, k.G = Gn, k.b = b - bY;
        }
        return k;
      };
      constexpr int W = kThreads / 32;
      int b = warp;
      for (; b + W < bY + bX; b += 2 * W) {
        const Blk k[2] = {blk(b), blk(b + W)};
        synthesis_blocks<T, 2>(Df, k, t0, Tc, M.seff, lane);
      }
      if (b < bY + bX) {
        const Blk k[1] = {blk(b)};
        synthesis_blocks<T, 1>(Df, k, t0, Tc, M.seff, lane);
      }
      __syncthreads();
      if (warp == 0 && u + 1 < u_end && args.stage_out)
        stage_rows<MODE, true>(mat_sm[1], args, smem, bar_out, u + 1, lane);
    }
  }
  if (failed) {
    // let copies already queued land before the shared memory is released
    if (tid == 0) {
      atomicAdd(&g_wait_timeouts, 1u);
      mbar_wait_bounded(bar_in, ph_in);
      if constexpr (SYN)
        if (args.stage_out) mbar_wait_bounded(bar_out, ph_out);
    }
    __syncthreads();
    return;
  }
  if (cur >= 0) ch.flush(plan, args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride, L, fsm, tid);
}

}  // namespace ffb
