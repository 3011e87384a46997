// Device code of libframefb: the batched tile kernel (S3-S6), the dC
// reduction and the merge kernel (S7).  Included by framefb_cuda.cu only.
//
// The frames of the GPU path have k = 16 and k*rho = d (every config of the
// paper's calibration k*rho = n, Sec. 4).  Their synthesis matrix is then a
// column permutation of blockdiag(D, ..., D), D the 32 x 32 realified DFT_16
// block scaled by 1/4 (Sec. 3.2 construction, appendix: Spectral Tetris rows
// of 16 ones, modulation by 16th roots of unity, realification).  So the
// projection onto frame coefficients of a 32-coordinate group is an inverse
// DFT_16 of its 16 complex values (x_{2j} + i x_{2j+1}) and the synthesis is a
// forward DFT_16; both run here as an exact radix-4 FFT in fp32 registers.
// The 1/4 of each side is folded into one scale s/16 applied at the end.
// The twiddles are read from the caller's device frame (column rho: subspace
// 1 of group 0 holds omega^j / 4 on coordinates 2j, 2j+1).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "framefb.h"
#include "plan_layout.h"

namespace ffb {

constexpr int kThreads = FRAMEFB_THREADS;
constexpr int kTmax = 4;     // tokens per tile
constexpr int kEreg = 16;    // chunk length held in registers
constexpr int kMaxMats = 256;

enum { MODE_F = 1, MODE_D = 2, MODE_C = 4 };

struct MatK {
  const void* X;
  void* dX;
  const void* dY;
  void* Y;
  const uint8_t* plan;
  const float* c_val;
  const float* tw_in;   // 32 floats: group-0 block of column rho of Phi_in
  const float* tw_out;  // same for Phi_out
  int64_t ldx, ldy;
  int32_t N, T, ubeg, ntiles;
  float seff;           // s / 16
  int32_t pad;
};

struct LaunchK {
  int32_t nmats, total_units, stride, pad;
  float* partial;       // [(grid + nmats) * stride] dC partial sums, slot = cta + matrix
  MatK m[kMaxMats];
};

struct ReduceMat {
  float* dC;
  int32_t ubeg, ntiles, nnz;
  float seff;
};

struct ReduceK {
  int32_t nmats, total_units, grid, stride;
  const float* partial;
  ReduceMat m[kMaxMats];
};

struct MergeK {
  const void* W0;
  void* Wout;
  const uint8_t* plan;
  const float* c_vals;
  const float* fin_val;
  const float* fout_val;
  int64_t ldw;
  int32_t m, n, rho_in, rho_out, nnz, T;
  float seff;
};

// ---------------------------------------------------------------------------
// radix-4 FFT_16 in registers.  SIGN = +1: sum_j x_j w^{+jk} (analysis,
// inverse DFT); SIGN = -1: forward DFT (synthesis).  Output k lands in slot
// 4 (k mod 4) + k / 4.
// ---------------------------------------------------------------------------
struct Tw {
  float c1, s1, c2, s2, c3, s3, c6, s6, c9, s9;  // omega^m = c_m + i s_m, omega = e^{2 pi i/16}
};

__device__ __forceinline__ Tw load_tw(const float* v) {
  Tw w;
  w.c1 = 4.f * __ldg(v + 2);
  w.s1 = -4.f * __ldg(v + 3);
  w.c2 = 4.f * __ldg(v + 4);
  w.s2 = -4.f * __ldg(v + 5);
  w.c3 = 4.f * __ldg(v + 6);
  w.s3 = -4.f * __ldg(v + 7);
  w.c6 = 4.f * __ldg(v + 12);
  w.s6 = -4.f * __ldg(v + 13);
  w.c9 = 4.f * __ldg(v + 18);
  w.s9 = -4.f * __ldg(v + 19);
  return w;
}

template <int SIGN>
__device__ __forceinline__ void cmul(float& xr, float& xi, float c, float s) {
  const float ss = SIGN > 0 ? s : -s;
  const float r = fmaf(xr, c, -xi * ss);
  const float i = fmaf(xr, ss, xi * c);
  xr = r;
  xi = i;
}

template <int SIGN>
__device__ __forceinline__ void dft4(float& ar, float& ai, float& br, float& bi, float& cr, float& ci, float& dr,
                                     float& di) {
  const float t0r = ar + cr, t0i = ai + ci;
  const float t1r = ar - cr, t1i = ai - ci;
  const float t2r = br + dr, t2i = bi + di;
  const float t3r = br - dr, t3i = bi - di;
  // (b - d) * W4, W4 = SIGN * i
  const float ur = SIGN > 0 ? -t3i : t3i;
  const float ui = SIGN > 0 ? t3r : -t3r;
  ar = t0r + t2r;
  ai = t0i + t2i;
  cr = t0r - t2r;
  ci = t0i - t2i;
  br = t1r + ur;
  bi = t1i + ui;
  dr = t1r - ur;
  di = t1i - ui;
}

template <int SIGN>
__device__ __forceinline__ void fft16(float (&xr)[16], float (&xi)[16], const Tw& w) {
#pragma unroll
  for (int n2 = 0; n2 < 4; ++n2)
    dft4<SIGN>(xr[n2], xi[n2], xr[4 + n2], xi[4 + n2], xr[8 + n2], xi[8 + n2], xr[12 + n2], xi[12 + n2]);
  // slot 4 k1 + n2 holds y[n2][k1]; multiply by W^{n2 k1}
  cmul<SIGN>(xr[5], xi[5], w.c1, w.s1);
  cmul<SIGN>(xr[9], xi[9], w.c2, w.s2);
  cmul<SIGN>(xr[13], xi[13], w.c3, w.s3);
  cmul<SIGN>(xr[6], xi[6], w.c2, w.s2);
  {  // W^4 = SIGN * i
    const float r = xr[10], i = xi[10];
    xr[10] = SIGN > 0 ? -i : i;
    xi[10] = SIGN > 0 ? r : -r;
  }
  cmul<SIGN>(xr[14], xi[14], w.c6, w.s6);
  cmul<SIGN>(xr[7], xi[7], w.c3, w.s3);
  cmul<SIGN>(xr[11], xi[11], w.c6, w.s6);
  cmul<SIGN>(xr[15], xi[15], w.c9, w.s9);
#pragma unroll
  for (int k1 = 0; k1 < 4; ++k1)
    dft4<SIGN>(xr[4 * k1], xi[4 * k1], xr[4 * k1 + 1], xi[4 * k1 + 1], xr[4 * k1 + 2], xi[4 * k1 + 2],
               xr[4 * k1 + 3], xi[4 * k1 + 3]);
}

__device__ __forceinline__ constexpr int slot_of(int k) { return 4 * (k & 3) + (k >> 2); }

// ---------------------------------------------------------------------------
// 32-element row segments of activations: load as 16 complex values
// (x_{2j}, x_{2j+1}), and read-modify-write y += seff * delta.
// ---------------------------------------------------------------------------
template <typename Elem>
struct Seg;

template <>
struct Seg<__nv_bfloat16> {
  uint4 q[4];
  __device__ __forceinline__ void load_stream(const void* p) {
    const uint4* s = reinterpret_cast<const uint4*>(p);
#pragma unroll
    for (int i = 0; i < 4; ++i) q[i] = __ldcs(s + i);
  }
  __device__ __forceinline__ void load(const void* p) {
    const uint4* s = reinterpret_cast<const uint4*>(p);
#pragma unroll
    for (int i = 0; i < 4; ++i) q[i] = s[i];
  }
  __device__ __forceinline__ uint32_t word(int j) const {
    const uint4& v = q[j >> 2];
    return (j & 3) == 0 ? v.x : (j & 3) == 1 ? v.y : (j & 3) == 2 ? v.z : v.w;
  }
  __device__ __forceinline__ void unpack(float (&xr)[16], float (&xi)[16]) const {
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const uint32_t w = word(j);
      xr[j] = __uint_as_float(w << 16);
      xi[j] = __uint_as_float(w & 0xFFFF0000u);
    }
  }
  // y_{2j} += seff * dr[slot_of(j)], y_{2j+1} += seff * di[slot_of(j)], stored to p
  __device__ __forceinline__ void add_store(void* p, const float (&dr)[16], const float (&di)[16], float seff) {
    uint32_t out[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const uint32_t w = word(j);
      const float lo = fmaf(seff, dr[slot_of(j)], __uint_as_float(w << 16));
      const float hi = fmaf(seff, di[slot_of(j)], __uint_as_float(w & 0xFFFF0000u));
      const __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
      out[j] = *reinterpret_cast<const uint32_t*>(&b);
    }
    uint4* d = reinterpret_cast<uint4*>(p);
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] = make_uint4(out[4 * i], out[4 * i + 1], out[4 * i + 2], out[4 * i + 3]);
  }
};

template <>
struct Seg<float> {
  float4 q[8];
  __device__ __forceinline__ void load_stream(const void* p) {
    const float4* s = reinterpret_cast<const float4*>(p);
#pragma unroll
    for (int i = 0; i < 8; ++i) q[i] = __ldcs(s + i);
  }
  __device__ __forceinline__ void load(const void* p) {
    const float4* s = reinterpret_cast<const float4*>(p);
#pragma unroll
    for (int i = 0; i < 8; ++i) q[i] = s[i];
  }
  __device__ __forceinline__ float re(int j) const { return (j & 1) ? q[j >> 1].z : q[j >> 1].x; }
  __device__ __forceinline__ float im(int j) const { return (j & 1) ? q[j >> 1].w : q[j >> 1].y; }
  __device__ __forceinline__ void unpack(float (&xr)[16], float (&xi)[16]) const {
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      xr[j] = re(j);
      xi[j] = im(j);
    }
  }
  __device__ __forceinline__ void add_store(void* p, const float (&dr)[16], const float (&di)[16], float seff) {
    float4* d = reinterpret_cast<float4*>(p);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int j0 = 2 * i, j1 = 2 * i + 1;
      d[i] = make_float4(fmaf(seff, dr[slot_of(j0)], re(j0)), fmaf(seff, di[slot_of(j0)], im(j0)),
                         fmaf(seff, dr[slot_of(j1)], re(j1)), fmaf(seff, di[slot_of(j1)], im(j1)));
    }
  }
};

// Store the 32 coefficients of one group (analysis output, slot order) into a
// swizzled shared-memory token row: chunk c = (V_{2c}, V_{2c+1}) complex.
__device__ __forceinline__ void store_group(float* row, int g, const float (&xr)[16], const float (&xi)[16]) {
  float* base = row + 32 * g;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int p0 = slot_of(2 * c), p1 = slot_of(2 * c + 1);
    *reinterpret_cast<float4*>(base + 4 * (c ^ (g & 7))) = make_float4(xr[p0], xi[p0], xr[p1], xi[p1]);
  }
}

// Read the 32 row sums of one group back in natural complex order.
__device__ __forceinline__ void load_group(const float* row, int g, float (&xr)[16], float (&xi)[16]) {
  const float* base = row + 32 * g;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const float4 v = *reinterpret_cast<const float4*>(base + 4 * (c ^ (g & 7)));
    xr[2 * c] = v.x;
    xi[2 * c] = v.y;
    xr[2 * c + 1] = v.z;
    xi[2 * c + 1] = v.w;
  }
}

__device__ __forceinline__ const FfbPlanHeader& hdr(const uint8_t* plan) {
  return *reinterpret_cast<const FfbPlanHeader*>(plan);
}
template <typename T>
__device__ __forceinline__ const T* table(const uint8_t* plan, int32_t off) {
  return reinterpret_cast<const T*>(plan + off);
}

__device__ __forceinline__ int32_t cta_of_unit(int64_t u, int64_t grid, int64_t units) {
  return static_cast<int32_t>(((u + 1) * grid - 1) / units);
}

// Write this thread's dC partial sums of one matrix to its workspace slot.
template <bool C, bool REG, int E>
__device__ __forceinline__ void flush_dc(const uint8_t* plan, int EG, float* dst, const float (&dc)[E],
                                         const float* dcs, int tid) {
  if constexpr (C) {
    const int32_t* gq = table<int32_t>(plan, hdr(plan).off_gq);
    if constexpr (REG) {
#pragma unroll
      for (int e = 0; e < E; ++e) {
        if (e < EG) {
          const int32_t q = __ldg(gq + e * kThreads + tid);
          if (q >= 0) dst[q] = dc[e];
        }
      }
    } else {
      for (int e = 0; e < EG; ++e) {
        const int32_t q = __ldg(gq + e * kThreads + tid);
        if (q >= 0) dst[q] = dcs[e * kThreads + tid];
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Tile kernel.  Persistent CTAs walk a contiguous range of units (matrix,
// tile of T tokens), matrix-major.  Per tile:
//   A  analysis: V = X Phi_in, U = dY Phi_out for every group touched by the
//      support (FFT_16 per token and group), into shared memory;
//   B1 coefficient SpMM by balanced chunks: row sums of c V[b] for Y (RZ),
//      column sums of c U[a] for dX (RG), and dC += U[a] V[b];
//   B2 fix-up of rows/columns whose entries were split between chunks;
//   B3 synthesis: FFT_16 of RZ / RG per group and y += (s/16) * result.
// dC accumulates over the CTA's tiles of a matrix and is written to the
// workspace slot (cta + matrix) when the CTA leaves the matrix.
// ---------------------------------------------------------------------------
template <typename Elem, int MODE, bool REG>
__global__ void __launch_bounds__(kThreads, 1) tile_kernel(const __grid_constant__ LaunchK args) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  constexpr bool NEED_V = F || C, NEED_U = D || C;
  constexpr int E = REG ? kEreg : 1;
  constexpr size_t ELEM = sizeof(Elem);
  extern __shared__ float4 smem4[];
  float* smem = reinterpret_cast<float*>(smem4);
  const int tid = threadIdx.x;

  const int64_t units = args.total_units;
  const int64_t u_begin = (static_cast<int64_t>(blockIdx.x) * units) / gridDim.x;
  const int64_t u_end = (static_cast<int64_t>(blockIdx.x + 1) * units) / gridDim.x;
  if (u_begin >= u_end) return;

  // register-resident chunk (REG) -- by row for Y, by column for dX / dC
  uint32_t zb[E], ga[E], gb[E];
  float zc[E], gc[E], dc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    zb[e] = ga[e] = gb[e] = 0;
    zc[e] = gc[e] = dc[e] = 0.f;
  }

  int j = 0;
  while (j + 1 < args.nmats && u_begin >= args.m[j].ubeg + args.m[j].ntiles) ++j;
  int cur = -1;
  const uint8_t* plan = nullptr;
  FfbTileLayout L{};
  Tw tw_in{}, tw_out{};
  int EZ = 0, EG = 0, Gn = 0, Gm = 0, nfixZ = 0, nfixG = 0, T = 1;
  float* dcs = nullptr;

  for (int64_t u = u_begin; u < u_end; ++u) {
    while (u >= args.m[j].ubeg + args.m[j].ntiles) ++j;
    const MatK& M = args.m[j];
    if (j != cur) {
      if (cur >= 0) flush_dc<C, REG, E>(plan, EG, args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride, dc, dcs, tid);
      cur = j;
      plan = M.plan;
      const FfbPlanHeader& h = hdr(plan);
      EZ = h.EZ;
      EG = h.EG;
      Gn = h.Gn;
      Gm = h.Gm;
      nfixZ = h.nfixZ;
      nfixG = h.nfixG;
      T = M.T;
      FfbPlanHeader hc = h;
      L = ffb_tile_layout(hc, MODE, T, C && !REG);
      tw_in = load_tw(M.tw_in);
      tw_out = load_tw(M.tw_out);
      __syncthreads();  // every thread is done with the previous matrix's shared memory
      for (int i = tid; i < L.total - L.oRZ; i += kThreads) smem[L.oRZ + i] = 0.f;
      dcs = smem + L.oDC;
      if constexpr (REG) {
        const int32_t* tzb = table<int32_t>(plan, h.off_zb);
        const int32_t* tzq = table<int32_t>(plan, h.off_zq);
        const int32_t* tga = table<int32_t>(plan, h.off_ga);
        const int32_t* tgb = table<int32_t>(plan, h.off_gb);
        const int32_t* tgq = table<int32_t>(plan, h.off_gq);
#pragma unroll
        for (int e = 0; e < E; ++e) {
          zb[e] = FFB_NO_STORE << 16;
          ga[e] = FFB_NO_STORE << 16;
          gb[e] = 0;
          zc[e] = gc[e] = dc[e] = 0.f;
          if (F && e < EZ) {
            zb[e] = static_cast<uint32_t>(__ldg(tzb + e * kThreads + tid));
            const int32_t q = __ldg(tzq + e * kThreads + tid);
            zc[e] = q >= 0 ? __ldg(M.c_val + q) : 0.f;
          }
          if ((D || C) && e < EG) {
            ga[e] = static_cast<uint32_t>(__ldg(tga + e * kThreads + tid));
            gb[e] = static_cast<uint32_t>(__ldg(tgb + e * kThreads + tid));
            const int32_t q = __ldg(tgq + e * kThreads + tid);
            gc[e] = (D && q >= 0) ? __ldg(M.c_val + q) : 0.f;
          }
        }
      }
      __syncthreads();
    }

    const int64_t t0 = static_cast<int64_t>(u - M.ubeg) * T;
    const int64_t left = static_cast<int64_t>(M.N) - t0;
    const int Tc = static_cast<int>(left < T ? left : T);
    float* V = smem + L.oV;
    float* U = smem + L.oU;
    float* RZ = smem + L.oRZ;
    float* RG = smem + L.oRG;
    const uint32_t* zmask = table<uint32_t>(plan, hdr(plan).off_zmask);
    const uint32_t* gmask = table<uint32_t>(plan, hdr(plan).off_gmask);

    // ---- A: analysis ------------------------------------------------------
    {
      const int gA = (NEED_V ? Gn : 0) + (NEED_U ? Gm : 0);
      for (int task = tid; task < Tc * gA; task += kThreads) {
        const int t = task / gA;
        int g = task - t * gA;
        const bool isV = NEED_V && g < (NEED_V ? Gn : 0);
        if (!isV && NEED_V) g -= Gn;
        if (isV) {
          if (__ldg(gmask + g) == 0u) continue;
          Seg<Elem> s;
          s.load_stream(static_cast<const char*>(M.X) + ((t0 + t) * M.ldx + 32 * g) * ELEM);
          float xr[16], xi[16];
          s.unpack(xr, xi);
          fft16<+1>(xr, xi, tw_in);
          store_group(V + t * L.sV, g, xr, xi);
        } else {
          if (__ldg(zmask + g) == 0u) continue;
          Seg<Elem> s;
          s.load_stream(static_cast<const char*>(M.dY) + ((t0 + t) * M.ldy + 32 * g) * ELEM);
          float xr[16], xi[16];
          s.unpack(xr, xi);
          fft16<+1>(xr, xi, tw_out);
          store_group(U + t * L.sU, g, xr, xi);
        }
      }
    }
    __syncthreads();

    // ---- B1: coefficient SpMM / SDDMM over this thread's chunk -------------
    // Y side (by row): RZ[st] = sum over a run of equal rows of c * V[b].
    // dX side (by column): RG[st] = sum over a run of equal columns of c * U[a];
    // dC: dc += U[a] V[b] summed over the tile's tokens.
    if constexpr (F) {
      float acc[kTmax] = {0.f, 0.f, 0.f, 0.f};
      auto step = [&](uint32_t pk, float c) {
        const uint32_t bo = pk & 0xFFFFu, st = pk >> 16;
#pragma unroll
        for (int t = 0; t < kTmax; ++t)
          if (t < Tc) acc[t] = fmaf(c, V[t * L.sV + bo], acc[t]);
        if (st != FFB_NO_STORE) {
#pragma unroll
          for (int t = 0; t < kTmax; ++t) {
            if (t < Tc) RZ[t * L.sRZ + st] = acc[t];
            acc[t] = 0.f;
          }
        }
      };
      if constexpr (REG) {
#pragma unroll
        for (int e = 0; e < E; ++e)
          if (e < EZ) step(zb[e], zc[e]);
      } else {
        const int32_t* tzb = table<int32_t>(plan, hdr(plan).off_zb);
        const int32_t* tzq = table<int32_t>(plan, hdr(plan).off_zq);
        for (int e = 0; e < EZ; ++e) {
          const uint32_t pk = static_cast<uint32_t>(__ldg(tzb + e * kThreads + tid));
          const int32_t q = __ldg(tzq + e * kThreads + tid);
          step(pk, q >= 0 ? __ldg(M.c_val + q) : 0.f);
        }
      }
    }
    if constexpr (D || C) {
      float acc[kTmax] = {0.f, 0.f, 0.f, 0.f};
      auto step = [&](uint32_t pa, uint32_t pb, float c) -> float {
        const uint32_t ao = pa & 0xFFFFu, st = pa >> 16;
        float dcv = 0.f;
#pragma unroll
        for (int t = 0; t < kTmax; ++t) {
          if (t < Tc) {
            const float uv = U[t * L.sU + ao];
            if constexpr (D) acc[t] = fmaf(c, uv, acc[t]);
            if constexpr (C) dcv = fmaf(uv, V[t * L.sV + pb], dcv);
          }
        }
        if constexpr (D) {
          if (st != FFB_NO_STORE) {
#pragma unroll
            for (int t = 0; t < kTmax; ++t) {
              if (t < Tc) RG[t * L.sRG + st] = acc[t];
              acc[t] = 0.f;
            }
          }
        }
        return dcv;
      };
      if constexpr (REG) {
#pragma unroll
        for (int e = 0; e < E; ++e)
          if (e < EG) {
            const float dcv = step(ga[e], gb[e], gc[e]);
            if constexpr (C) dc[e] += dcv;
          }
      } else {
        const int32_t* tga = table<int32_t>(plan, hdr(plan).off_ga);
        const int32_t* tgb = table<int32_t>(plan, hdr(plan).off_gb);
        const int32_t* tgq = table<int32_t>(plan, hdr(plan).off_gq);
        for (int e = 0; e < EG; ++e) {
          const uint32_t pa = static_cast<uint32_t>(__ldg(tga + e * kThreads + tid));
          const uint32_t pb = static_cast<uint32_t>(__ldg(tgb + e * kThreads + tid));
          float c = 0.f;
          if constexpr (D) {
            const int32_t q = __ldg(tgq + e * kThreads + tid);
            c = q >= 0 ? __ldg(M.c_val + q) : 0.f;
          }
          const float dcv = step(pa, pb, c);
          if constexpr (C) dcs[e * kThreads + tid] += dcv;
        }
      }
    }
    if constexpr (F || D) {
      // ---- B2: rows / columns split between chunks ----------------------
      const int nfix = (F ? nfixZ : 0) + (D ? nfixG : 0);
      if (nfix > 0) {
        __syncthreads();
        for (int i = tid; i < nfix; i += kThreads) {
          const bool z = F && i < (F ? nfixZ : 0);
          const int4 it = z ? __ldg(table<int4>(plan, hdr(plan).off_fixZ) + i)
                            : __ldg(table<int4>(plan, hdr(plan).off_fixG) + (i - (F ? nfixZ : 0)));
          float* R = z ? RZ : RG;
          const int stride = z ? L.sRZ : L.sRG;
          for (int t = 0; t < Tc; ++t) {
            float sacc = R[t * stride + it.x];
            for (int c2 = 0; c2 < it.z; ++c2) sacc += R[t * stride + it.y + c2];
            R[t * stride + it.x] = sacc;
          }
        }
      }
      __syncthreads();

      // ---- B3: synthesis and accumulate into Y / dX ----------------------
      const int gS = (F ? Gm : 0) + (D ? Gn : 0);
      for (int task = tid; task < Tc * gS; task += kThreads) {
        const int t = task / gS;
        int g = task - t * gS;
        const bool isY = F && g < (F ? Gm : 0);
        if (!isY && F) g -= Gm;
        if (isY) {
          if (__ldg(zmask + g) == 0u) continue;
          char* yp = static_cast<char*>(M.Y) + ((t0 + t) * M.ldy + 32 * g) * ELEM;
          Seg<Elem> s;
          s.load(yp);
          float xr[16], xi[16];
          load_group(RZ + t * L.sRZ, g, xr, xi);
          fft16<-1>(xr, xi, tw_out);
          s.add_store(yp, xr, xi, M.seff);
        } else {
          if (__ldg(gmask + g) == 0u) continue;
          char* xp = static_cast<char*>(M.dX) + ((t0 + t) * M.ldx + 32 * g) * ELEM;
          Seg<Elem> s;
          s.load(xp);
          float xr[16], xi[16];
          load_group(RG + t * L.sRG, g, xr, xi);
          fft16<-1>(xr, xi, tw_in);
          s.add_store(xp, xr, xi, M.seff);
        }
      }
    }
    // The next tile's analysis writes V/U only: ordered after this tile's
    // B1 reads by the barrier above (or the one below for dC-only runs).
    if constexpr (!(F || D)) __syncthreads();
  }
  if (cur >= 0)
    flush_dc<C, REG, E>(plan, EG, args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride, dc, dcs, tid);
}

// dC_q = (s/16) * sum over the CTAs that visited the matrix, in CTA order.
__global__ void __launch_bounds__(256) dc_reduce_kernel(const __grid_constant__ ReduceK r) {
  const int j = blockIdx.y;
  const ReduceMat& M = r.m[j];
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= M.nnz) return;
  float s = 0.f;
  if (M.ntiles > 0) {
    const int32_t c0 = cta_of_unit(M.ubeg, r.grid, r.total_units);
    const int32_t c1 = cta_of_unit(static_cast<int64_t>(M.ubeg) + M.ntiles - 1, r.grid, r.total_units);
    for (int32_t c = c0; c <= c1; ++c) s += r.partial[static_cast<size_t>(c + j) * r.stride + q];
  }
  M.dC[q] = M.seff * s;
}

// ---------------------------------------------------------------------------
// Merge: W_t[32g + i][32h + jl] = W0 + (s/16) sum_{e in block (g,h)} c_e
// Dout[i][a_e] Din[jl][b_e], D = 4 x the group-0 block of each frame staged in
// shared memory.  One CTA per (out group g, tenant t); a thread owns a column.
// ---------------------------------------------------------------------------
template <typename Elem>
__global__ void __launch_bounds__(256) merge_kernel(const __grid_constant__ MergeK a) {
  __shared__ float Din[32][33];
  __shared__ float Dout[32][33];
  for (int idx = threadIdx.x; idx < 1024; idx += blockDim.x) {
    const int w = idx & 31, x = idx >> 5, i = x >> 1, s = x & 1;
    Dout[w][x] = 4.f * __ldg(a.fout_val + 32 * (i * a.rho_out + s) + w);
    Din[w][x] = 4.f * __ldg(a.fin_val + 32 * (i * a.rho_in + s) + w);
  }
  __syncthreads();
  const int g = blockIdx.x, t = blockIdx.y;
  const FfbPlanHeader& h = hdr(a.plan);
  const int32_t* blkptr = table<int32_t>(a.plan, h.off_blkptr);
  const int2* blkent = table<int2>(a.plan, h.off_blkent);
  const float* cv = a.c_vals + static_cast<size_t>(t) * a.nnz;
  const Elem* W0 = static_cast<const Elem*>(a.W0);
  Elem* Wt = static_cast<Elem*>(a.Wout) + static_cast<size_t>(t) * a.m * a.ldw;
  for (int jc = threadIdx.x; jc < a.n; jc += blockDim.x) {
    const int hh = jc >> 5, jl = jc & 31;
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0.f;
    const int e0 = __ldg(blkptr + g * h.Gn + hh), e1 = __ldg(blkptr + g * h.Gn + hh + 1);
    for (int e = e0; e < e1; ++e) {
      const int2 en = __ldg(blkent + e);
      const int al = en.x & 31, bl = (en.x >> 8) & 31;
      const float w = __ldg(cv + en.y) * Din[jl][bl];
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] = fmaf(w, Dout[i][al], acc[i]);
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const size_t off = static_cast<size_t>(32 * g + i) * a.ldw + jc;
      const float v = fmaf(a.seff, acc[i], static_cast<float>(W0[off]));
      Wt[off] = static_cast<Elem>(v);
    }
  }
}

}  // namespace ffb
