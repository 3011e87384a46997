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
// 1 of group 0 holds omega^j / 4 on coordinates 2j, 2j+1).  This exact FFT
// serves fp32 activations; bf16 activations use the tensor-core kernel of
// framefb_mma.cuh.
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
  const float* fval_in;   // device fp32 CSC values of Phi_in (every column holds 32 entries)
  const float* fval_out;  // same for Phi_out
  int64_t ldx, ldy;
  int32_t N, T, ubeg, ntiles;
  float seff;             // s / 16
  int32_t rho_in, rho_out;
  int32_t n, m;           // in / out features
};

struct LaunchK {
  int32_t nmats, total_units, stride, pad;
  float* partial;       // [(grid + nmats) * stride] dC partial sums, slot = cta + matrix
  // shared-memory map of the bf16 tensor-core kernel (bytes): the staged
  // input rows (X then dY of the tile) at stg_in, the staged output rows (Y
  // then dX) at stg_out when stage_out is set (else read from global
  // memory), the fp32 region of the tile layout at fbase, two mbarriers
  int32_t stg_in, stg_out, stage_out, fbase, mbar, pad2;
  // pipelined kernel: one fp32 set layout for every matrix of the launch
  // (offsets of U, RZ, RG and the set size in floats, from the largest n, m
  // and overflow counts), so that sets of consecutive tiles of different
  // matrices never overlap
  int32_t set_oU, set_oRZ, set_oRG, set_total;
  int32_t fixc, fixc_items;  // pipelined kernel: fix-up item cache (bytes offset, capacity)
  MatK m[kMaxMats];
};

struct ReduceMat {
  float* dC;
  const int32_t* qlist;  // a plan's part: the entries' indices into dC (nnz of them), else null
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
// 32-element fp32 row segments of activations: load as 16 complex values
// (x_{2j}, x_{2j+1}), and read-modify-write y += seff * delta.
// ---------------------------------------------------------------------------
template <typename Elem>
struct Seg;

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
// token row laid out by ffb_slot: float4 chunk j (pairs 2j, 2j + 1) goes to
// chunk j ^ ((j >> 2) & 1) ^ 4 (g odd), its two pairs swapped when g is odd.
__device__ __forceinline__ void store_group(float* row, int g, const float (&xr)[16], const float (&xi)[16]) {
  float* base = row + 32 * g;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int p0 = slot_of(2 * c), p1 = slot_of(2 * c + 1);
    const float4 v = (g & 1) ? make_float4(xr[p1], xi[p1], xr[p0], xi[p0]) : make_float4(xr[p0], xi[p0], xr[p1], xi[p1]);
    *reinterpret_cast<float4*>(base + 4 * (c ^ ((c >> 2) & 1) ^ ((g & 1) << 2))) = v;
  }
}

// Read the 32 row sums of one group back in natural complex order.
__device__ __forceinline__ void load_group(const float* row, int g, float (&xr)[16], float (&xi)[16]) {
  const float* base = row + 32 * g;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const float4 v = *reinterpret_cast<const float4*>(base + 4 * (c ^ ((c >> 2) & 1) ^ ((g & 1) << 2)));
    const bool sw = g & 1;
    xr[2 * c] = sw ? v.z : v.x;
    xi[2 * c] = sw ? v.w : v.y;
    xr[2 * c + 1] = sw ? v.x : v.z;
    xi[2 * c + 1] = sw ? v.y : v.w;
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

// ---------------------------------------------------------------------------
// Sparse phase shared by both tile kernels.  A thread owns one chunk of the
// support ordered by row (for Y) and one ordered by column (for dX and dC).
// REG: the chunk (at most kEreg entries) lives in registers for the whole
// matrix; otherwise it is streamed from the plan on every tile and the dC
// accumulators live in shared memory.
// ---------------------------------------------------------------------------
// Per-slot token vectors of the sparse phase: TT tokens of one slot.
// MINOR (token-minor) with TT = 2 uses one 8-byte access; otherwise TT
// scalar accesses at stride `stride` (token-major) or 1 (token-minor, TT = 1).
template <int TT, bool MINOR>
struct Vecs {
  struct type {
    float v[TT];
  };
  static __device__ __forceinline__ type zero() {
    type r;
#pragma unroll
    for (int t = 0; t < TT; ++t) r.v[t] = 0.f;
    return r;
  }
  static __device__ __forceinline__ type load(const type* base, uint32_t slot, int stride) {
    const float* b = reinterpret_cast<const float*>(base);
    type r;
#pragma unroll
    for (int t = 0; t < TT; ++t) r.v[t] = MINOR ? b[slot * TT + t] : b[t * stride + slot];
    return r;
  }
  static __device__ __forceinline__ void store(type* base, uint32_t slot, int stride, const type& x) {
    float* b = reinterpret_cast<float*>(base);
#pragma unroll
    for (int t = 0; t < TT; ++t) {
      if (MINOR)
        b[slot * TT + t] = x.v[t];
      else
        b[t * stride + slot] = x.v[t];
    }
  }
  static __device__ __forceinline__ void fma(type& acc, float c, const type& x) {
#pragma unroll
    for (int t = 0; t < TT; ++t) acc.v[t] = fmaf(c, x.v[t], acc.v[t]);
  }
  static __device__ __forceinline__ float dot(const type& a, const type& b) {
    float s = 0.f;
#pragma unroll
    for (int t = 0; t < TT; ++t) s = fmaf(a.v[t], b.v[t], s);
    return s;
  }
};

template <>
struct Vecs<2, true> {
  using type = float2;
  static __device__ __forceinline__ float2 zero() { return make_float2(0.f, 0.f); }
  static __device__ __forceinline__ float2 load(const float2* base, uint32_t slot, int) { return base[slot]; }
  static __device__ __forceinline__ void store(float2* base, uint32_t slot, int, const float2& x) { base[slot] = x; }
  static __device__ __forceinline__ void fma(float2& acc, float c, const float2& x) {
    acc.x = fmaf(c, x.x, acc.x);
    acc.y = fmaf(c, x.y, acc.y);
  }
  static __device__ __forceinline__ float dot(const float2& a, const float2& b) { return fmaf(a.x, b.x, a.y * b.y); }
};

// FLIP: fold the sign pattern S = diag(+1, -1, +1, ...) of the row / column
// index into the coefficient values (the tensor-core synthesis reuses the
// analysis block through D^T = S D S, so it wants S Z and S G).
template <int MODE, bool REG, bool FLIP = false>
struct Chunk {
  static constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  static constexpr int E = REG ? kEreg : 1;
  // zb: V slot of b | RZ slot of the store target << 16 (FFB_NO_STORE: none)
  // ga: U slot of a | RG slot of the store target << 16;  gb: V slot of b
  uint32_t zb[E], ga[E], gb[E];
  float zc[E], gc[E];
  int EZ, EG, n, m;

  // coefficient value with the parity sign of plan word w (bit 15) folded in
  static __device__ __forceinline__ float signed_c(float c, uint32_t w) {
    return (FLIP && (w & 0x8000u)) ? -c : c;
  }

  // plan word (index | parity << 15 | target << 16) -> (slot | slot << 16)
  static __device__ __forceinline__ uint32_t slots(uint32_t w, int Klo, int Khi) {
    const uint32_t lo = w & 0x7FFFu, hi = w >> 16;
    const uint32_t slo = static_cast<uint32_t>(ffb_slot(static_cast<int32_t>(lo), Klo));
    const uint32_t shi = hi == FFB_NO_STORE ? FFB_NO_STORE : static_cast<uint32_t>(ffb_slot(static_cast<int32_t>(hi), Khi));
    return slo | (shi << 16);
  }

  __device__ __forceinline__ void load(const uint8_t* plan, const float* c_val, int tid) {
    const FfbPlanHeader& h = hdr(plan);
    EZ = h.EZ;
    EG = h.EG;
    n = h.n;
    m = h.m;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      zb[e] = FFB_NO_STORE << 16;
      ga[e] = FFB_NO_STORE << 16;
      gb[e] = 0;
      zc[e] = gc[e] = 0.f;
    }
    if constexpr (REG) {
      const int32_t* tzb = table<int32_t>(plan, h.off_zb);
      const int32_t* tzq = table<int32_t>(plan, h.off_zq);
      const int32_t* tga = table<int32_t>(plan, h.off_ga);
      const int32_t* tgb = table<int32_t>(plan, h.off_gb);
      const int32_t* tgq = table<int32_t>(plan, h.off_gq);
#pragma unroll
      for (int e = 0; e < E; ++e) {
        if (F && e < EZ) {
          const uint32_t w = static_cast<uint32_t>(__ldg(tzb + e * kThreads + tid));
          zb[e] = slots(w, n, m);
          const int32_t q = __ldg(tzq + e * kThreads + tid);
          zc[e] = q >= 0 ? signed_c(__ldg(c_val + q), w) : 0.f;
        }
        if ((D || C) && e < EG) {
          const uint32_t w = static_cast<uint32_t>(__ldg(tga + e * kThreads + tid));
          ga[e] = slots(w, m, n);
          gb[e] = static_cast<uint32_t>(ffb_slot(__ldg(tgb + e * kThreads + tid), n));
          const int32_t q = __ldg(tgq + e * kThreads + tid);
          gc[e] = (D && q >= 0) ? signed_c(__ldg(c_val + q), w) : 0.f;
        }
      }
    }
  }

  // One block of B entries of the row side from the register chunk or the
  // streamed tables: (plan word as slots, c).
  __device__ __forceinline__ void z_entry(const uint8_t* plan, const float* c_val, int tid, int e, uint32_t& w,
                                          float& c) const {
    if constexpr (REG) {
      (void)plan;
      (void)c_val;
      (void)tid;
      w = zb[e];
      c = zc[e];
    } else {
      const uint32_t raw = static_cast<uint32_t>(__ldg(table<int32_t>(plan, hdr(plan).off_zb) + e * kThreads + tid));
      w = slots(raw, n, m);
      const int32_t q = __ldg(table<int32_t>(plan, hdr(plan).off_zq) + e * kThreads + tid);
      c = q >= 0 ? signed_c(__ldg(c_val + q), raw) : 0.f;
    }
  }
  __device__ __forceinline__ void g_entry(const uint8_t* plan, const float* c_val, int tid, int e, uint32_t& wa,
                                          uint32_t& wb, float& c) const {
    if constexpr (REG) {
      (void)plan;
      (void)c_val;
      (void)tid;
      wa = ga[e];
      wb = gb[e];
      c = gc[e];
    } else {
      const uint32_t raw = static_cast<uint32_t>(__ldg(table<int32_t>(plan, hdr(plan).off_ga) + e * kThreads + tid));
      wa = slots(raw, m, n);
      wb = static_cast<uint32_t>(ffb_slot(__ldg(table<int32_t>(plan, hdr(plan).off_gb) + e * kThreads + tid), n));
      c = 0.f;
      if constexpr (D) {
        const int32_t q = __ldg(table<int32_t>(plan, hdr(plan).off_gq) + e * kThreads + tid);
        c = q >= 0 ? signed_c(__ldg(c_val + q), raw) : 0.f;
      }
    }
  }

  // Y side (by row): RZ[st] = sum over a run of equal rows of c V[b].
  // dX side (by column): RG[st] = sum over a run of equal columns of c U[a].
  // dC: dc += sum over the tile's tokens of U[a] V[b].
  // TT tokens in the tile.  Element (token t, slot s) lives at s * TT + t
  // (MINOR: token-minor, one vector access per slot) or t * stride + s.
  // V / U (read) and RZ / RG (written) are disjoint regions: the restrict
  // pointers let the loads of a block of entries issue ahead of the stores
  // of the previous block.
  template <int TT, bool MINOR>
  __device__ __forceinline__ void z_block(const uint8_t* plan, const float* c_val, int tid, int e0,
                                          const typename Vecs<TT, MINOR>::type* __restrict__ V,
                                          typename Vecs<TT, MINOR>::type* __restrict__ RZ, int sV, int sRZ,
                                          typename Vecs<TT, MINOR>::type& acc) const {
    using Vec = typename Vecs<TT, MINOR>::type;
    constexpr int B = FFB_ENTRY_BLOCK;
    uint32_t w[B];
    float c[B];
    Vec v[B];
#pragma unroll
    for (int e = 0; e < B; ++e) {
      if (REG || e0 + e < EZ) {
        z_entry(plan, c_val, tid, e0 + e, w[e], c[e]);
      } else {
        w[e] = FFB_NO_STORE << 16;
        c[e] = 0.f;
      }
      v[e] = Vecs<TT, MINOR>::load(V, w[e] & 0xFFFFu, sV);
    }
#pragma unroll
    for (int e = 0; e < B; ++e) {
      Vecs<TT, MINOR>::fma(acc, c[e], v[e]);
      const uint32_t st = w[e] >> 16;
      if (st != FFB_NO_STORE) {
        Vecs<TT, MINOR>::store(RZ, st, sRZ, acc);
        acc = Vecs<TT, MINOR>::zero();
      }
    }
  }

  template <int TT, bool MINOR>
  __device__ __forceinline__ void g_block(const uint8_t* plan, const float* c_val, int tid, int e0,
                                          const typename Vecs<TT, MINOR>::type* __restrict__ U,
                                          const typename Vecs<TT, MINOR>::type* __restrict__ V,
                                          typename Vecs<TT, MINOR>::type* __restrict__ RG, float* __restrict__ dcs,
                                          int sU, int sV, int sRG, typename Vecs<TT, MINOR>::type& acc) const {
    using Vec = typename Vecs<TT, MINOR>::type;
    constexpr int B = FFB_ENTRY_BLOCK;
    uint32_t wa[B], wb[B];
    float c[B];
    Vec uu[B], vv[B];
#pragma unroll
    for (int e = 0; e < B; ++e) {
      if (REG || e0 + e < EG) {
        g_entry(plan, c_val, tid, e0 + e, wa[e], wb[e], c[e]);
      } else {
        wa[e] = FFB_NO_STORE << 16;
        wb[e] = 0;
        c[e] = 0.f;
      }
      uu[e] = Vecs<TT, MINOR>::load(U, wa[e] & 0xFFFFu, sU);
      if constexpr (C) vv[e] = Vecs<TT, MINOR>::load(V, wb[e], sV);
    }
    float dsum[B];
#pragma unroll
    for (int e = 0; e < B; ++e) {
      if constexpr (C) dsum[e] = Vecs<TT, MINOR>::dot(uu[e], vv[e]);
      if constexpr (D) {
        Vecs<TT, MINOR>::fma(acc, c[e], uu[e]);
        const uint32_t st = wa[e] >> 16;
        if (st != FFB_NO_STORE) {
          Vecs<TT, MINOR>::store(RG, st, sRG, acc);
          acc = Vecs<TT, MINOR>::zero();
        }
      }
    }
    if constexpr (C) {
#pragma unroll
      for (int e = 0; e < B; ++e) dcs[(e0 + e) * kThreads + tid] += dsum[e];
    }
  }

  // Y side (by row): RZ[st] = sum over a run of equal rows of c V[b].
  // dX side (by column): RG[st] = sum over a run of equal columns of c U[a].
  // dC: dc += sum over the tile's tokens of U[a] V[b].
  // TT tokens in the tile.  Element (token t, slot s) lives at s * TT + t
  // (MINOR: token-minor, one vector access per slot) or t * stride + s.
  // V / U (read) and RZ / RG (written) are disjoint regions: the restrict
  // pointers let the loads of a block of entries issue ahead of the stores
  // of the previous block.
  template <int TT, bool MINOR>
  __device__ __forceinline__ void sparse_tt(const uint8_t* plan, const float* c_val, int tid, const FfbTileLayout& L,
                                            float* fsm) {
    using Vec = typename Vecs<TT, MINOR>::type;
    const Vec* V = reinterpret_cast<const Vec*>(fsm + L.oV);
    const Vec* U = reinterpret_cast<const Vec*>(fsm + L.oU);
    Vec* RZ = reinterpret_cast<Vec*>(fsm + L.oRZ);
    Vec* RG = reinterpret_cast<Vec*>(fsm + L.oRG);
    float* dcs = fsm + L.oDC;
    constexpr int B = FFB_ENTRY_BLOCK;
    static_assert(kEreg % B == 0, "register chunk must hold whole blocks");
    if constexpr (F) {
      Vec acc = Vecs<TT, MINOR>::zero();
      if constexpr (REG) {
#pragma unroll
        for (int e0 = 0; e0 < E; e0 += B)
          if (e0 < EZ) z_block<TT, MINOR>(plan, c_val, tid, e0, V, RZ, L.sV, L.sRZ, acc);
      } else {
        for (int e0 = 0; e0 < EZ; e0 += B) z_block<TT, MINOR>(plan, c_val, tid, e0, V, RZ, L.sV, L.sRZ, acc);
      }
    }
    if constexpr (D || C) {
      Vec acc = Vecs<TT, MINOR>::zero();
      if constexpr (REG) {
#pragma unroll
        for (int e0 = 0; e0 < E; e0 += B)
          if (e0 < EG) g_block<TT, MINOR>(plan, c_val, tid, e0, U, V, RG, dcs, L.sU, L.sV, L.sRG, acc);
      } else {
        for (int e0 = 0; e0 < EG; e0 += B)
          g_block<TT, MINOR>(plan, c_val, tid, e0, U, V, RG, dcs, L.sU, L.sV, L.sRG, acc);
      }
    }
  }

  template <bool MINOR>
  __device__ __forceinline__ void sparse(const uint8_t* plan, const float* c_val, int tid, const FfbTileLayout& L,
                                         float* fsm, int Tc) {
    switch (Tc) {
      case 1: sparse_tt<1, MINOR>(plan, c_val, tid, L, fsm); break;
      case 2: sparse_tt<2, MINOR>(plan, c_val, tid, L, fsm); break;
      case 3: sparse_tt<3, MINOR>(plan, c_val, tid, L, fsm); break;
      default: sparse_tt<4, MINOR>(plan, c_val, tid, L, fsm); break;
    }
  }

  // Write this thread's dC partial sums of one matrix to its workspace slot
  // (the accumulators live in shared memory, one column per thread).
  __device__ __forceinline__ void flush(const uint8_t* plan, float* dst, const FfbTileLayout& L, const float* fsm,
                                        int tid) {
    if constexpr (C) {
      const int32_t* gq = table<int32_t>(plan, hdr(plan).off_gq);
      const float* dcs = fsm + L.oDC;
      for (int e = 0; e < EG; ++e) {
        const int32_t q = __ldg(gq + e * kThreads + tid);
        if (q >= 0) dst[q] = dcs[e * kThreads + tid];
      }
    }
  }
};

// Rows (columns) of C whose entries were split between chunks: add the
// later pieces, stored in overflow slots, to the first piece.  Needs a
// barrier before (pieces written) and after (sums complete).  Element
// (token t, slot s) at s * T + t (minor) or t * stride + s.
template <int MODE, bool MINOR, int NT = kThreads>
__device__ __forceinline__ void fixup(const uint8_t* plan, const FfbTileLayout& L, float* fsm, int T, int Tc,
                                      int tid) {
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D;
  const FfbPlanHeader& h = hdr(plan);
  const int nfZ = F ? h.nfixZ : 0, nfG = D ? h.nfixG : 0;
  for (int i = tid; i < nfZ + nfG; i += NT) {
    const bool z = i < nfZ;
    const int4 it = z ? __ldg(table<int4>(plan, h.off_fixZ) + i) : __ldg(table<int4>(plan, h.off_fixG) + (i - nfZ));
    float* R = fsm + (z ? L.oRZ : L.oRG);
    const int stride = z ? L.sRZ : L.sRG;
    const int dst = ffb_slot(it.x, z ? h.m : h.n);
    for (int t = 0; t < Tc; ++t) {
      float* Rt = MINOR ? R + t : R + t * stride;
      const int sc = MINOR ? T : 1;
      float sacc = Rt[dst * sc];
      for (int c2 = 0; c2 < it.z; ++c2) sacc += Rt[(it.y + c2) * sc];
      Rt[dst * sc] = sacc;
    }
  }
}

__device__ __forceinline__ int fix_count(const uint8_t* plan, int mode) {
  const FfbPlanHeader& h = hdr(plan);
  return ((mode & MODE_F) ? h.nfixZ : 0) + ((mode & MODE_D) ? h.nfixG : 0);
}

// ---------------------------------------------------------------------------
// fp32 tile kernel (exact radix-4 FFT_16 on CUDA cores).  Persistent CTAs
// walk a contiguous range of units (matrix, tile of T tokens), matrix-major:
//   A  analysis: V = X Phi_in, U = dY Phi_out per 32-coordinate group;
//   B1 the sparse phase (Chunk::sparse); B2 fix-up;
//   B3 synthesis: FFT_16 of RZ / RG per group and y += (s/16) * result.
// dC accumulates over the CTA's tiles of a matrix and is written to the
// workspace slot (cta + matrix) when the CTA leaves the matrix.
// ---------------------------------------------------------------------------
template <int MODE, bool REG>
__global__ void __launch_bounds__(kThreads, 1) fft_tile_kernel(const __grid_constant__ LaunchK args) {
  using Elem = float;
  constexpr bool F = MODE & MODE_F, D = MODE & MODE_D, C = MODE & MODE_C;
  constexpr bool NEED_V = F || C, NEED_U = D || C;
  constexpr size_t ELEM = sizeof(Elem);
  extern __shared__ float4 smem4[];
  float* fsm = reinterpret_cast<float*>(smem4);
  const int tid = threadIdx.x;

  const int64_t units = args.total_units;
  const int64_t u_begin = (static_cast<int64_t>(blockIdx.x) * units) / gridDim.x;
  const int64_t u_end = (static_cast<int64_t>(blockIdx.x + 1) * units) / gridDim.x;
  if (u_begin >= u_end) return;

  Chunk<MODE, REG> ch;
  int j = 0;
  while (j + 1 < args.nmats && u_begin >= args.m[j].ubeg + args.m[j].ntiles) ++j;
  int cur = -1;
  const uint8_t* plan = nullptr;
  FfbTileLayout L{};
  Tw tw_in{}, tw_out{};
  int Gn = 0, Gm = 0, T = 1;

  for (int64_t u = u_begin; u < u_end; ++u) {
    while (u >= args.m[j].ubeg + args.m[j].ntiles) ++j;
    const MatK& M = args.m[j];
    if (j != cur) {
      if (cur >= 0) ch.flush(plan, args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride, L, fsm, tid);
      cur = j;
      plan = M.plan;
      const FfbPlanHeader& h = hdr(plan);
      Gn = h.Gn;
      Gm = h.Gm;
      T = M.T;
      FfbPlanHeader hc = h;
      L = ffb_tile_layout(hc, MODE, T, C);
      tw_in = load_tw(M.fval_in + 32 * M.rho_in);
      tw_out = load_tw(M.fval_out + 32 * M.rho_out);
      __syncthreads();  // every thread is done with the previous matrix's shared memory
      for (int i = tid; i < L.total - L.oRZ; i += kThreads) fsm[L.oRZ + i] = 0.f;
      ch.load(plan, M.c_val, tid);
      __syncthreads();
    }

    const int64_t t0 = static_cast<int64_t>(u - M.ubeg) * T;
    const int64_t left = static_cast<int64_t>(M.N) - t0;
    const int Tc = static_cast<int>(left < T ? left : T);
    float* V = fsm + L.oV;
    float* U = fsm + L.oU;
    float* RZ = fsm + L.oRZ;
    float* RG = fsm + L.oRG;
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

    // ---- B1: sparse phase -------------------------------------------------
    ch.template sparse<false>(plan, M.c_val, tid, L, fsm, Tc);
    if constexpr (F || D) {
      // ---- B2: fix-up ---------------------------------------------------
      if (fix_count(plan, MODE) > 0) {
        __syncthreads();
        fixup<MODE, false>(plan, L, fsm, T, Tc, tid);
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
    // sparse-phase reads by the barrier above (or the one below for dC-only runs).
    if constexpr (!(F || D)) __syncthreads();
  }
  if (cur >= 0) ch.flush(plan, args.partial + static_cast<size_t>(blockIdx.x + cur) * args.stride, L, fsm, tid);
}

// dC_q = (s/16) * sum over the CTAs that visited the matrix, in CTA order
// (a plan's part: q over its entries' indices).
__global__ void __launch_bounds__(256) dc_reduce_kernel(const __grid_constant__ ReduceK r) {
  const int j = blockIdx.y;
  const ReduceMat& M = r.m[j];
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.nnz) return;
  const int q = M.qlist ? __ldg(M.qlist + i) : i;
  float s = 0.f;
  if (M.ntiles > 0) {
    const int32_t c0 = cta_of_unit(M.ubeg, r.grid, r.total_units);
    const int32_t c1 = cta_of_unit(static_cast<int64_t>(M.ubeg) + M.ntiles - 1, r.grid, r.total_units);
    for (int32_t c = c0; c <= c1; ++c) s += r.partial[static_cast<size_t>(c + j) * r.stride + q];
  }
  M.dC[q] = M.seff * s;
}

// ---------------------------------------------------------------------------
// Merge (Sec. 3.4 "Storage efficiency", Alg. 1 step 6 per tenant):
//   W_t[32g + i][32h + j] = W0[..] + (s/16) sum_{e in block (g,h)} c_{t,e} Dout[i][a_e] Din[j][b_e],
// D = 4 x the group-0 block of each frame (k = 16, k*rho = d frames), staged
// once per CTA.  Work items are (out group g, tenant t, a run of four 32 x 32
// blocks h of that row); each warp takes items grid-stride (any number of
// tenants).  A warp first stages its item's entries (the blocks (g, .) are
// contiguous in the plan) and the tenant's values in its own slice of
// shared memory, so no CTA barrier ties the warps together and one warp's
// staging latency hides behind the others' arithmetic.  A
// lane owns one 16-byte chunk of one row per row pass: lanes (row l / CPR,
// chunk l % CPR), CPR = 16-byte chunks per 32-element row (4 bf16, 8 fp32),
// so a warp's store covers whole 64- or 128-byte row segments.  Bound: HBM
// (W_t written once; W0 and the plan are L2-resident across tenants).
// ---------------------------------------------------------------------------
template <typename Elem>
struct MergeIO;
template <>
struct MergeIO<__nv_bfloat16> {
  static constexpr int kPer = 8;  // elements per 16-byte chunk
  static __device__ __forceinline__ void unpack(const uint4& q, float (&x)[8]) {
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[2 * i] = __uint_as_float(w[i] << 16);
      x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
  static __device__ __forceinline__ uint4 pack(const float (&x)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = __floats2bfloat162_rn(x[2 * i], x[2 * i + 1]);
      w[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
};
template <>
struct MergeIO<float> {
  static constexpr int kPer = 4;
  static __device__ __forceinline__ void unpack(const uint4& q, float (&x)[4]) {
    x[0] = __uint_as_float(q.x);
    x[1] = __uint_as_float(q.y);
    x[2] = __uint_as_float(q.z);
    x[3] = __uint_as_float(q.w);
  }
  static __device__ __forceinline__ uint4 pack(const float (&x)[4]) {
    return make_uint4(__float_as_uint(x[0]), __float_as_uint(x[1]), __float_as_uint(x[2]), __float_as_uint(x[3]));
  }
};

constexpr int kMergeThreads = 256;
constexpr int kMergeWarps = kMergeThreads / 32;
constexpr int kMergeStage = 512;  // entries of one item a warp stages (longer rows read them from L2)
constexpr int kMergeBlocks = 4;   // 32 x 32 blocks per work item

template <typename Elem>
__global__ void __launch_bounds__(kMergeThreads, 2) merge_kernel(const __grid_constant__ MergeK a) {
  using IO = MergeIO<Elem>;
  constexpr int PER = IO::kPer;             // elements per lane chunk
  constexpr int CPR = 32 / PER;             // chunks per 32-element block row
  constexpr int RPP = 32 / CPR;             // rows per warp pass
  constexpr int PASSES = 32 / RPP;          // passes over the block's 32 rows
  __shared__ float DoutT[32][33];           // [a][i] = Dout[i][a]
  __shared__ __align__(16) float DinT[32][32];  // [b][j] = Din[j][b]
  __shared__ int32_t ent_s[kMergeWarps][kMergeStage];  // a_local | b_local << 8, per warp
  __shared__ float cv_s[kMergeWarps][kMergeStage];     // the tenant's value of each
  __shared__ int32_t bp_s[kMergeWarps][kMergeBlocks + 1];  // block boundaries of the item
  for (int idx = threadIdx.x; idx < 1024; idx += blockDim.x) {
    const int w = idx & 31, x = idx >> 5, i = x >> 1, s = x & 1;  // column x = 2i + s of the group block, row w
    DoutT[x][w] = 4.f * __ldg(a.fout_val + 32 * (i * a.rho_out + s) + w);
    DinT[x][w] = 4.f * __ldg(a.fin_val + 32 * (i * a.rho_in + s) + w);
  }
  __syncthreads();
  const FfbPlanHeader& h = hdr(a.plan);
  const int32_t* blkptr = table<int32_t>(a.plan, h.off_blkptr);
  const int2* blkent = table<int2>(a.plan, h.off_blkent);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rl = lane / CPR, cl = lane % CPR;  // row in the pass, chunk in the row
  int32_t* ent = ent_s[warp];
  float* cvw = cv_s[warp];
  int32_t* bp = bp_s[warp];
  const Elem* W0 = static_cast<const Elem*>(a.W0);
  // work items: (out group g, tenant t, run of kMergeBlocks blocks)
  const int nsub = (h.Gn + kMergeBlocks - 1) / kMergeBlocks;
  const int64_t items = static_cast<int64_t>(h.Gm) * nsub * a.T;
  for (int64_t it = static_cast<int64_t>(blockIdx.x) * kMergeWarps + warp; it < items;
       it += static_cast<int64_t>(gridDim.x) * kMergeWarps) {
    const int sub = static_cast<int>(it % nsub);
    const int g = static_cast<int>((it / nsub) % h.Gm);
    const int64_t t = it / (static_cast<int64_t>(nsub) * h.Gm);
    const int hb0 = sub * kMergeBlocks, hb1 = min(h.Gn, hb0 + kMergeBlocks);
    const float* cv = a.c_vals + t * a.nnz;
    Elem* Wt = static_cast<Elem*>(a.Wout) + t * static_cast<int64_t>(a.m) * a.ldw;
    const int eg0 = __ldg(blkptr + g * h.Gn + hb0), eg1 = __ldg(blkptr + g * h.Gn + hb1);
    const bool staged = eg1 - eg0 <= kMergeStage;
    __syncwarp();  // the warp's previous item is done with its slice
    if (staged) {
      for (int e = lane; e < eg1 - eg0; e += 32) {
        const int2 en = __ldg(blkent + eg0 + e);
        ent[e] = en.x;
        cvw[e] = __ldg(cv + en.y);
      }
      if (lane <= hb1 - hb0) bp[lane] = __ldg(blkptr + g * h.Gn + hb0 + lane);
    }
    __syncwarp();
    // W0 chunks one block ahead: their latency overlaps the previous block
    uint4 w0n[PASSES];
#pragma unroll
    for (int r = 0; r < PASSES; ++r)
      w0n[r] = __ldg(reinterpret_cast<const uint4*>(W0 + static_cast<int64_t>(32 * g + r * RPP + rl) * a.ldw +
                                                    32 * hb0 + cl * PER));
    for (int hb = hb0; hb < hb1; ++hb) {
      uint4 w0[PASSES];
#pragma unroll
      for (int r = 0; r < PASSES; ++r) w0[r] = w0n[r];
      if (hb + 1 < hb1) {
#pragma unroll
        for (int r = 0; r < PASSES; ++r)
          w0n[r] = __ldg(reinterpret_cast<const uint4*>(W0 + static_cast<int64_t>(32 * g + r * RPP + rl) * a.ldw +
                                                        32 * (hb + 1) + cl * PER));
      }
      float acc[PASSES][PER];
#pragma unroll
      for (int r = 0; r < PASSES; ++r)
#pragma unroll
        for (int j = 0; j < PER; ++j) acc[r][j] = 0.f;
      const int e0 = staged ? bp[hb - hb0] : __ldg(blkptr + g * h.Gn + hb);
      const int e1 = staged ? bp[hb - hb0 + 1] : __ldg(blkptr + g * h.Gn + hb + 1);
      for (int e = e0; e < e1; ++e) {
        int ex;
        float c;
        if (staged) {
          ex = ent[e - eg0];
          c = cvw[e - eg0];
        } else {
          const int2 en = __ldg(blkent + e);
          ex = en.x;
          c = __ldg(cv + en.y);
        }
        const int al = ex & 31, bl = (ex >> 8) & 31;
        float din[PER];
#pragma unroll
        for (int j = 0; j < PER; j += 4) {
          const float4 q = *reinterpret_cast<const float4*>(&DinT[bl][cl * PER + j]);
          din[j] = q.x;
          din[j + 1] = q.y;
          din[j + 2] = q.z;
          din[j + 3] = q.w;
        }
#pragma unroll
        for (int r = 0; r < PASSES; ++r) {
          const float u = c * DoutT[al][r * RPP + rl];
#pragma unroll
          for (int j = 0; j < PER; ++j) acc[r][j] = fmaf(u, din[j], acc[r][j]);
        }
      }
#pragma unroll
      for (int r = 0; r < PASSES; ++r) {
        const int64_t off = static_cast<int64_t>(32 * g + r * RPP + rl) * a.ldw + 32 * hb + cl * PER;
        float w[PER];
        IO::unpack(w0[r], w);
#pragma unroll
        for (int j = 0; j < PER; ++j) w[j] = fmaf(a.seff, acc[r][j], w[j]);
        *reinterpret_cast<uint4*>(Wt + off) = IO::pack(w);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// AdamW step on coefficient values (Appendix, hyperparameter tables: AdamW):
// elementwise over n fp32 values, 16 B read + 12 B written per element; a
// grid-stride loop over float4 chunks (VEC, all four arrays 16-byte aligned)
// or single values.  Bias corrections arrive as step_size = lr / (1 - b1^t)
// and inv_sqrt_bc2 = 1 / sqrt(1 - b2^t).
// ---------------------------------------------------------------------------
struct AdamWK {
  float* p;
  const float* g;
  float* m;
  float* v;
  int64_t n;
  float decay;  // 1 - lr * weight_decay
  float beta1, beta2, step_size, inv_sqrt_bc2, eps;
};

__device__ __forceinline__ void adamw_one(float& p, float g, float& m, float& v, const AdamWK& a) {
  p *= a.decay;
  m = fmaf(a.beta1, m, (1.f - a.beta1) * g);
  v = fmaf(a.beta2, v, (1.f - a.beta2) * g * g);
  const float denom = fmaf(sqrtf(v), a.inv_sqrt_bc2, a.eps);
  p -= a.step_size * (m / denom);
}

template <bool VEC>
__global__ void __launch_bounds__(256) adamw_kernel(const AdamWK a) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if constexpr (VEC) {
    const int64_t n4 = a.n >> 2;
    for (int64_t i = i0; i < n4; i += stride) {
      float4 p = reinterpret_cast<const float4*>(a.p)[i];
      const float4 g = __ldg(reinterpret_cast<const float4*>(a.g) + i);
      float4 m = reinterpret_cast<const float4*>(a.m)[i];
      float4 v = reinterpret_cast<const float4*>(a.v)[i];
      adamw_one(p.x, g.x, m.x, v.x, a);
      adamw_one(p.y, g.y, m.y, v.y, a);
      adamw_one(p.z, g.z, m.z, v.z, a);
      adamw_one(p.w, g.w, m.w, v.w, a);
      reinterpret_cast<float4*>(a.p)[i] = p;
      reinterpret_cast<float4*>(a.m)[i] = m;
      reinterpret_cast<float4*>(a.v)[i] = v;
    }
    for (int64_t i = (n4 << 2) + i0; i < a.n; i += stride) adamw_one(a.p[i], __ldg(a.g + i), a.m[i], a.v[i], a);
  } else {
    for (int64_t i = i0; i < a.n; i += stride) adamw_one(a.p[i], __ldg(a.g + i), a.m[i], a.v[i], a);
  }
}

}  // namespace ffb
