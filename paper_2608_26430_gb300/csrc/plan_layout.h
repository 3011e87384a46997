// Device image of a framefb plan: a header followed by int32 tables, all
// offsets in bytes from the start of the image, every table 16-byte aligned.
// Shared by the host builder (framefb_host.cpp) and the kernels (framefb_cuda.cu).
//
// Index spaces.  For the structured kernels (FFB_LAYOUT_GROUPS) a frame
// column in the paper's order c = i*rho + 2r + s (subspace i, Spectral
// Tetris row r, realified part s) is re-indexed group-major as
// x = 32 r + 2 i + s, so that group r (coordinates
// [32 r, 32 r + 32) of a k = 16, k*rho = d frame) owns the 32 contiguous
// columns [32 r, 32 r + 32): its coefficient vector is the 16 complex values
// (Re, Im interleaved) of the DFT_16 of that coordinate block.  For the dense
// path (FFB_LAYOUT_DENSE) the index is the paper's column c itself, and the
// 32-wide "groups" of the masks are blocks of 32 consecutive columns.
//
// The tables hold these group-major indices.  A store target t < K (K = m
// for the row side, n for the column side) is the index of the run's own
// row or column; t >= K is an overflow slot, kept after the K regular slots.
// Each kernel maps indices to its own shared-memory slots (ffb_slot below
// for the tile layouts) when it loads the tables.
#pragma once
#include <stdint.h>

#ifndef __CUDACC__
#ifndef __host__
#define __host__
#endif
#ifndef __device__
#define __device__
#endif
#endif

#define FFB_PLAN_MAGIC 0x50424646  /* "FFBP" */
#define FFB_PLAN_VERSION 3
#define FFB_LAYOUT_GROUPS 0        /* structured kernels: group-major column index (k = 16, k*rho = d) */
#define FFB_LAYOUT_DENSE 1         /* dense path: frame columns in the paper's order */
#define FFB_GROUP 32               /* real coordinates (and frame columns) per group */
#define FFB_NO_STORE 0xFFFFu
#define FFB_ENTRY_BLOCK 8          /* entries a thread loads together in the sparse phase */

struct FfbPlanHeader {
  int32_t magic, version;
  int32_t n, m;            // index spaces K_n, K_m (frame columns; = features when k*rho = d)
  int32_t Gn, Gm;          // groups of 32 on the input / output side
  int32_t nnz;
  int32_t P;               // threads the chunks were cut for
  int32_t EZ, EG;          // chunk length (entries per thread) by row / by column
  int32_t ovfZ, ovfG;      // overflow slots after the m (resp. n) row slots, multiple of 4
  int32_t nfixZ, nfixG;    // fix-up items (rows / columns split between chunks)
  int32_t off_zb, off_zq;  // [EZ][P]: b | parity(a) << 15 | store << 16, c index (-1 = padding)
  int32_t off_ga, off_gb, off_gq;  // [EG][P]: a | parity(b) << 15 | store << 16, b, c index
  int32_t off_fixZ, off_fixG;      // int4 {dst phys, first overflow slot, count, 0}
  int32_t off_zmask, off_gmask;    // uint32 per group: bit w = row (col) 32g+w is in the support
  int32_t off_blkptr;              // merge: [Gm*Gn + 1] entry ranges of each 32x32 block (g, h)
  int32_t off_blkent;              // merge: int2 {a_local | b_local << 8, c index}
  int32_t total_bytes;
  int32_t layout;          // FFB_LAYOUT_GROUPS or FFB_LAYOUT_DENSE (index space of the tables)
  int32_t d_in, d_out;     // features of the frames (= n, m for FFB_LAYOUT_GROUPS)
  int32_t nnz_full;        // size of the entry-index space q (the caller's nnz; > nnz for a part)
  int32_t off_qlist;       // a part: its entries' q (int32 [nnz]), else 0
  int32_t reserved;
};

// Slot of group-major index x (x < K) in a tile buffer.  Slots come in
// pairs (x even, x + 1); the 16 pairs of a group are permuted so that the
// MMA epilogue and prologue -- lane (g, t) touching pairs 4t..4t+3 of group
// G0 + g, g = 0..7 -- spread every quarter-warp over distinct banks, both
// with two tokens per slot (a pair is one 16-byte chunk) and with one (a
// 16-byte chunk holds two pairs; odd groups use the other half of the
// 128-byte line):
//     pair p of group r -> pair p ^ (((p >> 3) & 1) << 1) ^ (r & 1) ^ ((r & 1) << 3).
// Overflow slots (x >= K) are used as they are.
static inline __host__ __device__ int32_t ffb_slot(int32_t x, int32_t K) {
  if (x >= K) return x;
  const int32_t r = x >> 5, p = (x >> 1) & 15;
  const int32_t pp = p ^ (((p >> 3) & 1) << 1) ^ (r & 1) ^ ((r & 1) << 3);
  return (r << 5) | (pp << 1) | (x & 1);
}

// Shared-memory layout of one tile of T tokens (floats).  MODE bits:
// 1 = forward (Y), 2 = backward dX, 4 = coefficient gradient.  V = X Phi_in
// rows (n), U = dY Phi_out rows (m), RZ = coefficient-SpMM row sums for Y
// (m + ovfZ), RG = the same for dX (n + ovfG); DC = per-thread dC
// accumulators ([entry][thread]).
struct FfbTileLayout {
  int32_t sV, sU, sRZ, sRG;      // token-row strides
  int32_t oV, oU, oRZ, oRG, oDC; // region offsets
  int32_t total;                 // floats
};

static inline __host__ __device__ FfbTileLayout ffb_tile_layout(const FfbPlanHeader& h, int mode, int T,
                                                                bool dc_in_smem) {
  FfbTileLayout L;
  const bool fwd = mode & 1, bdx = mode & 2, gc = mode & 4;
  L.sV = h.n;
  L.sU = h.m;
  L.sRZ = h.m + h.ovfZ;
  L.sRG = h.n + h.ovfG;
  L.oV = 0;
  L.oU = L.oV + ((fwd || gc) ? T * L.sV : 0);
  L.oRZ = L.oU + ((bdx || gc) ? T * L.sU : 0);
  L.oRG = L.oRZ + (fwd ? T * L.sRZ : 0);
  L.oDC = L.oRG + (bdx ? T * L.sRG : 0);
  // whole blocks of entries: padding entries of the last block are updated too
  const int32_t eg = (h.EG + FFB_ENTRY_BLOCK - 1) / FFB_ENTRY_BLOCK * FFB_ENTRY_BLOCK;
  L.total = L.oDC + ((gc && dc_in_smem) ? eg * h.P : 0);
  return L;
}
