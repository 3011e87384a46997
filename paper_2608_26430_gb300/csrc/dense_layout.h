// Dense operand image of a frame for the generic (dense) path: the synthesis
// matrix Phi (d x K, K = k*rho columns) as the B operands of the tensor-core
// contractions, K-major so that every operand row is contiguous.
//   analysis   V = X Phi:    B row c = column c of Phi (d values), bf16 hi
//                             and bf16 lo parts (v = hi + lo to ~2^-16)
//   synthesis  Y = Z Phi^T:  B row j = row j of Phi (K values), fp32
//                             rounded to tf32 (round to nearest even)
// Rows are padded with zeros to 16-byte strides (TMA row pitch); every
// block starts on a 1024-byte boundary.  Shared by the host packer
// (framefb_host.cpp) and the dense-path launcher (framefb_dense.cu).
#pragma once
#include <stddef.h>
#include <stdint.h>

struct FfbDenseLayout {
  int64_t dp;      // bf16 elements per analysis row (d rounded up to 8)
  int64_t cp;      // fp32 elements per synthesis row (K rounded up to 4)
  int64_t off_hi;  // [K][dp] bf16
  int64_t off_lo;  // [K][dp] bf16
  int64_t off_sy;  // [d][cp] fp32
  int64_t total;   // bytes
};

static inline int64_t ffb_round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

static inline FfbDenseLayout ffb_dense_layout(int64_t d, int64_t K) {
  FfbDenseLayout L;
  L.dp = ffb_round_up(d, 8);
  L.cp = ffb_round_up(K, 4);
  const int64_t an = ffb_round_up(K * L.dp * 2, 1024);
  L.off_hi = 0;
  L.off_lo = an;
  L.off_sy = 2 * an;
  L.total = L.off_sy + ffb_round_up(d * L.cp * 4, 1024);
  return L;
}
