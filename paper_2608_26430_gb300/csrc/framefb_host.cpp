// Host side of libframefb: frame construction (S1), support sampling (S2),
// plan building and status strings.  Plain C++17, no CUDA calls.
#include "framefb.h"
#include "dense_layout.h"
#include "plan_layout.h"
#include "plan_internal.h"

#include <algorithm>
#include <atomic>
#include <memory>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <exception>
#include <new>
#include <system_error>
#include <unordered_set>
#include <thread>
#include <vector>

extern "C" const char* framefb_status_string(int32_t status) {
  switch (status) {
    case FRAMEFB_OK: return "ok";
    case FRAMEFB_EINVAL: return "invalid argument";
    case FRAMEFB_EUNSUPPORTED: return "unsupported parameters";
    case FRAMEFB_ENOMEM: return "out of host memory";
    case FRAMEFB_ECUDA: return "CUDA runtime error";
    case FRAMEFB_EWORKSPACE: return "workspace missing or too small";
    default: return "unknown status";
  }
}

extern "C" int32_t framefb_abi_version(void) { return FRAMEFB_ABI_VERSION; }

namespace {

// ---------------------------------------------------------------------------
// S1: Spectral Tetris (Sec. 3.2 step 1; appendix "Spectral Tetris").
// F is rho_c x d_c; every row must receive squared norm d_c/rho_c and every
// column unit norm.  Norms are tracked exactly in units of 1/rho_c: a row
// needs d_c units and a full entry 1 contributes rho_c units.  Ones are placed
// while at least rho_c units remain; a remainder 0 < x < 1 closes the row with
// T(x) = (1/sqrt2)[[sqrt x, sqrt x], [sqrt(2-x), -sqrt(2-x)]] in the next two
// columns, whose lower row hands 2 - x to the next row.
// ---------------------------------------------------------------------------
struct StRow { int32_t first, last; };

bool spectral_tetris(int32_t rho_c, int32_t d_c, std::vector<double>& F, std::vector<StRow>& sup) {
  if (rho_c < 1 || d_c < 2 * rho_c) return false;
  F.assign(static_cast<size_t>(rho_c) * d_c, 0.0);
  int64_t col = 0, handed = 0;
  for (int32_t r = 0; r < rho_c; ++r) {
    int64_t rem = static_cast<int64_t>(d_c) - handed;
    if (rem < 0) return false;
    while (rem >= rho_c) {
      if (col >= d_c) return false;
      F[static_cast<size_t>(r) * d_c + col] = 1.0;
      ++col;
      rem -= rho_c;
    }
    if (rem > 0) {
      if (r + 1 >= rho_c || col + 1 >= d_c) return false;
      const double top = std::sqrt(static_cast<double>(rem) / (2.0 * rho_c));
      const double bot = std::sqrt(static_cast<double>(2 * rho_c - rem) / (2.0 * rho_c));
      F[static_cast<size_t>(r) * d_c + col] = top;
      F[static_cast<size_t>(r) * d_c + col + 1] = top;
      F[static_cast<size_t>(r + 1) * d_c + col] = bot;
      F[static_cast<size_t>(r + 1) * d_c + col + 1] = -bot;
      col += 2;
      handed = 2 * static_cast<int64_t>(rho_c) - rem;
    } else {
      handed = 0;
    }
  }
  if (col != d_c) return false;
  sup.assign(rho_c, StRow{-1, -1});
  for (int32_t r = 0; r < rho_c; ++r) {
    for (int32_t j = 0; j < d_c; ++j) {
      if (F[static_cast<size_t>(r) * d_c + j] != 0.0) {
        if (sup[r].first < 0) sup[r].first = j;
        sup[r].last = j;
      }
    }
    if (sup[r].first < 0) return false;
  }
  return true;
}

template <typename T>
T* alloc_array(size_t n) {
  return static_cast<T*>(std::malloc(std::max<size_t>(n, 1) * sizeof(T)));
}

}  // namespace

extern "C" void framefb_frame_free(framefb_frame* f) {
  if (!f) return;
  std::free(f->csc_colptr);
  std::free(f->csc_rowidx);
  std::free(f->csc_val);
  std::free(f->csr_rowptr);
  std::free(f->csr_colidx);
  std::free(f->csr_val);
  std::free(f->grp_row0);
  std::free(f->grp_nrows);
  std::memset(f, 0, sizeof(*f));
}

// S1: (k, rho, d) tight fusion frame -- Sec. 3.2 steps (1)-(3), appendix example.
extern "C" framefb_status framefb_frame_build(int32_t d, const framefb_frame_params* params,
                                              framefb_frame* out) {
  if (!out) return FRAMEFB_EINVAL;
  std::memset(out, 0, sizeof(*out));
  if (!params) return FRAMEFB_EINVAL;
  const int32_t k = params->k, rho = params->rho;
  if (d <= 0 || (d & 1) || k < 1 || rho < 2 || (rho & 1)) return FRAMEFB_EINVAL;
  if (static_cast<int64_t>(k) * rho > (int64_t{1} << 30) || d > (1 << 30)) return FRAMEFB_EINVAL;
  const int32_t rho_c = rho / 2, d_c = d / 2;

  std::vector<double> F;
  std::vector<StRow> sup;
  try {
    if (!spectral_tetris(rho_c, d_c, F, sup)) return FRAMEFB_EUNSUPPORTED;
  } catch (const std::bad_alloc&) {
    return FRAMEFB_ENOMEM;
  }
  // Modulation is tight when no two columns of F sharing a row are congruent
  // mod k (the k-th-root sums cancel every other pair): k >= widest row support.
  for (const StRow& s : sup)
    if (s.last - s.first + 1 > k) return FRAMEFB_EUNSUPPORTED;

  const int32_t ncols = k * rho;
  int64_t nnz = 0;
  for (const StRow& s : sup) nnz += static_cast<int64_t>(k) * 2 * 2 * (s.last - s.first + 1);
  out->d = d;
  out->k = k;
  out->rho = rho;
  out->ncols = ncols;
  out->nnz = nnz;
  out->A = static_cast<double>(k) * rho / d;
  out->scale = params->parseval ? 1.0 / std::sqrt(out->A) : 1.0;
  out->ngroups = rho_c;
  out->dft_groups = (static_cast<int64_t>(k) * rho == d) ? 1 : 0;

  out->csc_colptr = alloc_array<int64_t>(ncols + 1);
  out->csc_rowidx = alloc_array<int32_t>(nnz);
  out->csc_val = alloc_array<double>(nnz);
  out->csr_rowptr = alloc_array<int64_t>(static_cast<size_t>(d) + 1);
  out->csr_colidx = alloc_array<int32_t>(nnz);
  out->csr_val = alloc_array<double>(nnz);
  out->grp_row0 = alloc_array<int32_t>(rho_c);
  out->grp_nrows = alloc_array<int32_t>(rho_c);
  if (!out->csc_colptr || !out->csc_rowidx || !out->csc_val || !out->csr_rowptr || !out->csr_colidx ||
      !out->csr_val || !out->grp_row0 || !out->grp_nrows) {
    framefb_frame_free(out);
    return FRAMEFB_ENOMEM;
  }
  for (int32_t r = 0; r < rho_c; ++r) {
    out->grp_row0[r] = 2 * sup[r].first;
    out->grp_nrows[r] = 2 * (sup[r].last - sup[r].first + 1);
  }

  // Modulation by omega^{(i j) mod k} (appendix "Modulation"), unit-norm
  // scaling by sqrt(rho_c/d_c), optional Parseval scaling, and realification
  // x + iy -> [[x, -y], [y, x]] applied to the frame-vector rows.
  const double two_pi = 6.283185307179586476925286766559;
  const double unit = std::sqrt(static_cast<double>(rho_c) / d_c) * out->scale;
  int64_t pos = 0;
  out->csc_colptr[0] = 0;
  for (int32_t c = 0; c < ncols; ++c) {
    const int32_t i = c / rho, r = (c % rho) / 2, s = c % 2;
    for (int32_t j = sup[r].first; j <= sup[r].last; ++j) {
      const double f = F[static_cast<size_t>(r) * d_c + j] * unit;
      const int64_t e = (static_cast<int64_t>(i) * j) % k;
      const double ang = two_pi * static_cast<double>(e) / k;
      const double zr = f * std::cos(ang), zi = f * std::sin(ang);
      out->csc_rowidx[pos] = 2 * j;
      out->csc_val[pos] = (s == 0) ? zr : zi;
      ++pos;
      out->csc_rowidx[pos] = 2 * j + 1;
      out->csc_val[pos] = (s == 0) ? -zi : zr;
      ++pos;
    }
    out->csc_colptr[c + 1] = pos;
  }
  // CSR by counting transpose (columns come out ascending within each row).
  std::vector<int64_t> fill(static_cast<size_t>(d) + 1, 0);
  for (int64_t q = 0; q < nnz; ++q) fill[out->csc_rowidx[q] + 1]++;
  for (int32_t j = 0; j < d; ++j) fill[j + 1] += fill[j];
  std::memcpy(out->csr_rowptr, fill.data(), (static_cast<size_t>(d) + 1) * sizeof(int64_t));
  for (int32_t c = 0; c < ncols; ++c) {
    for (int64_t q = out->csc_colptr[c]; q < out->csc_colptr[c + 1]; ++q) {
      const int64_t dst = fill[out->csc_rowidx[q]]++;
      out->csr_colidx[dst] = c;
      out->csr_val[dst] = out->csc_val[q];
    }
  }
  return FRAMEFB_OK;
}

// ---------------------------------------------------------------------------
// S2: support sampling (Sec. 3.3: random positions shared across layers).
// splitmix64 stream; uniform_int(R) = ((x >> 11) * R) >> 53 with a 128-bit
// product; uniform_01 = (x >> 11) * 2^-53; duplicates are discarded.
// ---------------------------------------------------------------------------
namespace {
struct SplitMix64 {
  uint64_t state;
  uint64_t next() {
    state += 0x9E3779B97F4A7C15ull;
    uint64_t z = state;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
  }
  uint64_t uniform_int(uint64_t r) {
    const unsigned __int128 p = static_cast<unsigned __int128>(next() >> 11) * r;
    return static_cast<uint64_t>(p >> 53);
  }
  double uniform_01() { return static_cast<double>(next() >> 11) * (1.0 / 9007199254740992.0); }
};
}  // namespace

extern "C" framefb_status framefb_support_build(int32_t rows, int32_t cols, int64_t nnz, uint64_t seed,
                                                int32_t mode, double zipf_s, int32_t k, int32_t* row,
                                                int32_t* col, int64_t* csr_rowptr, int32_t* csc_perm) {
  if (rows <= 0 || cols <= 0 || nnz < 0) return FRAMEFB_EINVAL;
  const int64_t total = static_cast<int64_t>(rows) * cols;
  if (nnz > total || nnz > (int64_t{1} << 31) - 1) return FRAMEFB_EINVAL;
  if (nnz > 0 && (!row || !col)) return FRAMEFB_EINVAL;
  if (mode == FRAMEFB_SUPPORT_BLOCKDIAG) {
    if (k < 1 || rows % k || cols % k) return FRAMEFB_EINVAL;
    if (nnz > static_cast<int64_t>(k) * (rows / k) * (cols / k)) return FRAMEFB_EINVAL;
  } else if (mode == FRAMEFB_SUPPORT_ZIPF_ROWS) {
    if (!(zipf_s > 0.0) || !std::isfinite(zipf_s)) return FRAMEFB_EINVAL;
  } else if (mode != FRAMEFB_SUPPORT_UNIFORM) {
    return FRAMEFB_EINVAL;
  }
  try {
    SplitMix64 rng{seed};
    std::vector<double> cdf;
    if (mode == FRAMEFB_SUPPORT_ZIPF_ROWS) {
      cdf.resize(rows);
      double acc = 0.0;
      for (int32_t r = 1; r <= rows; ++r) {
        acc += std::pow(static_cast<double>(r), -zipf_s);
        cdf[r - 1] = acc;
      }
    }
    std::unordered_set<uint64_t> seen;
    seen.reserve(static_cast<size_t>(nnz) * 2 + 1);
    std::vector<uint64_t> keys;
    keys.reserve(static_cast<size_t>(nnz));
    while (static_cast<int64_t>(keys.size()) < nnz) {
      uint64_t a, b;
      if (mode == FRAMEFB_SUPPORT_UNIFORM) {
        const uint64_t p = rng.uniform_int(static_cast<uint64_t>(total));
        a = p / cols;
        b = p % cols;
      } else if (mode == FRAMEFB_SUPPORT_ZIPF_ROWS) {
        const double u = rng.uniform_01() * cdf.back();
        a = static_cast<uint64_t>(std::upper_bound(cdf.begin(), cdf.end(), u) - cdf.begin());
        if (a >= static_cast<uint64_t>(rows)) a = rows - 1;
        b = rng.uniform_int(static_cast<uint64_t>(cols));
      } else {
        const uint64_t i = rng.uniform_int(static_cast<uint64_t>(k));
        const uint64_t rb = rows / k, cb = cols / k;
        a = i * rb + rng.uniform_int(rb);
        b = i * cb + rng.uniform_int(cb);
      }
      const uint64_t key = a * static_cast<uint64_t>(cols) + b;
      if (seen.insert(key).second) keys.push_back(key);
    }
    std::sort(keys.begin(), keys.end());
    for (int64_t q = 0; q < nnz; ++q) {
      row[q] = static_cast<int32_t>(keys[q] / cols);
      col[q] = static_cast<int32_t>(keys[q] % cols);
    }
    if (csr_rowptr) {
      std::fill(csr_rowptr, csr_rowptr + rows + 1, 0);
      for (int64_t q = 0; q < nnz; ++q) csr_rowptr[row[q] + 1]++;
      for (int32_t a = 0; a < rows; ++a) csr_rowptr[a + 1] += csr_rowptr[a];
    }
    if (csc_perm) {
      std::vector<int32_t> perm(static_cast<size_t>(nnz));
      for (int64_t q = 0; q < nnz; ++q) perm[q] = static_cast<int32_t>(q);
      std::sort(perm.begin(), perm.end(), [&](int32_t x, int32_t y) {
        return col[x] != col[y] ? col[x] < col[y] : row[x] < row[y];
      });
      std::memcpy(csc_perm, perm.data(), static_cast<size_t>(nnz) * sizeof(int32_t));
    }
  } catch (const std::bad_alloc&) {
    return FRAMEFB_ENOMEM;
  }
  return FRAMEFB_OK;
}

// ---------------------------------------------------------------------------
// Dense operand image of a frame (dense_layout.h).
// ---------------------------------------------------------------------------
namespace {

inline uint32_t float_bits(float x) {
  uint32_t u;
  std::memcpy(&u, &x, 4);
  return u;
}
inline float bits_float(uint32_t u) {
  float x;
  std::memcpy(&x, &u, 4);
  return x;
}
// Round to nearest, ties to even, keeping the top `keep` bits of the fp32
// pattern (finite inputs): 16 gives bf16, 19 gives tf32.
inline uint32_t round_bits(float x, int keep) {
  const int drop = 32 - keep;
  uint32_t u = float_bits(x);
  u += ((1u << (drop - 1)) - 1u) + ((u >> drop) & 1u);
  return u & ~((1u << drop) - 1u);
}

}  // namespace

extern "C" size_t framefb_frame_dense_bytes(const framefb_frame* f) {
  if (!f || f->d <= 0 || f->ncols <= 0 || !f->csc_colptr || !f->csc_rowidx || !f->csc_val) return 0;
  return static_cast<size_t>(ffb_dense_layout(f->d, f->ncols).total);
}

extern "C" framefb_status framefb_frame_dense_pack(const framefb_frame* f, void* out, size_t bytes) {
  const size_t need = framefb_frame_dense_bytes(f);
  if (need == 0 || !out || bytes < need) return FRAMEFB_EINVAL;
  const FfbDenseLayout L = ffb_dense_layout(f->d, f->ncols);
  uint8_t* base = static_cast<uint8_t*>(out);
  std::memset(base, 0, need);
  uint16_t* hi = reinterpret_cast<uint16_t*>(base + L.off_hi);
  uint16_t* lo = reinterpret_cast<uint16_t*>(base + L.off_lo);
  float* sy = reinterpret_cast<float*>(base + L.off_sy);
  for (int32_t c = 0; c < f->ncols; ++c) {
    for (int64_t e = f->csc_colptr[c]; e < f->csc_colptr[c + 1]; ++e) {
      const int32_t j = f->csc_rowidx[e];
      const double v = f->csc_val[e];
      const uint32_t h = round_bits(static_cast<float>(v), 16);
      const uint32_t l = round_bits(static_cast<float>(v - static_cast<double>(bits_float(h))), 16);
      hi[static_cast<int64_t>(c) * L.dp + j] = static_cast<uint16_t>(h >> 16);
      lo[static_cast<int64_t>(c) * L.dp + j] = static_cast<uint16_t>(l >> 16);
      sy[static_cast<int64_t>(j) * L.cp + c] = bits_float(round_bits(static_cast<float>(v), 19));
    }
  }
  return FRAMEFB_OK;
}

// ---------------------------------------------------------------------------
// Plan: the support re-indexed group-major and cut into per-thread chunks.
// ---------------------------------------------------------------------------
namespace {

// Paper column c = i*rho + 2r + s  ->  group-major x = 32 r + 2 i + s (k = 16).
inline int32_t group_major(int32_t c, int32_t rho) {
  const int32_t i = c / rho, rr = c % rho;
  return FFB_GROUP * (rr / 2) + 2 * i + (rr & 1);
}

struct Entry { int32_t key0, key1, q; };

// Banks of the default (two-token) tensor-core kernel's coefficient buffers.
// RZ / RG: 4-byte stores to the canonical K-major core-matrix layout (group
// r, coefficient c at float 256 (r / 8) + 32 (c / 4) + 4 (r % 8) + c % 4;
// overflow slots x >= K at x), bank = word mod 32 over a warp.
inline int32_t store_bank(int32_t x, int32_t K) { return x >= K ? (x & 31) : (((x >> 5) & 7) * 4 + (x & 3)); }
// V / U: 8-byte gathers (both tokens of a coefficient) from the layout in
// which group r's 16-byte chunks (two coefficients) are permuted by r mod 8:
// float2 index 32 r + 2 ((c / 2) xor (r mod 8)) + c mod 2; a half-warp's
// requests are served together, bank pair = float2 index mod 16.
inline int32_t gather_bank(int32_t x) {
  const int32_t r = x >> 5, c = x & 31;
  return (2 * ((c >> 1) ^ (r & 7)) + (c & 1)) & 15;
}

// Shared-memory banks one coefficient path touches per entry: the 8-byte
// gather of the other index and the reload of the key's own input where the
// key changes (dC, column path only), both per half-warp; the 4-byte run-sum
// stores at a piece end, per warp.
struct PathBanks {
  std::vector<int8_t> gather, key, store;  // per entry; key empty: no reload
};

// Arrange `ent` (sorted by key0, key1) into P chunks of E entries so that
// every run of equal key0 stays inside one chunk where its length allows:
// runs longer than E first fill whole chunks, then the pieces go, longest
// first, to the chunk whose free room fits them most tightly (best fit
// decreasing); a piece that fits nowhere is split over the roomiest chunks.
// The pieces are then moved (equal-length pieces swapped between chunks,
// entries reordered inside a piece) by a deterministic annealing search that
// lowers shared-memory wavefronts: for every SpMM instruction (32 consecutive
// chunks at one entry step) it counts the wavefronts of the gathers and key
// reloads (per half-warp: the largest number of lanes on one bank pair) and
// of the two run-sum stores (per warp: the largest number on one bank), plus
// a small sum-of-squares term over the same bank counts that keeps the
// search moving on plateaus of the wavefront count.  Half of the swaps start
// from a lane that conflicts in a random instruction.
// A chunk's pieces are consecutive, so each piece sums in registers and
// stores once, at its last position: the first piece of a key (in chunk
// order) writes the key's own slot, later pieces write overflow slots
// base + o, contiguous per key, which the fix-up list {key, first overflow
// slot, count, 0} adds in.  With no run longer than E and enough room,
// nothing overflows.
// Outputs: pos[p * E + e] = entry index or -1 (padding), store[entry] = its
// store target or FFB_NO_STORE.
void pack_runs(const std::vector<Entry>& ent, int32_t P, int32_t E, int32_t base, int32_t nkeys,
               const PathBanks& bk, int32_t moves, std::vector<int32_t>& pos, std::vector<int32_t>& store,
               std::vector<int32_t>& fix, int32_t& novf) {
  const int32_t nnz = static_cast<int32_t>(ent.size());
  pos.assign(static_cast<size_t>(P) * E, -1);
  store.assign(nnz, FFB_NO_STORE);
  fix.clear();
  novf = 0;
  if (nnz == 0 || E == 0) return;
  struct Piece { int32_t start, len; };
  std::vector<Piece> pieces;
  std::vector<std::vector<Piece>> chunk(P);
  std::vector<int32_t> room(P, E);
  int32_t next_full = 0;  // chunks handed out whole to long runs
  for (int32_t i = 0; i < nnz;) {
    int32_t j = i + 1;
    while (j < nnz && ent[j].key0 == ent[i].key0) ++j;
    int32_t start = i, len = j - i;
    while (len >= E && next_full < P) {
      chunk[next_full].push_back(Piece{start, E});
      room[next_full++] = 0;
      start += E;
      len -= E;
    }
    if (len > 0) pieces.push_back(Piece{start, len});
    i = j;
  }
  std::stable_sort(pieces.begin(), pieces.end(), [](const Piece& x, const Piece& y) { return x.len > y.len; });
  // bucket[c] = chunks with free room c (taken from the back)
  std::vector<std::vector<int32_t>> bucket(E + 1);
  for (int32_t c = P - 1; c >= next_full; --c) bucket[E].push_back(c);
  auto take = [&](int32_t c) {
    const int32_t id = bucket[c].back();
    bucket[c].pop_back();
    return id;
  };
  for (size_t k = 0; k < pieces.size(); ++k) {
    Piece pc = pieces[k];
    while (pc.len > 0) {
      int32_t c = pc.len;
      while (c <= E && bucket[c].empty()) ++c;
      if (c > E) {  // nowhere whole: fill the roomiest chunk and go on with the rest
        c = pc.len - 1;
        while (c > 0 && bucket[c].empty()) --c;
        if (c == 0) return;  // cannot happen: P * E >= nnz
      }
      const int32_t id = take(c);
      const int32_t put = std::min(pc.len, c);
      chunk[id].push_back(Piece{pc.start, put});
      room[id] = c - put;
      bucket[room[id]].push_back(id);
      pc.start += put;
      pc.len -= put;
    }
  }

  // placed pieces: chunk, offset, entries in order; grid of entry indices
  struct Placed { int32_t col, off, len; std::vector<int32_t> ents; };
  std::vector<Placed> pl;
  std::vector<int32_t>& grid = pos;  // [p * E + e]
  std::vector<int32_t> piece_of(nnz, -1);
  for (int32_t p = 0; p < P; ++p) {
    int32_t e = 0;
    for (const Piece& pc : chunk[p]) {
      Placed q{p, e, pc.len, {}};
      for (int32_t t = 0; t < pc.len; ++t) {
        q.ents.push_back(pc.start + t);
        grid[static_cast<size_t>(p) * E + e + t] = pc.start + t;
        piece_of[pc.start + t] = static_cast<int32_t>(pl.size());
      }
      e += pc.len;
      pl.push_back(std::move(q));
    }
  }

  // bank-conflict search.  An instruction is a group of 32 chunks at one
  // step; its bank counts (gathers and key reloads per half-warp, stores per
  // warp) are kept per instruction and updated cell by cell as pieces move.
  const bool has_key = !bk.key.empty();
  const int32_t W = (P + 31) / 32;
  struct Counts {
    uint8_t g[2][16], k[2][16], s[32];
  };
  std::vector<Counts> cnt(static_cast<size_t>(W) * E);
  std::memset(cnt.data(), 0, cnt.size() * sizeof(Counts));
  auto is_end = [&](int32_t idx, int32_t e) {
    const Placed& q = pl[piece_of[idx]];
    return q.off + q.len - 1 == e;
  };
  // add (d = 1) or remove (d = -1) what the entry at chunk p, step e puts in
  // its instruction; the key reload counts on every lane (the kernel loads it
  // on all lanes and keeps it where the key changes)
  auto cell = [&](int32_t p, int32_t e, int d) {
    const int32_t idx = grid[static_cast<size_t>(p) * E + e];
    if (idx < 0) return;
    Counts& c = cnt[static_cast<size_t>(p >> 5) * E + e];
    const int h = (p >> 4) & 1;
    c.g[h][bk.gather[idx]] = static_cast<uint8_t>(c.g[h][bk.gather[idx]] + d);
    if (has_key) c.k[h][bk.key[idx]] = static_cast<uint8_t>(c.k[h][bk.key[idx]] + d);
    if (is_end(idx, e)) c.s[bk.store[idx]] = static_cast<uint8_t>(c.s[bk.store[idx]] + d);
  };
  // 16 x wavefronts + 4 x sum of squared bank counts of one instruction
  auto cost_of = [](const Counts& c) {
    int32_t wf = 0, sq = 0;
    for (int h = 0; h < 2; ++h) {
      int32_t mg = 0, mk = 0;
      for (int b = 0; b < 16; ++b) {
        mg = std::max<int32_t>(mg, c.g[h][b]);
        mk = std::max<int32_t>(mk, c.k[h][b]);
        sq += c.g[h][b] * c.g[h][b] + c.k[h][b] * c.k[h][b];
      }
      wf += mg + mk;
    }
    int32_t ms = 0;
    for (int b = 0; b < 32; ++b) {
      ms = std::max<int32_t>(ms, c.s[b]);
      sq += 2 * c.s[b] * c.s[b];  // two stores: one per token
    }
    wf += 2 * ms;
    return 16 * wf + 4 * sq;
  };
  for (int32_t p = 0; p < P; ++p)
    for (int32_t e = 0; e < E; ++e) cell(p, e, 1);
  std::vector<int32_t> gcost(cnt.size());
  for (size_t g = 0; g < cnt.size(); ++g) gcost[g] = cost_of(cnt[g]);

  std::vector<std::vector<int32_t>> by_len(E + 1);
  std::vector<int32_t> multi;  // pieces of two or more entries
  for (size_t k = 0; k < pl.size(); ++k) {
    by_len[pl[k].len].push_back(static_cast<int32_t>(k));
    if (pl[k].len >= 2) multi.push_back(static_cast<int32_t>(k));
  }
  SplitMix64 rng{0x6A09E667F3BCC909ull ^ static_cast<uint64_t>(nnz)};
  const int64_t iters = std::min<int64_t>(static_cast<int64_t>(nnz) * moves, 60000000);
  std::vector<std::pair<int32_t, int32_t>> cells;
  std::vector<int32_t> groups, newcost;
  auto add_cell = [&](int32_t p, int32_t e) {
    cells.emplace_back(p, e);
    const int32_t g = (p >> 5) * E + e;
    if (std::find(groups.begin(), groups.end(), g) == groups.end()) groups.push_back(g);
  };
  // tries a move: `apply` performs it and, called again, undoes it
  auto attempt = [&](double T, auto&& apply) {
    int32_t before = 0;
    for (const int32_t g : groups) before += gcost[g];
    for (const auto& c : cells) cell(c.first, c.second, -1);
    apply();
    for (const auto& c : cells) cell(c.first, c.second, 1);
    int32_t after = 0;
    newcost.clear();
    for (const int32_t g : groups) {
      newcost.push_back(cost_of(cnt[g]));
      after += newcost.back();
    }
    const int32_t d = after - before;
    if (d > 0 && rng.uniform_01() >= std::exp(-d / (3.0 * T + 1e-9))) {
      for (const auto& c : cells) cell(c.first, c.second, -1);
      apply();
      for (const auto& c : cells) cell(c.first, c.second, 1);
      return;
    }
    for (size_t k = 0; k < groups.size(); ++k) gcost[groups[k]] = newcost[k];
  };
  for (int64_t it = 0; it < iters; ++it) {
    const double T = 1.0 - static_cast<double>(it) / static_cast<double>(iters);  // temperature
    cells.clear();
    groups.clear();
    const bool within = !multi.empty() && (rng.next() & 3) == 0;
    if (within) {
      // reorder two entries of one piece (one run: the key reloads stay)
      Placed& q = pl[multi[rng.uniform_int(multi.size())]];
      const int32_t i = static_cast<int32_t>(rng.uniform_int(q.len)), j = static_cast<int32_t>(rng.uniform_int(q.len));
      if (i == j) continue;
      add_cell(q.col, q.off + i);
      add_cell(q.col, q.off + j);
      attempt(T, [&]() {
        std::swap(q.ents[i], q.ents[j]);
        grid[static_cast<size_t>(q.col) * E + q.off + i] = q.ents[i];
        grid[static_cast<size_t>(q.col) * E + q.off + j] = q.ents[j];
      });
    } else {
      // swap two pieces of the same length between chunks
      int32_t a = static_cast<int32_t>(rng.uniform_int(pl.size()));
      if (rng.next() & 1) {
        // a piece holding a lane whose gather shares a bank pair in a random instruction
        const int32_t w = static_cast<int32_t>(rng.uniform_int(W)), e = static_cast<int32_t>(rng.uniform_int(E));
        const Counts& c = cnt[static_cast<size_t>(w) * E + e];
        int32_t cand[32], nc = 0;
        for (int32_t l = 0; l < 32 && 32 * w + l < P; ++l) {
          const int32_t idx = grid[static_cast<size_t>(32 * w + l) * E + e];
          if (idx >= 0 && c.g[l >> 4][bk.gather[idx]] > 1) cand[nc++] = idx;
        }
        if (nc == 0) continue;
        a = piece_of[cand[rng.uniform_int(nc)]];
      }
      const std::vector<int32_t>& same = by_len[pl[a].len];
      if (same.size() < 2) continue;
      const int32_t b = same[rng.uniform_int(same.size())];
      if (a == b || pl[a].col == pl[b].col) continue;
      for (int32_t t = 0; t < pl[a].len; ++t) {
        add_cell(pl[a].col, pl[a].off + t);
        add_cell(pl[b].col, pl[b].off + t);
      }
      attempt(T, [&]() {
        std::swap(pl[a].col, pl[b].col);
        std::swap(pl[a].off, pl[b].off);
        for (const int32_t k : {a, b})
          for (int32_t t = 0; t < pl[k].len; ++t) grid[static_cast<size_t>(pl[k].col) * E + pl[k].off + t] = pl[k].ents[t];
      });
    }
  }

  // own / overflow targets: the first piece of a key in chunk order owns the key's slot
  std::vector<int32_t> order(pl.size());
  for (size_t k = 0; k < pl.size(); ++k) order[k] = static_cast<int32_t>(k);
  std::sort(order.begin(), order.end(), [&](int32_t x, int32_t y) {
    return pl[x].col != pl[y].col ? pl[x].col < pl[y].col : pl[x].off < pl[y].off;
  });
  std::vector<int32_t> owner(nkeys, -1), n_ovf(nkeys, 0), first_ovf(nkeys, 0), used(nkeys, 0);
  for (const int32_t k : order) {
    const int32_t key = ent[pl[k].ents[0]].key0;
    if (owner[key] < 0)
      owner[key] = k;
    else
      ++n_ovf[key];
  }
  for (int32_t key = 0; key < nkeys; ++key) {
    if (n_ovf[key] == 0) continue;
    first_ovf[key] = novf;
    fix.push_back(key);
    fix.push_back(base + novf);
    fix.push_back(n_ovf[key]);
    fix.push_back(0);
    novf += n_ovf[key];
  }
  for (const int32_t k : order) {
    const int32_t last = pl[k].ents[pl[k].len - 1];
    const int32_t key = ent[last].key0;
    store[last] = owner[key] == k ? key : base + first_ovf[key] + used[key]++;
  }
}

inline int32_t align16(size_t x) { return static_cast<int32_t>((x + 15) & ~size_t{15}); }

}  // namespace

namespace {

// Plan image of the entries byrow (key0 = row a, key1 = column b, q = the
// entry's index into the caller's C values and dC) and bycol (key0 = b,
// key1 = a) over index spaces n (columns) and m (rows): chunks cut for
// FRAMEFB_THREADS threads, store targets, fix-ups, group masks, merge block
// lists.  nnz_full: the size of the q index space (the caller's nnz).
// moves: moves per entry of the bank-placement search (0: none; the
// default kernel's structured plans).
framefb_status build_plan_image(int32_t n, int32_t m, bool structured, int32_t moves, int32_t d_in, int32_t d_out,
                                std::vector<Entry>& byrow, std::vector<Entry>& bycol, int32_t nnz_full,
                                std::vector<uint8_t>& image) {
  const int32_t P = FRAMEFB_THREADS;
  const int32_t nz = static_cast<int32_t>(byrow.size());
  const int32_t Gn = (n + FFB_GROUP - 1) / FFB_GROUP, Gm = (m + FFB_GROUP - 1) / FFB_GROUP;
  auto lt = [](const Entry& x, const Entry& y) { return x.key0 != y.key0 ? x.key0 < y.key0 : x.key1 < y.key1; };
  std::sort(byrow.begin(), byrow.end(), lt);
  std::sort(bycol.begin(), bycol.end(), lt);
  const int32_t EZ = (nz + P - 1) / P, EG = EZ;

  std::vector<int32_t> posZ, storeZ, fixZ, posG, storeG, fixG;
  int32_t novfZ = 0, novfG = 0;
  // banks of the default kernel's slots: row path gathers V[b] and stores
  // Z[a]; column path gathers U[a], reloads V[b] where b changes and stores
  // G[b]
  PathBanks bkZ, bkG;
  bkZ.gather.resize(nz);
  bkZ.store.resize(nz);
  for (int32_t q = 0; q < nz; ++q) {
    bkZ.gather[q] = static_cast<int8_t>(gather_bank(byrow[q].key1));
    bkZ.store[q] = static_cast<int8_t>(store_bank(byrow[q].key0, m));
  }
  bkG.gather.resize(nz);
  bkG.key.resize(nz);
  bkG.store.resize(nz);
  for (int32_t q = 0; q < nz; ++q) {
    bkG.gather[q] = static_cast<int8_t>(gather_bank(bycol[q].key1));
    bkG.key[q] = static_cast<int8_t>(gather_bank(bycol[q].key0));
    bkG.store[q] = static_cast<int8_t>(store_bank(bycol[q].key0, n));
  }
  // the two paths are independent searches: run them side by side (in
  // sequence if no thread can be started); exceptions reach the caller's
  // handler after the join
  {
    std::exception_ptr ez, eg;
    auto run_z = [&]() {
      try {
        pack_runs(byrow, P, EZ, m, m, bkZ, moves, posZ, storeZ, fixZ, novfZ);
      } catch (...) {
        ez = std::current_exception();
      }
    };
    std::thread tz;
    try {
      tz = std::thread(run_z);
    } catch (const std::system_error&) {
      run_z();
    }
    try {
      pack_runs(bycol, P, EG, n, n, bkG, moves, posG, storeG, fixG, novfG);
    } catch (...) {
      eg = std::current_exception();
    }
    if (tz.joinable()) tz.join();
    if (ez) std::rethrow_exception(ez);
    if (eg) std::rethrow_exception(eg);
  }

  // store targets (own slots and overflow slots) are 16-bit fields
  if (m + novfZ >= static_cast<int32_t>(FFB_NO_STORE) || n + novfG >= static_cast<int32_t>(FFB_NO_STORE))
    return FRAMEFB_EUNSUPPORTED;
  FfbPlanHeader h;
  std::memset(&h, 0, sizeof(h));
  h.layout = structured ? FFB_LAYOUT_GROUPS : FFB_LAYOUT_DENSE;
  h.d_in = d_in;
  h.d_out = d_out;
  h.magic = FFB_PLAN_MAGIC;
  h.version = FFB_PLAN_VERSION;
  h.n = n;
  h.m = m;
  h.Gn = Gn;
  h.Gm = Gm;
  h.nnz = nz;
  h.P = P;
  h.EZ = EZ;
  h.EG = EG;
  h.ovfZ = (novfZ + 3) & ~3;
  h.ovfG = (novfG + 3) & ~3;
  h.nfixZ = static_cast<int32_t>(fixZ.size() / 4);
  h.nfixG = static_cast<int32_t>(fixG.size() / 4);
  h.nnz_full = nnz_full;

  size_t off = align16(sizeof(FfbPlanHeader));
  auto take = [&](size_t bytes) { const int32_t o = static_cast<int32_t>(off); off = align16(off + bytes); return o; };
  const size_t ezp = static_cast<size_t>(EZ) * P, egp = static_cast<size_t>(EG) * P;
  h.off_zb = take(ezp * 4);
  h.off_zq = take(ezp * 4);
  h.off_ga = take(egp * 4);
  h.off_gb = take(egp * 4);
  h.off_gq = take(egp * 4);
  h.off_fixZ = take(fixZ.size() * 4);
  h.off_fixG = take(fixG.size() * 4);
  h.off_zmask = take(static_cast<size_t>(Gm) * 4);
  h.off_gmask = take(static_cast<size_t>(Gn) * 4);
  const size_t nblk = static_cast<size_t>(Gm) * Gn;
  h.off_blkptr = take((nblk + 1) * 4);
  h.off_blkent = take(static_cast<size_t>(nz) * 8);
  if (off > static_cast<size_t>(INT32_MAX)) return FRAMEFB_EUNSUPPORTED;
  h.total_bytes = static_cast<int32_t>(off);

  image.assign(off, 0);
  uint8_t* base = image.data();
  auto arr = [&](int32_t o) { return reinterpret_cast<int32_t*>(base + o); };
  std::memcpy(base, &h, sizeof(h));

  // Per-thread chunk tables, entry-major ([e][p]) so that a warp reading
  // entry e of its 32 threads touches 128 contiguous bytes.
  int32_t* zb = arr(h.off_zb);
  int32_t* zq = arr(h.off_zq);
  int32_t* ga = arr(h.off_ga);
  int32_t* gb = arr(h.off_gb);
  int32_t* gq = arr(h.off_gq);
  for (int32_t p = 0; p < P; ++p) {
    for (int32_t e = 0; e < EZ; ++e) {
      const int32_t idx = posZ[static_cast<size_t>(p) * EZ + e];
      const size_t slot = static_cast<size_t>(e) * P + p;
      if (idx >= 0) {
        zb[slot] = byrow[idx].key1 | ((byrow[idx].key0 & 1) << 15) | (storeZ[idx] << 16);
        zq[slot] = byrow[idx].q;
      } else {
        zb[slot] = (FFB_NO_STORE << 16);
        zq[slot] = -1;
      }
    }
    for (int32_t e = 0; e < EG; ++e) {
      const int32_t idx = posG[static_cast<size_t>(p) * EG + e];
      const size_t slot = static_cast<size_t>(e) * P + p;
      if (idx >= 0) {
        ga[slot] = bycol[idx].key1 | ((bycol[idx].key0 & 1) << 15) | (storeG[idx] << 16);
        gb[slot] = bycol[idx].key0;
        gq[slot] = bycol[idx].q;
      } else {
        ga[slot] = (FFB_NO_STORE << 16);
        gb[slot] = 0;
        gq[slot] = -1;
      }
    }
  }
  if (!fixZ.empty()) std::memcpy(arr(h.off_fixZ), fixZ.data(), fixZ.size() * 4);
  if (!fixG.empty()) std::memcpy(arr(h.off_fixG), fixG.data(), fixG.size() * 4);
  uint32_t* zmask = reinterpret_cast<uint32_t*>(arr(h.off_zmask));
  uint32_t* gmask = reinterpret_cast<uint32_t*>(arr(h.off_gmask));
  for (int32_t q = 0; q < nz; ++q) {
    zmask[byrow[q].key0 >> 5] |= 1u << (byrow[q].key0 & 31);
    gmask[bycol[q].key0 >> 5] |= 1u << (bycol[q].key0 & 31);
  }
  // Merge: entries grouped by 32 x 32 block (out group g, in group h).
  int32_t* blkptr = arr(h.off_blkptr);
  int32_t* blkent = arr(h.off_blkent);
  std::vector<int32_t> cnt(nblk + 1, 0);
  for (int32_t q = 0; q < nz; ++q) cnt[static_cast<size_t>(byrow[q].key0 >> 5) * Gn + (byrow[q].key1 >> 5) + 1]++;
  for (size_t b = 0; b < nblk; ++b) cnt[b + 1] += cnt[b];
  std::memcpy(blkptr, cnt.data(), (nblk + 1) * 4);
  for (int32_t q = 0; q < nz; ++q) {  // byrow is sorted by (a, b): entries stay ordered inside a block
    const size_t b = static_cast<size_t>(byrow[q].key0 >> 5) * Gn + (byrow[q].key1 >> 5);
    const int32_t dst = cnt[b]++;
    blkent[2 * dst] = (byrow[q].key0 & 31) | ((byrow[q].key1 & 31) << 8);
    blkent[2 * dst + 1] = byrow[q].q;
  }
  return FRAMEFB_OK;
}

// Sub-plans of a structured plan beyond the fused tcgen05 kernels' limits
// (more than kSubEntries entries, so longer chunks than the register chunk,
// or an output side of more than kSubGroups groups): the output side cut
// into blocks of whole groups (at most kSubGroups, a multiple of 8), and the
// entries of a block, in row-major order, into runs of at most kSubEntries.  A
// sub-plan is the plan of its run over its two blocks (group-major indices
// less the blocks' first columns) and keeps the caller's entry indices q.
constexpr int32_t kSubGroups = 128;
constexpr int32_t kSubEntries = 16 * FRAMEFB_THREADS;
// moves per entry of the bank-placement search: a whole plan, a part
constexpr int32_t kMovesWhole = 4000, kMovesPart = 1500;

struct Block { int32_t g0, g1; };  // groups [g0, g1)

std::vector<Block> side_blocks(int32_t G) {
  const int32_t nb = (G + kSubGroups - 1) / kSubGroups;
  const int32_t w = ((G + nb - 1) / nb + 7) / 8 * 8;
  std::vector<Block> out;
  for (int32_t g0 = 0; g0 < G; g0 += w) out.push_back(Block{g0, std::min(G, g0 + w)});
  return out;
}

inline size_t align256(size_t x) { return (x + 255) & ~size_t{255}; }

}  // namespace

extern "C" framefb_status framefb_plan_build(const framefb_frame* fin, const framefb_frame* fout,
                                             const int32_t* row, const int32_t* col, int64_t nnz,
                                             framefb_plan** out) {
  if (!out) return FRAMEFB_EINVAL;
  *out = nullptr;
  if (!fin || !fout || nnz < 0 || (nnz > 0 && (!row || !col))) return FRAMEFB_EINVAL;
  if (fin->ncols <= 0 || fout->ncols <= 0 || fin->d <= 0 || fout->d <= 0) return FRAMEFB_EINVAL;
  // structured kernels: both frames k = 16 with k*rho = d (32-coordinate
  // DFT_16 groups); every other frame pair goes to the dense path
  auto groups16 = [](const framefb_frame* f) {
    return f->dft_groups && f->k == 16 && f->ncols == f->d && f->d % FFB_GROUP == 0;
  };
  const bool structured = groups16(fin) && groups16(fout);
  const int32_t n = fin->ncols, m = fout->ncols;            // index spaces K_n, K_m
  if (n > 32768 || m > 32768) return FRAMEFB_EUNSUPPORTED;  // 15-bit indices, 16-bit store targets
  if (nnz > static_cast<int64_t>(m) * n || nnz > (1 << 24)) return FRAMEFB_EINVAL;
  const int32_t nz = static_cast<int32_t>(nnz);
  for (int32_t q = 0; q < nz; ++q) {
    if (row[q] < 0 || row[q] >= m || col[q] < 0 || col[q] >= n) return FRAMEFB_EINVAL;
    if (q > 0) {
      const int64_t prev = static_cast<int64_t>(row[q - 1]) * n + col[q - 1];
      const int64_t cur = static_cast<int64_t>(row[q]) * n + col[q];
      if (cur <= prev) return FRAMEFB_EINVAL;  // not sorted row-major or duplicated
    }
  }
  try {
    std::vector<Entry> byrow(nz), bycol(nz);
    for (int32_t q = 0; q < nz; ++q) {
      const int32_t a = structured ? group_major(row[q], fout->rho) : row[q];
      const int32_t b = structured ? group_major(col[q], fin->rho) : col[q];
      byrow[q] = Entry{a, b, q};
      bycol[q] = Entry{b, a, q};
    }
    const std::vector<Entry> ent = byrow;  // (a, b, q) in the caller's order
    const int32_t Gn = (n + FFB_GROUP - 1) / FFB_GROUP, Gm = (m + FFB_GROUP - 1) / FFB_GROUP;
    // the fused tcgen05 kernels take the plan whole, or run its parts (the
    // whole plan then serves the other kernels only: no bank placement).
    // Parts need the input side in one block: blocks of the input side would
    // each hold a partial sum of every row's entries, and the bf16 output
    // rounded once per part would then lose more than the tolerance of the
    // bf16 path where a row's partial sums are larger than its sum
    // (heavy-tailed supports); runs of entries keep a row together but for
    // the row at a run boundary.
    const bool parts = structured && nz > 0 && Gn <= kSubGroups && (nz > kSubEntries || Gm > kSubGroups);
    std::vector<uint8_t> image;
    framefb_status st =
        build_plan_image(n, m, structured, structured && !parts ? kMovesWhole : 0, fin->d, fout->d, byrow, bycol, nz, image);
    if (st != FRAMEFB_OK) return st;
    framefb_plan* plan = new framefb_plan;
    std::unique_ptr<framefb_plan> guard(plan);
    plan->image = std::move(image);
    if (parts) {
      const std::vector<Block> bo = side_blocks(Gm), bi = side_blocks(Gn);
      // the parts' entries first; their plans are built side by side
      struct Job { std::vector<Entry> r, c, blk; int32_t n0, m0, nv, mv; std::vector<uint8_t> image; framefb_status st; };
      std::vector<Job> jobs;
      for (const Block& ob : bo) {
        for (const Block& ib : bi) {
          std::vector<Entry> blk;  // (a, b, q) of the block pair, block-local indices
          for (const Entry& e : ent) {
            const int32_t ga = e.key0 / FFB_GROUP, gb = e.key1 / FFB_GROUP;
            if (ga >= ob.g0 && ga < ob.g1 && gb >= ib.g0 && gb < ib.g1)
              blk.push_back(Entry{e.key0 - FFB_GROUP * ob.g0, e.key1 - FFB_GROUP * ib.g0, e.q});
          }
          if (blk.empty()) continue;
          std::sort(blk.begin(), blk.end(), [](const Entry& x, const Entry& y) {
            return x.key0 != y.key0 ? x.key0 < y.key0 : x.key1 < y.key1;
          });
          const int32_t cnt = static_cast<int32_t>(blk.size());
          const int32_t runs = (cnt + kSubEntries - 1) / kSubEntries;
          for (int32_t r = 0; r < runs; ++r) {
            const int32_t e0 = static_cast<int32_t>(static_cast<int64_t>(cnt) * r / runs);
            const int32_t e1 = static_cast<int32_t>(static_cast<int64_t>(cnt) * (r + 1) / runs);
            Job jb;
            jb.r.assign(blk.begin() + e0, blk.begin() + e1);
            jb.c.resize(jb.r.size());
            for (size_t i = 0; i < jb.r.size(); ++i) jb.c[i] = Entry{jb.r[i].key1, jb.r[i].key0, jb.r[i].q};
            jb.blk = jb.r;  // (a, b, q) in row-major order: the part's entry list
            jb.n0 = FFB_GROUP * ib.g0;
            jb.m0 = FFB_GROUP * ob.g0;
            jb.nv = FFB_GROUP * (ib.g1 - ib.g0);
            jb.mv = FFB_GROUP * (ob.g1 - ob.g0);
            jb.st = FRAMEFB_OK;
            jobs.push_back(std::move(jb));
          }
        }
      }
      {
        std::vector<std::exception_ptr> err(jobs.size());
        auto work = [&](size_t i) {
          try {
            Job& jb = jobs[i];
            jb.st = build_plan_image(jb.nv, jb.mv, true, kMovesPart, fin->d, fout->d, jb.r, jb.c, nz, jb.image);
          } catch (...) {
            err[i] = std::current_exception();
          }
        };
        const size_t hw = std::max<size_t>(1, std::thread::hardware_concurrency() / 2);  // each build runs two threads
        std::vector<std::thread> pool;
        std::atomic<size_t> next{0};
        auto loop = [&]() {
          for (size_t i = next++; i < jobs.size(); i = next++) work(i);
        };
        for (size_t t = 0; t + 1 < std::min(hw, jobs.size()); ++t) {
          try {
            pool.emplace_back(loop);
          } catch (const std::system_error&) {
            break;
          }
        }
        loop();
        for (std::thread& t : pool) t.join();
        for (const std::exception_ptr& e : err)
          if (e) std::rethrow_exception(e);
      }
      for (Job& jb : jobs) {
        if (jb.st != FRAMEFB_OK) return jb.st;
        FfbSubPlan sp{};
        sp.plan = new framefb_plan;
        std::unique_ptr<framefb_plan> sguard(sp.plan);
        sp.plan->image = std::move(jb.image);
        sp.n0 = jb.n0;
        sp.m0 = jb.m0;
        sp.nq = static_cast<int32_t>(jb.blk.size());
        // the part's image ends with its entries' q; it sits in the device
        // image after the whole plan, 256-byte aligned
        std::vector<uint8_t>& pim = sp.plan->image;
        const size_t qo = (pim.size() + 15) & ~size_t{15};
        if (qo + 4 * static_cast<size_t>(sp.nq) > static_cast<size_t>(INT32_MAX)) return FRAMEFB_EUNSUPPORTED;
        pim.resize(qo + 4 * static_cast<size_t>(sp.nq), 0);
        int32_t* ql = reinterpret_cast<int32_t*>(pim.data() + qo);
        for (int32_t i = 0; i < sp.nq; ++i) ql[i] = jb.blk[i].q;
        FfbPlanHeader* ph = reinterpret_cast<FfbPlanHeader*>(pim.data());
        ph->off_qlist = static_cast<int32_t>(qo);
        ph->total_bytes = static_cast<int32_t>(pim.size());
        sp.dev_off = align256(plan->image.size());
        sp.q_off = sp.dev_off + qo;
        plan->image.resize(sp.dev_off + pim.size(), 0);
        std::memcpy(plan->image.data() + sp.dev_off, pim.data(), pim.size());
        plan->subs.push_back(sp);
        sguard.release();
      }
    }
    *out = guard.release();
  } catch (const std::bad_alloc&) {
    return FRAMEFB_ENOMEM;
  }
  return FRAMEFB_OK;
}

extern "C" int32_t framefb_plan_parts(const framefb_plan* plan, framefb_plan_part* parts, int32_t max_parts) {
  if (!plan) return 0;
  const int32_t n = static_cast<int32_t>(plan->subs.size());
  for (int32_t i = 0; i < n && i < max_parts && parts; ++i) {
    const FfbSubPlan& sp = plan->subs[i];
    const FfbPlanHeader* h = reinterpret_cast<const FfbPlanHeader*>(sp.plan->image.data());
    parts[i].image_offset = static_cast<int64_t>(sp.dev_off);
    parts[i].image_bytes = static_cast<int64_t>(sp.plan->image.size());
    parts[i].q_offset = static_cast<int64_t>(sp.q_off);
    parts[i].nnz = sp.nq;
    parts[i].n0 = sp.n0;
    parts[i].m0 = sp.m0;
    parts[i].n = h->n;
    parts[i].m = h->m;
  }
  return n;
}

extern "C" size_t framefb_plan_bytes(const framefb_plan* plan) { return plan ? plan->image.size() : 0; }
extern "C" const void* framefb_plan_data(const framefb_plan* plan) { return plan ? plan->image.data() : nullptr; }
extern "C" void framefb_plan_free(framefb_plan* plan) { delete plan; }
