// Launchers of libframefb: argument validation, tiling, workspace sizing and
// the launches of the tile, dC-reduction and merge kernels.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "framefb.h"
#include "framefb_dense.h"
#include "framefb_kernels.cuh"
#include "framefb_mma.cuh"
#include "framefb_tc.cuh"
#include "framefb_tc2.cuh"
#include "framefb_tc2p.cuh"
#include "plan_internal.h"
#include "plan_layout.h"

namespace {

using ffb::kMaxMats;

// kernel parameters of the tensor-core launches (CUDA 12.1+: 32764 bytes)
static_assert(sizeof(ffb::TcLaunchK) <= 32764, "tensor-core launch parameters exceed the parameter space");
using ffb::kThreads;
using ffb::kTmax;

constexpr int kSmemBudget = 227 * 1024;  // dynamic shared memory per CTA on sm_103a

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

const FfbPlanHeader* plan_header(const framefb_plan* p) {
  if (!p || p->image.size() < sizeof(FfbPlanHeader)) return nullptr;
  const FfbPlanHeader* h = reinterpret_cast<const FfbPlanHeader*>(p->image.data());
  if (h->magic != FFB_PLAN_MAGIC || h->version != FFB_PLAN_VERSION || h->P != kThreads) return nullptr;
  if (static_cast<size_t>(h->total_bytes) > p->image.size()) return nullptr;  // (parts follow the plan)
  return h;
}

// Plan of the structured kernels (group-major index space), else NULL.
const FfbPlanHeader* groups_header(const framefb_plan* p) {
  const FfbPlanHeader* h = plan_header(p);
  return h && h->layout == FFB_LAYOUT_GROUPS ? h : nullptr;
}

bool frame_ok(const framefb_dev_frame* f, int32_t d) {
  return f && f->dft_groups && f->k == 16 && f->d == d && f->ncols == d && f->rho * 16 == d && f->val &&
         f->colptr && f->rowidx;
}

struct Prepared {
  ffb::LaunchK* args;  // heap: too large for the stack of some callers
  ffb::TcLaunchK* tcargs;
  ffb::ReduceK* red;
  int grid;
  size_t smem;
  size_t ws_bytes;
  bool reg;
  bool tc;    // bf16: pipelined kernel on tcgen05 tensor cores
  bool tc2;   // bf16: the same, two tokens per unit
  bool pack;  // tc2: some matrix packs several token pairs per unit
  bool seg;   // tc2: the launch carries a segment table (mixed tenants)
  int T;      // tile tokens of the bf16 kernel
  int threads;
};

void* tc_kernel_ptr(int mode) {
  switch (mode) {
    case 1: return reinterpret_cast<void*>(ffb::tc_tile_kernel<1>);
    case 2: return reinterpret_cast<void*>(ffb::tc_tile_kernel<2>);
    case 4: return reinterpret_cast<void*>(ffb::tc_tile_kernel<4>);
    case 6: return reinterpret_cast<void*>(ffb::tc_tile_kernel<6>);
    case 7: return reinterpret_cast<void*>(ffb::tc_tile_kernel<7>);
    default: return nullptr;
  }
}

// forward of the two-token kernels with a segment table (mixed tenants)
void* tc2_seg_kernel_ptr(bool pack) {
  return pack ? reinterpret_cast<void*>(ffb::tc2p_tile_kernel<1, true>)
              : reinterpret_cast<void*>(ffb::tc2_tile_kernel<1, true>);
}

// two-token kernel, or its packed form (several token pairs per unit)
void* tc2_kernel_ptr(int mode, bool pack) {
#define FFB_TC2(M) \
  case M:          \
    return pack ? reinterpret_cast<void*>(ffb::tc2p_tile_kernel<M>) : reinterpret_cast<void*>(ffb::tc2_tile_kernel<M>);
  switch (mode) {
    FFB_TC2(1)
    FFB_TC2(2)
    FFB_TC2(4)
    FFB_TC2(6)
    FFB_TC2(7)
    default: return nullptr;
  }
#undef FFB_TC2
}

// Token pairs per slot of the two-token kernel for a plan: P tokens of a
// slot share one 128-lane tile (lane p G + g), so P G <= 128 on both sides;
// at most kTc2MaxPairs; 1 for plans with more entries per chunk than the
// packed kernel holds in registers.
constexpr int kTc2MaxPairs = 8;
int tc2_pairs(const FfbPlanHeader& h) {
  if (h.EZ > ffb::kEregPack || h.EG > ffb::kEregPack) return 1;
  const int G = std::max(h.Gn, h.Gm);
  return std::max(1, std::min(kTc2MaxPairs, 128 / std::max(G, 1)));
}
bool pack_allowed() {
  const char* e = std::getenv("FRAMEFB_PACK");
  return !(e && std::strcmp(e, "0") == 0);
}

// bf16 activations: tensor-core kernel with staged rows (tile of T = 1 or 2
// tokens); fp32: exact FFT kernel.
void* tile_kernel_ptr(framefb_dtype dt, int mode, bool reg, int T) {
#define FFB_MMA(M) \
  case M:          \
    return reg ? (T == 2 ? reinterpret_cast<void*>(ffb::mma_tile_kernel<M, true, 2>)            \
                         : reinterpret_cast<void*>(ffb::mma_tile_kernel<M, true, 1>))           \
               : (T == 2 ? reinterpret_cast<void*>(ffb::mma_tile_kernel<M, false, 2>)           \
                         : reinterpret_cast<void*>(ffb::mma_tile_kernel<M, false, 1>));
#define FFB_FFT(M) \
  case M:          \
    return reg ? reinterpret_cast<void*>(ffb::fft_tile_kernel<M, true>) : reinterpret_cast<void*>(ffb::fft_tile_kernel<M, false>);
  if (dt == FRAMEFB_BF16) {
    if (T != 1 && T != 2) return nullptr;
    switch (mode) {
      FFB_MMA(1)
      FFB_MMA(2)
      FFB_MMA(4)
      FFB_MMA(6)
      FFB_MMA(7)
      default: return nullptr;
    }
  }
  switch (mode) {
    FFB_FFT(1)
    FFB_FFT(2)
    FFB_FFT(4)
    FFB_FFT(6)
    FFB_FFT(7)
    default: return nullptr;
  }
#undef FFB_MMA
#undef FFB_FFT
}

inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Shared-memory map of the bf16 kernel for a uniform tile of T tokens: the
// input rows (X, dY), the output rows (Y, dX) when stage_out, the fp32 tile
// layout (largest over the matrices), two mbarriers.  Each region is sized
// for the largest matrix; a matrix packs its rows from the region's start.
// Returns the total bytes.
size_t mma_smem_map(const framefb_mat* mats, int32_t nmats, int32_t ops, bool reg, int T, bool stage_out,
                    ffb::LaunchK* a) {
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  size_t in = 0, out = 0, fp32 = 0;
  for (int32_t j = 0; j < nmats; ++j) {
    const FfbPlanHeader* h = plan_header(mats[j].plan);
    const size_t rx = round_up(2 * static_cast<size_t>(h->n), 128), ry = round_up(2 * static_cast<size_t>(h->m), 128);
    in = std::max(in, T * (((F || C) ? rx : 0) + ((D || C) ? ry : 0)));
    if (stage_out) out = std::max(out, T * ((F ? ry : 0) + (D ? rx : 0)));
    fp32 = std::max<size_t>(fp32, static_cast<size_t>(ffb_tile_layout(*h, ops, T, C).total) * 4);
  }
  const size_t fbase = round_up(in + out, 128);
  const size_t mbar = round_up(fbase + fp32, 16);
  if (a) {
    a->stg_in = 0;
    a->stg_out = static_cast<int32_t>(in);
    a->stage_out = stage_out ? 1 : 0;
    a->fbase = static_cast<int32_t>(fbase);
    a->mbar = static_cast<int32_t>(mbar);
  }
  return mbar + 16;
}

// Shared-memory map of the tensor-core pipelined kernel: a ring of S stages
// (one token row of X then dY, each landed by a tensor copy as a swizzled
// K-major operand padded to whole 128-group tiles), B operands (8 KB), two
// fp32 sets in the canonical tf32 layout (RZ / RG padded to whole tiles), the
// fix-up item cache, S + 1 mbarriers.  Returns the total bytes, or 0 when a
// matrix does not fit the kernel's shape rules.
size_t tc_smem_map(const framefb_mat* mats, int32_t nmats, int32_t ops, int S, ffb::TcLaunchK* a) {
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  const bool needV = F || C, needU = D || C;
  size_t nfix = 0;
  int32_t nmax = 0, mmax = 0, ovfZ = 0, ovfG = 0;
  for (int32_t j = 0; j < nmats; ++j) {
    const FfbPlanHeader* h = plan_header(mats[j].plan);
    if (h->Gn % 8 || h->Gm % 8 || h->Gn > 128 * ffb::kTcMaxTiles || h->Gm > 128 * ffb::kTcMaxTiles) return 0;
    nmax = std::max(nmax, h->n);
    mmax = std::max(mmax, h->m);
    ovfZ = std::max(ovfZ, h->ovfZ);
    ovfG = std::max(ovfG, h->ovfG);
    nfix = std::max<size_t>(nfix, (F ? h->nfixZ : 0) + (D ? h->nfixG : 0));
  }
  auto tiles = [](int32_t d) { return static_cast<size_t>((d / 32 + 127) / 128); };
  const size_t xbox = needV ? tiles(nmax) * 8192 : 0;
  const size_t stage = xbox + (needU ? tiles(mmax) * 8192 : 0);
  const size_t bops = S * stage;
  const size_t fbase = bops + 8192;
  // set layout (floats)
  const size_t oU = needV ? nmax : 0;
  const size_t oRZ = round_up(oU + (needU ? mmax : 0), 32);
  const size_t szRZ = F ? round_up(std::max<size_t>(tiles(mmax) * 128 * 32, mmax + ovfZ), 32) : 0;
  const size_t oRG = oRZ + szRZ;
  const size_t szRG = D ? round_up(std::max<size_t>(tiles(nmax) * 128 * 32, nmax + ovfG), 32) : 0;
  const size_t set = oRG + szRG;
  const size_t fixc = fbase + 2 * set * 4;
  const size_t mbar = round_up(fixc + 16 * nfix, 16);
  if (a) {
    a->S = S;
    a->stage = static_cast<int32_t>(stage);
    a->xbox_u = static_cast<int32_t>(xbox);
    a->bops = static_cast<int32_t>(bops);
    a->fbase = static_cast<int32_t>(fbase);
    a->set_oU = static_cast<int32_t>(oU);
    a->set_oRZ = static_cast<int32_t>(oRZ);
    a->set_oRG = static_cast<int32_t>(oRG);
    a->set_total = static_cast<int32_t>(set);
    a->fixc = static_cast<int32_t>(fixc);
    a->fixc_items = static_cast<int32_t>(nfix);
    a->mbar = static_cast<int32_t>(mbar);
  }
  return mbar + 8 * static_cast<size_t>(S + 1);
}

// Shared-memory map of the two-token tensor-core kernel and its packed
// form: a ring of S stages (two slots of X rows, then two of dY, each a
// swizzled K-major operand of one 128-lane tile: one token row, or P of them
// when packed), B operands (8 KB), the V/U sets (float2 per coefficient:
// both tokens of a pair; unpacked: V over the largest n, then U; packed: one
// set of n + m per pair), one RZ/RG set per slot in the canonical tf32
// layout (P canonical blocks padded to a whole tile, then the pairs'
// overflow slots), the fix-up item cache, S + 2 mbarriers.  P of matrix j is
// pairs[j] (all 1 unless pack).  Returns the total bytes, or 0 when a matrix
// does not fit the shape rules (group counts a multiple of 8 and at most
// 128, P G <= 128).
size_t tc2_smem_map(const framefb_mat* mats, int32_t nmats, int32_t ops, int S, const int* pairs, bool pack,
                    ffb::TcLaunchK* a) {
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  const bool needV = F || C, needU = D || C;
  size_t nfix = 0, vuset = 0, szRZ = 0, szRG = 0;
  int32_t nmax = 0, mmax = 0;
  for (int32_t j = 0; j < nmats; ++j) {
    const FfbPlanHeader* h = plan_header(mats[j].plan);
    const size_t P = static_cast<size_t>(pairs[j]);
    if (h->Gn % 8 || h->Gm % 8 || h->Gn > 128 || h->Gm > 128) return 0;
    if (P < 1 || (!pack && P != 1) || P * h->Gn > 128 || P * h->Gm > 128) return 0;
    nmax = std::max(nmax, h->n);
    mmax = std::max(mmax, h->m);
    vuset = std::max(vuset, P * static_cast<size_t>(h->n + h->m));
    if (F) szRZ = std::max(szRZ, P * static_cast<size_t>(h->m + h->ovfZ));
    if (D) szRG = std::max(szRG, P * static_cast<size_t>(h->n + h->ovfG));
    nfix = std::max<size_t>(nfix, (F ? h->nfixZ : 0) + (D ? h->nfixG : 0));
  }
  const size_t tok_x = needV ? 8192 : 0, tok_u = needU ? 8192 : 0;
  const size_t stage = 2 * tok_x + 2 * tok_u;
  const size_t bops = S * stage;
  const size_t vu = bops + 8192;
  const size_t oU = pack ? 0 : (needV ? nmax : 0);  // float2 units; packed: per matrix
  if (!pack) vuset = oU + (needU ? mmax : 0);
  const size_t rzg = vu + round_up(vuset * 8, 128);
  szRZ = F ? round_up(std::max<size_t>(128 * 32, szRZ), 32) : 0;
  szRG = D ? round_up(std::max<size_t>(128 * 32, szRG), 32) : 0;
  const size_t rzg_tok = szRZ + szRG;  // floats
  const size_t fixc = rzg + 2 * rzg_tok * 4;
  const size_t mbar = round_up(fixc + 16 * nfix, 16);
  if (a) {
    a->S = S;
    a->stage = static_cast<int32_t>(stage);
    a->xbox_u = static_cast<int32_t>(2 * tok_x);
    a->tok_x = static_cast<int32_t>(tok_x);
    a->tok_u = static_cast<int32_t>(tok_u);
    a->bops = static_cast<int32_t>(bops);
    a->vu = static_cast<int32_t>(vu);
    a->set_oU = static_cast<int32_t>(oU);
    a->rzg = static_cast<int32_t>(rzg);
    a->set_oRZ = 0;
    a->set_oRG = static_cast<int32_t>(szRZ);
    a->rzg_tok = static_cast<int32_t>(rzg_tok);
    a->fixc = static_cast<int32_t>(fixc);
    a->fixc_items = static_cast<int32_t>(nfix);
    a->mbar = static_cast<int32_t>(mbar);
  }
  return mbar + 8 * static_cast<size_t>(S + 3);  // stages, analysis, synthesis, RZ/RG written
}

using ffb_host::encode_tiled;
using ffb_host::EncodeTiledFn;

// Tensor map of the bf16 rows of one activation tensor (d features, N
// tokens, leading dimension ld elements): {32 coordinates, d / 32 groups, N
// tokens}, box {32, d / 32, rows} (rows consecutive tokens, one row per
// group, token-major), 64-byte swizzle.
bool encode_rows(CUtensorMap* map, const void* base, int32_t d, int32_t N, int64_t ld, int32_t rows = 1) {
  const EncodeTiledFn fn = encode_tiled();
  if (!fn) return false;
  const cuuint64_t dims[3] = {32, static_cast<cuuint64_t>(d / 32), static_cast<cuuint64_t>(N)};
  const cuuint64_t strides[2] = {64, static_cast<cuuint64_t>(ld) * 2};
  const cuuint32_t box[3] = {32, static_cast<cuuint32_t>(d / 32), static_cast<cuuint32_t>(rows)};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Kernel choice for bf16: the two-token tensor-core kernel wherever it
// applies (register-resident plans, group counts a multiple of 8 and at most
// 128, its shared-memory map fits; packed units where a side has at most 64
// groups, unless FRAMEFB_PACK=0), else the one-token tensor-core kernel
// (group counts up to 256), else the one-phase-at-a-time tile kernel.
// FRAMEFB_KERNEL=tc2, =tc or =tile selects one of them where it applies
// (for comparison and tests).
bool kernel_is(const char* name) {
  const char* e = std::getenv("FRAMEFB_KERNEL");
  return e && std::strcmp(e, name) == 0;
}
bool tc_allowed() { return !kernel_is("tile"); }
bool tc2_allowed() { return tc_allowed() && !kernel_is("tc"); }

// Segments of a mixed-tenant forward: tokens [start[i], start[i + 1]) of
// every matrix belong to tenant tenant[i].
struct SegTable {
  int32_t nseg;
  const int32_t* start;
  const int32_t* tenant;
};

// Validate one chunk of matrices and fill the launch parameters.  With a
// segment table the chunk must run on a two-token kernel with one pair
// count for all its matrices (else FRAMEFB_EUNSUPPORTED).
framefb_status prepare(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dt, Prepared& P,
                       const SegTable* seg = nullptr) {
  const size_t esz = dt == FRAMEFB_BF16 ? 2 : 4;
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  std::memset(P.args, 0, sizeof(ffb::LaunchK));
  std::memset(P.red, 0, sizeof(ffb::ReduceK));
  bool reg = true;
  int32_t nnz_max = 0;
  for (int32_t j = 0; j < nmats; ++j) {
    const FfbPlanHeader* h = groups_header(mats[j].plan);
    if (!h) return FRAMEFB_EINVAL;
    if (h->EZ > ffb::kEreg || h->EG > ffb::kEreg) reg = false;
    nnz_max = std::max({nnz_max, h->nnz, h->nnz_full});  // dC partial slots are indexed by q
  }
  int64_t units = 0;
  size_t smem = 0;
  int T_mma = 0;
  bool tc = false, tc2 = false;
  int pairs[ffb::kTcMaxMats];
  bool pack = false;
  if (dt == FRAMEFB_BF16 && reg && tc2_allowed() && nmats <= ffb::kTcMaxMats && encode_tiled()) {
    // two-token tensor-core kernel: two stages; small dimensions pack
    // several token pairs per unit
    for (int32_t j = 0; j < nmats; ++j) {
      pairs[j] = pack_allowed() ? tc2_pairs(*plan_header(mats[j].plan)) : 1;
      pack = pack || pairs[j] > 1;
    }
    int dev = 0, optin = 0;
    cudaFuncAttributes fa{};
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
        cudaFuncGetAttributes(&fa, tc2_kernel_ptr(ops, pack)) != cudaSuccess)
      return FRAMEFB_ECUDA;
    size_t budget = static_cast<size_t>(optin) - fa.sharedSizeBytes;
    size_t need = tc2_smem_map(mats, nmats, ops, 2, pairs, pack, nullptr);
    if (pack && (need == 0 || need > budget)) {
      // packed sets do not fit: unpacked units
      for (int32_t j = 0; j < nmats; ++j) pairs[j] = 1;
      pack = false;
      if (cudaFuncGetAttributes(&fa, tc2_kernel_ptr(ops, pack)) != cudaSuccess) return FRAMEFB_ECUDA;
      budget = static_cast<size_t>(optin) - fa.sharedSizeBytes;
      need = tc2_smem_map(mats, nmats, ops, 2, pairs, pack, nullptr);
    }
    if (need > 0 && need <= budget) {
      tc2 = true;
      T_mma = 2;
      std::memset(P.tcargs, 0, sizeof(ffb::TcLaunchK));
      smem = tc2_smem_map(mats, nmats, ops, 2, pairs, pack, P.tcargs);
    }
  }
  if (dt == FRAMEFB_BF16 && reg && !tc2 && tc_allowed() && nmats <= ffb::kTcMaxMats && encode_tiled()) {
    // tensor-core pipelined kernel: deepest staging ring (2..4) that fits
    int dev = 0, optin = 0;
    cudaFuncAttributes fa{};
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
        cudaFuncGetAttributes(&fa, tc_kernel_ptr(ops)) != cudaSuccess)
      return FRAMEFB_ECUDA;
    const size_t budget = static_cast<size_t>(optin) - fa.sharedSizeBytes;
    for (int S = 4; S >= 2 && !tc; --S) {
      const size_t need = tc_smem_map(mats, nmats, ops, S, nullptr);
      if (need > 0 && need <= budget) {
        tc = true;
        T_mma = 1;
        std::memset(P.tcargs, 0, sizeof(ffb::TcLaunchK));
        smem = tc_smem_map(mats, nmats, ops, S, P.tcargs);
      }
    }
  }
  if (dt == FRAMEFB_BF16 && !tc && !tc2) {
    // one tile size for the launch; stage the output rows too when they fit,
    // else the synthesis reads them from global memory
    bool staged = false;
    for (int pass = 0; pass < 2 && !T_mma; ++pass) {
      const bool stage_out = pass == 0;
      for (int T = 2; T >= 1 && !T_mma; --T)
        if (mma_smem_map(mats, nmats, ops, reg, T, stage_out, nullptr) <= static_cast<size_t>(kSmemBudget)) {
          T_mma = T;
          staged = stage_out;
        }
    }
    if (!T_mma) return FRAMEFB_EUNSUPPORTED;
    smem = mma_smem_map(mats, nmats, ops, reg, T_mma, staged, P.args);
  }
  if (seg) {
    if (!tc2 || ops != FRAMEFB_OP_FORWARD || seg->nseg > ffb::kTcMaxSeg) return FRAMEFB_EUNSUPPORTED;
    for (int32_t j = 1; j < nmats; ++j)
      if (pairs[j] != pairs[0]) return FRAMEFB_EUNSUPPORTED;
  }
  for (int32_t j = 0; j < nmats; ++j) {
    const framefb_mat& M = mats[j];
    const FfbPlanHeader* h = plan_header(M.plan);
    if (M.N < 0 || M.n <= 0 || M.m <= 0) return FRAMEFB_EINVAL;
    // (a plan's part covers blocks of the frames' features: n, m < d)
    if (!frame_ok(M.fin, h->d_in) || !frame_ok(M.fout, h->d_out)) return FRAMEFB_EINVAL;
    if (h->n != M.n || h->m != M.m) return FRAMEFB_EINVAL;
    if (!M.plan_dev || !aligned16(M.plan_dev)) return FRAMEFB_EINVAL;
    if (!std::isfinite(M.scale)) return FRAMEFB_EINVAL;
    if ((F || D) && h->nnz > 0 && !M.c_val) return FRAMEFB_EINVAL;
    const bool needX = F || C, needdY = D || C;
    if (M.N > 0) {
      if ((needX || D) && (M.ldx < M.n || (M.ldx * esz) % 16)) return FRAMEFB_EINVAL;
      if ((needdY || F) && (M.ldy < M.m || (M.ldy * esz) % 16)) return FRAMEFB_EINVAL;
      if (needX && (!M.X || !aligned16(M.X))) return FRAMEFB_EINVAL;
      if (needdY && (!M.dY || !aligned16(M.dY))) return FRAMEFB_EINVAL;
      if (F && (!M.Y || !aligned16(M.Y))) return FRAMEFB_EINVAL;
      if (D && (!M.dX || !aligned16(M.dX))) return FRAMEFB_EINVAL;
    }
    if (C && h->nnz > 0 && !M.dC) return FRAMEFB_EINVAL;
    // tokens per tile: as many as fit in shared memory, at most kTmax
    int T = tc2 ? 2 * pairs[j] : T_mma;
    if (dt != FRAMEFB_BF16) {
      T = kTmax;
      while (T > 1 && ffb_tile_layout(*h, ops, T, C).total * 4 > kSmemBudget) --T;
      const size_t bytes = static_cast<size_t>(ffb_tile_layout(*h, ops, T, C).total) * 4;
      if (bytes > static_cast<size_t>(kSmemBudget)) return FRAMEFB_EUNSUPPORTED;
      smem = std::max(smem, bytes);
    }
    int32_t ntiles = (M.N + T - 1) / T;
    if (seg) {  // the segments' runs of units
      int64_t nt = 0;
      for (int32_t i = 0; i < seg->nseg; ++i) nt += (seg->start[i + 1] - seg->start[i] + T - 1) / T;
      if (nt > INT32_MAX / 2) return FRAMEFB_EUNSUPPORTED;
      ntiles = static_cast<int32_t>(nt);
    }
    ffb::MatK& K = P.args->m[j];
    K.X = M.X;
    K.dX = M.dX;
    K.dY = M.dY;
    K.Y = M.Y;
    K.plan = static_cast<const uint8_t*>(M.plan_dev);
    K.c_val = M.c_val;
    K.fval_in = M.fin->val;
    K.fval_out = M.fout->val;
    K.rho_in = M.fin->rho;
    K.rho_out = M.fout->rho;
    K.n = M.n;
    K.m = M.m;
    K.ldx = M.ldx;
    K.ldy = M.ldy;
    K.N = M.N;
    K.T = T;
    K.ubeg = static_cast<int32_t>(units);
    K.ntiles = ntiles;
    K.seff = M.scale / 16.f;
    ffb::ReduceMat& R = P.red->m[j];
    R.dC = M.dC;
    R.qlist = h->off_qlist ? reinterpret_cast<const int32_t*>(static_cast<const uint8_t*>(M.plan_dev) + h->off_qlist)
                           : nullptr;
    R.ubeg = K.ubeg;
    R.ntiles = ntiles;
    R.nnz = h->nnz;
    R.seff = K.seff;
    units += ntiles;
    if (units > INT32_MAX / 2) return FRAMEFB_EUNSUPPORTED;
  }
  if (seg) {
    ffb::TcLaunchK& A = *P.tcargs;
    const int32_t T = 2 * pairs[0];
    A.nseg = seg->nseg;
    A.seg_u0[0] = 0;
    for (int32_t i = 0; i < seg->nseg; ++i) {
      A.seg_tok[i] = seg->start[i];
      A.seg_tenant[i] = seg->tenant[i];
      A.seg_u0[i + 1] = A.seg_u0[i] + (seg->start[i + 1] - seg->start[i] + T - 1) / T;
    }
    A.seg_tok[seg->nseg] = seg->start[seg->nseg];
  }
  P.args->nmats = nmats;
  P.args->total_units = static_cast<int32_t>(units);
  P.args->stride = (nnz_max + 63) & ~63;
  if (tc || tc2) {
    ffb::TcLaunchK& A = *P.tcargs;
    A.nmats = nmats;
    A.total_units = P.args->total_units;
    A.stride = P.args->stride;
    for (int32_t j = 0; j < nmats; ++j) {
      A.m[j] = P.args->m[j];
      const framefb_mat& M = mats[j];
      if (M.N == 0) continue;
      const int32_t rows = tc2 ? pairs[j] : 1;
      if ((F || C) && !encode_rows(&A.maps[2 * j], M.X, M.n, M.N, M.ldx, rows)) return FRAMEFB_ECUDA;
      if ((D || C) && !encode_rows(&A.maps[2 * j + 1], M.dY, M.m, M.N, M.ldy, rows)) return FRAMEFB_ECUDA;
    }
  }
  P.red->nmats = nmats;
  P.red->total_units = static_cast<int32_t>(units);
  P.red->stride = P.args->stride;
  P.reg = reg;
  P.tc = tc;
  P.tc2 = tc2;
  P.pack = tc2 && pack;
  P.seg = seg != nullptr;
  P.threads = (tc || tc2) ? ffb::kTcThreads : kThreads;
  P.T = T_mma;
  P.smem = std::max<size_t>(smem, 16);
  P.grid = 0;
  P.ws_bytes = 0;
  if (units == 0) return FRAMEFB_OK;
  void* fn = P.seg ? tc2_seg_kernel_ptr(P.pack)
             : tc2 ? tc2_kernel_ptr(ops, P.pack) : tc ? tc_kernel_ptr(ops) : tile_kernel_ptr(dt, ops, reg, T_mma);
  if (!fn) return FRAMEFB_EINVAL;
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FRAMEFB_ECUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return FRAMEFB_ECUDA;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(P.smem)) !=
      cudaSuccess)
    return FRAMEFB_ECUDA;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, P.threads, P.smem) != cudaSuccess)
    return FRAMEFB_ECUDA;
  if (per_sm < 1) return FRAMEFB_EUNSUPPORTED;
  P.grid = static_cast<int>(std::min<int64_t>(static_cast<int64_t>(sms) * per_sm, units));
  P.red->grid = P.grid;
  if (C) P.ws_bytes = static_cast<size_t>(P.grid + nmats) * P.args->stride * sizeof(float) + 256;
  return FRAMEFB_OK;
}

struct Buffers {
  std::vector<uint8_t> a, t, r;
  Buffers() : a(sizeof(ffb::LaunchK)), t(sizeof(ffb::TcLaunchK) + 64), r(sizeof(ffb::ReduceK)) {}
  Prepared prep() {
    Prepared p{};
    p.args = reinterpret_cast<ffb::LaunchK*>(a.data());
    // tensor maps want 64-byte alignment
    const uintptr_t ta = (reinterpret_cast<uintptr_t>(t.data()) + 63) & ~uintptr_t{63};
    p.tcargs = reinterpret_cast<ffb::TcLaunchK*>(ta);
    p.red = reinterpret_cast<ffb::ReduceK*>(r.data());
    return p;
  }
};

// Matrices in the launch that starts at `mats` (`rest` left): the
// tensor-core kernel carries tensor maps in its parameters and takes at most
// kTcMaxMats; the chunk is that short only when the kernel applies to it.
int32_t chunk_len(const framefb_mat* mats, int32_t rest, framefb_dtype dt) {
  if (dt == FRAMEFB_BF16 && tc_allowed()) {
    // matrices of one pair count only (units of equal cost in a launch; the
    // caller's order is sorted by it), in launches of equal size (at most 64
    // matrices each): no small tail launch
    int32_t run = rest;
    if (tc2_allowed() && pack_allowed()) {
      const FfbPlanHeader* h0 = plan_header(mats[0].plan);
      run = 1;
      while (h0 && run < rest) {
        const FfbPlanHeader* h = plan_header(mats[run].plan);
        if (!h || tc2_pairs(*h) != tc2_pairs(*h0)) break;
        ++run;
      }
    }
    const int32_t launches = (run + ffb::kTcMaxMats - 1) / ffb::kTcMaxMats;
    const int32_t k = (run + launches - 1) / launches;
    bool ok = true;
    for (int32_t j = 0; j < k && ok; ++j) {
      const FfbPlanHeader* h = plan_header(mats[j].plan);
      ok = h && h->EZ <= ffb::kEreg && h->EG <= ffb::kEreg && h->Gn % 8 == 0 && h->Gm % 8 == 0 &&
           h->Gn <= 128 * ffb::kTcMaxTiles && h->Gm <= 128 * ffb::kTcMaxTiles;
    }
    if (ok) return k;
  }
  return std::min(rest, kMaxMats);
}

bool ops_ok(int32_t ops) { return ops == 1 || ops == 2 || ops == 4 || ops == 6 || ops == 7; }

}  // namespace

namespace {

size_t structured_workspace(const framefb_mat* mats, int32_t nmats, int32_t ops) {
  if (nmats <= 0) return 0;
  Buffers b;
  size_t need = 0;
  // the workspace depends on the launch chunking, the kernel and its grid,
  // all of which depend on the dtype: the larger need of the two dtypes the
  // matrices are valid for (the descriptors carry no dtype)
  bool any = false;
  for (const framefb_dtype dt : {FRAMEFB_BF16, FRAMEFB_F32}) {
    size_t need_dt = 0;
    bool ok = true;
    for (int32_t j0 = 0, nm = 0; j0 < nmats && ok; j0 += nm) {
      nm = chunk_len(mats + j0, nmats - j0, dt);
      Prepared P = b.prep();
      ok = prepare(mats + j0, nm, ops, dt, P) == FRAMEFB_OK;
      need_dt = std::max(need_dt, P.ws_bytes);
    }
    if (ok) {
      any = true;
      need = std::max(need, need_dt);
    }
  }
  return any ? need : 0;
}

// Validate every launch chunk of the structured matrices; *need = the
// workspace the largest chunk needs.
framefb_status structured_check(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype,
                                size_t* need, const SegTable* seg = nullptr) {
  *need = 0;
  Buffers b;
  for (int32_t j0 = 0, nm = 0; j0 < nmats; j0 += nm) {
    nm = chunk_len(mats + j0, nmats - j0, dtype);
    Prepared P = b.prep();
    const framefb_status s = prepare(mats + j0, nm, ops, dtype, P, seg);
    if (s != FRAMEFB_OK) return s;
    *need = std::max(*need, P.ws_bytes);
  }
  return FRAMEFB_OK;
}

// Queue the structured kernels (after structured_check).
framefb_status structured_run(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype, void* ws,
                              cudaStream_t st, const SegTable* seg = nullptr) {
  Buffers b;
  for (int32_t j0 = 0, nm = 0; j0 < nmats; j0 += nm) {
    nm = chunk_len(mats + j0, nmats - j0, dtype);
    Prepared P = b.prep();
    const framefb_status s = prepare(mats + j0, nm, ops, dtype, P, seg);
    if (s != FRAMEFB_OK) return s;
    if (P.grid == 0) {
      if (ops & FRAMEFB_OP_GRAD_COEFF) {  // no tokens: the gradient is zero
        for (int32_t j = 0; j < nm; ++j)
          if (P.red->m[j].nnz > 0 &&
              cudaMemsetAsync(P.red->m[j].dC, 0, sizeof(float) * P.red->m[j].nnz, st) != cudaSuccess)
            return FRAMEFB_ECUDA;
      }
      continue;
    }
    P.args->partial = static_cast<float*>(ws);
    P.tcargs->partial = static_cast<float*>(ws);
    P.red->partial = static_cast<const float*>(ws);
    void* fn = P.seg   ? tc2_seg_kernel_ptr(P.pack)
               : P.tc2 ? tc2_kernel_ptr(ops, P.pack)
               : P.tc  ? tc_kernel_ptr(ops)
                       : tile_kernel_ptr(dtype, ops, P.reg, P.T);
    void* kargs[] = {(P.tc || P.tc2) ? static_cast<void*>(P.tcargs) : static_cast<void*>(P.args)};
    if (cudaLaunchKernel(fn, dim3(P.grid), dim3(P.threads), kargs, P.smem, st) != cudaSuccess)
      return FRAMEFB_ECUDA;
    if (ops & FRAMEFB_OP_GRAD_COEFF) {
      int nnz_max = 0;
      for (int32_t j = 0; j < nm; ++j) nnz_max = std::max(nnz_max, P.red->m[j].nnz);
      if (nnz_max > 0) {
        void* rargs[] = {P.red};
        const dim3 rg((nnz_max + 255) / 256, nm);
        if (cudaLaunchKernel(reinterpret_cast<void*>(ffb::dc_reduce_kernel), rg, dim3(256), rargs, 0, st) !=
            cudaSuccess)
          return FRAMEFB_ECUDA;
      }
    }
  }
  return FRAMEFB_OK;
}

framefb_status structured_names(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype,
                                std::vector<std::string>& names) {
  Buffers b;
  for (int32_t j0 = 0, nm = 0; j0 < nmats; j0 += nm) {
    nm = chunk_len(mats + j0, nmats - j0, dtype);
    Prepared P = b.prep();
    const framefb_status s = prepare(mats + j0, nm, ops, dtype, P);
    if (s != FRAMEFB_OK) return s;
    if (P.grid == 0) continue;
    std::string k = P.pack  ? "tc2p_tile_kernel"
                    : P.tc2 ? "tc2_tile_kernel"
                    : P.tc  ? "tc_tile_kernel"
                            : (dtype == FRAMEFB_BF16 ? "mma_tile_kernel" : "fft_tile_kernel");
    k += "<" + std::to_string(ops) + ">";
    if (std::find(names.begin(), names.end(), k) == names.end()) names.push_back(k);
  }
  return FRAMEFB_OK;
}


// The fused tcgen05 kernels take the plan: register-resident chunks and
// group counts a multiple of 8, at most 256 per side.
bool fused_tc_ok(const FfbPlanHeader& h) {
  return h.EZ <= ffb::kEreg && h.EG <= ffb::kEreg && h.Gn % 8 == 0 && h.Gm % 8 == 0 &&
         h.Gn <= 128 * ffb::kTcMaxTiles && h.Gm <= 128 * ffb::kTcMaxTiles;
}

bool parts_allowed() {
  const char* e = std::getenv("FRAMEFB_PARTS");
  return !(e && std::strcmp(e, "0") == 0);
}

// Matrices of a call split by path, each in call order: the fused kernels
// (structured plans they take, fp32, or rows with padding), the plans' parts
// on the fused tcgen05 kernels (bf16 structured plans the kernels do not
// take whole, with parts, and tokens; FRAMEFB_PARTS=0 sends them to the
// contraction path), and the contraction path of framefb_dense.cu
// (dense-layout plans, and the other bf16 structured plans the fused
// tcgen05 kernels do not take, with unpadded rows).  FRAMEFB_KERNEL=tile
// keeps every structured plan on the warp-MMA kernel.
framefb_status split_paths(const framefb_mat* mats, int32_t nmats, framefb_dtype dt, std::vector<framefb_mat>& grp,
                           std::vector<framefb_mat>& den, std::vector<framefb_mat>* prt = nullptr) {
  try {
    for (int32_t j = 0; j < nmats; ++j) {
      const framefb_mat& M = mats[j];
      const FfbPlanHeader* h = plan_header(M.plan);
      if (!h) return FRAMEFB_EINVAL;
      const bool big = h->layout == FFB_LAYOUT_GROUPS && dt == FRAMEFB_BF16 && tc_allowed() && !fused_tc_ok(*h);
      if (big && prt && parts_allowed() && !M.plan->subs.empty() && M.N > 0) {
        prt->push_back(M);
        continue;
      }
      const bool split = big && M.ldx == M.n && M.ldy == M.m;
      (h->layout == FFB_LAYOUT_DENSE || split ? den : grp).push_back(M);
    }
    // the two-token kernel's units carry P token pairs of a matrix (P = 1
    // for large dimensions): matrices of one P launch together, largest P
    // first (results do not depend on the order of the matrices)
    if (dt == FRAMEFB_BF16 && tc2_allowed() && pack_allowed())
      std::stable_sort(grp.begin(), grp.end(), [](const framefb_mat& x, const framefb_mat& y) {
        return tc2_pairs(*plan_header(x.plan)) > tc2_pairs(*plan_header(y.plan));
      });
  } catch (const std::bad_alloc&) {
    return FRAMEFB_ENOMEM;
  }
  return FRAMEFB_OK;
}

// The launch waves of the structured matrices: wave 0 holds the matrices
// the fused kernels take whole; the matrices with parts run as their parts,
// one matrix of the fused kernels per part (its blocks of X, dY, Y and dX,
// the part's plan, the whole c_val and dC indexed by the part's entries).
// ΔW is linear in C, so Y and dX take the sum of the parts' contributions;
// parts of one matrix that write the same features of Y (forward) or dX
// (backward dx) read-modify-write the same bytes and go to successive waves
// (greedily), so that no launch holds both.
framefb_status plan_waves(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dt,
                          std::vector<std::vector<framefb_mat>>& waves, std::vector<framefb_mat>& den) {
  std::vector<framefb_mat> grp, prt;
  framefb_status s = split_paths(mats, nmats, dt, grp, den, &prt);
  if (s != FRAMEFB_OK) return s;
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX;
  const size_t esz = dt == FRAMEFB_BF16 ? 2 : 4;
  try {
    waves.assign(1, std::move(grp));
    for (const framefb_mat& M : prt) {
      const std::vector<FfbSubPlan>& sub = M.plan->subs;
      std::vector<int32_t> wave(sub.size(), 0);
      for (size_t i = 0; i < sub.size(); ++i) {
        auto clash = [&](size_t k) {
          return (F && sub[k].m0 == sub[i].m0) || (D && sub[k].n0 == sub[i].n0);
        };
        int32_t w = 0;
        for (bool busy = true; busy; ) {
          busy = false;
          for (size_t k = 0; k < i && !busy; ++k) busy = wave[k] == w && clash(k);
          if (busy) ++w;
        }
        wave[i] = w;
        framefb_mat V = M;
        const FfbPlanHeader* h = plan_header(sub[i].plan);
        if (!h) return FRAMEFB_EINVAL;
        V.n = h->n;
        V.m = h->m;
        V.X = M.X ? static_cast<const uint8_t*>(M.X) + esz * sub[i].n0 : nullptr;
        V.dX = M.dX ? static_cast<uint8_t*>(M.dX) + esz * sub[i].n0 : nullptr;
        V.dY = M.dY ? static_cast<const uint8_t*>(M.dY) + esz * sub[i].m0 : nullptr;
        V.Y = M.Y ? static_cast<uint8_t*>(M.Y) + esz * sub[i].m0 : nullptr;
        V.plan = sub[i].plan;
        V.plan_dev = M.plan_dev ? static_cast<const uint8_t*>(M.plan_dev) + sub[i].dev_off : nullptr;
        if (static_cast<size_t>(w) >= waves.size()) waves.resize(w + 1);
        waves[w].push_back(V);
      }
    }
  } catch (const std::bad_alloc&) {
    return FRAMEFB_ENOMEM;
  }
  return FRAMEFB_OK;
}

}  // namespace

extern "C" size_t framefb_workspace_size(const framefb_mat* mats, int32_t nmats, int32_t ops) {
  if (!mats || nmats <= 0 || !ops_ok(ops)) return 0;
  // the routing depends on the dtype: the larger need of the two
  size_t need = 0;
  for (const framefb_dtype dt : {FRAMEFB_BF16, FRAMEFB_F32}) {
    std::vector<std::vector<framefb_mat>> waves;
    std::vector<framefb_mat> den;
    if (plan_waves(mats, nmats, ops, dt, waves, den) != FRAMEFB_OK) return 0;
    size_t dneed = 0;
    if (!den.empty() &&
        ffb_host::dense_check(den.data(), static_cast<int32_t>(den.size()), ops, dt, &dneed) != FRAMEFB_OK)
      continue;
    need = std::max(need, dneed);
    for (const std::vector<framefb_mat>& w : waves)
      need = std::max(need, structured_workspace(w.data(), static_cast<int32_t>(w.size()), ops));
  }
  return need;
}

extern "C" framefb_status framefb_run(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype,
                                      void* ws, size_t ws_bytes, void* stream) {
  if (nmats < 0 || (nmats > 0 && !mats) || !ops_ok(ops)) return FRAMEFB_EINVAL;
  if (dtype != FRAMEFB_F32 && dtype != FRAMEFB_BF16) return FRAMEFB_EINVAL;
  if (nmats == 0) return FRAMEFB_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  std::vector<std::vector<framefb_mat>> waves;
  std::vector<framefb_mat> den;
  framefb_status s = plan_waves(mats, nmats, ops, dtype, waves, den);
  if (s != FRAMEFB_OK) return s;
  // validate everything before queueing anything; the waves and the two
  // paths run one after the other on the stream and share the workspace
  size_t need = 0;
  for (const std::vector<framefb_mat>& w : waves) {
    size_t gneed = 0;
    s = structured_check(w.data(), static_cast<int32_t>(w.size()), ops, dtype, &gneed);
    if (s != FRAMEFB_OK) return s;
    need = std::max(need, gneed);
  }
  size_t dneed = 0;
  s = ffb_host::dense_check(den.data(), static_cast<int32_t>(den.size()), ops, dtype, &dneed);
  if (s != FRAMEFB_OK) return s;
  need = std::max(need, dneed);
  if (need > 0) {
    if (!ws || ws_bytes < need) return FRAMEFB_EWORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) & 255u) return FRAMEFB_EINVAL;
  }
  for (const std::vector<framefb_mat>& w : waves) {
    s = structured_run(w.data(), static_cast<int32_t>(w.size()), ops, dtype, ws, st);
    if (s != FRAMEFB_OK) return s;
  }
  return ffb_host::dense_run(den.data(), static_cast<int32_t>(den.size()), ops, dtype, ws, ws_bytes, st);
}

extern "C" framefb_status framefb_kernel_names(const framefb_mat* mats, int32_t nmats, int32_t ops,
                                               framefb_dtype dtype, char* buf, size_t len) {
  if (!buf || len == 0) return FRAMEFB_EINVAL;
  buf[0] = '\0';
  if (nmats < 0 || (nmats > 0 && !mats) || !ops_ok(ops)) return FRAMEFB_EINVAL;
  if (dtype != FRAMEFB_F32 && dtype != FRAMEFB_BF16) return FRAMEFB_EINVAL;
  std::vector<std::vector<framefb_mat>> waves;
  std::vector<framefb_mat> den;
  framefb_status s = plan_waves(mats, nmats, ops, dtype, waves, den);
  if (s != FRAMEFB_OK) return s;
  std::vector<std::string> names;
  for (const std::vector<framefb_mat>& w : waves) {
    s = structured_names(w.data(), static_cast<int32_t>(w.size()), ops, dtype, names);
    if (s != FRAMEFB_OK) return s;
  }
  if (!den.empty()) {
    size_t need = 0;
    s = ffb_host::dense_check(den.data(), static_cast<int32_t>(den.size()), ops, dtype, &need);
    if (s != FRAMEFB_OK) return s;
    ffb_host::dense_kernel_names(den.data(), static_cast<int32_t>(den.size()), ops, names);
  }
  std::string out;
  for (const std::string& k : names) out += (out.empty() ? "" : ",") + k;
  if (out.size() + 1 > len) return FRAMEFB_EINVAL;
  std::memcpy(buf, out.c_str(), out.size() + 1);
  return FRAMEFB_OK;
}

extern "C" framefb_status framefb_forward(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype, void* ws,
                                          size_t ws_bytes, void* stream) {
  return framefb_run(mats, nmats, FRAMEFB_OP_FORWARD, dtype, ws, ws_bytes, stream);
}
extern "C" framefb_status framefb_backward_dx(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                              void* ws, size_t ws_bytes, void* stream) {
  return framefb_run(mats, nmats, FRAMEFB_OP_BACKWARD_DX, dtype, ws, ws_bytes, stream);
}
extern "C" framefb_status framefb_grad_coeff(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype, void* ws,
                                             size_t ws_bytes, void* stream) {
  return framefb_run(mats, nmats, FRAMEFB_OP_GRAD_COEFF, dtype, ws, ws_bytes, stream);
}
extern "C" framefb_status framefb_backward(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype, void* ws,
                                           size_t ws_bytes, void* stream) {
  return framefb_run(mats, nmats, FRAMEFB_OP_BACKWARD_DX | FRAMEFB_OP_GRAD_COEFF, dtype, ws, ws_bytes, stream);
}
extern "C" framefb_status framefb_fused_fwd_bwd(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                                void* ws, size_t ws_bytes, void* stream) {
  return framefb_run(mats, nmats, FRAMEFB_OP_FORWARD | FRAMEFB_OP_BACKWARD_DX | FRAMEFB_OP_GRAD_COEFF, dtype, ws,
                     ws_bytes, stream);
}

extern "C" framefb_status framefb_merge(const void* W0, framefb_dtype dtype, int32_t m, int32_t n, int64_t ldw,
                                        const framefb_dev_frame* fin, const framefb_dev_frame* fout,
                                        const framefb_plan* plan, const void* plan_dev, const float* c_vals,
                                        int32_t T, float scale, void* Wout, void* stream) {
  if (dtype != FRAMEFB_F32 && dtype != FRAMEFB_BF16) return FRAMEFB_EINVAL;
  const FfbPlanHeader* h = plan_header(plan);
  if (!h || m <= 0 || n <= 0 || T < 0) return FRAMEFB_EINVAL;
  if (h->layout != FFB_LAYOUT_GROUPS) return FRAMEFB_EUNSUPPORTED;  // the merge kernel takes DFT_16-group frames
  if (h->m != m || h->n != n) return FRAMEFB_EINVAL;
  if (!frame_ok(fin, n) || !frame_ok(fout, m)) return FRAMEFB_EINVAL;
  const size_t esz = dtype == FRAMEFB_BF16 ? 2 : 4;
  if (ldw < n || (ldw * esz) % 16 || !std::isfinite(scale)) return FRAMEFB_EINVAL;
  if (T == 0) return FRAMEFB_OK;
  if (!W0 || !Wout || !plan_dev || !aligned16(W0) || !aligned16(Wout) || !aligned16(plan_dev)) return FRAMEFB_EINVAL;
  if (h->nnz > 0 && !c_vals) return FRAMEFB_EINVAL;
  {  // Wout must not overlap W0
    const uintptr_t w0 = reinterpret_cast<uintptr_t>(W0), w1 = w0 + static_cast<size_t>(m) * ldw * esz;
    const uintptr_t o0 = reinterpret_cast<uintptr_t>(Wout), o1 = o0 + static_cast<size_t>(T) * m * ldw * esz;
    if (o0 < w1 && w0 < o1) return FRAMEFB_EINVAL;
  }
  ffb::MergeK a{};
  a.W0 = W0;
  a.Wout = Wout;
  a.plan = static_cast<const uint8_t*>(plan_dev);
  a.c_vals = c_vals;
  a.fin_val = fin->val;
  a.fout_val = fout->val;
  a.ldw = ldw;
  a.m = m;
  a.n = n;
  a.rho_in = fin->rho;
  a.rho_out = fout->rho;
  a.nnz = h->nnz;
  a.T = T;
  a.seff = scale / 16.f;
  void* kargs[] = {&a};
  void* fn = dtype == FRAMEFB_BF16 ? reinterpret_cast<void*>(ffb::merge_kernel<__nv_bfloat16>)
                                   : reinterpret_cast<void*>(ffb::merge_kernel<float>);
  // grid-stride over (out group, tenant) items: as many CTAs as are resident
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, ffb::kMergeThreads, 0) != cudaSuccess)
    return FRAMEFB_ECUDA;
  // one warp per (out group, tenant, run of blocks) item
  const int64_t items =
      static_cast<int64_t>(h->Gm) * T * ((h->Gn + ffb::kMergeBlocks - 1) / ffb::kMergeBlocks);
  const int64_t grid = std::max<int64_t>(
      1, std::min<int64_t>((items + ffb::kMergeWarps - 1) / ffb::kMergeWarps, static_cast<int64_t>(sms) * std::max(per_sm, 1)));
  if (cudaLaunchKernel(fn, dim3(static_cast<unsigned>(grid)), dim3(ffb::kMergeThreads), kargs, 0,
                       static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return FRAMEFB_ECUDA;
  return FRAMEFB_OK;
}

extern "C" framefb_status framefb_forward_tenants(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                                  const int32_t* seg_start, const int32_t* seg_tenant, int32_t nseg,
                                                  int32_t ntenants, void* stream) {
  if (nmats < 0 || (nmats > 0 && !mats) || nseg < 0 || ntenants <= 0 || !seg_start || (nseg > 0 && !seg_tenant))
    return FRAMEFB_EINVAL;
  if (seg_start[0] != 0) return FRAMEFB_EINVAL;
  for (int32_t i = 0; i < nseg; ++i)
    if (seg_start[i + 1] < seg_start[i] || seg_tenant[i] < 0 || seg_tenant[i] >= ntenants) return FRAMEFB_EINVAL;
  const int32_t N = seg_start[nseg];
  for (int32_t j = 0; j < nmats; ++j)
    if (!plan_header(mats[j].plan) || mats[j].N != N) return FRAMEFB_EINVAL;
  // the segment table in the kernel parameters: units stay inside segments,
  // one launch per chunk of matrices, where every chunk runs on a two-token
  // kernel (FRAMEFB_SEG_KERNEL=0 takes the per-segment path below)
  const char* env = std::getenv("FRAMEFB_SEG_KERNEL");
  if (dtype == FRAMEFB_BF16 && nmats > 0 && nseg > 0 && nseg <= ffb::kTcMaxSeg && !(env && std::strcmp(env, "0") == 0)) {
    std::vector<framefb_mat> grp, den;
    framefb_status s = split_paths(mats, nmats, dtype, grp, den);
    if (s != FRAMEFB_OK) return s;
    if (den.empty()) {
      const SegTable st{nseg, seg_start, seg_tenant};
      size_t need = 0;
      s = structured_check(grp.data(), static_cast<int32_t>(grp.size()), FRAMEFB_OP_FORWARD, dtype, &need, &st);
      if (s == FRAMEFB_OK)
        return structured_run(grp.data(), static_cast<int32_t>(grp.size()), FRAMEFB_OP_FORWARD, dtype, nullptr,
                              static_cast<cudaStream_t>(stream), &st);
      if (s != FRAMEFB_EUNSUPPORTED) return s;
    }
  }
  // else the segments of all matrices run as the matrices of one framefb_run call
  if (static_cast<int64_t>(nmats) * nseg > INT32_MAX) return FRAMEFB_EINVAL;
  std::vector<framefb_mat> seg;
  try {
    seg.reserve(static_cast<size_t>(nmats) * static_cast<size_t>(nseg));
  } catch (const std::bad_alloc&) {
    return FRAMEFB_ENOMEM;
  }
  const size_t esz = dtype == FRAMEFB_BF16 ? 2 : 4;
  for (int32_t j = 0; j < nmats; ++j) {
    const framefb_mat& M = mats[j];
    const FfbPlanHeader* h = plan_header(M.plan);
    if (!h || M.N != N) return FRAMEFB_EINVAL;
    for (int32_t i = 0; i < nseg; ++i) {
      const int32_t t0 = seg_start[i], len = seg_start[i + 1] - seg_start[i];
      if (len == 0) continue;
      framefb_mat S = M;
      S.N = len;
      S.X = M.X ? static_cast<const uint8_t*>(M.X) + static_cast<size_t>(t0) * M.ldx * esz : nullptr;
      S.Y = M.Y ? static_cast<uint8_t*>(M.Y) + static_cast<size_t>(t0) * M.ldy * esz : nullptr;
      S.dX = nullptr;
      S.dY = nullptr;
      S.dC = nullptr;
      S.c_val = M.c_val ? M.c_val + static_cast<size_t>(seg_tenant[i]) * h->nnz : nullptr;
      seg.push_back(S);
    }
  }
  return framefb_run(seg.data(), static_cast<int32_t>(seg.size()), FRAMEFB_OP_FORWARD, dtype, nullptr, 0, stream);
}

extern "C" framefb_status framefb_adamw(float* param, const float* grad, float* m, float* v, int64_t n,
                                        const framefb_adamw_params* hp, int64_t step, void* stream) {
  if (n < 0 || step < 1 || !hp) return FRAMEFB_EINVAL;
  const double lr = hp->lr, b1 = hp->beta1, b2 = hp->beta2, eps = hp->eps, wd = hp->weight_decay;
  if (!(lr >= 0) || !(b1 >= 0 && b1 < 1) || !(b2 >= 0 && b2 < 1) || !(eps > 0) || !(wd >= 0) || !std::isfinite(lr) ||
      !std::isfinite(eps) || !std::isfinite(wd))
    return FRAMEFB_EINVAL;
  if (n == 0) return FRAMEFB_OK;
  const float* ptrs[4] = {param, grad, m, v};
  bool vec = true;
  for (const float* q : ptrs) {
    if (!q || reinterpret_cast<uintptr_t>(q) % 4) return FRAMEFB_EINVAL;
    vec = vec && aligned16(q);
  }
  ffb::AdamWK a{};
  a.p = param;
  a.g = grad;
  a.m = m;
  a.v = v;
  a.n = n;
  a.decay = static_cast<float>(1.0 - lr * wd);
  a.beta1 = hp->beta1;
  a.beta2 = hp->beta2;
  a.step_size = static_cast<float>(lr / (1.0 - std::pow(b1, static_cast<double>(step))));
  a.inv_sqrt_bc2 = static_cast<float>(1.0 / std::sqrt(1.0 - std::pow(b2, static_cast<double>(step))));
  a.eps = hp->eps;
  const int64_t work = vec ? (n + 3) / 4 : n;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return FRAMEFB_ECUDA;
  const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((work + 255) / 256, static_cast<int64_t>(sms) * 8));
  void* kargs[] = {&a};
  void* fn = vec ? reinterpret_cast<void*>(ffb::adamw_kernel<true>) : reinterpret_cast<void*>(ffb::adamw_kernel<false>);
  if (cudaLaunchKernel(fn, dim3(static_cast<unsigned>(blocks)), dim3(256), kargs, 0, static_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return FRAMEFB_ECUDA;
  return FRAMEFB_OK;
}

extern "C" double framefb_linear_warmup_lr(int64_t i, int64_t total, int64_t warmup, double lr_max) {
  if (i < 0 || total < 0 || warmup < 0) return 0.0;
  if (i < warmup) return lr_max * static_cast<double>(i) / static_cast<double>(warmup);
  if (total <= warmup) return 0.0;
  return lr_max * std::max(0.0, static_cast<double>(total - i) / static_cast<double>(total - warmup));
}

// ---------------------------------------------------------------------------
// Workspace-free variant of framefb_run for callers that cannot allocate
// device memory: the dC partial sums live in this file-scope device array.
// Host code must not use `g_static_ws` as an address (it names a host-side
// stand-in); the device address is looked up once per device below.
// ---------------------------------------------------------------------------
static __device__ __align__(256) unsigned char g_static_ws[FRAMEFB_STATIC_WS_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_static_ws_mu;
struct StaticWsEntry {
  CUcontext ctx;  // context the address was looked up in
  void* ptr;
};
StaticWsEntry g_static_ws_cache[kMaxDevices] = {};

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
CtxGetCurrentFn ctx_get_current() {
  static const CtxGetCurrentFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<CtxGetCurrentFn>(nullptr);
    return reinterpret_cast<CtxGetCurrentFn>(p);
  }();
  return fn;
}

// Device address of g_static_ws in the current context of the current
// device.  It is looked up on the first call in a context and cached with
// that context: after a device reset or a new primary context the module is
// loaded again, the array may move, and the next call looks it up afresh.
framefb_status static_ws_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FRAMEFB_ECUDA;
  const CtxGetCurrentFn get = ctx_get_current();
  CUcontext ctx = nullptr;
  if (!get || get(&ctx) != CUDA_SUCCESS) return FRAMEFB_ECUDA;
  std::lock_guard<std::mutex> lock(g_static_ws_mu);
  StaticWsEntry& e = g_static_ws_cache[dev];
  if (!ctx || !e.ptr || e.ctx != ctx) {
    // the lookup also makes the runtime's context current when none is yet
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_ws) != cudaSuccess || !p) return FRAMEFB_ECUDA;
    if (get(&ctx) != CUDA_SUCCESS || !ctx) return FRAMEFB_ECUDA;
    e.ctx = ctx;
    e.ptr = p;
  }
  *out = e.ptr;
  return FRAMEFB_OK;
}
}  // namespace

extern "C" framefb_status framefb_run_static_ws(const framefb_mat* mats, int32_t nmats, int32_t ops,
                                                framefb_dtype dtype, void* stream) {
  if (nmats < 0 || (nmats > 0 && !mats) || !ops_ok(ops)) return FRAMEFB_EINVAL;
  if (dtype != FRAMEFB_F32 && dtype != FRAMEFB_BF16) return FRAMEFB_EINVAL;
  void* ws = nullptr;
  const framefb_status s = static_ws_address(&ws);
  if (s != FRAMEFB_OK) return s;
  // framefb_run rejects a need above FRAMEFB_STATIC_WS_BYTES with FRAMEFB_EWORKSPACE
  return framefb_run(mats, nmats, ops, dtype, ws, FRAMEFB_STATIC_WS_BYTES, stream);
}

extern "C" framefb_status framefb_wait_timeouts(uint32_t* count) {
  if (!count) return FRAMEFB_EINVAL;
  uint32_t structured = 0, dense = 0;
  if (cudaMemcpyFromSymbol(&structured, ffb::g_wait_timeouts, sizeof(uint32_t)) != cudaSuccess) return FRAMEFB_ECUDA;
  const framefb_status s = ffb_host::dense_wait_timeouts(&dense);
  if (s != FRAMEFB_OK) return s;
  *count = structured + dense;
  return FRAMEFB_OK;
}
