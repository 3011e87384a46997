// Launchers of the contraction path of libframefb: validation, workspace
// sizing, tensor maps, and per matrix and token chunk the sequence analysis
// GEMM -> coefficient SpMM -> synthesis GEMM, then the deterministic dC
// reduction (framefb_dense.cuh).  It serves two kinds of matrices:
//   dense    frames outside the structured kernels (rho = 2, T blocks):
//            Phi is a dense d x K operand, GEMMs over (tokens x K);
//   grouped  k = 16, k*rho = d frames whose plans or sizes the fused tcgen05
//            kernels do not take (more than 16 entries per plan column, more
//            than 256 groups): Phi is block diagonal with one 32 x 32 block,
//            so the GEMMs run over (token, group) rows with K = 32 -- the
//            activation rows viewed as [N * d/32][32], which needs rows
//            without padding (leading dimension = features).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <utility>
#include <vector>

#include "dense_layout.h"
#include "framefb.h"
#include "framefb_dense.cuh"
#include "framefb_dense.h"
#include "plan_internal.h"
#include "plan_layout.h"

namespace ffb_host {

EncodeTiledFn encode_tiled() {
  static const EncodeTiledFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<EncodeTiledFn>(nullptr);
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}

namespace {

namespace fd = ffb::dense;

constexpr int kAnBN = 128;          // dense analysis tile columns (bf16 hi + lo operands)
constexpr int kSyBN = 256;          // dense synthesis tile columns (tf32 operand)
constexpr int kGrBN = 32;           // grouped GEMMs: one 32-coefficient group per row
constexpr int64_t kChunk = 8192;    // tokens per pass: bounds the workspace
constexpr int kSmemOptin = 227 * 1024;
constexpr size_t kBlockBytes = 8192;  // group block operands of one frame (hi, lo, sy)

using AnShape = fd::GemmShape<fd::KIND_BF16_HILO, kAnBN>;
using SyShape = fd::GemmShape<fd::KIND_TF32, kSyBN>;
using GrAnShape = fd::GemmShape<fd::KIND_BF16_HILO, kGrBN>;
using GrSyShape = fd::GemmShape<fd::KIND_TF32, kGrBN>;

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline int64_t rup(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

const FfbPlanHeader* header_of(const framefb_plan* p) {
  if (!p || p->image.size() < sizeof(FfbPlanHeader)) return nullptr;
  const FfbPlanHeader* h = reinterpret_cast<const FfbPlanHeader*>(p->image.data());
  if (h->magic != FFB_PLAN_MAGIC || h->version != FFB_PLAN_VERSION || h->P != fd::kSpmmThreads) return nullptr;
  if (static_cast<size_t>(h->total_bytes) > p->image.size()) return nullptr;  // (parts follow the plan)
  return h;
}

// One SpMM pass: the MODE bits it runs, its tokens per unit and shared memory.
struct SpmmPass {
  int mode, TT;
  size_t smem;
  int32_t oV, oU, oRZ, oRG, oDC;
};

// Shared-memory map of a SpMM pass (floats), 0 bytes when it does not fit.
SpmmPass spmm_pass(const FfbPlanHeader& h, int mode, int TT) {
  const bool F = mode & 1, D = mode & 2, C = mode & 4;
  SpmmPass s{mode, TT, 0, 0, 0, 0, 0, 0};
  int64_t off = 0;
  auto take = [&](int64_t floats) {
    const int32_t o = static_cast<int32_t>(off);
    off = rup(off + floats, 4);
    return o;
  };
  s.oV = take((F || C) ? rup(h.n, 4) * TT : 0);
  s.oU = take((D || C) ? rup(h.m, 4) * TT : 0);
  s.oRZ = take(F ? rup(h.m + h.ovfZ, 4) * TT : 0);
  s.oRG = take(D ? rup(h.n + h.ovfG, 4) * TT : 0);
  s.oDC = take(0);  // the dC sums live in registers
  const size_t bytes = static_cast<size_t>(off) * 4;
  s.smem = bytes <= static_cast<size_t>(kSmemOptin) ? std::max<size_t>(bytes, 16) : 0;
  return s;
}

// The SpMM passes of `ops`: one pass when everything fits, else the column
// path with dC and then the row path; empty when even one token per unit
// does not fit.
std::vector<SpmmPass> spmm_passes(const FfbPlanHeader& h, int32_t ops) {
  const int all = ops & 7;
  for (int TT = 2; TT >= 1; --TT) {
    const SpmmPass s = spmm_pass(h, all, TT);
    if (s.smem) return {s};
  }
  const int col = all & 6, row = all & 1;
  std::vector<SpmmPass> out;
  for (const int m : {col, row}) {
    if (!m) continue;
    SpmmPass best{};
    for (int TT = 2; TT >= 1 && !best.smem; --TT) best = spmm_pass(h, m, TT);
    if (!best.smem) return {};
    out.push_back(best);
  }
  return out;
}

// Register chunk length of the SpMM for a plan (0: more entries per column
// than the kernels hold).
int spmm_e(const FfbPlanHeader& h) {
  const int e = std::max(h.EZ, h.EG);
  return e <= 8 ? 8 : e <= 16 ? 16 : e <= 32 ? 32 : 0;
}

// Geometry of one matrix.  Workspace of a call: the group block operands of
// its grouped matrices' frames (kBlockBytes each, two per matrix), then one
// matrix region (the largest), reused matrix after matrix:
//   V [Nc][ldv], U [Nc][ldu], Z [Nc][ldu], G [Nc][ldv] fp32, dC partials.
struct Geom {
  const FfbPlanHeader* h;
  bool grouped;
  int64_t Nc;       // tokens per chunk
  int64_t nchunks;
  int64_t ldv, ldu;  // floats per row of the K_n-wide and the K_m-wide buffers
  int32_t grid;     // SpMM CTAs of a full chunk
  int32_t stride;   // dC partial slot stride (floats)
  std::vector<SpmmPass> passes;
  size_t off_u, off_z, off_g, off_part, bytes;
};

framefb_status geom_of(const framefb_mat& M, int32_t ops, int sms, Geom& g) {
  g.h = header_of(M.plan);
  if (!g.h) return FRAMEFB_EINVAL;
  const FfbPlanHeader& h = *g.h;
  g.grouped = h.layout == FFB_LAYOUT_GROUPS;
  g.Nc = std::min<int64_t>(std::max<int32_t>(M.N, 1), kChunk);
  g.nchunks = M.N > 0 ? (M.N + g.Nc - 1) / g.Nc : 0;
  // grouped rows are viewed as 32-float groups: no padding allowed
  g.ldv = g.grouped ? h.n : rup(h.n, 4);
  g.ldu = g.grouped ? h.m : rup(h.m, 4);
  g.passes = spmm_passes(h, ops);
  if (g.passes.empty() || spmm_e(h) == 0) return FRAMEFB_EUNSUPPORTED;  // at most 32 entries per plan column
  int tt = 2;
  for (const SpmmPass& p : g.passes) tt = std::min(tt, p.TT);
  const int64_t units = (g.Nc + tt - 1) / tt;
  // one CTA per SM: each CTA loads its plan chunk into registers once
  g.grid = static_cast<int32_t>(std::max<int64_t>(1, std::min<int64_t>(units, sms)));
  g.stride = (h.nnz + 63) & ~63;
  const size_t rv = rup(static_cast<size_t>(g.Nc) * g.ldv * 4, 256), ru = rup(static_cast<size_t>(g.Nc) * g.ldu * 4, 256);
  g.off_u = rv;
  g.off_z = g.off_u + ru;
  g.off_g = g.off_z + ru;
  g.off_part = g.off_g + rv;
  const size_t part = (ops & FRAMEFB_OP_GRAD_COEFF) && h.nnz > 0
                          ? static_cast<size_t>(g.nchunks) * g.grid * g.stride * 4
                          : 0;
  g.bytes = g.off_part + rup(part, 256);
  return FRAMEFB_OK;
}

int sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return sms;
}

bool groups16(const framefb_dev_frame* f, int32_t d) {
  return f && f->dft_groups && f->k == 16 && f->d == d && f->ncols == d && f->rho * 16 == d && f->val;
}

bool check_mat(const framefb_mat& M, int32_t ops, const FfbPlanHeader& h) {
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  const framefb_dev_frame* fi = M.fin;
  const framefb_dev_frame* fo = M.fout;
  if (!fi || !fo) return false;
  const bool grouped = h.layout == FFB_LAYOUT_GROUPS;
  if (grouped) {
    if (!groups16(fi, M.n) || !groups16(fo, M.m) || h.n != M.n || h.m != M.m) return false;
  } else {
    if (!fi->dense || !fo->dense || !aligned16(fi->dense) || !aligned16(fo->dense)) return false;
    if (h.layout != FFB_LAYOUT_DENSE || h.n != fi->ncols || h.m != fo->ncols) return false;
    if (h.d_in != M.n || h.d_out != M.m || fi->d != M.n || fo->d != M.m) return false;
  }
  if (M.N < 0 || !std::isfinite(M.scale)) return false;
  if ((F || D) && h.nnz > 0 && !M.c_val) return false;
  if (C && h.nnz > 0 && !M.dC) return false;
  if (M.N == 0) return true;
  const bool needX = F || C, needdY = D || C;
  if ((needX || D) && (M.ldx < M.n || (M.ldx * 2) % 16 || (grouped && M.ldx != M.n))) return false;
  if ((needdY || F) && (M.ldy < M.m || (M.ldy * 2) % 16 || (grouped && M.ldy != M.m))) return false;
  if (needX && (!M.X || !aligned16(M.X))) return false;
  if (needdY && (!M.dY || !aligned16(M.dY))) return false;
  if (F && (!M.Y || !aligned16(M.Y))) return false;
  if (D && (!M.dX || !aligned16(M.dX))) return false;
  return true;
}

// Distinct frames of the grouped matrices, in first-use order (their group
// blocks occupy the start of the workspace).
std::vector<const framefb_dev_frame*> block_frames(const framefb_mat* mats, int32_t nmats) {
  std::vector<const framefb_dev_frame*> out;
  for (int32_t j = 0; j < nmats; ++j) {
    const FfbPlanHeader* h = header_of(mats[j].plan);
    if (!h || h->layout != FFB_LAYOUT_GROUPS) continue;
    for (const framefb_dev_frame* f : {mats[j].fin, mats[j].fout})
      if (std::find(out.begin(), out.end(), f) == out.end()) out.push_back(f);
  }
  return out;
}

// 2-D tensor map of a row-major [rows][cols] matrix (pitch in bytes), box
// {128 bytes of columns, box_rows rows}, 128-byte swizzle, zeros outside.
bool encode_2d(CUtensorMap* map, CUtensorMapDataType type, int esz, const void* base, int64_t cols, int64_t rows,
               int64_t pitch, int box_rows) {
  const EncodeTiledFn fn = encode_tiled();
  if (!fn || cols <= 0 || rows <= 0) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(pitch)};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(fd::kRowBytes / esz), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, type, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

void* spmm_kernel_ptr(int mode, int TT, int E) {
#define FFB_SPMM_E(M, T)                                                   \
  return E == 8    ? reinterpret_cast<void*>(fd::dense_spmm_kernel<M, T, 8>)  \
         : E == 16 ? reinterpret_cast<void*>(fd::dense_spmm_kernel<M, T, 16>) \
                   : reinterpret_cast<void*>(fd::dense_spmm_kernel<M, T, 32>);
#define FFB_SPMM(M)         \
  case M:                   \
    if (TT == 2) {          \
      FFB_SPMM_E(M, 2)      \
    } else {                \
      FFB_SPMM_E(M, 1)      \
    }
  if (E != 8 && E != 16 && E != 32) return nullptr;
  switch (mode) {  // single passes take ops & 7; split passes the column part (& 6) and the row part (1)
    FFB_SPMM(1)
    FFB_SPMM(2)
    FFB_SPMM(4)
    FFB_SPMM(6)
    FFB_SPMM(7)
    default: return nullptr;
  }
#undef FFB_SPMM
#undef FFB_SPMM_E
}

struct GemmKind {
  void* fn;
  uint32_t smem;
  int bn;
  int per_sm;  // CTAs per SM the kernel's shared memory allows
};
GemmKind an_kernel(bool grouped) {
  if (grouped)
    return {reinterpret_cast<void*>(fd::dense_gemm_kernel<fd::KIND_BF16_HILO, fd::EPI_STORE_F32, kGrBN>),
            GrAnShape::SMEM, kGrBN, 2};
  return {reinterpret_cast<void*>(fd::dense_gemm_kernel<fd::KIND_BF16_HILO, fd::EPI_STORE_F32, kAnBN>),
          AnShape::SMEM, kAnBN, 1};
}
GemmKind sy_kernel(bool grouped) {
  if (grouped)
    return {reinterpret_cast<void*>(fd::dense_gemm_kernel<fd::KIND_TF32, fd::EPI_ACCUM_BF16, kGrBN>),
            GrSyShape::SMEM, kGrBN, 2};
  return {reinterpret_cast<void*>(fd::dense_gemm_kernel<fd::KIND_TF32, fd::EPI_ACCUM_BF16, kSyBN>),
          SyShape::SMEM, kSyBN, 1};
}

// Queue one contraction launch over `L` (problems filled, tiles counted).
framefb_status launch_gemm(const GemmKind& k, fd::GemmLaunch& L, int sms, cudaStream_t st) {
  if (L.total_tiles == 0) return FRAMEFB_OK;
  if (cudaFuncSetAttribute(k.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(k.smem)) != cudaSuccess)
    return FRAMEFB_ECUDA;
  const int grid = std::min(L.total_tiles, sms * k.per_sm);
  void* args[] = {&L};
  if (cudaLaunchKernel(k.fn, dim3(grid), dim3(fd::kGemmThreads), args, k.smem, st) != cudaSuccess)
    return FRAMEFB_ECUDA;
  return FRAMEFB_OK;
}

// Append a problem to a launch: out[M][N] (+)= A[M][K] B[N][K]^T.
void add_problem(fd::GemmLaunch& L, int BN, void* out, int64_t ldo, int64_t M, int64_t N, int64_t K, float alpha) {
  fd::GemmProblem& P = L.p[L.nprob];
  P.out = out;
  P.ldo = ldo;
  P.M = static_cast<int32_t>(M);
  P.N = static_cast<int32_t>(N);
  P.K = static_cast<int32_t>(K);
  P.nt = static_cast<int32_t>((N + BN - 1) / BN);
  P.tile0 = L.total_tiles;
  P.alpha = alpha;
  L.total_tiles += static_cast<int32_t>((M + fd::kBM - 1) / fd::kBM) * P.nt;
  ++L.nprob;
}

// Tensor maps of the analysis operands of one side: activations A (tokens
// t0 .. t0 + Nc of `act`, d features, leading dimension ld) and the frame's
// B operands.  grouped: A viewed as [Nc * d/32][32], B = the group block.
bool an_maps(fd::GemmProblem& P, bool grouped, const void* act, int64_t ld, int64_t t0, int64_t Nc, int64_t d,
             int64_t K, const framefb_dev_frame* f, const uint8_t* blocks) {
  const __nv_bfloat16* a = static_cast<const __nv_bfloat16*>(act) + t0 * ld;
  if (grouped)
    return encode_2d(&P.a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, a, 32, Nc * (d / 32), 64, fd::kBM) &&
           encode_2d(&P.b0, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, blocks, 32, 32, 64, kGrBN) &&
           encode_2d(&P.b1, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, blocks + 2048, 32, 32, 64, kGrBN);
  const FfbDenseLayout Lf = ffb_dense_layout(d, K);
  const uint8_t* di = static_cast<const uint8_t*>(f->dense);
  return encode_2d(&P.a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, a, d, Nc, ld * 2, fd::kBM) &&
         encode_2d(&P.b0, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, di + Lf.off_hi, d, K, Lf.dp * 2, kAnBN) &&
         encode_2d(&P.b1, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, di + Lf.off_lo, d, K, Lf.dp * 2, kAnBN);
}

// Tensor maps of the synthesis operands of one side: the row sums R
// ([Nc][ldr] fp32, K columns) and the frame's synthesis operand.
bool sy_maps(fd::GemmProblem& P, bool grouped, const float* R, int64_t ldr, int64_t Nc, int64_t d, int64_t K,
             const framefb_dev_frame* f, const uint8_t* blocks) {
  if (grouped)
    return encode_2d(&P.a, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, R, 32, Nc * (K / 32), 128, fd::kBM) &&
           encode_2d(&P.b0, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, blocks + 4096, 32, 32, 128, kGrBN);
  const FfbDenseLayout Lf = ffb_dense_layout(d, K);
  const uint8_t* di = static_cast<const uint8_t*>(f->dense);
  return encode_2d(&P.a, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, R, K, Nc, ldr * 4, fd::kBM) &&
         encode_2d(&P.b0, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, di + Lf.off_sy, K, d, Lf.cp * 4, kSyBN);
}

}  // namespace

framefb_status dense_check(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dt, size_t* ws_need) {
  *ws_need = 0;
  if (nmats == 0) return FRAMEFB_OK;
  if (dt != FRAMEFB_BF16) return FRAMEFB_EUNSUPPORTED;  // this path takes bf16 activations
  if (!encode_tiled()) return FRAMEFB_ECUDA;
  const int sms = sm_count();
  if (sms <= 0) return FRAMEFB_ECUDA;
  size_t region = 0;
  bool work = false;
  for (int32_t j = 0; j < nmats; ++j) {
    Geom g;
    const framefb_status s = geom_of(mats[j], ops, sms, g);
    if (s != FRAMEFB_OK) return s;
    if (!check_mat(mats[j], ops, *g.h)) return FRAMEFB_EINVAL;
    if (mats[j].N > 0 || ((ops & FRAMEFB_OP_GRAD_COEFF) && g.h->nnz > 0)) {
      region = std::max(region, g.bytes);
      work = true;
    }
  }
  const std::vector<const framefb_dev_frame*> fr = block_frames(mats, nmats);
  if (work) *ws_need = rup(fr.size() * kBlockBytes, 256) + region;
  return FRAMEFB_OK;
}

framefb_status dense_run(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dt, void* ws,
                         size_t ws_bytes, cudaStream_t st) {
  (void)dt;
  (void)ws_bytes;
  if (nmats == 0) return FRAMEFB_OK;
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  const int sms = sm_count();
  if (sms <= 0) return FRAMEFB_ECUDA;
  uint8_t* w = static_cast<uint8_t*>(ws);
  // group block operands of the grouped matrices' frames
  const std::vector<const framefb_dev_frame*> fr = block_frames(mats, nmats);
  for (size_t i0 = 0; i0 < fr.size(); i0 += 8) {
    fd::GroupBlockArgs a;
    std::memset(&a, 0, sizeof(a));
    const int nb = static_cast<int>(std::min<size_t>(8, fr.size() - i0));
    for (int i = 0; i < nb; ++i) {
      a.val[i] = fr[i0 + i]->val;
      a.rho[i] = fr[i0 + i]->rho;
      a.out[i] = w + (i0 + i) * kBlockBytes;
    }
    void* args[] = {&a};
    if (cudaLaunchKernel(reinterpret_cast<void*>(fd::group_block_kernel), dim3(nb), dim3(1024), args, 0, st) !=
        cudaSuccess)
      return FRAMEFB_ECUDA;
  }
  auto block_of = [&](const framefb_dev_frame* f) {
    const size_t i = std::find(fr.begin(), fr.end(), f) - fr.begin();
    return w + i * kBlockBytes;
  };
  uint8_t* region = w + rup(fr.size() * kBlockBytes, 256);
  for (int32_t j = 0; j < nmats; ++j) {
    const framefb_mat& M = mats[j];
    Geom g;
    if (geom_of(M, ops, sms, g) != FRAMEFB_OK) return FRAMEFB_EINVAL;
    const FfbPlanHeader& h = *g.h;
    const bool gr = g.grouped;
    const int64_t Kn = h.n, Km = h.m;
    float* V = reinterpret_cast<float*>(region);
    float* U = reinterpret_cast<float*>(region + g.off_u);
    float* Z = reinterpret_cast<float*>(region + g.off_z);
    float* G = reinterpret_cast<float*>(region + g.off_g);
    float* part = reinterpret_cast<float*>(region + g.off_part);
    const uint8_t* bi = gr ? block_of(M.fin) : nullptr;
    const uint8_t* bo = gr ? block_of(M.fout) : nullptr;
    // grouped GEMMs run over (token, group) rows with 32 columns
    const int64_t an_ld_v = gr ? 32 : g.ldv, an_ld_u = gr ? 32 : g.ldu;
    int32_t slots = 0;
    for (int64_t c = 0; c < g.nchunks; ++c) {
      const int64_t t0 = c * g.Nc, Nc = std::min<int64_t>(g.Nc, M.N - t0);
      {  // analysis: V = X Phi_in, U = dY Phi_out
        const GemmKind k = an_kernel(gr);
        fd::GemmLaunch L;
        std::memset(&L, 0, sizeof(L));
        if (F || C) {
          if (!an_maps(L.p[L.nprob], gr, M.X, M.ldx, t0, Nc, M.n, Kn, M.fin, bi)) return FRAMEFB_ECUDA;
          add_problem(L, k.bn, V, an_ld_v, gr ? Nc * (Kn / 32) : Nc, gr ? 32 : Kn, gr ? 32 : M.n, 1.f);
        }
        if (D || C) {
          if (!an_maps(L.p[L.nprob], gr, M.dY, M.ldy, t0, Nc, M.m, Km, M.fout, bo)) return FRAMEFB_ECUDA;
          add_problem(L, k.bn, U, an_ld_u, gr ? Nc * (Km / 32) : Nc, gr ? 32 : Km, gr ? 32 : M.m, 1.f);
        }
        const framefb_status s = launch_gemm(k, L, sms, st);
        if (s != FRAMEFB_OK) return s;
      }
      for (const SpmmPass& p : g.passes) {  // coefficient SpMM and dC partials
        fd::SpmmLaunch a;
        std::memset(&a, 0, sizeof(a));
        a.plan = static_cast<const uint8_t*>(M.plan_dev);
        a.c_val = M.c_val;
        a.V = V;
        a.U = U;
        a.Z = Z;
        a.G = G;
        a.partial = part;
        a.ldv = a.ldg = g.ldv;
        a.ldu = a.ldz = g.ldu;
        a.N = static_cast<int32_t>(Nc);
        a.stride = g.stride;
        a.slot0 = slots;
        a.oV = p.oV;
        a.oU = p.oU;
        a.oRZ = p.oRZ;
        a.oRG = p.oRG;
        a.oDC = p.oDC;
        const int64_t units = (Nc + p.TT - 1) / p.TT;
        const int grid = static_cast<int>(std::min<int64_t>(units, g.grid));
        void* fn = spmm_kernel_ptr(p.mode, p.TT, spmm_e(h));
        if (!fn ||
            cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(p.smem)) !=
                cudaSuccess)
          return FRAMEFB_ECUDA;
        void* args[] = {&a};
        if (cudaLaunchKernel(fn, dim3(grid), dim3(fd::kSpmmThreads), args, p.smem, st) != cudaSuccess)
          return FRAMEFB_ECUDA;
        if (p.mode & 4) slots += grid;
      }
      if (F || D) {  // synthesis: Y += s Z Phi_out^T, dX += s G Phi_in^T
        const GemmKind k = sy_kernel(gr);
        fd::GemmLaunch L;
        std::memset(&L, 0, sizeof(L));
        if (F) {
          fd::GemmProblem& P = L.p[L.nprob];
          if (!sy_maps(P, gr, Z, g.ldu, Nc, M.m, Km, M.fout, bo)) return FRAMEFB_ECUDA;
          P.b1 = P.b0;
          __nv_bfloat16* y = static_cast<__nv_bfloat16*>(M.Y) + t0 * M.ldy;
          add_problem(L, k.bn, y, gr ? 32 : M.ldy, gr ? Nc * (M.m / 32) : Nc, gr ? 32 : M.m, gr ? 32 : Km, M.scale);
        }
        if (D) {
          fd::GemmProblem& P = L.p[L.nprob];
          if (!sy_maps(P, gr, G, g.ldv, Nc, M.n, Kn, M.fin, bi)) return FRAMEFB_ECUDA;
          P.b1 = P.b0;
          __nv_bfloat16* x = static_cast<__nv_bfloat16*>(M.dX) + t0 * M.ldx;
          add_problem(L, k.bn, x, gr ? 32 : M.ldx, gr ? Nc * (M.n / 32) : Nc, gr ? 32 : M.n, gr ? 32 : Kn, M.scale);
        }
        const framefb_status s = launch_gemm(k, L, sms, st);
        if (s != FRAMEFB_OK) return s;
      }
    }
    if (C && h.nnz > 0) {
      if (slots == 0) {  // no tokens: the gradient is zero
        if (cudaMemsetAsync(M.dC, 0, sizeof(float) * h.nnz, st) != cudaSuccess) return FRAMEFB_ECUDA;
      } else {
        const float* pp = part;
        int32_t ns = slots, stride = g.stride, nnz = h.nnz;
        float alpha = M.scale;
        float* dC = M.dC;
        void* args[] = {&pp, &ns, &stride, &nnz, &alpha, &dC};
        if (cudaLaunchKernel(reinterpret_cast<void*>(fd::dense_dc_reduce_kernel), dim3((nnz + 255) / 256),
                             dim3(256), args, 0, st) != cudaSuccess)
          return FRAMEFB_ECUDA;
      }
    }
  }
  return FRAMEFB_OK;
}

void dense_kernel_names(const framefb_mat* mats, int32_t nmats, int32_t ops, std::vector<std::string>& out) {
  const bool F = ops & FRAMEFB_OP_FORWARD, D = ops & FRAMEFB_OP_BACKWARD_DX, C = ops & FRAMEFB_OP_GRAD_COEFF;
  std::vector<std::string> k;
  for (int32_t j = 0; j < nmats; ++j) {
    const FfbPlanHeader* h = header_of(mats[j].plan);
    if (!h || mats[j].N == 0) continue;
    const std::string sfx = h->layout == FFB_LAYOUT_GROUPS ? "<grouped>" : "";
    if (h->layout == FFB_LAYOUT_GROUPS) k.push_back("group_block_kernel");
    k.push_back("dense_gemm_kernel<bf16_hilo>" + sfx);
    k.push_back("dense_spmm_kernel<" + std::to_string(ops & 7) + ">");
    if (F || D) k.push_back("dense_gemm_kernel<tf32>" + sfx);
    if (C) k.push_back("dense_dc_reduce_kernel");
  }
  for (const std::string& s : k)
    if (std::find(out.begin(), out.end(), s) == out.end()) out.push_back(s);
}

framefb_status dense_wait_timeouts(uint32_t* count) {
  if (cudaMemcpyFromSymbol(count, fd::g_dense_timeouts, sizeof(uint32_t)) != cudaSuccess) return FRAMEFB_ECUDA;
  return FRAMEFB_OK;
}

}  // namespace ffb_host
