// Host interface between the launchers of libframefb (framefb_cuda.cu) and
// the dense path (framefb_dense.cu).  Internal: not part of the C ABI.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <string>
#include <vector>

#include "framefb.h"

namespace ffb_host {

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link
// against the driver library); NULL when the driver does not provide it.
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled();

// Validate the dense-path matrices of a call (plans with FFB_LAYOUT_DENSE)
// and report the workspace they need (bytes; the matrices run one after
// another and share it).
framefb_status dense_check(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dt, size_t* ws_need);

// Queue the dense path of every matrix on `st` (after dense_check).
framefb_status dense_run(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dt, void* ws,
                         size_t ws_bytes, cudaStream_t st);

// Kernels dense_run launches for `ops` (appended to `out`, no duplicates).
void dense_kernel_names(const framefb_mat* mats, int32_t nmats, int32_t ops, std::vector<std::string>& out);

// Bounded waits of the dense kernels that gave up on the current device.
framefb_status dense_wait_timeouts(uint32_t* count);

}  // namespace ffb_host
