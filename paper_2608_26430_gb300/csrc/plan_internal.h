// Host-only definition of the opaque framefb_plan handle (shared by the host
// builder and the launcher, never seen by callers).
#pragma once
#include <stddef.h>
#include <stdint.h>
#include <vector>

struct framefb_plan;

// A part of a plan beyond the fused tcgen05 kernels' limits: the plan of a
// run of the support over a block of input and a block of output features.
struct FfbSubPlan {
  framefb_plan* plan;  // host copy of its image (sizes and checks)
  size_t dev_off;      // its image in the parent's device image
  size_t q_off;        // its entries' indices into the caller's C / dC (int32 [nq]) in the parent's image
  int32_t n0, m0;      // first input / output feature of its blocks
  int32_t nq;          // its entries
};

struct framefb_plan {
  std::vector<uint8_t> image;  // device image: FfbPlanHeader and its tables, then the parts
  std::vector<FfbSubPlan> subs;
  framefb_plan() = default;
  framefb_plan(const framefb_plan&) = delete;
  framefb_plan& operator=(const framefb_plan&) = delete;
  ~framefb_plan() {
    for (FfbSubPlan& sp : subs) delete sp.plan;
  }
};
