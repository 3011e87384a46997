// Host-only definition of the opaque framefb_plan handle (shared by the host
// builder and the launcher, never seen by callers).
#pragma once
#include <stdint.h>
#include <vector>

struct framefb_plan {
  std::vector<uint8_t> image;  // device image: FfbPlanHeader followed by its tables
};
