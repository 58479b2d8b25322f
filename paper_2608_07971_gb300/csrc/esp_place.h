// Host entry points of the placement kernels used only by test hooks (internal).
#pragma once

#include "esp_kernels.h"

namespace esp {

// launch_place_res with the grid barrier held: the arrival counter starts at 0xC0C0C0C0, about 2^30
// arrivals short of any target the kernel waits for, so no CTA passes the first barrier, every
// CTA's bounded wait runs out and the solve reports a timeout (failure detection without a fault).
cudaError_t launch_place_res_held(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a,
                                  const PlaceRes &pr, cudaStream_t stream);

}  // namespace esp
