// Launch-plan query of the whole-sequence forward beyond ForwardPlan (pbb_forward.cu).
#pragma once

#include "pbb_internal.h"

namespace pbb {

// The query tiles (of 128 rows) one persistent CTA of the forward works on at once for these
// sizes on the current device: 2 where the paired-item kernel runs, else 1.
cudaError_t plan_forward_query_tiles(const ForwardArgs& a, int* query_tiles);

}  // namespace pbb
