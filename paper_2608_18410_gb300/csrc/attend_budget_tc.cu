// attend_budget_tc.cu -- the tensor-core attention (attend_tc.cuh) over a
// budget cache (per-token counts K_i, Sec. 3.5): the instance with three
// whole-row value gatherers.
#include "attend_tc.cuh"

namespace rs {

cudaError_t launch_attend_tc_budget(const AttendArgs &a) { return launch_attend_impl<true>(a); }

}  // namespace rs
