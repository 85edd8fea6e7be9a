// attend_tc.cu -- the tensor-core attention (attend_tc.cuh) for fixed-k
// caches, and the entry point that dispatches budget caches (per-token
// counts) to attend_budget_tc.cu.
#include "attend_tc.cuh"

namespace rs {

bool attend_tc_supported(const rolesub_shape *s)
{
    // unit records hold h in 10 bits and l in 14
    return s->dtype == ROLESUB_BF16 && s->head_dim == kDh && s->num_groups == kG && s->num_heads <= 1024 &&
           s->num_layers <= 16384;
}

cudaError_t launch_attend_tc(const AttendArgs &a)
{
    return a.k_tok ? launch_attend_tc_budget(a) : launch_attend_impl<false>(a);
}

}  // namespace rs
