// selftest.cu -- a self-test of the bounded mbarrier wait that every
// tensor-core kernel of the library uses (sm100.cuh). The paper has no
// counterpart: this is the library's failure handling.
//
// One CTA of two warps initialises an mbarrier that nothing ever arrives on.
// Warp 0's elected lane waits on it through the same loop as the production
// waits, with the caller's short limit: the wait runs out, records
// ROLESUB_ETIMEOUT and the site in the status word and raises the CTA's
// abort flag. Warp 1's lane waits with the production limit (about two
// seconds) and must come back at once through that flag, as the other roles
// of a kernel do when one of its waits gives up. No copy or tensor-core
// operation is in flight, so the kernel simply returns.
#include "internal.h"
#include "sm100.cuh"

namespace rs {
namespace {

constexpr int kSiteLeader = 900;    // the wait that runs out
constexpr int kSiteFollower = 901;  // the wait ended by the abort flag

__global__ void __launch_bounds__(64, 1)
    k_wait_selftest(uint64_t limit_ns, int32_t *status, int64_t *out)
{
    using namespace sm100;
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
        const uint64_t t0 = global_ns();
        bool ok;
        if (warp == 0) {
            ok = mbar_wait_loop(smem_u32(&bar), 0, status, &abort_flag, kSiteLeader, limit_ns);
        } else {
            // starts after the leader has given up or while it waits; either
            // way the abort flag ends it within one sleep hint
            ok = mbar_wait(smem_u32(&bar), 0, status, &abort_flag, kSiteFollower);
        }
        out[2 * warp] = ok ? 1 : 0;
        out[2 * warp + 1] = (int64_t)(global_ns() - t0);
    }
    __syncthreads();
    if (threadIdx.x == 0) asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(smem_u32(&bar)) : "memory");
}

}  // namespace
}  // namespace rs

extern "C" rolesub_status rolesub_wait_selftest(int64_t limit_ns, void *workspace, int64_t *out, void *stream)
{
    if (limit_ns < 1000 || limit_ns > (int64_t)rs::sm100::kWaitLimitNs) return ROLESUB_EINVAL;
    if (!workspace || !out) return ROLESUB_EINVAL;
    if (((uintptr_t)workspace | (uintptr_t)out) & 15) return ROLESUB_EINVAL;
    rs::k_wait_selftest<<<1, 64, 0, (cudaStream_t)stream>>>((uint64_t)limit_ns, (int32_t *)workspace, out);
    rs::count_launches(1);
    return cudaGetLastError() == cudaSuccess ? ROLESUB_OK : ROLESUB_ECUDA;
}
