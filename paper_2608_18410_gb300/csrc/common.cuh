// common.cuh -- device helpers shared by the RoleSub kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "rolesub.h"

namespace rs {

// Status word at the start of every workspace: {code, detail}.
constexpr size_t kStatusBytes = 256;

__device__ __forceinline__ void report(int32_t *status, int32_t code, int32_t detail)
{
    if (status && atomicCAS(status, 0, code) == 0) atomicExch(status + 1, detail);
}

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }

template <class T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x)
{
    return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Device-side view of a plan blob (pointers into the device copy).
struct PlanDev {
    const rolesub_segment *segs;
    const rolesub_episode *eps;
    const int32_t *row_seg;
    const int32_t *routed;
    const int32_t *stored;
    const int32_t *route_tiles;
};

}  // namespace rs
