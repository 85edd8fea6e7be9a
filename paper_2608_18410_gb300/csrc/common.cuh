// common.cuh -- device helpers shared by the RoleSub kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "rolesub.h"

namespace rs {

// Status word at the start of every workspace: {code, detail}.
constexpr size_t kStatusBytes = 256;

// Programmatic dependent launch. A kernel started by launch_pdl may begin
// while its predecessor in the stream still runs: it must call pdl_wait()
// before touching anything the predecessor writes (pdl_wait returns once the
// predecessor has completed and its writes are visible; at once for a kernel
// launched the ordinary way). pdl_trigger() lets this kernel's own dependent
// be scheduled early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Loads of what the kernel before this one writes, in a kernel started by
// launch_pdl. Such a kernel is resident while its predecessor still writes,
// so that data must not be read through a const __restrict__ pointer or
// __ldg: the compiler may then take the read-only (non-coherent) path and
// move the load above pdl_wait(), and the kernel reads stale values (found on
// the language context, which the bias kernels read as soon as a small
// pooling grid let them start). These are ordinary global loads in asm
// volatile, so they stay after the wait.
__device__ __forceinline__ float ld_dep(const float *p)
{
    float v;
    asm volatile("ld.global.f32 %0, [%1];" : "=f"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ float4 ld_dep(const float4 *p)
{
    float4 v;
    asm volatile("ld.global.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p)
                 : "memory");
    return v;
}

__device__ __forceinline__ uint4 ld_dep(const uint4 *p)
{
    uint4 v;
    asm volatile("ld.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p)
                 : "memory");
    return v;
}

__device__ __forceinline__ uint32_t ld_dep(const uint8_t *p)
{
    uint32_t v;
    asm volatile("ld.global.u8 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

template <class... P, class... A>
inline cudaError_t launch_pdl(void (*kern)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              A &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<A>(args)...);
}

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
