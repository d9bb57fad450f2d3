// common.cuh -- small device helpers shared by the libreco kernels (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace reco {

// Bits of the sticky device error word (read and cleared by reco_check).
enum : unsigned {
    ERR_LEN = 1u,    // a unit length outside its valid range
    ERR_KEEP = 2u,   // a keep count outside [w, len]
    ERR_ID = 4u,     // a reflection id outside [0, V)
    ERR_TOKEN = 8u,  // an answer token outside [0, V)
    ERR_ROOM = 16u,  // no room to append a decoded row
    ERR_INTERNAL = 32u,  // an internal consistency check failed (the access was skipped)
    ERR_NORM = 64u,  // a window row's log-normaliser passed to scoring is not finite
};

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ void raise_error(unsigned *err, unsigned bit) { atomicOr(err, bit); }

__device__ __forceinline__ float to_float(float x) { return x; }
__device__ __forceinline__ float to_float(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_float(float x);
template <> __device__ __forceinline__ float from_float<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float x)
{
    return __float2bfloat16_rn(x);
}

// Programmatic dependent launch.  Kernels launched with launch_pdl() may be scheduled
// while the previous kernel in the stream drains; each one calls wait_prior_grid()
// before it reads anything a previous kernel wrote (it returns at once when the launch
// was an ordinary one).  No kernel signals its dependents early, so a dependent grid
// starts only as the previous one's blocks exit: what overlaps is launch processing and
// the part of a kernel before its wait.
__device__ __forceinline__ void wait_prior_grid() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// 2^x on the MUFU pipe (ex2.approx.ftz.f32).
__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int warp_sum_int(int v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Combine two (max, sum) pairs of a log2-domain online softmax.
__device__ __forceinline__ void lse_merge(float &m, float &s, float m2, float s2)
{
    float mn = fmaxf(m, m2);
    if (mn == -INFINITY) return;  // both empty
    s = s * fast_exp2(m - mn) + s2 * fast_exp2(m2 - mn);
    m = mn;
}

// Read-only 16-byte global load that bypasses L1 allocation (streamed data).
__device__ __forceinline__ uint4 ld_stream_u4(const void *p)
{
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

}  // namespace reco
