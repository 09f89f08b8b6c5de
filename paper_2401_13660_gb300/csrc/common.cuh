// Device helpers shared by the selective-scan kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "internal.h"

namespace mbscan {

constexpr float kLog2e = 1.4426950408889634f;
constexpr unsigned kFull = 0xffffffffu;

// 2^x on the SFU (MUFU.EX2), flushing subnormal results to zero.
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

constexpr float kLn2 = 0.6931471805599453f;

// log2(x) on the SFU (MUFU.LG2).
__device__ __forceinline__ float lg2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Delta = softplus(v) = log(1 + e^v) (Eq. 3), with u = e^v from the SFU:
//  * u < 2^-5: log1p(u) by its Taylor series to u^3 (truncation < 8e-6 relative);
//  * otherwise: ln 2 * log2(1 + u) on the SFU, where 1 + u >= 1.03 carries no
//    cancellation (relative error < 1e-5 at the switch point, falling above);
//  * v > 15: v itself (the dropped log1p(e^-v) < 3.1e-7 is below fp32 resolution).
__device__ __forceinline__ float softplus(float v) {
    const float u = ex2(v * kLog2e);
    const float series = u * fmaf(u, fmaf(u, 0.33333334f, -0.5f), 1.f);
    const float logw = lg2(1.f + u) * kLn2;
    const float r = u < 0.03125f ? series : logw;
    return v > 15.f ? v : r;
}

// silu(z) = z * sigmoid(z), the Swish gate of the Mamba block. For z < -88
// e^-z overflows to inf and the quotient is -0, the correctly rounded limit.
__device__ __forceinline__ float silu(float z) {
    return __fdividef(z, 1.f + ex2(-z * kLog2e));
}

// Element loads of the input dtype, widened to fp32.
__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

template <typename T> __device__ __forceinline__ float ldg1(const T *p) { return to_f32(__ldg(p)); }

// Four consecutive elements starting at p (8-byte aligned for bf16, 16 for fp32).
__device__ __forceinline__ float4 ldg4(const float *p) { return __ldg(reinterpret_cast<const float4 *>(p)); }
__device__ __forceinline__ float4 ldg4(const __nv_bfloat16 *p) {
    uint2 u = __ldg(reinterpret_cast<const uint2 *>(p));
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

// Two consecutive elements starting at p (4-byte aligned for bf16, 8 for fp32).
__device__ __forceinline__ float2 ldg2(const float *p) { return __ldg(reinterpret_cast<const float2 *>(p)); }
__device__ __forceinline__ float2 ldg2(const __nv_bfloat16 *p) {
    unsigned u = __ldg(reinterpret_cast<const unsigned *>(p));
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}

// ---- Programmatic dependent launch. Kernels launched with launch_pdl may
// start while the previous kernel on the stream is still draining; each such
// kernel runs pdl_wait() before its first global-memory read or write, which
// returns once every prerequisite grid has completed and its writes are
// visible, so only shared-memory set-up and L2 prefetches (hints that return
// no data) overlap the predecessor. pdl_trigger() lets the
// next kernel launch before this one completes (it still waits for it). Only
// the persistent decode step and the single-wave fused convolution +
// x-projection issue it: a grid of many short-lived CTAs that triggers early
// lets the next grid's CTAs take SM slots as they free up, which leaves SMs
// unevenly loaded when that grid fills less than every slot (measured:
// back-to-back prefills of 448 CTAs, 822 -> 990 us).
#ifndef MB_PDL
#define MB_PDL 1
#endif
__device__ __forceinline__ void pdl_wait() {
#if MB_PDL
    asm volatile("griddepcontrol.wait;" ::: "memory");
#endif
}
__device__ __forceinline__ void pdl_trigger() {
#if MB_PDL
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
#endif
}

// Launch `kern` on `s`; with overlap = true it may start during the previous
// kernel's tail (see pdl_wait). The decode step and the fused convolution +
// x-projection with its reduction use the overlap (whole-model decode 2.92 ->
// 2.89 ms); next to cuBLAS kernels (which trigger early) the short element-wise
// kernels measured slower with it (3.32 -> 3.38 ms), so they launch plainly.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(bool overlap, void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = (MB_PDL && overlap) ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// Record the first device-side error of a call in the workspace status block.
__device__ __forceinline__ void report(StatusBlock *sb, int code, long long detail) {
    if (sb == nullptr) return;
    if (atomicCAS(&sb->code, 0, code) == 0) {
        sb->detail = detail;
        __threadfence();
    }
}

}  // namespace mbscan
