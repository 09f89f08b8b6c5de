// Decode-side kernels of the selective-scan layer core: the batched
// single-byte recurrent step and the rollback gather of speculative decoding
// (MambaByte Section 6.3 and Algorithm 1). The verify scan shares the prefill
// kernel (prefill.cu).
//
// Both are HBM-streaming kernels. A (batch row, channel) pair owns 16 fp32
// states (64 contiguous bytes). In the step kernel four lanes share a channel,
// each holding 4 states in one float4, so a warp moves 512 contiguous bytes
// of state per instruction; each lane group serves kSlots channels so that
// every lane has kSlots independent 16-byte state loads in flight.
#include "common.cuh"
#include "tma.cuh"

namespace mbscan {
namespace {

constexpr int kStepThreads = 256;
constexpr int kSlots = 4;                                       // channels per lane group
constexpr int kStepChPerWarp = 8 * kSlots;                      // 32
constexpr int kStepChPerCta = kStepChPerWarp * (kStepThreads / 32);  // 256

// Lane q of a 4-lane group holds the group's shares part[0..3] (one per
// slot); return the full 4-lane sum of slot q (two shuffle rounds).
__device__ __forceinline__ float reduce_slots(const float (&part)[4], int q) {
    const bool hi = (q & 2) != 0;
    float k0 = hi ? part[2] : part[0], k1 = hi ? part[3] : part[1];
    const float s0 = hi ? part[0] : part[2], s1 = hi ? part[1] : part[3];
    k0 += __shfl_xor_sync(kFull, s0, 2);
    k1 += __shfl_xor_sync(kFull, s1, 2);
    const bool odd = (q & 1) != 0;
    const float keep = odd ? k1 : k0, send = odd ? k0 : k1;
    return keep + __shfl_xor_sync(kFull, send, 1);
}

// ---------------------------------------------------------------------------
// mb_step: state[b, d, :] <- one recurrence step (Eq. 2 with L = 1), y[b, 0, d].
// Lane (g, q) of a warp: slot j covers channel wbase + 8 j + g, states 4q..4q+3.
// The lane computes the channel scalars (Delta, Delta*x, D*x, silu z) only for
// slot q and hands Delta, Delta*x to its group by shuffle; after the 4-lane
// reduction it also owns slot q's output.
template <typename T>
__global__ void __launch_bounds__(kStepThreads, 4) step_kernel(ScanParams p) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane >> 2, q = lane & 3;
    const int64_t D = p.d_inner;
    const int64_t nchan = p.batch * D;
    const int64_t wbase = (int64_t)blockIdx.x * kStepChPerCta + warp * kStepChPerWarp;
    const T *x = static_cast<const T *>(p.x);
    const T *z = static_cast<const T *>(p.z);
    const T *dt = static_cast<const T *>(p.dt);
    const T *Bm = static_cast<const T *>(p.B);
    const T *Cm = static_cast<const T *>(p.C);
    float4 *state = reinterpret_cast<float4 *>(p.h_out);

    float4 h[kSlots];
#pragma unroll
    for (int j = 0; j < kSlots; ++j) {
        const int64_t ch = wbase + 8 * j + g;
        h[j] = ch < nchan ? __ldcs(state + ch * (kDState / 4) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
    }

    // channel scalars of slot q
    const int64_t mc = wbase + 8 * q + g;
    const bool mok = mc < nchan;
    const int64_t md = mok ? mc % D : 0;
    float delta = 0.f, gx = 0.f, xd = 0.f, sz = 1.f;
    if (mok) {
        const float xv = ldg1(x + mc);
        delta = softplus(ldg1(dt + mc) + (p.dt_bias ? __ldg(p.dt_bias + md) : 0.f));
        gx = delta * xv;
        xd = (p.D ? __ldg(p.D + md) : 0.f) * xv;
        if (z) sz = silu(ldg1(z + mc));
    }

    float part[kSlots];
#pragma unroll
    for (int j = 0; j < kSlots; ++j) {
        const int64_t ch = wbase + 8 * j + g;
        const int64_t cch = ch < nchan ? ch : 0;
        const int64_t b = cch / D, d = cch - b * D;
        const float dj = __shfl_sync(kFull, delta, 4 * g + j);
        const float gj = __shfl_sync(kFull, gx, 4 * g + j);
        const float4 av = ldg4(p.A + d * kDState + 4 * q);
        const float4 bv = ldg4(Bm + b * kDState + 4 * q);
        const float4 cv = ldg4(Cm + b * kDState + 4 * q);
        float2 h01 = make_float2(h[j].x, h[j].y), h23 = make_float2(h[j].z, h[j].w);
        const float2 dd = make_float2(dj, dj), gg = make_float2(gj, gj);
        const float2 e01 = mul2(dd, make_float2(av.x * kLog2e, av.y * kLog2e));
        const float2 e23 = mul2(dd, make_float2(av.z * kLog2e, av.w * kLog2e));
        h01 = fma2(make_float2(ex2(e01.x), ex2(e01.y)), h01, mul2(make_float2(bv.x, bv.y), gg));
        h23 = fma2(make_float2(ex2(e23.x), ex2(e23.y)), h23, mul2(make_float2(bv.z, bv.w), gg));
        h[j] = make_float4(h01.x, h01.y, h23.x, h23.y);
        const float2 acc = fma2(make_float2(cv.z, cv.w), h23, mul2(make_float2(cv.x, cv.y), h01));
        part[j] = acc.x + acc.y;
    }
    const float ysum = reduce_slots(part, q);

#pragma unroll
    for (int j = 0; j < kSlots; ++j) {
        const int64_t ch = wbase + 8 * j + g;
        if (ch < nchan) __stcs(state + ch * (kDState / 4) + q, h[j]);
    }
    if (mok) static_cast<T *>(p.y)[mc] = from_f32<T>((ysum + xd) * sz);
}

// ---------------------------------------------------------------------------
// mb_rollback: h_out[s] = accept[s] == 0 ? h0[s] : h_all[s, accept[s] - 1].
// Each thread copies kRbVec float4s of one stream (per_stream is a multiple of
// 4 float4s since d_inner * 16 floats = 4 * d_inner float4s).
constexpr int kRbThreads = 256;
constexpr int kRbVec = 4;

__global__ void __launch_bounds__(kRbThreads)
rollback_kernel(const float4 *h0 /* may alias h_out */, const float4 *__restrict__ h_all,
                const int32_t *__restrict__ accept, float4 *h_out, int64_t batch, int64_t k,
                int64_t per_stream /* float4s */, StatusBlock *status) {
    const int64_t i0 = ((int64_t)blockIdx.x * kRbThreads + threadIdx.x) * kRbVec;
    if (i0 >= batch * per_stream) return;
    const int64_t s = i0 / per_stream;
    const int64_t j0 = i0 - s * per_stream;
    const int a = __ldg(accept + s);
    if (a < 0 || a > k) {
        if (j0 == 0) report(status, 1 /* MB_ERR_INVALID_ARG */, s);
        return;
    }
    float4 v[kRbVec];
    const float4 *src = a == 0 ? (h0 ? h0 + i0 : nullptr) : h_all + (s * k + (a - 1)) * per_stream + j0;
#pragma unroll
    for (int u = 0; u < kRbVec; ++u) v[u] = src ? __ldcs(src + u) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int u = 0; u < kRbVec; ++u) h_out[i0 + u] = v[u];
}

}  // namespace

cudaError_t launch_step(const ScanParams &p, bool bf16, cudaStream_t s) {
    const int64_t nchan = p.batch * p.d_inner;
    const int64_t grid = (nchan + kStepChPerCta - 1) / kStepChPerCta;
    if (grid == 0) return cudaSuccess;
    if (bf16)
        step_kernel<__nv_bfloat16><<<(unsigned)grid, kStepThreads, 0, s>>>(p);
    else
        step_kernel<float><<<(unsigned)grid, kStepThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_rollback(const float *h0, const float *h_all, const int32_t *accept,
                            float *h_out, int64_t batch, int64_t k, int64_t d_inner,
                            StatusBlock *status, cudaStream_t s) {
    const int64_t per = d_inner * kDState / 4;
    const int64_t threads = batch * per / kRbVec;
    if (threads == 0) return cudaSuccess;
    const int64_t grid = (threads + kRbThreads - 1) / kRbThreads;
    rollback_kernel<<<(unsigned)grid, kRbThreads, 0, s>>>(
        reinterpret_cast<const float4 *>(h0), reinterpret_cast<const float4 *>(h_all), accept,
        reinterpret_cast<float4 *>(h_out), batch, k, per, status);
    return cudaGetLastError();
}

}  // namespace mbscan
