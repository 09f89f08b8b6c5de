// Decode-side kernels of the selective-scan layer core: the batched
// single-byte recurrent step, the speculative-decoding verify scan that keeps
// every per-position state, and the rollback gather (MambaByte Section 3,
// Section 6.3 and Algorithm 1).
//
// All three are HBM-streaming kernels: a (batch row, channel) pair owns 16
// fp32 states (64 contiguous bytes). Four lanes share one channel, each lane
// holding 4 states in one float4, so that a warp moves 512 contiguous bytes of
// state per instruction. The channel's scalars (dt, x, z) are broadcast to the
// four lanes; C.h is reduced over the four lanes with two xor-shuffles.
#include "common.cuh"

namespace mbscan {
namespace {

constexpr int kThreads = 256;         // 64 channels per CTA per channel slot
constexpr int kChanPerCta = kThreads / 4;

// One time step of one channel on one lane (states 4q..4q+3). Returns this
// lane's share of C.h.
__device__ __forceinline__ float lane_update(float4 &h, const float4 a2, float delta, float dx,
                                            const float4 b, const float4 c) {
    h.x = fmaf(ex2(delta * a2.x), h.x, b.x * dx);
    h.y = fmaf(ex2(delta * a2.y), h.y, b.y * dx);
    h.z = fmaf(ex2(delta * a2.z), h.z, b.z * dx);
    h.w = fmaf(ex2(delta * a2.w), h.w, b.w * dx);
    return fmaf(c.x, h.x, fmaf(c.y, h.y, fmaf(c.z, h.z, c.w * h.w)));
}

// ---------------------------------------------------------------------------
// mb_step: state[b, d, :] <- one recurrence step; y[b, 0, d]. CPT channels per
// thread (strided by kChanPerCta) keep several 16-byte state loads in flight.
template <typename T, int CPT>
__global__ void __launch_bounds__(kThreads) step_kernel(ScanParams p) {
    const int q = threadIdx.x & 3;
    const int64_t nchan = p.batch * p.d_inner;
    const int64_t base = (int64_t)blockIdx.x * (kChanPerCta * CPT) + (threadIdx.x >> 2);
    const T *x = static_cast<const T *>(p.x);
    const T *z = static_cast<const T *>(p.z);
    const T *dt = static_cast<const T *>(p.dt);
    const T *Bm = static_cast<const T *>(p.B);
    const T *Cm = static_cast<const T *>(p.C);
    T *y = static_cast<T *>(p.y);

    float4 h[CPT];
    bool ok[CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        const int64_t ch = base + (int64_t)j * kChanPerCta;
        ok[j] = ch < nchan;
        h[j] = ok[j] ? __ldcs(reinterpret_cast<const float4 *>(p.h_out + ch * kDState) + q)
                     : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        const int64_t ch = base + (int64_t)j * kChanPerCta;
        const int64_t b = ok[j] ? ch / p.d_inner : 0;
        const int64_t d = ok[j] ? ch - b * p.d_inner : 0;
        const int64_t i = ok[j] ? ch : 0;  // [b, 0, d] with seqlen 1
        const float xv = ldg1(x + i);
        const float v = ldg1(dt + i) + (p.dt_bias ? __ldg(p.dt_bias + d) : 0.f);
        const float delta = softplus(v);
        float4 a2 = ldg4(p.A + d * kDState + 4 * q);
        a2.x *= kLog2e; a2.y *= kLog2e; a2.z *= kLog2e; a2.w *= kLog2e;
        const float4 bv = ldg4(Bm + b * kDState + 4 * q);
        const float4 cv = ldg4(Cm + b * kDState + 4 * q);
        float part = lane_update(h[j], a2, delta, delta * xv, bv, cv);
        part += __shfl_xor_sync(kFull, part, 1);
        part += __shfl_xor_sync(kFull, part, 2);
        if (ok[j]) {
            __stcs(reinterpret_cast<float4 *>(p.h_out + ch * kDState) + q, h[j]);
            if (q == 0) {
                float out = part + (p.D ? __ldg(p.D + d) : 0.f) * xv;
                if (z) out *= silu(ldg1(z + i));
                y[i] = from_f32<T>(out);
            }
        }
    }
}

// ---------------------------------------------------------------------------
// mb_scan_verify: from h0, scan k drafted bytes; write every state to h_all.
template <typename T>
__global__ void __launch_bounds__(kThreads) verify_kernel(ScanParams p) {
    const int q = threadIdx.x & 3;
    const int64_t nchan = p.batch * p.d_inner;
    const int64_t ch = (int64_t)blockIdx.x * kChanPerCta + (threadIdx.x >> 2);
    const bool ok = ch < nchan;
    const int64_t b = ok ? ch / p.d_inner : 0;
    const int64_t d = ok ? ch - b * p.d_inner : 0;
    const int64_t L = p.seqlen, D = p.d_inner;
    const T *x = static_cast<const T *>(p.x);
    const T *z = static_cast<const T *>(p.z);
    const T *dt = static_cast<const T *>(p.dt);
    const T *Bm = static_cast<const T *>(p.B);
    const T *Cm = static_cast<const T *>(p.C);
    T *y = static_cast<T *>(p.y);

    float4 h = (ok && p.h0) ? __ldg(reinterpret_cast<const float4 *>(p.h0 + ch * kDState) + q)
                            : make_float4(0.f, 0.f, 0.f, 0.f);
    float4 a2 = ldg4(p.A + d * kDState + 4 * q);
    a2.x *= kLog2e; a2.y *= kLog2e; a2.z *= kLog2e; a2.w *= kLog2e;
    const float bias = p.dt_bias ? __ldg(p.dt_bias + d) : 0.f;
    const float Dd = p.D ? __ldg(p.D + d) : 0.f;

#pragma unroll 4
    for (int64_t t = 0; t < L; ++t) {
        const int64_t i = (b * L + t) * D + d;
        const float xv = ldg1(x + i);
        const float delta = softplus(ldg1(dt + i) + bias);
        const float4 bv = ldg4(Bm + (b * L + t) * kDState + 4 * q);
        const float4 cv = ldg4(Cm + (b * L + t) * kDState + 4 * q);
        float part = lane_update(h, a2, delta, delta * xv, bv, cv);
        part += __shfl_xor_sync(kFull, part, 1);
        part += __shfl_xor_sync(kFull, part, 2);
        if (ok) {
            __stcs(reinterpret_cast<float4 *>(p.h_out + ((b * L + t) * D + d) * kDState) + q, h);
            if (q == 0) {
                float out = part + Dd * xv;
                if (z) out *= silu(ldg1(z + i));
                y[i] = from_f32<T>(out);
            }
        }
    }
}

// ---------------------------------------------------------------------------
// mb_rollback: h_out[s] = accept[s] == 0 ? h0[s] : h_all[s, accept[s] - 1].
__global__ void __launch_bounds__(kThreads)
rollback_kernel(const float4 *__restrict__ h0, const float4 *__restrict__ h_all,
                const int32_t *__restrict__ accept, float4 *h_out, int64_t batch, int64_t k,
                int64_t per_stream /* float4s */, StatusBlock *status) {
    const int64_t total = batch * per_stream;
    for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * kThreads) {
        const int64_t s = i / per_stream;
        const int64_t j = i - s * per_stream;
        const int a = __ldg(accept + s);
        if (a < 0 || a > k) {
            if (j == 0) report(status, 1 /* MB_ERR_INVALID_ARG */, s);
            continue;
        }
        float4 v;
        if (a == 0)
            v = h0 ? __ldg(h0 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
        else
            v = __ldcs(h_all + (s * k + (a - 1)) * per_stream + j);
        h_out[i] = v;
    }
}

}  // namespace

cudaError_t launch_step(const ScanParams &p, bool bf16, cudaStream_t s) {
    constexpr int CPT = 2;
    const int64_t nchan = p.batch * p.d_inner;
    const int64_t grid = (nchan + kChanPerCta * CPT - 1) / (kChanPerCta * CPT);
    if (grid == 0) return cudaSuccess;
    if (bf16)
        step_kernel<__nv_bfloat16, CPT><<<(unsigned)grid, kThreads, 0, s>>>(p);
    else
        step_kernel<float, CPT><<<(unsigned)grid, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_verify(const ScanParams &p, bool bf16, cudaStream_t s) {
    const int64_t nchan = p.batch * p.d_inner;
    const int64_t grid = (nchan + kChanPerCta - 1) / kChanPerCta;
    if (grid == 0 || p.seqlen == 0) return cudaSuccess;
    if (bf16)
        verify_kernel<__nv_bfloat16><<<(unsigned)grid, kThreads, 0, s>>>(p);
    else
        verify_kernel<float><<<(unsigned)grid, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_rollback(const float *h0, const float *h_all, const int32_t *accept,
                            float *h_out, int64_t batch, int64_t k, int64_t d_inner,
                            StatusBlock *status, cudaStream_t s) {
    const int64_t per = d_inner * kDState / 4;
    const int64_t total = batch * per;
    if (total == 0) return cudaSuccess;
    int64_t grid = (total + kThreads - 1) / kThreads;
    if (grid > 152 * 16) grid = 152 * 16;
    rollback_kernel<<<(unsigned)grid, kThreads, 0, s>>>(
        reinterpret_cast<const float4 *>(h0), reinterpret_cast<const float4 *>(h_all), accept,
        reinterpret_cast<float4 *>(h_out), batch, k, per, status);
    return cudaGetLastError();
}

}  // namespace mbscan
