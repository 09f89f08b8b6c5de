// The element-wise steps of a MambaByte block around the selective scan, for
// recurrent decoding (Figure 6: the Mamba block; Table 6: "Pre-SSM 1D
// convolution"): the residual add with RMS normalisation that opens a block,
// and one step of the causal depthwise convolution with its SiLU. Both are
// HBM-streaming kernels over [batch, width] rows.
#include "common.cuh"

namespace mbscan {
namespace {

// Eight consecutive elements of the input dtype, widened (16 B for bf16).
__device__ __forceinline__ void load8(const __nv_bfloat16 *p, float (&v)[8]) {
    const uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
    const unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        v[2 * j] = __uint_as_float(w[j] << 16);
        v[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
}
__device__ __forceinline__ void load8(const float *p, float (&v)[8]) {
    const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
// Plain (coherent) loads for buffers the kernel also writes.
__device__ __forceinline__ void ld8(const __nv_bfloat16 *p, float (&v)[8]) {
    const uint4 u = *reinterpret_cast<const uint4 *>(p);
    const unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        v[2 * j] = __uint_as_float(w[j] << 16);
        v[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
}
__device__ __forceinline__ void ld8(const float *p, float (&v)[8]) {
    const float4 a = reinterpret_cast<const float4 *>(p)[0];
    const float4 b = reinterpret_cast<const float4 *>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void store8(__nv_bfloat16 *p, const float (&v)[8]) {
    uint4 u;
    unsigned *w = &u.x;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
        w[j] = *reinterpret_cast<const unsigned *>(&h);
    }
    *reinterpret_cast<uint4 *>(p) = u;
}
__device__ __forceinline__ void store8(float *p, const float (&v)[8]) {
    reinterpret_cast<float4 *>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4 *>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// residual[b] += add[b] (when given); out[b] = residual[b] / sqrt(mean(residual[b]^2) + eps) * w.
// One CTA per row, blockDim = 32 * ceil(groups / 32) (<= 1024) so that each
// thread usually owns one 8-element group, which it keeps in registers
// between the sum of squares and the scaling; wider rows loop and re-read.
template <typename T>
__global__ void __launch_bounds__(1024) rmsnorm_kernel(const T *__restrict__ add, float *residual,
                                                       const float *__restrict__ w, float eps,
                                                       T *__restrict__ out, int64_t width) {
    __shared__ float red[32];
    pdl_wait();
    const int64_t row = blockIdx.x;
    float *r = residual + row * width;
    const int groups = (int)(width / 8);
    float v0[8];
    float ss = 0.f;
    for (int g = threadIdx.x; g < groups; g += blockDim.x) {
        float v[8];
        ld8(r + 8 * g, v);
        if (add) {
            float a[8];
            load8(add + row * width + 8 * g, a);
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] += a[j];
            store8(r + 8 * g, v);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) ss = fmaf(v[j], v[j], ss);
        if (g == (int)threadIdx.x) {
#pragma unroll
            for (int j = 0; j < 8; ++j) v0[j] = v[j];
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(kFull, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) tot += red[i];
    const float scale = rsqrtf(tot / (float)width + eps);
    for (int g = threadIdx.x; g < groups; g += blockDim.x) {
        float v[8], wv[8], o[8];
        if (g == (int)threadIdx.x) {
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = v0[j];
        } else {
            ld8(r + 8 * g, v);
        }
        load8(w + 8 * g, wv);
#pragma unroll
        for (int j = 0; j < 8; ++j) o[j] = v[j] * scale * wv[j];
        store8(out + row * width + 8 * g, o);
    }
}

constexpr int kConvThreads = 256;
#ifndef MB_CONV_ROWS
#define MB_CONV_ROWS 2
#endif
constexpr int kConvRows = MB_CONV_ROWS;   // batch rows per thread (the weights are loaded once for them)

// One decode step of the causal depthwise convolution (kernel 4) and SiLU:
//   out[b,d] = silu(sum_{j<3} w[d,j] state[b,j,d] + w[d,3] x[b,d] + bias[d]),
// then the window moves: state[b,0] <- state[b,1], state[b,1] <- state[b,2],
// state[b,2] <- x[b]. state: [batch, 3, width] in the input dtype (the last
// three inputs, oldest first). Thread: 8 channels of kConvRows rows.
template <typename T>
__global__ void __launch_bounds__(kConvThreads) conv_step_kernel(const T *__restrict__ x, T *state,
                                                                 const float *__restrict__ w,
                                                                 const float *__restrict__ bias,
                                                                 T *__restrict__ out, int64_t batch,
                                                                 int64_t width) {
    pdl_wait();
    const int64_t groups = width / 8;
    const int64_t rowblocks = (batch + kConvRows - 1) / kConvRows;
    const int64_t i = (int64_t)blockIdx.x * kConvThreads + threadIdx.x;
    if (i >= rowblocks * groups) return;
    const int64_t rb = i / groups, d0 = (i - rb * groups) * 8;
    float4 wj[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) wj[j] = __ldg(reinterpret_cast<const float4 *>(w + (d0 + j) * 4));
    float bv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (bias) load8(bias + d0, bv);
#pragma unroll
    for (int u = 0; u < kConvRows; ++u) {
        const int64_t b = rb * kConvRows + u;
        if (b >= batch) break;
        float xv[8], s0[8], s1[8], s2[8], o[8];
        load8(x + b * width + d0, xv);
        T *st = state + b * 3 * width + d0;
        ld8(st, s0);
        ld8(st + width, s1);
        ld8(st + 2 * width, s2);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            float acc = bv[j];
            acc = fmaf(wj[j].x, s0[j], acc);
            acc = fmaf(wj[j].y, s1[j], acc);
            acc = fmaf(wj[j].z, s2[j], acc);
            acc = fmaf(wj[j].w, xv[j], acc);
            o[j] = silu(acc);
        }
        store8(out + b * width + d0, o);
        store8(st, s1);
        store8(st + width, s2);
        store8(st + 2 * width, xv);
    }
}

}  // namespace

cudaError_t launch_rmsnorm(const void *add, float *residual, const float *w, float eps, void *out,
                           int64_t batch, int64_t width, bool bf16, cudaStream_t s) {
    if (batch == 0 || width == 0) return cudaSuccess;
    const int64_t groups = width / 8;
    const unsigned threads = (unsigned)(groups >= 1024 ? 1024 : 32 * ((groups + 31) / 32));
    if (bf16)
        return launch_pdl(false, rmsnorm_kernel<__nv_bfloat16>, dim3((unsigned)batch), dim3(threads), 0, s,
                          static_cast<const __nv_bfloat16 *>(add), residual, w, eps,
                          static_cast<__nv_bfloat16 *>(out), width);
    return launch_pdl(false, rmsnorm_kernel<float>, dim3((unsigned)batch), dim3(threads), 0, s,
                      static_cast<const float *>(add), residual, w, eps, static_cast<float *>(out), width);
}

cudaError_t launch_conv_step(const void *x, void *state, const float *w, const float *bias, void *out,
                             int64_t batch, int64_t width, bool bf16, cudaStream_t s) {
    const int64_t n = ((batch + kConvRows - 1) / kConvRows) * (width / 8);
    if (n == 0) return cudaSuccess;
    const unsigned grid = (unsigned)((n + kConvThreads - 1) / kConvThreads);
    if (bf16)
        return launch_pdl(false, conv_step_kernel<__nv_bfloat16>, dim3(grid), dim3(kConvThreads), 0, s,
                          static_cast<const __nv_bfloat16 *>(x), static_cast<__nv_bfloat16 *>(state), w, bias,
                          static_cast<__nv_bfloat16 *>(out), batch, width);
    return launch_pdl(false, conv_step_kernel<float>, dim3(grid), dim3(kConvThreads), 0, s,
                      static_cast<const float *>(x), static_cast<float *>(state), w, bias,
                      static_cast<float *>(out), batch, width);
}

}  // namespace mbscan
