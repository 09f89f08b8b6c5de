// Bifurcation of speculative decoding (MambaByte Algorithm 1): for every
// stream, count how many leading drafted bytes fall in the verifier's top-beta
// candidates. The count a[s] is what the rollback (and the corrector loop)
// resumes from: the state after a[s] accepted bytes.
//
// rank_p(b) = 1 + #{v in 0..255 : logit[v] > logit[b]} (ties share the better
// rank; a NaN logit is never larger). Drafted byte i is accepted when
// rank <= beta; a[s] = the first i (0-based) that is not accepted, else k.
//
// One CTA per stream, one warp per drafted position: warp w decides
// positions w, w + kAccWarps, ... (lane l compares the 8 logits 8l .. 8l+7
// with the drafted byte's logit, the warp sums the counts); the CTA then takes
// the first rejected position. Positions are decided kAccWarps at a time, and
// later groups are skipped once a rejection is found.
#include "common.cuh"

namespace mbscan {
namespace {

constexpr int kAccWarps = 16;

__device__ __forceinline__ void load8(const float *p, float (&v)[8]) {
    const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void load8(const __nv_bfloat16 *p, float (&v)[8]) {
    const uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
    const unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        v[2 * j] = __uint_as_float(w[j] << 16);
        v[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
}

template <typename T>
__global__ void __launch_bounds__(32 * kAccWarps) accept_kernel(const T *__restrict__ logits,
                                                                const uint8_t *__restrict__ drafted,
                                                                int64_t k, int beta,
                                                                int32_t *__restrict__ accept) {
    __shared__ int first_reject;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t s = blockIdx.x;
    if (threadIdx.x == 0) first_reject = (int)k;
    __syncthreads();
    pdl_wait();
    for (int64_t base = 0; base < k; base += kAccWarps) {
        const int64_t i = base + warp;
        if (i < k) {
            const T *row = logits + (s * k + i) * 256;
            const int byte = __ldg(drafted + s * k + i);
            const float target = to_f32(row[byte]);
            float v[8];
            load8(row + 8 * lane, v);
            int greater = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) greater += v[j] > target ? 1 : 0;
            const int rank = 1 + __reduce_add_sync(kFull, greater);
            if (rank > beta && lane == 0) atomicMin(&first_reject, (int)i);
        }
        __syncthreads();
        const bool done = first_reject < (int)k;
        __syncthreads();   // every thread has read it before the next group can lower it
        if (done) break;   // uniform
    }
    if (threadIdx.x == 0) accept[s] = first_reject;
}

}  // namespace

cudaError_t launch_accept(const void *logits, bool bf16, const uint8_t *drafted, int64_t streams,
                          int64_t k, int beta, int32_t *accept, cudaStream_t s) {
    if (streams == 0) return cudaSuccess;
    const unsigned grid = (unsigned)streams;
    if (bf16)
        return launch_pdl(false, accept_kernel<__nv_bfloat16>, dim3(grid), dim3(32 * kAccWarps), 0, s,
                          static_cast<const __nv_bfloat16 *>(logits), drafted, k, beta, accept);
    return launch_pdl(false, accept_kernel<float>, dim3(grid), dim3(32 * kAccWarps), 0, s,
                      static_cast<const float *>(logits), drafted, k, beta, accept);
}

}  // namespace mbscan
