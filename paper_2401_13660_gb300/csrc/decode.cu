// Decode-side kernels of the selective-scan layer core: the batched
// single-byte recurrent step and the rollback gather of speculative decoding
// (MambaByte Section 6.3 and Algorithm 1). The verify scan shares the prefill
// kernel (prefill.cu).
//
// Both are HBM-streaming kernels. A (batch row, channel) pair owns 16 fp32
// states (64 contiguous bytes). In the step kernel four lanes share a channel,
// each holding 4 states in one float4, so a warp moves 512 contiguous bytes
// of state per instruction.
#include <string.h>

#include <atomic>
#include <mutex>

#include "common.cuh"
#include "tma.cuh"

namespace mbscan {
namespace {

constexpr int kStepConsumers = 8;                          // consumer warps
constexpr int kStepThreads = 32 * (kStepConsumers + 1);    // + one producer warp
constexpr int kStepCh = 8 * kStepConsumers;                // 64 channels per tile
constexpr int kStepRows = 4;                               // batch rows per tile
#ifndef MB_STEP_STAGES
#define MB_STEP_STAGES 4
#endif
constexpr int kStepStages = MB_STEP_STAGES;
// Tiles per CTA whose state is prefetched into L2 before the dependency wait
// (measured at batch 256 x 4608: 1 / 2 / 4 tiles took the back-to-back step
// from 27.6 to 26.4 / 25.8 / 25.8 us and the whole-model decode, where a GEMM
// precedes each step, from 2.885 to 2.849 / 2.834 / 2.926 ms).
constexpr int kStepPrefetch = 2;

// One tile of the decode step in shared memory (TMA destinations; every member
// offset is a multiple of 128 bytes for both dtypes).
template <typename T>
struct StepStage {
    float state[kStepRows][kStepCh][kDState];   // 16 KB
    T x[kStepRows][kStepCh];
    T dt[kStepRows][kStepCh];
    T z[kStepRows][kStepCh];
    T B[kStepRows][kDState];
    T C[kStepRows][kDState];
};

template <typename T>
struct StepSmem {
    StepStage<T> st[kStepStages];
    uint64_t full[kStepStages];
    uint64_t empty[kStepStages];
};

struct StepArgs {
    CUtensorMap tm_state, tm_x, tm_dt, tm_z, tm_B, tm_C;
    // resume: initial state of row s from h0 (tm_state over p.h0, box of one
    // row) or from h_all[s, accept[s]-1] (tm_hall)
    CUtensorMap tm_hall;
    const int32_t *accept;
    int64_t k;
    ScanParams p;
    int ntiles, ntiles_d, has_gate, has_h0;
};

// Resume: the drafted-byte index whose state row s starts from (0 .. k-1),
// -1 for the cached state h0, or -2 when accept[s] is outside [0, k].
__device__ __forceinline__ int resume_index(const StepArgs &a, int64_t s) {
    const int acc = __ldg(a.accept + s);
    return (acc < 0 || acc > a.k) ? -2 : acc - 1;
}

// Lane q of a 4-lane group holds the group's shares part[0..3] (one per row of
// the tile); return the full 4-lane sum of row q (two shuffle rounds, the
// lanes of a group are adjacent).
__device__ __forceinline__ float reduce_rows(const float (&part)[kStepRows], int q) {
    const bool hi = (q & 2) != 0;
    float k0 = hi ? part[2] : part[0], k1 = hi ? part[3] : part[1];
    const float s0 = hi ? part[0] : part[2], s1 = hi ? part[1] : part[3];
    k0 += __shfl_xor_sync(kFull, s0, 2);
    k1 += __shfl_xor_sync(kFull, s1, 2);
    const bool odd = (q & 1) != 0;
    const float keep = odd ? k1 : k0, send = odd ? k0 : k1;
    return keep + __shfl_xor_sync(kFull, send, 1);
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Four consecutive shared-memory elements of the input dtype, widened.
__device__ __forceinline__ float4 lds4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 lds4(const __nv_bfloat16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

// ---------------------------------------------------------------------------
// mb_step: state[b, d, :] <- one recurrence step (Eq. 2 with L = 1), y[b, 0, d].
// Persistent, warp-specialised streaming kernel. The work is cut into tiles
// of 64 channels x 4 batch rows (16 KB of state); CTA i takes tiles i, i + grid,
// ... A producer warp streams each tile's state, x, dt, z, B and C into a
// kStepStages-deep shared-memory ring with TMA; 8 consumer warps compute it.
// Consumer lane (g, q) of warp w serves channel d0 + 8 w + g, states 4q..4q+3,
// for the tile's 4 rows; lane q evaluates the channel scalars (Delta, Delta*x,
// D*x, silu z) of row q only and shares Delta, Delta*x by shuffle, and after
// the 4-lane reduction owns row q's output. New states go straight from
// registers to global memory (512 contiguous bytes per warp and row). The
// round-robin order changes the channel block from tile to tile, so each
// lane loads its channel's A row, dt_bias and D one tile ahead. Launched with
// programmatic dependent launch, the producer prefetches its first tiles'
// state into L2 while the previous kernel drains.
// kResume (speculative decoding, after the bifurcation of Algorithm 1): row s
// starts from h0[s] or h_all[s, accept[s]-1] instead of the state itself, so
// the rollback needs no copy of its own; rows with an accept count outside
// [0, k] are reported and left untouched.
// Minimum CTAs per SM: those its shared memory allows (3 for bf16, 2 for fp32).
template <typename T, bool kResume>
__global__ void __launch_bounds__(kStepThreads, sizeof(T) == 2 ? 3 : 2) step_kernel(const __grid_constant__ StepArgs a) {
    extern __shared__ unsigned char smem_dyn[];
    StepSmem<T> &s = smem_aligned<StepSmem<T>>(smem_dyn);
    const ScanParams &p = a.p;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t D = p.d_inner;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStepStages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kStepConsumers);
        }
        fence_mbar_init();
    }
    __syncthreads();
    pdl_trigger();   // persistent grid: the next kernel's CTAs take the SMs as this one drains
    // The state of this CTA's first kStepPrefetch tiles is prefetched into L2
    // before the wait for the previous kernel: the first loads after the wait
    // then come from L2 instead of paying the DRAM latency while the previous
    // kernel drains. A prefetch returns nothing, so whatever that kernel still
    // writes is seen by the loads after the wait.
    if (!kResume && warp == kStepConsumers && lane == 0) {
        for (int j = 0; j < kStepPrefetch; ++j) {
            const int k = blockIdx.x + j * gridDim.x;
            if (k >= a.ntiles) break;
            tma_prefetch_3d(&a.tm_state, 0, (k % a.ntiles_d) * kStepCh, (k / a.ntiles_d) * kStepRows);
        }
    }
    pdl_wait();      // everything below reads or writes global memory

    if (warp == kStepConsumers) {
        // ---- producer
        if (lane == 0) {
            constexpr uint32_t st_bytes = kStepRows * kStepCh * kDState * 4;
            constexpr uint32_t tok = kStepRows * kStepCh * sizeof(T), bc = kStepRows * kDState * sizeof(T);
            const uint32_t bytes = st_bytes + (a.has_gate ? 3 : 2) * tok + 2 * bc;
            for (int j = 0;; ++j) {
                const int k = blockIdx.x + j * gridDim.x;
                if (k >= a.ntiles) break;
                const int si = j % kStepStages;
                if (j >= kStepStages &&
                    !mbar_wait(&s.empty[si], (uint32_t)((j / kStepStages - 1) & 1))) {
                    report(p.status, 4 /* MB_ERR_TIMEOUT */, k);
                    break;
                }
                const int d0 = (k % a.ntiles_d) * kStepCh, b0 = (k / a.ntiles_d) * kStepRows;
                StepStage<T> &t = s.st[si];
                mbar_arrive_expect_tx(&s.full[si], bytes);
                if constexpr (kResume) {
                    for (int u = 0; u < kStepRows; ++u) {
                        const int64_t bs = b0 + u;
                        int r = bs < p.batch ? resume_index(a, bs) : -2;
                        if (r == -2 && bs < p.batch && d0 == 0) report(p.status, 1 /* MB_ERR_INVALID_ARG */, bs);
                        if (r == -1 && a.has_h0)
                            tma_load_3d(&t.state[u][0][0], &a.tm_state, &s.full[si], 0, d0, (int)bs);
                        else   // h_all row r; r < 0 (no h0, or a row left untouched) reads zeros
                            tma_load_4d(&t.state[u][0][0], &a.tm_hall, &s.full[si], 0, d0, r < 0 ? -1 : r,
                                        (int)bs);
                    }
                } else {
                    tma_load_3d(&t.state[0][0][0], &a.tm_state, &s.full[si], 0, d0, b0);
                }
                tma_load_2d(&t.x[0][0], &a.tm_x, &s.full[si], d0, b0);
                tma_load_2d(&t.dt[0][0], &a.tm_dt, &s.full[si], d0, b0);
                if (a.has_gate) tma_load_2d(&t.z[0][0], &a.tm_z, &s.full[si], d0, b0);
                tma_load_2d(&t.B[0][0], &a.tm_B, &s.full[si], 0, b0);
                tma_load_2d(&t.C[0][0], &a.tm_C, &s.full[si], 0, b0);
            }
        }
        return;
    }

    // ---- consumers
    const int g = lane >> 2, q = lane & 3;
    const int c = warp * 8 + g;
    float4 *state = reinterpret_cast<float4 *>(p.h_out);
    T *y = static_cast<T *>(p.y);
    // Channel constants (A row, dt_bias, D) of the next tile, loaded one tile
    // ahead so that their latency overlaps the current tile.
    float4 nav = make_float4(0.f, 0.f, 0.f, 0.f);
    float nbias = 0.f, ndsk = 0.f;
    auto load_const = [&](int k) {
        nav = make_float4(0.f, 0.f, 0.f, 0.f);
        nbias = ndsk = 0.f;
        if (k < a.ntiles) {
            const int64_t dn = (int64_t)(k % a.ntiles_d) * kStepCh + c;
            if (dn < D) {
                nav = ldg4(p.A + dn * kDState + 4 * q);
                nbias = p.dt_bias ? __ldg(p.dt_bias + dn) : 0.f;
                ndsk = p.D ? __ldg(p.D + dn) : 0.f;
            }
        }
    };
    load_const(blockIdx.x);
    for (int j = 0;; ++j) {
        const int k = blockIdx.x + j * gridDim.x;
        if (k >= a.ntiles) break;
        const int si = j % kStepStages;
        const float2 a01 = make_float2(nav.x * kLog2e, nav.y * kLog2e);
        const float2 a23 = make_float2(nav.z * kLog2e, nav.w * kLog2e);
        const float bias = nbias, dsk = ndsk;
        load_const(k + gridDim.x);
        if (!mbar_wait(&s.full[si], (uint32_t)((j / kStepStages) & 1))) {
            if (lane == 0) report(p.status, 4 /* MB_ERR_TIMEOUT */, k);
            break;
        }
        const int64_t d0 = (int64_t)(k % a.ntiles_d) * kStepCh, b0 = (int64_t)(k / a.ntiles_d) * kStepRows;
        const int64_t d = d0 + c;
        const bool dok = d < D;
        const StepStage<T> &t = s.st[si];
        float4 h[kStepRows];
#pragma unroll
        for (int u = 0; u < kStepRows; ++u) h[u] = lds4(&t.state[u][c][4 * q]);
        // channel scalars of row q
        const float xv = to_f32(t.x[q][c]);
        const float delta = softplus(to_f32(t.dt[q][c]) + bias);
        const float gx = delta * xv, xd = dsk * xv;
        const float sz = a.has_gate ? silu(to_f32(t.z[q][c])) : 1.f;
        float part[kStepRows];
#pragma unroll
        for (int u = 0; u < kStepRows; ++u) {
            const int src = (lane & ~3) | u;
            const float du = __shfl_sync(kFull, delta, src);
            const float gu = __shfl_sync(kFull, gx, src);
            const float4 bv = lds4(&t.B[u][4 * q]);
            const float4 cv = lds4(&t.C[u][4 * q]);
            const float2 dd2 = make_float2(du, du), gg = make_float2(gu, gu);
            const float2 e01 = mul2(dd2, a01), e23 = mul2(dd2, a23);
            float2 h01 = make_float2(h[u].x, h[u].y), h23 = make_float2(h[u].z, h[u].w);
            h01 = fma2(make_float2(ex2(e01.x), ex2(e01.y)), h01, mul2(make_float2(bv.x, bv.y), gg));
            h23 = fma2(make_float2(ex2(e23.x), ex2(e23.y)), h23, mul2(make_float2(bv.z, bv.w), gg));
            h[u] = make_float4(h01.x, h01.y, h23.x, h23.y);
            const float2 acc = fma2(make_float2(cv.z, cv.w), h23, mul2(make_float2(cv.x, cv.y), h01));
            part[u] = acc.x + acc.y;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.empty[si]);   // this warp is done with the stage
#pragma unroll
        for (int u = 0; u < kStepRows; ++u) {
            const int64_t b = b0 + u;
            bool ok = dok && b < p.batch;
            if constexpr (kResume) ok = ok && resume_index(a, b) != -2;
            if (ok) __stcs(state + (b * D + d) * (kDState / 4) + q, h[u]);
        }
        const float ysum = reduce_rows(part, q);
        const int64_t b = b0 + q;
        bool yok = dok && b < p.batch;
        if constexpr (kResume) yok = yok && resume_index(a, b) != -2;
        if (yok) y[b * D + d] = from_f32<T>((ysum + xd) * sz);
    }
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
    pdl_wait();
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

template <typename T, bool kResume>
cudaError_t launch_step_typed(const ScanParams &p, const float *h_all, const int32_t *accept, int64_t k,
                              cudaStream_t s) {
    const int es = sizeof(T);
    StepArgs a;
    memset(&a, 0, sizeof(a));
    a.p = p;
    a.accept = accept;
    a.k = k;
    a.has_h0 = p.h0 != nullptr;
    a.has_gate = p.z != nullptr;
    a.ntiles_d = (int)((p.d_inner + kStepCh - 1) / kStepCh);
    a.ntiles = a.ntiles_d * (int)((p.batch + kStepRows - 1) / kStepRows);
    const uint64_t sdims[3] = {kDState, (uint64_t)p.d_inner, (uint64_t)p.batch};
    const uint64_t sstr[2] = {kDState * 4, (uint64_t)p.d_inner * kDState * 4};
    const uint32_t sbox[3] = {kDState, kStepCh, kStepRows};
    const uint64_t tdims[2] = {(uint64_t)p.d_inner, (uint64_t)p.batch};
    const uint64_t tstr[1] = {(uint64_t)p.d_inner * es};
    const uint32_t tbox[2] = {kStepCh, kStepRows};
    const uint64_t bdims[2] = {kDState, (uint64_t)p.batch};
    const uint64_t bstr[1] = {(uint64_t)p.bc_stride * es};
    const uint32_t bbox[2] = {kDState, kStepRows};
    bool ok_maps = true;
    if constexpr (kResume) {
        // one row per load: h0 [batch, D, 16] and h_all [batch, k, D, 16]
        const uint32_t rbox[3] = {kDState, kStepCh, 1};
        const uint64_t hdims[4] = {kDState, (uint64_t)p.d_inner, (uint64_t)k, (uint64_t)p.batch};
        const uint64_t hstr[3] = {kDState * 4, (uint64_t)p.d_inner * kDState * 4,
                                  (uint64_t)k * p.d_inner * kDState * 4};
        const uint32_t hbox[4] = {kDState, kStepCh, 1, 1};
        ok_maps = (!p.h0 || encode_tmap(&a.tm_state, p.h0, 4, 3, sdims, sstr, rbox)) &&
                  encode_tmap(&a.tm_hall, h_all, 4, 4, hdims, hstr, hbox);
    } else {
        ok_maps = encode_tmap(&a.tm_state, p.h_out, 4, 3, sdims, sstr, sbox);
    }
    if (!ok_maps ||
        !encode_tmap(&a.tm_x, p.x, es, 2, tdims, tstr, tbox) ||
        !encode_tmap(&a.tm_dt, p.dt, es, 2, tdims, tstr, tbox) ||
        (p.z && !encode_tmap(&a.tm_z, p.z, es, 2, tdims, tstr, tbox)) ||
        !encode_tmap(&a.tm_B, p.B, es, 2, bdims, bstr, bbox) ||
        !encode_tmap(&a.tm_C, p.C, es, 2, bdims, bstr, bbox))
        return cudaErrorInvalidValue;
    const size_t smem = sizeof(StepSmem<T>) + 128;
    auto kern = step_kernel<T, kResume>;
    // Device limits, computed once per device (per instantiation) and published
    // through `ready`: SMs, resident CTAs per SM, shared memory per SM and
    // reserved per CTA.
    struct Limits {
        std::atomic<int> ready;
        int sms, per;
        size_t smem_sm, smem_reserved, smem_optin;
    };
    constexpr int kMaxDevices = 64;
    static Limits lim[kMaxDevices];
    static std::mutex init_mu;
    int dev = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    Limits &l = lim[dev];
    if (!l.ready.load(std::memory_order_acquire)) {
        std::lock_guard<std::mutex> guard(init_mu);
        if (!l.ready.load(std::memory_order_relaxed)) {
            int n = 0, r = 0, sm_bytes = 0, rsv = 0, optin = 0;
            if ((e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess ||
                (e = cudaDeviceGetAttribute(&sm_bytes, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev)) !=
                    cudaSuccess ||
                (e = cudaDeviceGetAttribute(&rsv, cudaDevAttrReservedSharedMemoryPerBlock, dev)) != cudaSuccess ||
                (e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess)
                return e;
            // the padded requests below stay within the opt-in maximum
            if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, optin)) != cudaSuccess)
                return e;
            if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, kern, kStepThreads, smem)) != cudaSuccess)
                return e;
            l.sms = n > 0 ? n : 1;
            l.per = r > 0 ? r : 1;
            l.smem_sm = (size_t)sm_bytes;
            l.smem_reserved = (size_t)rsv;
            l.smem_optin = (size_t)optin;
            l.ready.store(1, std::memory_order_release);
        }
    }
    const int sms = l.sms, per = l.per;
    const size_t smem_sm = l.smem_sm, smem_reserved = l.smem_reserved, smem_optin = l.smem_optin;
    const int ctas = sms * per;
    const int grid = a.ntiles < ctas ? a.ntiles : ctas;
    // A grid of at most one wave needs only m = ceil(tiles / SMs) CTAs per SM.
    // Left to the resident limit, the block scheduler stacks up to `per` of
    // them on some SMs while others stay idle; asking for more than
    // 1 / (m + 1) of an SM's shared memory per CTA spreads them instead.
    size_t smem_launch = smem;
    const int m = (grid + sms - 1) / sms;
    if (m < per) {
        const size_t spread = smem_sm / (size_t)(m + 1) - smem_reserved + 128;
        if (spread > smem_launch && spread <= smem_optin) smem_launch = spread;
    }
    return launch_pdl(true, kern, dim3(grid), dim3(kStepThreads), smem_launch, s, a);
}

}  // namespace

cudaError_t launch_step(const ScanParams &p, bool bf16, cudaStream_t s) {
    if (p.batch == 0 || p.d_inner == 0) return cudaSuccess;
    return bf16 ? launch_step_typed<__nv_bfloat16, false>(p, nullptr, nullptr, 0, s)
                : launch_step_typed<float, false>(p, nullptr, nullptr, 0, s);
}

cudaError_t launch_step_resume(const ScanParams &p, bool bf16, const float *h_all,
                               const int32_t *accept, int64_t k, cudaStream_t s) {
    if (p.batch == 0 || p.d_inner == 0) return cudaSuccess;
    return bf16 ? launch_step_typed<__nv_bfloat16, true>(p, h_all, accept, k, s)
                : launch_step_typed<float, true>(p, h_all, accept, k, s);
}

cudaError_t launch_rollback(const float *h0, const float *h_all, const int32_t *accept,
                            float *h_out, int64_t batch, int64_t k, int64_t d_inner,
                            StatusBlock *status, cudaStream_t s) {
    const int64_t per = d_inner * kDState / 4;
    const int64_t threads = batch * per / kRbVec;
    if (threads == 0) return cudaSuccess;
    const int64_t grid = (threads + kRbThreads - 1) / kRbThreads;
    return launch_pdl(false, rollback_kernel, dim3((unsigned)grid), dim3(kRbThreads), 0, s,
                      reinterpret_cast<const float4 *>(h0), reinterpret_cast<const float4 *>(h_all), accept,
                      reinterpret_cast<float4 *>(h_out), batch, k, per, status);
}

}  // namespace mbscan
