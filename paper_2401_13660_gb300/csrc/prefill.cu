// Prefill scan of the selective-scan layer core (MambaByte Section 2,
// "Implementation: parallel scans"; Eq. 2-3; Table 6 output and gating).
//
// Work decomposition. Every (batch row, channel) pair is an independent
// linear recurrence over L steps with a 16-float state, so the kernel is
// channel-parallel and runs each channel's recurrence sequentially in time
// (the cheapest evaluation order in operations: one FMA per state per step;
// a time-parallel scan with the associative operator of Section 2 would add
// work per element). A CTA owns kCh channels of one batch row; four lanes per
// channel each hold 4 of the 16 states in registers (fp32) for the whole
// sequence.
//
// Per chunk of kT time steps the CTA
//   1. loads the raw dt, x, z [kT, kCh] and B, C [kT, 16] tiles (coalesced,
//      issued one chunk ahead into registers so the loads overlap the scan),
//   2. converts them once per (t, channel) into shared memory:
//      (Delta, Delta*x) with Delta = softplus(dt + bias), D*x, z, and B, C as
//      fp32 (so the softplus is paid once per channel-byte, not per lane),
//   3. scans: per step and state, Abar = 2^(Delta * A*log2 e) on the SFU and
//      h = Abar*h + B*(Delta*x); each lane writes its share of C.h,
//   4. reduces the four shares per (t, channel), adds D*x, applies silu(z)
//      and stores y (32 consecutive channels per warp store).
// Steps past L are padded with Delta = 0, which leaves the state unchanged.
#include "common.cuh"

namespace mbscan {
namespace {

constexpr int kCh = 32;              // channels per CTA
constexpr int kT = 16;               // time steps per chunk
constexpr int kThreads = kCh * 4;    // four lanes per channel

struct Smem {
    float2 dd[2][kT][kCh];   // (Delta, Delta*x)
    float bm[2][kT][kDState];
    float cm[2][kT][kDState];
    float zg[2][kT][kCh];    // gate input z
    float xd[2][kT][kCh];    // D*x
    float part[kT][kCh * 4]; // per-lane shares of C.h
};

// Raw chunk held in registers between the global load and the conversion.
struct Raw {
    float4 dt, x, z;   // 4 consecutive channels at one time step
    float2 b, c;       // 2 consecutive states at one time step
};

template <typename T>
__device__ __forceinline__ Raw load_chunk(const ScanParams &p, int64_t b, int64_t d0, int64_t t0) {
    const int tid = threadIdx.x;
    const int t = tid >> 3;               // 0..15
    const int c4 = (tid & 7) * 4;         // 0..28
    const int64_t tt = t0 + t;
    Raw r;
    const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
    if (tt < p.seqlen && d0 + c4 < p.d_inner) {
        const int64_t i = (b * p.seqlen + tt) * p.d_inner + d0 + c4;
        r.dt = ldg4(static_cast<const T *>(p.dt) + i);
        r.x = ldg4(static_cast<const T *>(p.x) + i);
        r.z = p.z ? ldg4(static_cast<const T *>(p.z) + i) : zero4;
    } else {
        r.dt = zero4; r.x = zero4; r.z = zero4;
    }
    const int n2 = (tid & 7) * 2;
    if (tt < p.seqlen) {
        const int64_t j = (b * p.seqlen + tt) * kDState + n2;
        r.b = ldg2(static_cast<const T *>(p.B) + j);
        r.c = ldg2(static_cast<const T *>(p.C) + j);
    } else {
        r.b = make_float2(0.f, 0.f); r.c = make_float2(0.f, 0.f);
    }
    return r;
}

__device__ __forceinline__ void convert_store(Smem &s, int buf, const Raw &r, int64_t b,
                                              int64_t d0, int64_t t0, const ScanParams &p) {
    const int tid = threadIdx.x;
    const int t = tid >> 3;
    const int c4 = (tid & 7) * 4;
    const bool valid = (t0 + t < p.seqlen) && (d0 + c4 < p.d_inner);
    const float dtv[4] = {r.dt.x, r.dt.y, r.dt.z, r.dt.w};
    const float xv[4] = {r.x.x, r.x.y, r.x.z, r.x.w};
    const float zv[4] = {r.z.x, r.z.y, r.z.z, r.z.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        float delta = 0.f, dx = 0.f, xdv = 0.f;
        if (valid) {
            const int64_t d = d0 + c4 + j;
            delta = softplus(dtv[j] + (p.dt_bias ? __ldg(p.dt_bias + d) : 0.f));
            dx = delta * xv[j];
            xdv = (p.D ? __ldg(p.D + d) : 0.f) * xv[j];
        }
        s.dd[buf][t][c4 + j] = make_float2(delta, dx);
        s.xd[buf][t][c4 + j] = xdv;
        s.zg[buf][t][c4 + j] = zv[j];
    }
    const int n2 = (tid & 7) * 2;
    s.bm[buf][t][n2] = r.b.x;
    s.bm[buf][t][n2 + 1] = r.b.y;
    s.cm[buf][t][n2] = r.c.x;
    s.cm[buf][t][n2 + 1] = r.c.y;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) prefill_kernel(ScanParams p) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    Smem &s = *reinterpret_cast<Smem *>(smem_raw);
    const int tid = threadIdx.x;
    const int64_t b = blockIdx.y;
    const int64_t d0 = (int64_t)blockIdx.x * kCh;
    const int c = tid >> 2;   // channel within the CTA (scan role)
    const int q = tid & 3;    // state quarter
    const int64_t d = d0 + c;
    const bool chan_ok = d < p.d_inner;

    float4 h = make_float4(0.f, 0.f, 0.f, 0.f);
    float4 a2 = h;
    if (chan_ok) {
        if (p.h0) h = __ldg(reinterpret_cast<const float4 *>(p.h0 + (b * p.d_inner + d) * kDState) + q);
        a2 = ldg4(p.A + d * kDState + 4 * q);
        a2.x *= kLog2e; a2.y *= kLog2e; a2.z *= kLog2e; a2.w *= kLog2e;
    }

    const int64_t nchunks = (p.seqlen + kT - 1) / kT;
    Raw r = load_chunk<T>(p, b, d0, 0);
    convert_store(s, 0, r, b, d0, 0, p);
    __syncthreads();

    T *y = static_cast<T *>(p.y);
    const bool gate = p.z != nullptr;
    for (int64_t ci = 0; ci < nchunks; ++ci) {
        const int buf = (int)(ci & 1);
        const int64_t t0 = ci * kT;
        if (ci + 1 < nchunks) r = load_chunk<T>(p, b, d0, t0 + kT);

#pragma unroll 4
        for (int t = 0; t < kT; ++t) {
            const float2 dd = s.dd[buf][t][c];
            const float4 bv = *reinterpret_cast<const float4 *>(&s.bm[buf][t][4 * q]);
            const float4 cv = *reinterpret_cast<const float4 *>(&s.cm[buf][t][4 * q]);
            h.x = fmaf(ex2(dd.x * a2.x), h.x, bv.x * dd.y);
            h.y = fmaf(ex2(dd.x * a2.y), h.y, bv.y * dd.y);
            h.z = fmaf(ex2(dd.x * a2.z), h.z, bv.z * dd.y);
            h.w = fmaf(ex2(dd.x * a2.w), h.w, bv.w * dd.y);
            s.part[t][tid] = fmaf(cv.x, h.x, fmaf(cv.y, h.y, fmaf(cv.z, h.z, cv.w * h.w)));
        }
        __syncthreads();

        // Epilogue: warp w handles time steps w, w+4, ...; lane = channel.
        {
            const int ec = tid & 31;
            const int64_t ed = d0 + ec;
#pragma unroll
            for (int t = tid >> 5; t < kT; t += 4) {
                if (t0 + t < p.seqlen && ed < p.d_inner) {
                    const float4 pp = *reinterpret_cast<const float4 *>(&s.part[t][ec * 4]);
                    float out = (pp.x + pp.y) + (pp.z + pp.w) + s.xd[buf][t][ec];
                    if (gate) out *= silu(s.zg[buf][t][ec]);
                    y[(b * p.seqlen + t0 + t) * p.d_inner + ed] = from_f32<T>(out);
                }
            }
        }
        if (ci + 1 < nchunks) convert_store(s, buf ^ 1, r, b, d0, t0 + kT, p);
        __syncthreads();
    }

    if (p.h_out && chan_ok)
        reinterpret_cast<float4 *>(p.h_out + (b * p.d_inner + d) * kDState)[q] = h;
}

}  // namespace

cudaError_t launch_prefill(const ScanParams &p, bool bf16, cudaStream_t s) {
    if (p.batch == 0) return cudaSuccess;
    const dim3 grid((unsigned)((p.d_inner + kCh - 1) / kCh), (unsigned)p.batch);
    const size_t smem = sizeof(Smem);
    if (bf16) {
        auto k = prefill_kernel<__nv_bfloat16>;
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k<<<grid, kThreads, smem, s>>>(p);
    } else {
        auto k = prefill_kernel<float>;
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k<<<grid, kThreads, smem, s>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace mbscan
