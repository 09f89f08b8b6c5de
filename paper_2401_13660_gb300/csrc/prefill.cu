// Prefill scan of the selective-scan layer core (MambaByte Section 2,
// "Implementation: parallel scans"; Eq. 2-3; Table 6 output and gating), and
// the speculative-decoding verify scan (Algorithm 1), which is the same scan
// that also streams every per-position state to h_all.
//
// Work decomposition. Every (batch row, channel) pair is an independent
// linear recurrence over L steps with a 16-float state (A is diagonal, so the
// scan of Section 2 is element-wise). The kernel is channel-parallel and runs
// each channel's recurrence sequentially in time, the evaluation order with
// the fewest operations (one Abar, one FMA for h and one FMA for C.h per state
// and step); the associative operator of Section 2 is only needed to split a
// span, which the h0 / h_last interface does across calls.
//
// A CTA of kWarps warps owns CH = 32 kWarps / LPC channels of one batch row
// for the whole span (small CTAs spread the channels evenly over the SMs). LPC lanes share a channel, each keeping 16 / LPC of its fp32 states in
// registers. The state index varies slowest across a warp, so the 8 lanes of
// each quarter-warp read the same B, C values (a shared-memory broadcast).
//
// Pipeline, per chunk of kT = 16 time steps:
//  * one thread keeps a STAGES-deep ring of 3-D TMA tile loads in flight:
//    dt, x, z [kT x CH] and B, C [kT x 16], one mbarrier per stage (bounded
//    waits, tma.cuh);
//  * the CTA converts a chunk once per (t, channel) into fp32 in shared
//    memory: (Delta, Delta*x) with Delta = softplus(dt + bias), (D*x, silu z);
//  * each lane scans the chunk: Abar = 2^(Delta * A*log2 e) on the SFU for all
//    kT steps, then h = Abar*h + B*(Delta*x) and its share of C.h in packed
//    f32x2 arithmetic, reading B and C straight from the TMA tile in the input
//    dtype (for bf16 this halves the shared-memory bytes of the scan, whose
//    bandwidth is its limit); groups of LPC steps are reduced across the LPC
//    lanes of a channel with log2(LPC) shuffle rounds, each lane finishing one
//    output y = (C.h + D*x) * silu(z), which goes to a shared-memory tile that
//    one thread writes out with a TMA store.
//  Loop iteration i converts chunk i+1 and scans chunk i in one basic block,
//  so every warp has two independent instruction streams to interleave; one
//  CTA barrier per chunk orders them, after which the stage of chunk i is
//  refilled with chunk i + STAGES.
// Steps at or beyond L are converted with Delta = 0, which leaves h unchanged.
#include <string.h>

#include "common.cuh"
#include "tma.cuh"

namespace mbscan {
namespace {

constexpr int kT = 16;            // time steps per chunk
#ifndef MB_PREFILL_WARPS
#define MB_PREFILL_WARPS 4
#endif
constexpr int kWarps = MB_PREFILL_WARPS;   // warps per CTA
constexpr int kThreads = 32 * kWarps;
#ifndef MB_PREFILL_LPC
#define MB_PREFILL_LPC 4
#endif
constexpr int kPrefillLanesPerChannel = MB_PREFILL_LPC;
constexpr int kPrefillStages = 4;  // TMA ring depth for long spans
constexpr int kVerifyStages = 2;   // verify spans are short
#ifndef MB_VERIFY_MINB
#define MB_VERIFY_MINB 8   // verify CTAs per SM the register budget must allow (64 registers)
#endif

// Lane geometry: LPC lanes share one channel, each holding kSPL states.
template <int LPC>
struct Geom {
    static constexpr int kSPL = kDState / LPC;     // states per lane
    static constexpr int kPairs = kSPL / 2;        // float2 state pairs per lane
    static constexpr int kChPerWarp = 32 / LPC;
    static constexpr int kCh = kWarps * kChPerWarp;  // channels per CTA
};

template <typename T, int CH>
struct Raw {  // TMA destinations; every member offset is a multiple of 128 B
    T dt[kT][CH];
    T x[kT][CH];
    T z[kT][CH];
    T B[kT][kDState];
    T C[kT][kDState];
};

template <int CH>
struct Conv {
    float2 dg[kT][CH];          // (Delta, Delta*x)
    float2 xs[kT][CH];          // (D*x, silu(z)); silu(z) = 1 without a gate
};

template <typename T, int CH, int STAGES>
struct Smem {
    Raw<T, CH> raw[STAGES];
    Conv<CH> cv[2];
    T ys[2][kT][CH];            // output tiles, written out by TMA stores
    uint64_t full[STAGES];
};

struct PrefillArgs {
    CUtensorMap tm_dt, tm_x, tm_z, tm_B, tm_C, tm_y;
    ScanParams p;
    int has_gate;
};

template <typename T, int CH, int STAGES>
__device__ __forceinline__ void issue_chunk(Smem<T, CH, STAGES> &s, const PrefillArgs &a, int stage,
                                            int64_t chunk, int d0, int b) {
    constexpr uint32_t tok = kT * CH * sizeof(T), bc = kT * kDState * sizeof(T);
    const uint32_t bytes = (a.has_gate ? 3 : 2) * tok + 2 * bc;
    uint64_t *bar = &s.full[stage];
    mbar_arrive_expect_tx(bar, bytes);
    const int t = (int)(chunk * kT);
    Raw<T, CH> &r = s.raw[stage];
    tma_load_3d(&r.dt[0][0], &a.tm_dt, bar, d0, t, b);
    tma_load_3d(&r.x[0][0], &a.tm_x, bar, d0, t, b);
    if (a.has_gate) tma_load_3d(&r.z[0][0], &a.tm_z, bar, d0, t, b);
    tma_load_3d(&r.B[0][0], &a.tm_B, bar, 0, t, b);
    tma_load_3d(&r.C[0][0], &a.tm_C, bar, 0, t, b);
}

// Two adjacent channels of the input dtype, widened to fp32.
__device__ __forceinline__ float2 ld_pair(const float *p) { return *reinterpret_cast<const float2 *>(p); }
__device__ __forceinline__ float2 ld_pair(const __nv_bfloat16 *p) {
    const unsigned u = *reinterpret_cast<const unsigned *>(p);
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}

// Four adjacent elements of the input dtype from shared memory, widened.
__device__ __forceinline__ float4 ld_quad(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 ld_quad(const __nv_bfloat16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

// Per-thread constants of the conversion role: thread converts the adjacent
// channel pair (2 cp, 2 cp + 1) at steps th, th + kRows, ...
template <int CH>
struct ConvRole {
    static constexpr int kPairsPerRow = CH / 2;
    static constexpr int kRows = kThreads / kPairsPerRow;   // step rows per pass
    static constexpr int kPasses = kT / kRows;
    int cp, th;
    float2 bias, dsk;
    bool ok;
};

// Convert one chunk: raw TMA tiles -> fp32 (Delta, Delta*x), (D*x, silu z).
template <typename T, int CH>
__device__ __forceinline__ void convert(Conv<CH> &cv, const Raw<T, CH> &r, const ConvRole<CH> &cr,
                                        int64_t t0, int64_t L, bool gate) {
#pragma unroll
    for (int k = 0; k < ConvRole<CH>::kPasses; ++k) {
        const int t = cr.th + ConvRole<CH>::kRows * k;
        const int c = 2 * cr.cp;
        float4 dg = make_float4(0.f, 0.f, 0.f, 0.f), xs = make_float4(0.f, 1.f, 0.f, 1.f);
        if (cr.ok && t0 + t < L) {
            const float2 xv = ld_pair(&r.x[t][c]);
            const float2 dv = ld_pair(&r.dt[t][c]);
            const float d0 = softplus(dv.x + cr.bias.x), d1 = softplus(dv.y + cr.bias.y);
            dg = make_float4(d0, d0 * xv.x, d1, d1 * xv.y);
            xs.x = cr.dsk.x * xv.x;
            xs.z = cr.dsk.y * xv.y;
            if (gate) {
                const float2 zv = ld_pair(&r.z[t][c]);
                xs.y = silu(zv.x);
                xs.w = silu(zv.y);
            }
        }
        *reinterpret_cast<float4 *>(&cv.dg[t][c]) = dg;
        *reinterpret_cast<float4 *>(&cv.xs[t][c]) = xs;
    }
}

// Sum the LPC per-lane shares of C.h for LPC consecutive steps so that lane q
// ends with the full sum of step q of the group (a transposed reduction:
// log2(LPC) shuffle rounds per LPC steps instead of per step). The lanes of
// one channel are 32 / LPC apart (q is the slowest-varying lane index).
template <int LPC>
__device__ __forceinline__ float reduce_steps(const float (&part)[LPC], int q) {
    if constexpr (LPC == 2) {
        const float keep = q ? part[1] : part[0];
        const float send = q ? part[0] : part[1];
        return keep + __shfl_xor_sync(kFull, send, 16);
    } else {
        static_assert(LPC == 4, "LPC must be 2 or 4");
        const bool hi = (q & 2) != 0;
        float k0 = hi ? part[2] : part[0], k1 = hi ? part[3] : part[1];
        const float s0 = hi ? part[0] : part[2], s1 = hi ? part[1] : part[3];
        k0 += __shfl_xor_sync(kFull, s0, 16);
        k1 += __shfl_xor_sync(kFull, s1, 16);
        const bool odd = (q & 1) != 0;
        const float keep = odd ? k1 : k0, send = odd ? k0 : k1;
        return keep + __shfl_xor_sync(kFull, send, 8);
    }
}

template <typename T, int LPC, int STAGES, bool kStoreAll, bool kCkpt>
__global__ void __launch_bounds__(kThreads, kStoreAll ? MB_VERIFY_MINB : 1)
    prefill_kernel(const __grid_constant__ PrefillArgs a) {
    using G = Geom<LPC>;
    constexpr int CH = G::kCh;
    using S = Smem<T, CH, STAGES>;
    extern __shared__ unsigned char smem_dyn[];
    S &s = *reinterpret_cast<S *>((reinterpret_cast<uintptr_t>(smem_dyn) + 127) &
                                  ~static_cast<uintptr_t>(127));
    const ScanParams &p = a.p;
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    // blockIdx.x = batch row * channel tiles + channel tile (no 65535 limit on batch)
    const int ntd = (int)((p.d_inner + CH - 1) / CH);
    const int b = blockIdx.x / ntd;
    const int d0 = (blockIdx.x % ntd) * CH;
    const int64_t L = p.seqlen, D = p.d_inner;
    const int64_t nchunks = (L + kT - 1) / kT;
    const bool gate = a.has_gate != 0;

    if (tid == 0) {
        for (int st = 0; st < STAGES; ++st) mbar_init(&s.full[st], 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (tid == 0) {
        for (int st = 0; st < STAGES && st < nchunks; ++st) issue_chunk(s, a, st, st, d0, b);
    }

    // ---- conversion role
    ConvRole<CH> cr;
    cr.cp = tid % ConvRole<CH>::kPairsPerRow;
    cr.th = tid / ConvRole<CH>::kPairsPerRow;
    {
        const int64_t dc = d0 + 2 * cr.cp;   // D % 8 == 0: both channels valid or neither
        cr.ok = dc < D;
        cr.bias = (cr.ok && p.dt_bias) ? __ldg(reinterpret_cast<const float2 *>(p.dt_bias + dc))
                                       : make_float2(0.f, 0.f);
        cr.dsk = (cr.ok && p.D) ? __ldg(reinterpret_cast<const float2 *>(p.D + dc)) : make_float2(0.f, 0.f);
    }

    // ---- scan role: channel c, states kSPL*q .. kSPL*q + kSPL-1
    const int c = warp * G::kChPerWarp + lane % G::kChPerWarp;
    const int q = lane / G::kChPerWarp;
    const int64_t d = d0 + c;
    const bool chan_ok = d < D;
    float2 h[G::kPairs], a2[G::kPairs];
#pragma unroll
    for (int k = 0; k < G::kPairs; ++k) { h[k] = make_float2(0.f, 0.f); a2[k] = h[k]; }
    if (chan_ok) {
        const float2 *Ap = reinterpret_cast<const float2 *>(p.A + d * kDState + G::kSPL * q);
        const float2 *hp = reinterpret_cast<const float2 *>(p.h0 + ((int64_t)b * D + d) * kDState + G::kSPL * q);
#pragma unroll
        for (int k = 0; k < G::kPairs; ++k) {
            const float2 av = __ldg(Ap + k);
            a2[k] = make_float2(av.x * kLog2e, av.y * kLog2e);
            if (p.h0) h[k] = __ldg(hp + k);
        }
    }

    // ---- prologue: chunk 0
    bool ok = nchunks > 0 ? mbar_wait(&s.full[0], 0) : true;
    if (ok && nchunks > 0) convert(s.cv[0], s.raw[0], cr, 0, L, gate);
    if (__syncthreads_or(ok ? 0 : 1)) {
        if (tid == 0) {
            report(p.status, 4 /* MB_ERR_TIMEOUT */, 0);
            for (int j = 0; j < STAGES && j < nchunks; ++j) mbar_wait(&s.full[j], 0);
        }
        return;
    }

    for (int64_t i = 0; i < nchunks; ++i) {
        const int64_t t0 = i * kT;
        const bool has_next = i + 1 < nchunks;
        // (1) chunk i+1: wait for its tiles and convert them
        const int nst = (int)((i + 1) % STAGES);
        ok = has_next ? mbar_wait(&s.full[nst], (uint32_t)(((i + 1) / STAGES) & 1)) : true;
        if (has_next && ok) convert(s.cv[(i + 1) & 1], s.raw[nst], cr, t0 + kT, L, gate);

        // (2) chunk i: decays of all kT steps, recurrence, shares of C.h
        if constexpr (kCkpt) {   // state before chunk i, for the backward's recompute
            static_assert(kT == kCkptSteps, "checkpoints are taken per chunk");
            if (chan_ok) {
                float2 *dst = reinterpret_cast<float2 *>(
                    p.h_ckpt + (((int64_t)b * nchunks + i) * D + d) * kDState + G::kSPL * q);
#pragma unroll
                for (int k = 0; k < G::kPairs; k += 2)
                    *reinterpret_cast<float4 *>(dst + k) = make_float4(h[k].x, h[k].y, h[k + 1].x, h[k + 1].y);
            }
        }
        const Conv<CH> &cv = s.cv[i & 1];
        const Raw<T, CH> &rs = s.raw[i % STAGES];   // B, C straight from the TMA tile
        float2 ab[kT][G::kPairs];
        float gx[kT];
#pragma unroll
        for (int t = 0; t < kT; ++t) {
            const float2 dg = cv.dg[t][c];
            const float2 dd = make_float2(dg.x, dg.x);
            gx[t] = dg.y;
#pragma unroll
            for (int k = 0; k < G::kPairs; ++k) {
                const float2 e = mul2(dd, a2[k]);
                ab[t][k] = make_float2(ex2(e.x), ex2(e.y));
            }
        }
        float part[kT];
#pragma unroll
        for (int t = 0; t < kT; ++t) {
            const float2 gg = make_float2(gx[t], gx[t]);
            float2 bp[G::kPairs], cp[G::kPairs];
#pragma unroll
            for (int k = 0; k < G::kPairs; k += 2) {
                const float4 b4 = ld_quad(&rs.B[t][G::kSPL * q + 2 * k]);
                const float4 c4 = ld_quad(&rs.C[t][G::kSPL * q + 2 * k]);
                bp[k] = make_float2(b4.x, b4.y); bp[k + 1] = make_float2(b4.z, b4.w);
                cp[k] = make_float2(c4.x, c4.y); cp[k + 1] = make_float2(c4.z, c4.w);
            }
            float2 acc[2];
#pragma unroll
            for (int k = 0; k < G::kPairs; ++k) {
                h[k] = fma2(ab[t][k], h[k], mul2(bp[k], gg));
                acc[k & 1] = k < 2 ? mul2(cp[k], h[k]) : fma2(cp[k], h[k], acc[k & 1]);
            }
            const float2 sum = add2(acc[0], acc[1]);
            part[t] = sum.x + sum.y;
            if constexpr (kStoreAll) {
                if (chan_ok && t0 + t < L) {
                    float2 *dst = reinterpret_cast<float2 *>(
                        p.h_out + (((int64_t)b * L + t0 + t) * D + d) * kDState + G::kSPL * q);
#pragma unroll
                    for (int k = 0; k < G::kPairs; k += 2)
                        __stcs(reinterpret_cast<float4 *>(dst + k),
                               make_float4(h[k].x, h[k].y, h[k + 1].x, h[k + 1].y));
                }
            }
        }
        // (3) chunk i: reduce across the lanes of each channel, gate, stage y
        T(&ys)[kT][CH] = s.ys[i & 1];
#pragma unroll
        for (int m = 0; m < kT / LPC; ++m) {
            float grp[LPC];
#pragma unroll
            for (int u = 0; u < LPC; ++u) grp[u] = part[LPC * m + u];
            const float ysum = reduce_steps<LPC>(grp, q);
            const int t = LPC * m + q;
            const float2 xs = cv.xs[t][c];
            ys[t][c] = from_f32<T>((ysum + xs.x) * xs.y);
        }
        fence_proxy_async_smem();   // y tile -> visible to the TMA store below
        if (tid == 0) bulk_wait_read_all();   // the store of chunk i-1 no longer reads its tile
        if (__syncthreads_or(ok ? 0 : 1)) {
            if (tid == 0) {
                report(p.status, 4 /* MB_ERR_TIMEOUT */, i + 1);
                for (int64_t j = i + 1; j < i + STAGES && j < nchunks; ++j)
                    mbar_wait(&s.full[j % STAGES], (uint32_t)((j / STAGES) & 1));
                bulk_wait_all();
            }
            return;
        }
        if (tid == 0) {
            tma_store_3d(&a.tm_y, &ys[0][0], d0, (int)t0, b);
            bulk_commit();
            // stage i % STAGES (chunk i: converted last iteration, scanned
            // now) is free: refill it with chunk i + STAGES
            if (i + STAGES < nchunks) {
                fence_proxy_async_smem();
                issue_chunk(s, a, (int)(i % STAGES), i + STAGES, d0, b);
            }
        }
    }
    if (tid == 0) bulk_wait_all();

    if (!kStoreAll && p.h_out && chan_ok) {
        float2 *hp = reinterpret_cast<float2 *>(p.h_out + ((int64_t)b * D + d) * kDState + G::kSPL * q);
#pragma unroll
        for (int k = 0; k < G::kPairs; ++k) hp[k] = h[k];
    }
}

// ---------------------------------------------------------------------------
// Host side: tensor maps and the launch.

// [batch, L, inner] tensor with a (box_inner x kT x 1) box; rows (b, t) are
// `row` elements apart (row >= inner).
bool make_map(CUtensorMap *m, const void *base, bool bf16, int64_t batch, int64_t L, int64_t inner,
              int box_inner, int64_t row = 0) {
    const int64_t es = bf16 ? 2 : 4;
    if (row == 0) row = inner;
    const uint64_t dims[3] = {(uint64_t)inner, (uint64_t)L, (uint64_t)batch};
    const uint64_t strides[2] = {(uint64_t)(row * es), (uint64_t)(L * row * es)};
    const uint32_t box[3] = {(uint32_t)box_inner, (uint32_t)kT, 1};
    return encode_tmap(m, base, (int)es, 3, dims, strides, box);
}

template <typename T, int LPC, int STAGES, bool kStoreAll, bool kCkpt = false>
cudaError_t launch_typed(const ScanParams &p, cudaStream_t s) {
    constexpr int kCh = Geom<LPC>::kCh;
    const bool bf16 = sizeof(T) == 2;
    PrefillArgs a;
    memset(&a, 0, sizeof(a));
    a.p = p;
    a.has_gate = p.z != nullptr;
    if (!make_map(&a.tm_dt, p.dt, bf16, p.batch, p.seqlen, p.d_inner, kCh) ||
        !make_map(&a.tm_x, p.x, bf16, p.batch, p.seqlen, p.d_inner, kCh) ||
        (p.z && !make_map(&a.tm_z, p.z, bf16, p.batch, p.seqlen, p.d_inner, kCh)) ||
        !make_map(&a.tm_B, p.B, bf16, p.batch, p.seqlen, kDState, kDState, p.bc_stride) ||
        !make_map(&a.tm_C, p.C, bf16, p.batch, p.seqlen, kDState, kDState, p.bc_stride) ||
        !make_map(&a.tm_y, p.y, bf16, p.batch, p.seqlen, p.d_inner, kCh))
        return cudaErrorInvalidValue;
    const size_t smem = sizeof(Smem<T, kCh, STAGES>) + 128;
    auto k = prefill_kernel<T, LPC, STAGES, kStoreAll, kCkpt>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid((unsigned)(((p.d_inner + kCh - 1) / kCh) * p.batch));
    k<<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefill(const ScanParams &p, bool bf16, cudaStream_t s) {
    if (p.batch == 0 || p.d_inner == 0) return cudaSuccess;
    if (p.seqlen == 0) {
        // Nothing to scan: the final state is the initial state.
        if (!p.h_out) return cudaSuccess;
        const size_t bytes = (size_t)p.batch * p.d_inner * kDState * sizeof(float);
        if (p.h0) {
            if (p.h0 == p.h_out) return cudaSuccess;
            return cudaMemcpyAsync(p.h_out, p.h0, bytes, cudaMemcpyDeviceToDevice, s);
        }
        return cudaMemsetAsync(p.h_out, 0, bytes, s);
    }
    constexpr int LPC = kPrefillLanesPerChannel;
    return bf16 ? launch_typed<__nv_bfloat16, LPC, kPrefillStages, false>(p, s)
                : launch_typed<float, LPC, kPrefillStages, false>(p, s);
}

cudaError_t launch_prefill_ckpt(const ScanParams &p, bool bf16, cudaStream_t s) {
    if (p.batch == 0 || p.d_inner == 0) return cudaSuccess;
    if (p.seqlen == 0) return launch_prefill(p, bf16, s);   // no chunks: no checkpoints
    constexpr int LPC = kPrefillLanesPerChannel;
    return bf16 ? launch_typed<__nv_bfloat16, LPC, kPrefillStages, false, true>(p, s)
                : launch_typed<float, LPC, kPrefillStages, false, true>(p, s);
}

cudaError_t launch_verify(const ScanParams &p, bool bf16, cudaStream_t s) {
    if (p.batch == 0 || p.d_inner == 0 || p.seqlen == 0) return cudaSuccess;
    constexpr int LPC = kPrefillLanesPerChannel;
    if (p.seqlen <= kT)   // one chunk: a single ring stage suffices (smaller CTAs, more resident)
        return bf16 ? launch_typed<__nv_bfloat16, LPC, 1, true>(p, s)
                    : launch_typed<float, LPC, 1, true>(p, s);
    return bf16 ? launch_typed<__nv_bfloat16, LPC, kVerifyStages, true>(p, s)
                : launch_typed<float, LPC, kVerifyStages, true>(p, s);
}

}  // namespace mbscan
