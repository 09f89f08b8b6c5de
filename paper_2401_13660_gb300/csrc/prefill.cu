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
// for the whole span (small CTAs spread the channels evenly over the SMs).
// LPC lanes share a channel, each keeping 16 / LPC of its fp32 states in
// registers. The state index varies slowest across a warp, so the 8 lanes of
// each quarter-warp read the same B, C values (a shared-memory broadcast).
//
// Pipeline, per chunk of kT = 16 time steps:
//  * one thread keeps a STAGES-deep ring of 3-D TMA tile loads in flight:
//    dt, x, z [kT x CH] and B, C [kT x 16], one mbarrier per stage (bounded
//    waits, tma.cuh);
//  * the CTA converts a chunk once per (t, channel) into fp32 in shared
//    memory: (Delta, Delta*x) with Delta = softplus(dt + bias), (D*x, silu z);
//    a bf16 prefill also widens the chunk's B and C rows to fp32 once, so
//    that the scan does not convert them again in every lane;
//  * each lane scans the chunk: Abar = 2^(Delta * A*log2 e) on the SFU for all
//    kT steps, then h = Abar*h + B*(Delta*x) and its share of C.h in packed
//    f32x2 arithmetic, reading B and C (four states each) from those fp32
//    rows, or, in verify and for fp32 inputs, straight from the TMA tile in
//    the input dtype; groups of LPC steps are reduced across the LPC
//    lanes of a channel with log2(LPC) shuffle rounds, each lane finishing one
//    output y = (C.h + D*x) * silu(z), which goes to a shared-memory tile that
//    one thread writes out with a TMA store.
//  Loop iteration i converts chunk i+1 and scans chunk i in one basic block,
//  so every warp has two independent instruction streams to interleave; one
//  CTA barrier per chunk orders them, after which the stage of chunk i is
//  refilled with chunk i + STAGES.
// Steps at or beyond L are converted with Delta = 0, which leaves h unchanged.
//
// Fused Delta projection (kFuse, bf16): instead of a dt tile the ring holds the
// chunk's dt_low tile [kT x r] (W_R x of Eq. 3) and, once per CTA, the CTA's
// W_Delta rows [CH x r], both as 128-byte-swizzled TMA boxes; in the
// conversion step each warp forms the dt tile of its own 8 channels with r/16
// mma.sync m16n8k16 (fp32 accumulation), and its lanes convert the channel
// pairs and steps that the accumulator layout gives them.
#include <stddef.h>
#include <string.h>

#include <atomic>

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
// With the fused Delta projection and dt_rank > 64 each stage also holds two
// or more dt_low boxes: one stage less keeps 4 CTAs per SM.
constexpr int kPrefillStagesWide = 3;
constexpr int kVerifyStages = 2;   // verify spans are short
// Verify CTAs per SM the register budget must allow (5: 96 registers). The
// scan reads its shared tiles through shared-state-space loads, which the
// compiler may schedule ahead of the h_all stores; below 96 registers those
// early loads spill.
#ifndef MB_VERIFY_MINB
#define MB_VERIFY_MINB 5
#endif
#ifndef MB_VERIFY_FUSED_MINB
#define MB_VERIFY_FUSED_MINB 5   // the same with the Delta projection in the kernel
#endif

// Lane geometry: LPC lanes share one channel, each holding kSPL states.
template <int LPC>
struct Geom {
    static constexpr int kSPL = kDState / LPC;     // states per lane
    static constexpr int kPairs = kSPL / 2;        // float2 state pairs per lane
    static constexpr int kChPerWarp = 32 / LPC;
    static constexpr int kCh = kWarps * kChPerWarp;  // channels per CTA
};

template <typename T, int CH, bool kFuse>
struct alignas(128) Raw {  // TMA destinations; every member offset is a multiple of 128 B
    T x[kT][CH];
    T z[kT][CH];
    T B[kT][kDState];
    T C[kT][kDState];
    T dt[kFuse ? 1 : kT][CH];   // unused when Delta is projected in the kernel
};

template <int CH>
struct Conv {
    float2 dg[kT][CH];          // (Delta, Delta*x)
    float2 xs[kT][CH];          // (D*x, silu(z)); silu(z) = 1 without a gate
};

// B and C rows widened to fp32 once per chunk (bf16 prefill): the scan then
// reads four states of each with one shared load and no per-lane conversion.
// Verify spans are a single chunk, where the extra pass only lengthens the
// critical path; they read the bf16 tiles directly.
template <bool kWide>
struct alignas(16) WideBC {
    float B[kT][kDState];
    float C[kT][kDState];
};
template <>
struct WideBC<false> {};

template <typename T, bool kStoreAll>
constexpr bool kWideBC = sizeof(T) == 2 && !kStoreAll;

template <typename T, int CH, int STAGES, bool kFuse, bool kWide>
struct Smem {
    Raw<T, CH, kFuse> raw[STAGES];
    Conv<CH> cv[2];
    WideBC<kWide> wbc[2];       // with cv: chunk i in slot i % 2
    alignas(128) T ys[2][kT][CH];   // output tiles, written out by TMA stores
    uint64_t full[STAGES];
};

struct PrefillArgs {
    CUtensorMap tm_dt, tm_x, tm_z, tm_B, tm_C, tm_y;
    // fused Delta projection: dt_low [batch, L, r] and W_dt [D, r] in 64-wide,
    // 128-byte-swizzled boxes (kRankTile columns x kT rows, resp. x CH rows)
    CUtensorMap tm_dtl, tm_wdt;
    ScanParams p;
    int has_gate;
    int nbox;      // ceil(dt_rank / kRankTile)
    int grid_segs; // segments of L covered by the grid (blockIdx = (b, segment, channel tile))
};

// Shared-memory layout of the fused Delta projection, after the Smem struct:
// per stage nbox dt_low boxes (kT x 128 B), then the CTA's W_dt slice
// (nbox boxes of CH x 128 B); 1024-byte aligned for the 128-byte swizzle.
constexpr uint32_t kDtlBox = kT * 128;
template <int CH>
struct FuseLayout {
    static constexpr uint32_t kWBox = CH * 128;
    static uint32_t bytes(int stages, int nbox) { return 1024 + (uint32_t)nbox * (stages * kDtlBox + kWBox); }
};

// Byte offset of 16-byte chunk `chunk` of row `row` in a 128-byte-swizzled box.
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
    return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

template <typename T, int CH, int STAGES, bool kFuse, bool kWide>
__device__ __forceinline__ void issue_chunk(Smem<T, CH, STAGES, kFuse, kWide> &s, const PrefillArgs &a, int stage,
                                            int64_t chunk, int d0, int b, unsigned char *fz,
                                            uint32_t extra_bytes = 0) {
    constexpr uint32_t tok = kT * CH * sizeof(T), bc = kT * kDState * sizeof(T);
    const uint32_t bytes = (a.has_gate ? 2 : 1) * tok + 2 * bc + extra_bytes +
                           (kFuse ? (uint32_t)a.nbox * kDtlBox : tok);
    uint64_t *bar = &s.full[stage];
    mbar_arrive_expect_tx(bar, bytes);
    const int t = (int)(chunk * kT);
    Raw<T, CH, kFuse> &r = s.raw[stage];
    if constexpr (kFuse) {
        for (int bx = 0; bx < a.nbox; ++bx)
            tma_load_3d(fz + (stage * a.nbox + bx) * kDtlBox, &a.tm_dtl, bar, bx * kRankTile, t, b);
    } else {
        tma_load_3d(&r.dt[0][0], &a.tm_dt, bar, d0, t, b);
    }
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
// channel pair (2 cp, 2 cp + 1) at steps th, th + kRows, ... With the fused
// Delta projection the pairs follow the mma accumulator layout: warp w owns
// channels 8w .. 8w+7, lane l the pair 4w + l % 4 at steps l / 4 and l / 4 + 8.
template <int CH>
struct ConvRole {
    static constexpr int kPairsPerRow = CH / 2;
    static constexpr int kRows = kThreads / kPairsPerRow;   // step rows per pass
    static constexpr int kPasses = kT / kRows;
    int cp, th;
    float2 bias, dsk;
    bool ok;
};

// Delta before softplus for the fused projection (Eq. 3, W_Delta (W_R x)):
// warp w multiplies the chunk's dt_low tile [kT x r] by its 8 channels' W_dt
// rows [8 x r]^T on the tensor cores, r / 16 mma steps; both operands come
// from 128-byte-swizzled TMA boxes (dtl: this stage's dt_low boxes, w: the
// CTA's W_dt boxes). acc[0..1]: steps lane / 4, channels 8w + 2 (lane % 4) + {0, 1};
// acc[2..3]: the same channels at step lane / 4 + 8.
template <int CH>
__device__ __forceinline__ void project_delta(float (&acc)[4], uint32_t dtl, uint32_t w, int nks) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t tok = order_token();   // the operands are valid from here (after the stage's wait)
    dtl += tok;
    w += tok;
    acc[0] = acc[1] = acc[2] = acc[3] = 0.f;
    const int arow = lane & 15, achunk = lane >> 4;             // A: 4 matrices (rows 0-7 / 8-15, k 0-7 / 8-15)
    const int brow = 8 * warp + (lane & 7), bchunk = (lane >> 3) & 1;   // B: 2 matrices (k 0-7 / 8-15)
    for (int ks = 0; ks < nks; ++ks) {
        const int bx = ks >> 2, c0 = (ks & 3) * 2;
        uint32_t a[4], b[2];
        ldsm_x4(dtl + bx * kDtlBox + swz(arow, c0 + achunk), a);
        ldsm_x2(w + bx * FuseLayout<CH>::kWBox + swz(brow, c0 + bchunk), b);
        mma_bf16_16816(acc, a, b);
    }
}

struct FuseCtx {
    uint32_t dtl, w;   // shared addresses: this stage's dt_low boxes, the W_dt boxes
    int nks;           // dt_rank / 16
};

// Convert one chunk: raw TMA tiles -> fp32 (Delta, Delta*x), (D*x, silu z)
// and, with kWide, fp32 rows of B and C.
template <typename T, int CH, bool kFuse, bool kWide>
__device__ __forceinline__ void convert(Conv<CH> &cv, WideBC<kWide> &wbc, const Raw<T, CH, kFuse> &r,
                                        const ConvRole<CH> &cr, int64_t t0, int64_t L, bool gate,
                                        const FuseCtx &fx) {
    float acc[4];
    if constexpr (kFuse) project_delta<CH>(acc, fx.dtl, fx.w, fx.nks);
#pragma unroll
    for (int k = 0; k < ConvRole<CH>::kPasses; ++k) {
        const int t = cr.th + ConvRole<CH>::kRows * k;
        const int c = 2 * cr.cp;
        float4 dg = make_float4(0.f, 0.f, 0.f, 0.f), xs = make_float4(0.f, 1.f, 0.f, 1.f);
        if (cr.ok && t0 + t < L) {
            const float2 xv = ld_pair(&r.x[t][c]);
            float2 dv;
            if constexpr (kFuse) dv = make_float2(acc[2 * k], acc[2 * k + 1]);
            else dv = ld_pair(&r.dt[t][c]);
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
    if constexpr (kWide) {   // item (t, j): four states of B (j < 4) or C (j >= 4) at step t
        static_assert(kDState == 16, "quarter rows of B and C");
        constexpr int kItems = kT * 8, kRounds = (kItems + kThreads - 1) / kThreads;
#pragma unroll
        for (int u = 0; u < kRounds; ++u) {
            const int it = (int)threadIdx.x + u * kThreads;
            if (kItems % kThreads != 0 && it >= kItems) break;
            const int t = it >> 3, j = it & 7;
            const float4 v = ld_quad(j < 4 ? &r.B[t][4 * j] : &r.C[t][4 * (j - 4)]);
            *reinterpret_cast<float4 *>(j < 4 ? &wbc.B[t][4 * j] : &wbc.C[t][4 * (j - 4)]) = v;
        }
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

// kSummary (first pass of a time-split prefill): scan each segment of L from a
// zero state and record its end state and the product of its decays in the
// scratch (no outputs). The second pass is the plain kernel: its segment s
// starts from the state the summaries of segments 0 .. s-1 give (folded with
// the associative operator of Section 2: h <- P_s' * h + H_s').
template <typename T, int LPC, int STAGES, bool kStoreAll, bool kCkpt, bool kFuse, bool kSummary = false>
__global__ void __launch_bounds__(kThreads, kStoreAll ? (kFuse ? MB_VERIFY_FUSED_MINB : MB_VERIFY_MINB) : 1)
    prefill_kernel(const __grid_constant__ PrefillArgs a) {
    using G = Geom<LPC>;
    constexpr int CH = G::kCh;
    static_assert(!kFuse || (LPC == 4 && sizeof(T) == 2 && CH == 8 * kWarps),
                  "the fused Delta projection maps one 8-channel mma tile per warp (bf16)");
    constexpr bool kWide = kWideBC<T, kStoreAll>;
    using S = Smem<T, CH, STAGES, kFuse, kWide>;
    // every TMA source or destination in S starts on a 128-byte boundary
    using R = Raw<T, CH, kFuse>;
    static_assert(sizeof(R) % 128 == 0 && offsetof(R, z) % 128 == 0 && offsetof(R, B) % 128 == 0 &&
                      offsetof(R, C) % 128 == 0 && offsetof(R, dt) % 128 == 0 && offsetof(S, raw) % 128 == 0 &&
                      offsetof(S, ys) % 128 == 0 && (sizeof(T) * kT * CH) % 128 == 0,
                  "TMA tiles must be 128-byte aligned");
    extern __shared__ unsigned char smem_dyn[];
    S &s = smem_aligned<S>(smem_dyn);
    // fused Delta projection: dt_low stage boxes, then the W_dt boxes (1024-aligned)
    uint32_t fz_addr = 0;   // shared address of the first dt_low box
    unsigned char *fz = nullptr;
    FuseCtx fx{0u, 0u, 0};
    if constexpr (kFuse) {
        const uint32_t sbase = smem_u32(smem_dyn);
        fz_addr = (sbase + 128 + (uint32_t)sizeof(S) + 1023u) & ~1023u;
        fz = smem_dyn + (fz_addr - sbase);
        fx.w = fz_addr + (uint32_t)(STAGES * a.nbox) * kDtlBox;
        fx.nks = (int)(a.p.dt_rank / 16);
    }
    const ScanParams &p = a.p;
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    // blockIdx.x = (batch row, segment of L, channel tile), channel tile fastest;
    // only the plain prefill is ever split over L
    constexpr bool kSplit = !kStoreAll && !kFuse;
    const int ntd = (int)((p.d_inner + CH - 1) / CH);
    const int64_t L = p.seqlen, D = p.d_inner;
    const int64_t nchunks = (L + kT - 1) / kT;   // chunks of the whole span
    int seg = 0, b = (int)(blockIdx.x / ntd);
    int64_t nseg = 1, c0 = 0, nch = nchunks;    // this CTA's chunks: c0 .. c0 + nch - 1
    if constexpr (kSplit) {
        seg = (int)((blockIdx.x / ntd) % a.grid_segs);
        b = (int)(blockIdx.x / ntd / a.grid_segs);
        nseg = p.nseg > 1 ? p.nseg : 1;
        const int64_t cps = (nchunks + nseg - 1) / nseg;   // chunks per segment
        c0 = seg * cps;
        nch = nchunks - c0 < cps ? nchunks - c0 : cps;
    }
    const int d0 = (blockIdx.x % ntd) * CH;
    const bool gate = a.has_gate != 0;

    if (tid == 0) {
        for (int st = 0; st < STAGES; ++st) mbar_init(&s.full[st], 1);
        fence_mbar_init();
    }
    __syncthreads();
    pdl_wait();   // everything below reads or writes global memory
    // Resume: the state this row starts from (0: h0, a > 0: h_prev_all[b, a-1]).
    // An accept count outside [0, k_prev] is reported and the row left
    // untouched; the check comes before any copy is issued.
    int resume_a = 0;
    if (p.accept) {
        resume_a = __ldg(p.accept + b);   // one batch row per CTA: uniform
        if (resume_a < 0 || resume_a > p.k_prev) {
            if (tid == 0 && d0 == 0) report(p.status, 1 /* MB_ERR_INVALID_ARG */, b);
            return;
        }
    }
    if (tid == 0) {
        for (int st = 0; st < STAGES && st < nch; ++st) {
            // the CTA's W_dt slice rides on chunk 0's barrier (its bytes are
            // part of that arrival's expected count)
            const bool wslice = kFuse && st == 0;
            issue_chunk(s, a, st, c0 + st, d0, b, fz, wslice ? (uint32_t)a.nbox * FuseLayout<CH>::kWBox : 0u);
            if (wslice)
                for (int bx = 0; bx < a.nbox; ++bx)
                    tma_load_2d(fz + (uint32_t)(STAGES * a.nbox) * kDtlBox + (uint32_t)bx * FuseLayout<CH>::kWBox,
                                &a.tm_wdt, &s.full[0], bx * kRankTile, d0);
        }
    }

    // ---- conversion role
    ConvRole<CH> cr;
    if constexpr (kFuse) {
        cr.cp = 4 * warp + (lane & 3);
        cr.th = lane >> 2;
    } else {
        cr.cp = tid % ConvRole<CH>::kPairsPerRow;
        cr.th = tid / ConvRole<CH>::kPairsPerRow;
    }
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
        const float *hrow = resume_a > 0
                                ? p.h_prev_all + (((int64_t)b * p.k_prev + resume_a - 1) * D + d) * kDState
                                : (p.h0 ? p.h0 + ((int64_t)b * D + d) * kDState : nullptr);
        const float2 *hp = hrow ? reinterpret_cast<const float2 *>(hrow + G::kSPL * q) : nullptr;
#pragma unroll
        for (int k = 0; k < G::kPairs; ++k) {
            const float2 av = __ldg(Ap + k);
            a2[k] = make_float2(av.x * kLog2e, av.y * kLog2e);
            if (hp && !kSummary) h[k] = __ldg(hp + k);   // a summary starts from zero
        }
        if constexpr (kSplit && !kSummary) {   // segment s > 0 of a split span: fold the summaries before it
            for (int sp = 0; sp < seg; ++sp) {
                const int64_t off = (((int64_t)b * nseg + sp) * D + d) * kDState + G::kSPL * q;
                const float2 *hs_ = reinterpret_cast<const float2 *>(p.seg_h + off);
                const float2 *ps_ = reinterpret_cast<const float2 *>(p.seg_p + off);
#pragma unroll
                for (int k = 0; k < G::kPairs; ++k) h[k] = fma2(ps_[k], h[k], hs_[k]);
            }
        }
    }
    float2 prod[G::kPairs];   // kSummary: product of the segment's decays
#pragma unroll
    for (int k = 0; k < G::kPairs; ++k) prod[k] = make_float2(1.f, 1.f);

    // ---- prologue: chunk 0
    bool ok = nch > 0 ? mbar_wait(&s.full[0], 0) : true;
    if constexpr (kFuse) ok = __all_sync(kFull, ok);   // mma.sync needs the whole warp
    auto stage_fx = [&](int st) {   // the fused projection's operands for ring stage st
        FuseCtx f = fx;
        if constexpr (kFuse) f.dtl = fz_addr + (uint32_t)(st * a.nbox) * kDtlBox;
        return f;
    };
    if (ok && nch > 0) convert(s.cv[0], s.wbc[0], s.raw[0], cr, c0 * kT, L, gate, stage_fx(0));
    if (__syncthreads_or(ok ? 0 : 1)) {
        if (tid == 0) {
            report(p.status, 4 /* MB_ERR_TIMEOUT */, 0);
            for (int j = 0; j < STAGES && j < nch; ++j) mbar_wait(&s.full[j], 0);
        }
        return;
    }

    for (int64_t i = 0; i < nch; ++i) {   // i: chunk c0 + i of the span, ring slot i % STAGES
        const int64_t t0 = (c0 + i) * kT;
        const bool has_next = i + 1 < nch;
        // (1) chunk i+1: wait for its tiles and convert them
        const int nst = (int)((i + 1) % STAGES);
        ok = has_next ? mbar_wait(&s.full[nst], (uint32_t)(((i + 1) / STAGES) & 1)) : true;
        if constexpr (kFuse) ok = __all_sync(kFull, ok);
        if (has_next && ok)
            convert(s.cv[(i + 1) & 1], s.wbc[(i + 1) & 1], s.raw[nst], cr, t0 + kT, L, gate, stage_fx(nst));

        // (2) chunk i: decays of all kT steps, recurrence, shares of C.h
        if constexpr (kCkpt) {   // state before chunk i, for the backward's recompute
            static_assert(kT == kCkptSteps, "checkpoints are taken per chunk");
            if (chan_ok) {
                float2 *dst = reinterpret_cast<float2 *>(
                    p.h_ckpt + (((int64_t)b * nchunks + c0 + i) * D + d) * kDState + G::kSPL * q);
#pragma unroll
                for (int k = 0; k < G::kPairs; k += 2)
                    *reinterpret_cast<float4 *>(dst + k) = make_float4(h[k].x, h[k].y, h[k + 1].x, h[k + 1].y);
            }
        }
        const Conv<CH> &cv = s.cv[i & 1];
        const Raw<T, CH, kFuse> &rs = s.raw[i % STAGES];   // without kWide: B, C straight from the TMA tile
        const WideBC<kWide> &wb = s.wbc[i & 1];
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
                float4 b4, c4;
                if constexpr (kWide) {
                    b4 = *reinterpret_cast<const float4 *>(&wb.B[t][G::kSPL * q + 2 * k]);
                    c4 = *reinterpret_cast<const float4 *>(&wb.C[t][G::kSPL * q + 2 * k]);
                } else {
                    b4 = ld_quad(&rs.B[t][G::kSPL * q + 2 * k]);
                    c4 = ld_quad(&rs.C[t][G::kSPL * q + 2 * k]);
                }
                bp[k] = make_float2(b4.x, b4.y); bp[k + 1] = make_float2(b4.z, b4.w);
                cp[k] = make_float2(c4.x, c4.y); cp[k + 1] = make_float2(c4.z, c4.w);
            }
            float2 acc[2];
#pragma unroll
            for (int k = 0; k < G::kPairs; ++k) {
                h[k] = fma2(ab[t][k], h[k], mul2(bp[k], gg));
                if constexpr (kSummary) prod[k] = mul2(prod[k], ab[t][k]);
                else acc[k & 1] = k < 2 ? mul2(cp[k], h[k]) : fma2(cp[k], h[k], acc[k & 1]);
            }
            if constexpr (!kSummary) {
                const float2 sum = add2(acc[0], acc[1]);
                part[t] = sum.x + sum.y;
            }
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
        for (int m = 0; m < (kSummary ? 0 : kT / LPC); ++m) {
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
                report(p.status, 4 /* MB_ERR_TIMEOUT */, c0 + i + 1);
                for (int64_t j = i + 1; j < i + STAGES && j < nch; ++j)
                    mbar_wait(&s.full[j % STAGES], (uint32_t)((j / STAGES) & 1));
                bulk_wait_all();
            }
            return;
        }
        if (tid == 0) {
            if constexpr (!kSummary) {
                tma_store_3d(&a.tm_y, &ys[0][0], d0, (int)t0, b);
                bulk_commit();
            }
            // stage i % STAGES (chunk i: converted last iteration, scanned
            // now) is free: refill it with chunk i + STAGES
            if (i + STAGES < nch) {
                fence_proxy_async_smem();
                issue_chunk(s, a, (int)(i % STAGES), c0 + i + STAGES, d0, b, fz);
            }
        }
    }
    if (tid == 0) bulk_wait_all();

    if constexpr (kSummary) {   // this segment's end state from a zero start, and its decay product
        if (chan_ok) {
            const int64_t off = (((int64_t)b * nseg + seg) * D + d) * kDState + G::kSPL * q;
            float2 *hd = reinterpret_cast<float2 *>(p.seg_h + off);
            float2 *pd = reinterpret_cast<float2 *>(p.seg_p + off);
#pragma unroll
            for (int k = 0; k < G::kPairs; ++k) { hd[k] = h[k]; pd[k] = prod[k]; }
        }
    } else if (!kStoreAll && p.h_out && chan_ok && seg == nseg - 1) {   // the span's last state
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

template <typename T, int LPC, int STAGES, bool kStoreAll, bool kCkpt = false, bool kFuse = false>
cudaError_t launch_typed(const ScanParams &p, cudaStream_t s) {
    constexpr int kCh = Geom<LPC>::kCh;
    const bool bf16 = sizeof(T) == 2;
    PrefillArgs a;
    memset(&a, 0, sizeof(a));
    a.p = p;
    a.has_gate = p.z != nullptr;
    constexpr bool kSplittable = !kStoreAll && !kFuse;
    if (!kSplittable || p.nseg < 2 || !p.seg_h || !p.seg_p) a.p.nseg = 1;
    const int64_t nseg = a.p.nseg;
    size_t fuse_bytes = 0;
    if constexpr (kFuse) {
        // dt_low [batch, L, r] (rows dt_low_stride apart) and W_dt [D, r], both
        // in kRankTile-wide boxes with the 128-byte swizzle; columns past r read 0
        a.nbox = (int)((p.dt_rank + kRankTile - 1) / kRankTile);
        const uint64_t ldims[3] = {(uint64_t)p.dt_rank, (uint64_t)p.seqlen, (uint64_t)p.batch};
        const uint64_t lstr[2] = {(uint64_t)p.dt_low_stride * 2, (uint64_t)(p.seqlen * p.dt_low_stride) * 2};
        const uint32_t lbox[3] = {kRankTile, kT, 1};
        const uint64_t wdims[2] = {(uint64_t)p.dt_rank, (uint64_t)p.d_inner};
        const uint64_t wstr[1] = {(uint64_t)p.dt_rank * 2};
        const uint32_t wbox[2] = {kRankTile, (uint32_t)kCh};
        if (!encode_tmap(&a.tm_dtl, p.dt_low, 2, 3, ldims, lstr, lbox, 128) ||
            !encode_tmap(&a.tm_wdt, p.W_dt, 2, 2, wdims, wstr, wbox, 128))
            return cudaErrorInvalidValue;
        fuse_bytes = FuseLayout<kCh>::bytes(STAGES, a.nbox);
    } else {
        if (!make_map(&a.tm_dt, p.dt, bf16, p.batch, p.seqlen, p.d_inner, kCh)) return cudaErrorInvalidValue;
    }
    if (!make_map(&a.tm_x, p.x, bf16, p.batch, p.seqlen, p.d_inner, kCh) ||
        (p.z && !make_map(&a.tm_z, p.z, bf16, p.batch, p.seqlen, p.d_inner, kCh)) ||
        !make_map(&a.tm_B, p.B, bf16, p.batch, p.seqlen, kDState, kDState, p.bc_stride) ||
        !make_map(&a.tm_C, p.C, bf16, p.batch, p.seqlen, kDState, kDState, p.bc_stride) ||
        !make_map(&a.tm_y, p.y, bf16, p.batch, p.seqlen, p.d_inner, kCh))
        return cudaErrorInvalidValue;
    const size_t smem = sizeof(Smem<T, kCh, STAGES, kFuse, kWideBC<T, kStoreAll>>) + 128 + fuse_bytes;
    const int64_t ctas = ((p.d_inner + kCh - 1) / kCh) * p.batch;   // per segment of L
    cudaError_t e;
    if constexpr (kSplittable) {
        if (nseg > 1) {   // first pass: summaries of segments 0 .. nseg-2
            PrefillArgs a1 = a;
            a1.has_gate = 0;   // no outputs: the gate is not read
            a1.grid_segs = (int)(nseg - 1);
            auto k1 = prefill_kernel<T, LPC, STAGES, false, false, false, true>;
            if ((e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
                return e;
            if ((e = launch_pdl(false, k1, dim3((unsigned)(ctas * (nseg - 1))), dim3(kThreads), smem, s, a1)) !=
                cudaSuccess)
                return e;
        }
    }
    a.grid_segs = (int)nseg;
    auto k = prefill_kernel<T, LPC, STAGES, kStoreAll, kCkpt, kFuse>;
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(false, k, dim3((unsigned)(ctas * nseg)), dim3(kThreads), smem, s, a);
}

}  // namespace

// Time split: only when the batch rows and channel tiles give at most one CTA
// per SM (a CTA alone on an SM leaves most of its issue slots idle); then into
// as many segments as fill the resident slots (4 per SM for bf16, 3 for fp32),
// each at least kMinSegChunks chunks long. The summary pass repeats most of a
// scan, so at 1.7 CTAs per SM (batch 4 x 2048 channels) the split measured
// slower (604 -> 653 us) while batch 1 x 2048 channels x 8192 steps went
// 480 -> 180 us.
constexpr int64_t kMinSegChunks = 8;

int64_t prefill_segments(const ScanParams &p, bool bf16) {
    if (p.batch <= 0 || p.d_inner <= 0 || p.seqlen <= 0 || p.dt_low) return 1;
    constexpr int kMaxDevices = 64;
    static std::atomic<int> sm_count[kMaxDevices];   // per device, filled on first use (0: not yet)
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 1;
    int sms = sm_count[dev].load(std::memory_order_relaxed);
    if (sms == 0) {
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 1;
        sm_count[dev].store(sms, std::memory_order_relaxed);   // every writer stores the same value
    }
    constexpr int kCh = Geom<kPrefillLanesPerChannel>::kCh;
    const int64_t slots = (int64_t)sms * (bf16 ? 4 : 3);
    const int64_t ctas = p.batch * ((p.d_inner + kCh - 1) / kCh);
    if (ctas > sms) return 1;
    const int64_t nchunks = (p.seqlen + kT - 1) / kT;
    int64_t nseg = slots / ctas;
    if (nseg > nchunks / kMinSegChunks) nseg = nchunks / kMinSegChunks;
    if (nseg < 2) return 1;
    const int64_t cps = (nchunks + nseg - 1) / nseg;
    return (nchunks + cps - 1) / cps;   // no empty segment
}

size_t prefill_split_bytes(const ScanParams &p, int64_t nseg) {
    return nseg > 1 ? (size_t)(2 * p.batch * nseg * p.d_inner * kDState) * sizeof(float) : 0;
}

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
    if (p.dt_low)   // fused Delta projection (bf16 only; the API checks)
        return !bf16 ? cudaErrorInvalidValue
               : p.dt_rank <= kRankTile ? launch_typed<__nv_bfloat16, LPC, kPrefillStages, false, false, true>(p, s)
                                        : launch_typed<__nv_bfloat16, LPC, kPrefillStagesWide, false, false, true>(p, s);
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
    if (p.dt_low) {   // fused Delta projection (bf16 only; the API checks)
        if (!bf16) return cudaErrorInvalidValue;
        return p.seqlen <= kT ? launch_typed<__nv_bfloat16, LPC, 1, true, false, true>(p, s)
                              : launch_typed<__nv_bfloat16, LPC, kVerifyStages, true, false, true>(p, s);
    }
    if (p.seqlen <= kT)   // one chunk: a single ring stage suffices (smaller CTAs, more resident)
        return bf16 ? launch_typed<__nv_bfloat16, LPC, 1, true>(p, s)
                    : launch_typed<float, LPC, 1, true>(p, s);
    return bf16 ? launch_typed<__nv_bfloat16, LPC, kVerifyStages, true>(p, s)
                : launch_typed<float, LPC, kVerifyStages, true>(p, s);
}

}  // namespace mbscan
