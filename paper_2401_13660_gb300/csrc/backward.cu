// Backward of the selective-scan layer core: the training path (MambaByte
// trains through this scan, Section 2 "parallel scans"; Section 4 setup).
// Given the forward inputs, the state checkpoints of the training forward
// (the state before every kCkptSteps-step chunk) and dJ/dout, dJ/dh_last, it
// returns every input gradient. For each (batch row, channel), from t = L-1
// down to 0, with g = dJ/dh_t:
//   dy = dout * silu(z);  dz = dout * y * silu'(z);  g += dy * C_t
//   dC_t += dy * h_t (summed over channels);  S1 = sum_n g B_t
//   dx = dy * D + Delta * S1;  dDelta = x * S1 + sum_n (g Abar h_{t-1}) A
//   dB_t += g * Delta * x (summed over channels);  dA += (g Abar h_{t-1}) Delta
//   g *= Abar;  ddt = dDelta * sigmoid(dt + bias);  dbias += ddt;  dD += dy x
// and dh0 = g at the end.
//
// Work decomposition (the lane geometry of the forward kernel): a CTA of 4
// warps owns 32 channels of one batch row; lane = 8 q + c8 keeps the 4 states
// 4q .. 4q+3 of channel warp*8 + c8. Chunks of kCkptSteps steps are taken in
// reverse order through a ring of 3-D TMA tile loads (dt, x, z, dout, B, C).
// Per chunk:
//  * conversion (once per (t, channel pair)): Delta, Delta*x and dy into
//    shared memory; for bf16 inputs also the chunk's B and C rows, widened
//    to fp32 once instead of in every lane of both sweeps (x, needed only
//    where a step is finished, is read there from the input tile);
//  * recompute: from the chunk's checkpoint, the forward states of the 16
//    steps and each lane's share of C.h (for y); the states of the even steps
//    go to shared memory (one float4 per lane and even step): the sweep forms
//    an odd step's state again from the even state below it, with the decay
//    and inputs of that step that it needs anyway, bit for bit the same value
//    (half the shared-memory traffic of keeping every state: 3.41 -> 3.24 ms
//    on the 353M layer);
//  * reverse sweep: the adjoint g, dA in registers; per step the lane's
//    shares of dB, dC (8 values) are summed over the 8 channels of its
//    quarter-warp with a transposed 3-round shuffle reduction and left in
//    shared memory per warp; S1, S2 and y are summed over the 4 lanes of a
//    channel with a transposed 2-round reduction per 4 steps, after which lane
//    q finishes step 4m+q (dx, ddt, dz to output tiles written by TMA stores);
//    The finishing lane evaluates sigmoid(dt + bias) and silu'(z) itself from
//    the chunk's tiles;
//  * after the chunk's barrier (in the next iteration), the CTA's dB, dC sums
//    are sent to global memory with vector atomics.
// Two barriers per chunk (after the conversion, after the sweep) keep one
// conversion buffer and one dB/dC buffer, so that 4 CTAs fit on an SM.
// dA, dD, dbias are accumulated in registers and added atomically at the end
// (one contribution per batch row); dh0 is stored directly.
#include <stddef.h>
#include <string.h>

#include "common.cuh"
#include "tma.cuh"

namespace mbscan {
namespace {

constexpr int kBT = kCkptSteps;   // steps per chunk
constexpr int kBWarps = 4;
constexpr int kBThreads = 32 * kBWarps;
constexpr int kBCh = 8 * kBWarps;  // channels per CTA
constexpr int kBStages = 2;

template <typename T>
struct BRaw {  // TMA destinations; member offsets are multiples of 128 B
    T dt[kBT][kBCh];
    T x[kBT][kBCh];
    T z[kBT][kBCh];
    T dout[kBT][kBCh];
    T B[kBT][kDState];
    T C[kBT][kDState];
};

template <bool kWide>
struct BConv {
    float2 dg[kBT][kBCh];   // (Delta, Delta*x)
    float dy[kBT][kBCh];    // dJ/dy * silu(z)
};
// bf16 inputs: B and C rows widened to fp32 once per chunk (both sweeps read
// four states of each per step; the space comes from keeping x out of the
// conversion tile: the few readers of x take it from the input tile)
template <>
struct BConv<true> {
    float2 dg[kBT][kBCh];
    float dy[kBT][kBCh];
    float B[kBT][kDState];
    float C[kBT][kDState];
};

template <typename T>
struct BSmem {
    BRaw<T> raw[kBStages];
    BConv<sizeof(T) == 2> cv;
    float4 hs[kBT / 2][kBThreads];    // recomputed states of the chunk's even steps, per lane
    T gx[kBT][kBCh], gdt[kBT][kBCh], gz[kBT][kBCh];   // output tiles (TMA stores)
    float bc[kBT][32];   // per step: slot 8q + j, j < 4 dB[4q+j], else dC[4q+j-4]
    uint64_t full[kBStages];
};

struct BwdArgs {
    CUtensorMap tm_dt, tm_x, tm_z, tm_dout, tm_B, tm_C, tm_dx, tm_ddt, tm_dz;
    ScanParams p;
    GradParams g;
    int has_gate;
};

template <typename T>
__device__ __forceinline__ void issue_bchunk(BSmem<T> &s, const BwdArgs &a, int stage, int64_t chunk,
                                             int d0, int b) {
    constexpr uint32_t tok = kBT * kBCh * sizeof(T), bc = kBT * kDState * sizeof(T);
    const uint32_t bytes = (a.has_gate ? 4 : 3) * tok + 2 * bc;
    uint64_t *bar = &s.full[stage];
    mbar_arrive_expect_tx(bar, bytes);
    const int t = (int)(chunk * kBT);
    BRaw<T> &r = s.raw[stage];
    tma_load_3d(&r.dt[0][0], &a.tm_dt, bar, d0, t, b);
    tma_load_3d(&r.x[0][0], &a.tm_x, bar, d0, t, b);
    if (a.has_gate) tma_load_3d(&r.z[0][0], &a.tm_z, bar, d0, t, b);
    tma_load_3d(&r.dout[0][0], &a.tm_dout, bar, d0, t, b);
    tma_load_3d(&r.B[0][0], &a.tm_B, bar, 0, t, b);
    tma_load_3d(&r.C[0][0], &a.tm_C, bar, 0, t, b);
}

__device__ __forceinline__ float2 ld_pair(const float *p) { return *reinterpret_cast<const float2 *>(p); }
__device__ __forceinline__ float2 ld_pair(const __nv_bfloat16 *p) {
    const unsigned u = *reinterpret_cast<const unsigned *>(p);
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}
__device__ __forceinline__ float4 ld_quad(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 ld_quad(const __nv_bfloat16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

// sigmoid(v) = u / (1 + u) with u = e^v, 1 where u overflows (v > 15 gives
// 1 - 3e-7, below fp32 resolution of the product it scales).
__device__ __forceinline__ float sigmoid_v(float v) {
    if (v > 15.f) return 1.f;
    const float u = ex2(v * kLog2e);
    return __fdividef(u, 1.f + u);
}

// Conversion of one chunk by one thread: channel pair cp at steps th, th + 8
// (and, for bf16, a quarter row of B or C).
template <typename T>
__device__ __forceinline__ void bconvert(BConv<sizeof(T) == 2> &cv, const BRaw<T> &r, int cp, int th, float2 bias,
                                         bool ok, int64_t t0, int64_t L, bool gate) {
#pragma unroll
    for (int k = 0; k < kBT / 8; ++k) {
        const int t = th + 8 * k;
        const int c = 2 * cp;
        float4 dg = make_float4(0.f, 0.f, 0.f, 0.f);   // (Delta, Delta*x) of channels c, c + 1
        float2 dy = make_float2(0.f, 0.f);
        if (ok && t0 + t < L) {
            const float2 xv = ld_pair(&r.x[t][c]);
            const float2 dv = ld_pair(&r.dt[t][c]);
            const float2 ov = ld_pair(&r.dout[t][c]);
            const float d0 = softplus(dv.x + bias.x), d1 = softplus(dv.y + bias.y);   // as in the forward
            dy = ov;
            if (gate) {
                const float2 zv = ld_pair(&r.z[t][c]);
                dy = make_float2(ov.x * silu(zv.x), ov.y * silu(zv.y));
            }
            dg = make_float4(d0, d0 * xv.x, d1, d1 * xv.y);
        }
        *reinterpret_cast<float4 *>(&cv.dg[t][c]) = dg;
        *reinterpret_cast<float2 *>(&cv.dy[t][c]) = dy;
    }
    if constexpr (sizeof(T) == 2) {   // thread (t, j): four states of B (j < 4) or C (j >= 4) at step t
        static_assert(kBThreads == kBT * 8 && kDState == 16, "one quarter row of B or C per thread");
        const int t = threadIdx.x >> 3, j = threadIdx.x & 7;
        const float4 v = ld_quad(j < 4 ? &r.B[t][4 * j] : &r.C[t][4 * (j - 4)]);
        *reinterpret_cast<float4 *>(j < 4 ? &cv.B[t][4 * j] : &cv.C[t][4 * (j - 4)]) = v;
    }
}

// Four states of B and C at step t: the widened rows (bf16) or the tile (fp32).
template <typename T>
__device__ __forceinline__ void load_bc(const BConv<sizeof(T) == 2> &cv, const BRaw<T> &r, int t, int q,
                                        float4 &b4, float4 &c4) {
    if constexpr (sizeof(T) == 2) {
        b4 = *reinterpret_cast<const float4 *>(&cv.B[t][4 * q]);
        c4 = *reinterpret_cast<const float4 *>(&cv.C[t][4 * q]);
    } else {
        b4 = ld_quad(&r.B[t][4 * q]);
        c4 = ld_quad(&r.C[t][4 * q]);
    }
}

// Transposed sum over the 4 lanes of a channel (8 apart) for 4 consecutive
// steps: lane q ends with the full sum of step q.
__device__ __forceinline__ float reduce4(float p0, float p1, float p2, float p3, int q) {
    const bool hi = (q & 2) != 0;
    float k0 = hi ? p2 : p0, k1 = hi ? p3 : p1;
    const float s0 = hi ? p0 : p2, s1 = hi ? p1 : p3;
    k0 += __shfl_xor_sync(kFull, s0, 16);
    k1 += __shfl_xor_sync(kFull, s1, 16);
    const bool odd = (q & 1) != 0;
    const float keep = odd ? k1 : k0, send = odd ? k0 : k1;
    return keep + __shfl_xor_sync(kFull, send, 8);
}

// Transposed sum of 8 values over the 8 lanes c8 = 0..7 of a quarter-warp
// (lanes 1, 2, 4 apart): lane c8 ends with the sum of value c8.
__device__ __forceinline__ float reduce8(const float (&v)[8], int c8) {
    const bool h4 = (c8 & 4) != 0, h2 = (c8 & 2) != 0, h1 = (c8 & 1) != 0;
    float k[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float keep = h4 ? v[4 + i] : v[i], send = h4 ? v[i] : v[4 + i];
        k[i] = keep + __shfl_xor_sync(kFull, send, 4);
    }
    float k2[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const float keep = h2 ? k[2 + i] : k[i], send = h2 ? k[i] : k[2 + i];
        k2[i] = keep + __shfl_xor_sync(kFull, send, 2);
    }
    const float keep = h1 ? k2[1] : k2[0], send = h1 ? k2[0] : k2[1];
    return keep + __shfl_xor_sync(kFull, send, 1);
}

template <typename T>
__device__ __forceinline__ void store_out(T (&tile)[kBT][kBCh], int t, int c, float v) {
    tile[t][c] = from_f32<T>(v);
}

// dB, dC of one chunk: send the CTA's sums to global memory and clear the
// buffer for its next use (thread: step tid / 8, slots 4 sg .. 4 sg + 3).
__device__ __forceinline__ void flush_bc(float (&bc)[kBT][32], const GradParams &g, int64_t b, int64_t t0,
                                         int64_t L) {
    static_assert(kBT * 8 == kBThreads, "one thread per step and slot group");
    const int t = threadIdx.x >> 3, sg = threadIdx.x & 7;
    float4 &v = *reinterpret_cast<float4 *>(&bc[t][4 * sg]);
    if (t0 + t < L) {
        const int q = sg >> 1;
        float *dst = ((sg & 1) ? g.dC : g.dB) + ((b * L + t0 + t) * kDState + 4 * q);
        atomicAdd(reinterpret_cast<float4 *>(dst), v);
    }
    v = make_float4(0.f, 0.f, 0.f, 0.f);
}

template <typename T>
__global__ void __launch_bounds__(kBThreads, 4) backward_kernel(const __grid_constant__ BwdArgs a) {
    constexpr int S = kBStages;
    using R = BRaw<T>;
    using SM = BSmem<T>;
    // every TMA source or destination starts on a 128-byte boundary
    static_assert(sizeof(R) % 128 == 0 && offsetof(R, x) % 128 == 0 && offsetof(R, z) % 128 == 0 &&
                      offsetof(R, dout) % 128 == 0 && offsetof(R, B) % 128 == 0 && offsetof(R, C) % 128 == 0 &&
                      offsetof(SM, raw) % 128 == 0 && offsetof(SM, gx) % 128 == 0 &&
                      offsetof(SM, gdt) % 128 == 0 && offsetof(SM, gz) % 128 == 0,
                  "TMA tiles must be 128-byte aligned");
    extern __shared__ unsigned char smem_dyn[];
    BSmem<T> &s = smem_aligned<BSmem<T>>(smem_dyn);
    const ScanParams &p = a.p;
    const GradParams &gp = a.g;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ntd = (int)((p.d_inner + kBCh - 1) / kBCh);
    const int b = blockIdx.x / ntd;
    const int d0 = (blockIdx.x % ntd) * kBCh;
    const int64_t L = p.seqlen, D = p.d_inner;
    const int64_t nchunks = (L + kBT - 1) / kBT;   // >= 1: L > 0 here
    const bool gate = a.has_gate != 0;

    if (tid == 0) {
        for (int st = 0; st < S; ++st) mbar_init(&s.full[st], 1);
        fence_mbar_init();
    }
    for (int i = tid; i < kBT * 32; i += kBThreads) (&s.bc[0][0])[i] = 0.f;
    __syncthreads();
    pdl_wait();   // everything below reads or writes global memory
    // ring slot j holds chunk nchunks-1-j (reverse order)
    if (tid == 0)
        for (int j = 0; j < S && j < nchunks; ++j) issue_bchunk(s, a, j, nchunks - 1 - j, d0, b);

    // ---- conversion role: channel pair cp at steps th, th + 8
    const int cp = tid % (kBCh / 2), th = tid / (kBCh / 2);
    const int64_t dc = d0 + 2 * cp;
    const bool cok = dc < D;
    const float2 bias2 = (cok && p.dt_bias) ? __ldg(reinterpret_cast<const float2 *>(p.dt_bias + dc))
                                            : make_float2(0.f, 0.f);

    // ---- scan role: channel c, states 4q .. 4q+3
    const int c8 = lane & 7, q = lane >> 3;
    const int c = warp * 8 + c8;
    const int64_t d = d0 + c;
    const bool chan_ok = d < D;
    float2 a2[2], Ar[2], g[2], dA[2];
    float dsk = 0.f, dtb = 0.f, dD_acc = 0.f, db_acc = 0.f;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        a2[k] = make_float2(0.f, 0.f); Ar[k] = a2[k]; g[k] = a2[k]; dA[k] = a2[k];
    }
    if (chan_ok) {
        const float4 av = __ldg(reinterpret_cast<const float4 *>(p.A + d * kDState + 4 * q));
        Ar[0] = make_float2(av.x, av.y);
        Ar[1] = make_float2(av.z, av.w);
        a2[0] = make_float2(av.x * kLog2e, av.y * kLog2e);
        a2[1] = make_float2(av.z * kLog2e, av.w * kLog2e);
        dsk = p.D ? __ldg(p.D + d) : 0.f;
        dtb = p.dt_bias ? __ldg(p.dt_bias + d) : 0.f;
        if (gp.dh_last) {
            const float4 gv = __ldg(reinterpret_cast<const float4 *>(gp.dh_last + ((int64_t)b * D + d) * kDState + 4 * q));
            g[0] = make_float2(gv.x, gv.y);
            g[1] = make_float2(gv.z, gv.w);
        }
    }

    // checkpoint of chunk i, loaded one iteration ahead (its latency overlaps
    // the previous chunk's sweep)
    auto load_ckpt = [&](int64_t i) {
        return chan_ok ? __ldg(reinterpret_cast<const float4 *>(
                             gp.h_ckpt + (((int64_t)b * nchunks + i) * D + d) * kDState + 4 * q))
                       : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    float4 ck_next = load_ckpt(nchunks - 1);

    bool ok = true;
    for (int64_t j = 0; j < nchunks; ++j) {
        const int64_t i = nchunks - 1 - j;   // chunk of this iteration
        const int64_t t0 = i * kBT;
        // (1) wait for chunk i's tiles and convert them; dB, dC of chunk i + 1
        ok = mbar_wait(&s.full[j % S], (uint32_t)((j / S) & 1));
        if (ok) bconvert(s.cv, s.raw[j % S], cp, th, bias2, cok, t0, L, gate);
        if (j >= 1) flush_bc(s.bc, gp, b, t0 + kBT, L);
        if (__syncthreads_or(ok ? 0 : 1)) {
            if (tid == 0) {
                report(p.status, 4 /* MB_ERR_TIMEOUT */, j);
                int64_t last = j + S - 1;   // ring slots issued so far: 0 .. j+S-1
                if (last > nchunks - 1) last = nchunks - 1;
                for (int64_t jj = j; jj <= last; ++jj)
                    mbar_wait(&s.full[jj % S], (uint32_t)((jj / S) & 1));
                bulk_wait_all();
            }
            return;
        }

        // (2) chunk i
        const BConv<sizeof(T) == 2> &cv = s.cv;
        const BRaw<T> &rs = s.raw[j % S];
        const float2 hc[2] = {make_float2(ck_next.x, ck_next.y), make_float2(ck_next.z, ck_next.w)};
        if (i > 0) ck_next = load_ckpt(i - 1);
        // recompute the chunk's forward states (same arithmetic as the forward)
        float4(&hs)[kBT / 2][kBThreads] = s.hs;
        float yv[kBT / 4];   // lane q: share-summed y of step 4m + q
        {
            float2 h0v = hc[0], h1v = hc[1];
            float part[4];
#pragma unroll
            for (int t = 0; t < kBT; ++t) {
                const float2 av = cv.dg[t][c];
                const float2 dd = make_float2(av.x, av.x), gg = make_float2(av.y, av.y);
                const float2 e0 = mul2(dd, a2[0]), e1 = mul2(dd, a2[1]);
                float4 b4, c4;
                load_bc(cv, rs, t, q, b4, c4);
                h0v = fma2(make_float2(ex2(e0.x), ex2(e0.y)), h0v, mul2(make_float2(b4.x, b4.y), gg));
                h1v = fma2(make_float2(ex2(e1.x), ex2(e1.y)), h1v, mul2(make_float2(b4.z, b4.w), gg));
                if ((t & 1) == 0) hs[t / 2][tid] = make_float4(h0v.x, h0v.y, h1v.x, h1v.y);
                const float2 acc = fma2(make_float2(c4.z, c4.w), h1v, mul2(make_float2(c4.x, c4.y), h0v));
                part[t & 3] = acc.x + acc.y;
                if ((t & 3) == 3) yv[t >> 2] = reduce4(part[0], part[1], part[2], part[3], q);
            }
        }
        // reverse sweep over the chunk. Only the even steps' states were kept:
        // an odd step's state is one recurrence step from the even state below
        // it, with that step's decay and inputs, which the sweep forms anyway
        // (one step ahead), so the result is bit for bit the recompute's.
        float (&bcs)[kBT][32] = s.bc;
        float s1[4], s2[4];
        struct StepVals {
            float2 dd, gx, ab0, ab1;
            float4 b4, c4;
            float dyv;
        };
        auto stepvals = [&](int t) {
            StepVals v;
            const float2 av = cv.dg[t][c];   // (Delta, Delta*x)
            v.dd = make_float2(av.x, av.x);
            v.gx = make_float2(av.y, av.y);
            v.dyv = cv.dy[t][c];
            const float2 e0 = mul2(v.dd, a2[0]), e1 = mul2(v.dd, a2[1]);
            v.ab0 = make_float2(ex2(e0.x), ex2(e0.y));
            v.ab1 = make_float2(ex2(e1.x), ex2(e1.y));
            load_bc(cv, rs, t, q, v.b4, v.c4);
            return v;
        };
        auto advance = [&](const StepVals &v, float4 hp) {   // the forward step from hp
            const float2 n0 = fma2(v.ab0, make_float2(hp.x, hp.y), mul2(make_float2(v.b4.x, v.b4.y), v.gx));
            const float2 n1 = fma2(v.ab1, make_float2(hp.z, hp.w), mul2(make_float2(v.b4.z, v.b4.w), v.gx));
            return make_float4(n0.x, n0.y, n1.x, n1.y);
        };
        StepVals cur = stepvals(kBT - 1);
        float4 heven = hs[kBT / 2 - 1][tid];   // h_{kBT-2}
        float4 hcur = advance(cur, heven);     // h_{kBT-1}
#pragma unroll
        for (int t = kBT - 1; t >= 0; --t) {
            const float2 dd = cur.dd, gx = cur.gx;
            const float2 dy = make_float2(cur.dyv, cur.dyv);
            const float2 ab0 = cur.ab0, ab1 = cur.ab1;
            const float4 b4 = cur.b4, c4 = cur.c4;
            float4 hprev;
            StepVals nxt = cur;
            if (t == 0) {
                hprev = make_float4(hc[0].x, hc[0].y, hc[1].x, hc[1].y);
            } else if (t & 1) {
                hprev = heven;                   // h_{t-1}, even: kept
                nxt = stepvals(t - 1);
            } else {
                nxt = stepvals(t - 1);
                heven = hs[t / 2 - 1][tid];      // h_{t-2}
                hprev = advance(nxt, heven);     // h_{t-1}, odd
            }
            const float2 hp0 = make_float2(hprev.x, hprev.y), hp1 = make_float2(hprev.z, hprev.w);
            const float2 ht0 = make_float2(hcur.x, hcur.y), ht1 = make_float2(hcur.z, hcur.w);
            hcur = hprev;
            cur = nxt;
            g[0] = fma2(dy, make_float2(c4.x, c4.y), g[0]);
            g[1] = fma2(dy, make_float2(c4.z, c4.w), g[1]);
            const float2 dc0 = mul2(dy, ht0), dc1 = mul2(dy, ht1);
            const float2 sb = fma2(g[1], make_float2(b4.z, b4.w), mul2(g[0], make_float2(b4.x, b4.y)));
            const float2 db0 = mul2(g[0], gx), db1 = mul2(g[1], gx);
            const float2 ga0 = mul2(g[0], ab0), ga1 = mul2(g[1], ab1);
            const float2 w0 = mul2(ga0, hp0), w1 = mul2(ga1, hp1);
            const float2 sa = fma2(w1, Ar[1], mul2(w0, Ar[0]));
            dA[0] = fma2(w0, dd, dA[0]);
            dA[1] = fma2(w1, dd, dA[1]);
            g[0] = ga0;
            g[1] = ga1;
            s1[t & 3] = sb.x + sb.y;
            s2[t & 3] = sa.x + sa.y;
            const float v8[8] = {db0.x, db0.y, db1.x, db1.y, dc0.x, dc0.y, dc1.x, dc1.y};
            atomicAdd(&bcs[t][lane], reduce8(v8, c8));   // the 4 warps' shares
            if ((t & 3) == 0) {   // steps t .. t+3 done: finish step t + q on this lane
                const float S1 = reduce4(s1[0], s1[1], s1[2], s1[3], q);
                const float S2 = reduce4(s2[0], s2[1], s2[2], s2[3], q);
                const int tq = t + q;
                const bool live = chan_ok && t0 + tq < L;
                const float delta = cv.dg[tq][c].x, dyq = cv.dy[tq][c];
                const float xq = live ? to_f32(rs.x[tq][c]) : 0.f;
                const float sig = live ? sigmoid_v(to_f32(rs.dt[tq][c]) + dtb) : 0.f;
                float qz = 0.f;
                if (gate && live) {
                    const float zt = to_f32(rs.z[tq][c]);
                    const float sz = __fdividef(1.f, 1.f + ex2(-zt * kLog2e));
                    qz = to_f32(rs.dout[tq][c]) * sz * fmaf(zt, 1.f - sz, 1.f);
                }
                const float dx = fmaf(delta, S1, dyq * dsk);
                const float ddt = fmaf(xq, S1, S2) * sig;
                const float y = fmaf(dsk, xq, yv[t >> 2]);
                dD_acc = fmaf(dyq, xq, dD_acc);
                db_acc += ddt;
                store_out(s.gx, tq, c, dx);
                store_out(s.gdt, tq, c, ddt);
                if (gate) store_out(s.gz, tq, c, y * qz);
            }
        }
        fence_proxy_async_smem();   // output tiles -> visible to the TMA stores
        __syncthreads();
        if (tid == 0) {
            tma_store_3d(&a.tm_dx, &s.gx[0][0], d0, (int)t0, b);
            tma_store_3d(&a.tm_ddt, &s.gdt[0][0], d0, (int)t0, b);
            if (gate) tma_store_3d(&a.tm_dz, &s.gz[0][0], d0, (int)t0, b);
            bulk_commit();
            // slot j (chunk i) is converted and consumed: refill it with the
            // chunk of slot j + S
            if (j + S < nchunks) {
                fence_proxy_async_smem();
                issue_bchunk(s, a, (int)(j % S), nchunks - 1 - (j + S), d0, b);
            }
            // the output tiles are rewritten after the next conversion
            // barrier: wait until these stores have read them
            bulk_wait_read_all();
        }
    }
    // dB, dC of chunk 0
    flush_bc(s.bc, gp, b, 0, L);

    // per-channel sums: dD, dbias over the 4 lanes of the channel
    dD_acc += __shfl_xor_sync(kFull, dD_acc, 8);
    dD_acc += __shfl_xor_sync(kFull, dD_acc, 16);
    db_acc += __shfl_xor_sync(kFull, db_acc, 8);
    db_acc += __shfl_xor_sync(kFull, db_acc, 16);
    if (chan_ok) {
        atomicAdd(reinterpret_cast<float4 *>(gp.dA + d * kDState + 4 * q),
                  make_float4(dA[0].x, dA[0].y, dA[1].x, dA[1].y));
        if (gp.dh0)
            *reinterpret_cast<float4 *>(gp.dh0 + ((int64_t)b * D + d) * kDState + 4 * q) =
                make_float4(g[0].x, g[0].y, g[1].x, g[1].y);
        if (q == 0) {
            if (gp.dD) atomicAdd(gp.dD + d, dD_acc);
            if (gp.ddt_bias) atomicAdd(gp.ddt_bias + d, db_acc);
        }
    }
    if (tid == 0) bulk_wait_all();
}

bool make_map3(CUtensorMap *m, const void *base, bool bf16, int64_t batch, int64_t L, int64_t inner,
               int box_inner, int64_t row = 0) {
    const int64_t es = bf16 ? 2 : 4;
    if (row == 0) row = inner;
    const uint64_t dims[3] = {(uint64_t)inner, (uint64_t)L, (uint64_t)batch};
    const uint64_t strides[2] = {(uint64_t)(row * es), (uint64_t)(L * row * es)};
    const uint32_t box[3] = {(uint32_t)box_inner, (uint32_t)kBT, 1};
    return encode_tmap(m, base, (int)es, 3, dims, strides, box);
}

template <typename T>
cudaError_t launch_backward_typed(const ScanParams &p, const GradParams &g, cudaStream_t s) {
    const bool bf16 = sizeof(T) == 2;
    BwdArgs a;
    memset(&a, 0, sizeof(a));
    a.p = p;
    a.g = g;
    a.has_gate = p.z != nullptr;
    const int64_t Bn = p.batch, L = p.seqlen, D = p.d_inner;
    if (!make_map3(&a.tm_dt, p.dt, bf16, Bn, L, D, kBCh) || !make_map3(&a.tm_x, p.x, bf16, Bn, L, D, kBCh) ||
        (p.z && !make_map3(&a.tm_z, p.z, bf16, Bn, L, D, kBCh)) ||
        !make_map3(&a.tm_dout, g.dout, bf16, Bn, L, D, kBCh) ||
        !make_map3(&a.tm_B, p.B, bf16, Bn, L, kDState, kDState, p.bc_stride) ||
        !make_map3(&a.tm_C, p.C, bf16, Bn, L, kDState, kDState, p.bc_stride) ||
        !make_map3(&a.tm_dx, g.dx, bf16, Bn, L, D, kBCh) || !make_map3(&a.tm_ddt, g.ddt, bf16, Bn, L, D, kBCh) ||
        (p.z && !make_map3(&a.tm_dz, g.dz, bf16, Bn, L, D, kBCh)))
        return cudaErrorInvalidValue;
    const size_t smem = sizeof(BSmem<T>) + 128;
    auto k = backward_kernel<T>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid((unsigned)(((D + kBCh - 1) / kBCh) * Bn));
    e = launch_pdl(false, k, grid, dim3(kBThreads), smem, s, a);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_backward(const ScanParams &p, const GradParams &g, bool bf16, cudaStream_t s) {
    const int64_t Bn = p.batch, L = p.seqlen, D = p.d_inner;
    // The sums are accumulated atomically: clear them first.
    cudaError_t e;
    if (Bn * L > 0) {
        if ((e = cudaMemsetAsync(g.dB, 0, (size_t)(Bn * L * kDState) * 4, s)) != cudaSuccess) return e;
        if ((e = cudaMemsetAsync(g.dC, 0, (size_t)(Bn * L * kDState) * 4, s)) != cudaSuccess) return e;
    }
    if (D > 0) {
        if ((e = cudaMemsetAsync(g.dA, 0, (size_t)(D * kDState) * 4, s)) != cudaSuccess) return e;
        if (g.dD && (e = cudaMemsetAsync(g.dD, 0, (size_t)D * 4, s)) != cudaSuccess) return e;
        if (g.ddt_bias && (e = cudaMemsetAsync(g.ddt_bias, 0, (size_t)D * 4, s)) != cudaSuccess) return e;
    }
    if (Bn == 0 || D == 0) return cudaSuccess;
    if (L == 0) {   // nothing to scan: dJ/dh0 = dJ/dh_last
        if (!g.dh0) return cudaSuccess;
        const size_t bytes = (size_t)(Bn * D * kDState) * 4;
        if (g.dh_last) return cudaMemcpyAsync(g.dh0, g.dh_last, bytes, cudaMemcpyDeviceToDevice, s);
        return cudaMemsetAsync(g.dh0, 0, bytes, s);
    }
    return bf16 ? launch_backward_typed<__nv_bfloat16>(p, g, s) : launch_backward_typed<float>(p, g, s);
}

}  // namespace mbscan
