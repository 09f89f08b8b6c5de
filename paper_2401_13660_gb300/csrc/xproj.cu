// Decode-step convolution and x-projection of the Mamba block, fused
// (MambaByte Figure 6; Table 6 rows "Pre-SSM 1D convolution" and "Delta, B, C
// from input x"), for recurrent generation of a whole model:
//
//   xc[b, d]  = silu(w[d,0] s[b,0,d] + w[d,1] s[b,1,d] + w[d,2] s[b,2,d] + w[d,3] x[b,d] + bias[d])
//   window    : s[b,0] <- s[b,1], s[b,1] <- s[b,2], s[b,2] <- x[b]
//   out[b, n] = sum_d xc[b, d] W[n, d]        ([dt_low | B | C] = xc W_xproj^T)
//
// At decode batch sizes the projection is a narrow GEMM (n_out = dt_rank + 32
// columns, 176 for d_model 2304) over a long K (d_inner = 4608). The work is
// split over K: CTA (m, s) owns batch rows 64 m .. 64 m + 63 and channels
// 128 s .. 128 s + 127. One thread issues all of its global traffic as TMA
// copies at the start: the x tile, the three window tiles and the matching
// 128 columns of W (two 64-column boxes, 128-byte swizzle); the window and W
// tiles, which the preceding input GEMM does not produce, are first prefetched
// into L2 while that kernel drains (programmatic dependent launch). As soon as x and
// the window have landed, the shifted window goes back out as three TMA
// stores of the tiles just loaded (s1, s2, x), while the threads compute the
// convolution step from shared memory into the A operand (bf16, the same
// 128-byte swizzle), which a TMA store also writes out as xc. Four warps then
// multiply their 16 rows by all n_out columns with mma.sync m16n8k16 (bf16
// operands, fp32 accumulation) and store fp32 partial sums; a second kernel
// adds the K splits in a fixed order and rounds to bf16. Rows past the batch
// load as zeros and are never stored.
#include <string.h>

#include "common.cuh"
#include "tma.cuh"

namespace mbscan {
namespace {

constexpr int kXpRows = 64;       // batch rows per CTA (4 warps x 16)
constexpr int kXpK = 128;         // channels per CTA (the K split)
constexpr int kXpThreads = 128;
constexpr uint32_t kXpABox = kXpRows * 128;      // one 64-channel box of A: 64 rows of 128 bytes
constexpr uint32_t kXpTile = kXpRows * kXpK * 2;  // one [64 rows][128 channels] bf16 tile

struct XpArgs {
    CUtensorMap tm_w;            // W [n_out, width]: boxes {64 columns, n_out rows}, 128-byte swizzle
    CUtensorMap tm_x;            // x [batch, width]: boxes {128, 64}
    CUtensorMap tm_s;            // window [batch, 3, width]: boxes {128, 1, 64}
    CUtensorMap tm_xc;           // xc [batch, width]: boxes {64, 64}, 128-byte swizzle
    const float *cw, *cb;        // [width, 4]; [width] or null
    float *part;                 // [splits, batch, n_out]
    StatusBlock *status;
    int64_t batch;
};

// Byte offset of 16-byte chunk `chunk` of row `row` in a 128-byte-swizzled box
// (the layout TMA writes and reads for such a box at a 1024-byte boundary).
__device__ __forceinline__ uint32_t xswz(int row, int chunk) {
    return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ void unpack8(const uint4 u, float (&v)[8]) {
    const unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        v[2 * j] = __uint_as_float(w[j] << 16);
        v[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
}

template <int NT>   // n_out = 8 NT output columns
__global__ void __launch_bounds__(kXpThreads) conv_xproj_kernel(const __grid_constant__ XpArgs a) {
    constexpr int kNOut = 8 * NT;
    constexpr uint32_t kBBox = kNOut * 128;   // one 64-column box of W
    extern __shared__ unsigned char smem_dyn[];
    const uint32_t sbase = smem_u32(smem_dyn);
    unsigned char *As = smem_dyn + (((sbase + 1023u) & ~1023u) - sbase);   // the swizzled boxes want 1024 B
    unsigned char *Bs = As + 2 * kXpABox;
    unsigned char *Xs = Bs + 2 * kBBox;
    unsigned char *Ss = Xs + kXpTile;                                        // s0, s1, s2
    uint64_t *bar = reinterpret_cast<uint64_t *>(Ss + 3 * kXpTile);         // [0] x and window, [1] W
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int r0 = (int)(blockIdx.x * kXpRows), k0 = (int)(blockIdx.y * kXpK);
    if (tid == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (tid == 0) {   // the window and W tiles into L2 while the previous kernel (the input GEMM) drains
#pragma unroll
        for (int j = 0; j < 3; ++j) tma_prefetch_3d(&a.tm_s, k0, j, r0);
        tma_prefetch_2d(&a.tm_w, k0, 0);
        tma_prefetch_2d(&a.tm_w, k0 + 64, 0);
    }
    pdl_wait();   // everything below reads or writes global memory
    if (tid == 0) {
        mbar_arrive_expect_tx(&bar[0], 4 * kXpTile);
        tma_load_2d(Xs, &a.tm_x, &bar[0], k0, r0);
#pragma unroll
        for (int j = 0; j < 3; ++j) tma_load_3d(Ss + j * kXpTile, &a.tm_s, &bar[0], k0, j, r0);
        mbar_arrive_expect_tx(&bar[1], 2 * kBBox);
        tma_load_2d(Bs, &a.tm_w, &bar[1], k0, 0);
        tma_load_2d(Bs + kBBox, &a.tm_w, &bar[1], k0 + 64, 0);
    }
    pdl_trigger();   // one wave: the reduction's CTAs may take the SM slots this grid leaves free
    // the convolution weights of this thread's 8 channels (group g), loaded while the tiles land
    const int g = tid & 15;
    const int kc = k0 + 8 * g;
    float4 wj[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) wj[j] = __ldg(reinterpret_cast<const float4 *>(a.cw + (int64_t)(kc + j) * 4));
    float bv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (a.cb) {
        const float4 b0 = __ldg(reinterpret_cast<const float4 *>(a.cb + kc));
        const float4 b1 = __ldg(reinterpret_cast<const float4 *>(a.cb + kc) + 1);
        bv[0] = b0.x; bv[1] = b0.y; bv[2] = b0.z; bv[3] = b0.w;
        bv[4] = b1.x; bv[5] = b1.y; bv[6] = b1.z; bv[7] = b1.w;
    }
    if (!__syncthreads_and(mbar_wait(&bar[0], 0))) {
        if (tid == 0) {
            report(a.status, 4 /* MB_ERR_TIMEOUT */, blockIdx.y);
            mbar_wait(&bar[0], 0);   // copies may still be landing: wait (bounded) before leaving
            mbar_wait(&bar[1], 0);
        }
        return;
    }
    if (tid == 0) {   // the shifted window, straight from the tiles just loaded
        tma_store_3d(&a.tm_s, Ss + kXpTile, k0, 0, r0);
        tma_store_3d(&a.tm_s, Ss + 2 * kXpTile, k0, 1, r0);
        tma_store_3d(&a.tm_s, Xs, k0, 2, r0);
        bulk_commit();
    }

    // ---- the convolution step of channels kc .. kc + 7 for rows tid / 16 + 8 i,
    // i = 0..7, from shared memory; the same arithmetic as mb_conv1d_step
    {
        const int box = g >> 3, chunk = g & 7;
#pragma unroll 2
        for (int i = 0; i < kXpRows / 8; ++i) {
            const int r = (tid >> 4) + 8 * i;
            const uint32_t off = (uint32_t)(r * kXpK * 2 + 16 * g);
            float xv[8], s0[8], s1[8], s2[8];
            unpack8(*reinterpret_cast<const uint4 *>(Xs + off), xv);
            unpack8(*reinterpret_cast<const uint4 *>(Ss + off), s0);
            unpack8(*reinterpret_cast<const uint4 *>(Ss + kXpTile + off), s1);
            unpack8(*reinterpret_cast<const uint4 *>(Ss + 2 * kXpTile + off), s2);
            unsigned w[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float o[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int e = 2 * j + h;
                    float acc = bv[e];
                    acc = fmaf(wj[e].x, s0[e], acc);
                    acc = fmaf(wj[e].y, s1[e], acc);
                    acc = fmaf(wj[e].z, s2[e], acc);
                    acc = fmaf(wj[e].w, xv[e], acc);
                    o[h] = silu(acc);
                }
                const __nv_bfloat162 hb = __floats2bfloat162_rn(o[0], o[1]);
                w[j] = *reinterpret_cast<const unsigned *>(&hb);
            }
            *reinterpret_cast<uint4 *>(As + box * kXpABox + xswz(r, chunk)) = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
    fence_proxy_async_smem();   // the A tile -> visible to the TMA store of xc
    __syncthreads();
    if (tid == 0) {
        tma_store_2d(&a.tm_xc, As, k0, r0);
        tma_store_2d(&a.tm_xc, As + kXpABox, k0 + 64, r0);
        bulk_commit();
    }
    if (!__syncthreads_and(mbar_wait(&bar[1], 0))) {
        if (tid == 0) {
            report(a.status, 4 /* MB_ERR_TIMEOUT */, blockIdx.y);
            mbar_wait(&bar[1], 0);
            bulk_wait_all();
        }
        return;
    }

    // ---- warp w: rows 16 w .. 16 w + 15 of the tile, all n_out columns. The
    // operand addresses derive from a token taken after the waits above.
    const uint32_t tok = order_token();
    float acc[NT][4];
#pragma unroll
    for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    const uint32_t aaddr = smem_u32(As) + tok, baddr = smem_u32(Bs) + tok;
    const int arow = 16 * warp + (lane & 15), achunk = lane >> 4;
    const int brow = lane & 7, bchunk = (lane >> 3) & 1;
#pragma unroll
    for (int ks = 0; ks < kXpK / 16; ++ks) {
        const int bx = ks >> 2, c0 = (ks & 3) * 2;
        uint32_t af[4];
        ldsm_x4(aaddr + bx * kXpABox + xswz(arow, c0 + achunk), af);
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            uint32_t bf[2];
            ldsm_x2(baddr + bx * kBBox + xswz(8 * j + brow, c0 + bchunk), bf);
            mma_bf16_16816(acc[j], af, bf);
        }
    }
    // ---- fp32 partial sums of this K split: rows lane / 4 and lane / 4 + 8
    const int64_t ra = (int64_t)r0 + 16 * warp + (lane >> 2), rb = ra + 8;
    float *pbase = a.part + (int64_t)blockIdx.y * a.batch * kNOut;
#pragma unroll
    for (int j = 0; j < NT; ++j) {
        const int col = 8 * j + 2 * (lane & 3);
        if (ra < a.batch) *reinterpret_cast<float2 *>(pbase + ra * kNOut + col) = make_float2(acc[j][0], acc[j][1]);
        if (rb < a.batch) *reinterpret_cast<float2 *>(pbase + rb * kNOut + col) = make_float2(acc[j][2], acc[j][3]);
    }
    if (tid == 0) bulk_wait_read_all();   // the window and xc tiles stay valid until the stores have read them
}

// out = sum over the K splits of the partial sums, rounded to bf16. Block:
// 64 groups of four adjacent outputs x 4 interleaved subsets of the splits
// (subset q sums splits q, q + 4, ... in order); the four subset sums are then
// added in order q = 0..3, so the result does not depend on timing.
constexpr int kRedQuads = 64, kRedSub = 4, kRedThreads = kRedQuads * kRedSub;
__global__ void __launch_bounds__(kRedThreads) xproj_reduce_kernel(const float *__restrict__ part,
                                                                  __nv_bfloat16 *__restrict__ out,
                                                                  int64_t quads, int splits) {
    __shared__ float4 sub[kRedSub][kRedQuads];
    pdl_wait();
    const int qi = threadIdx.x % kRedQuads, q = threadIdx.x / kRedQuads;
    const int64_t i = (int64_t)blockIdx.x * kRedQuads + qi;
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < quads) {
        const float4 *p = reinterpret_cast<const float4 *>(part) + i;
#pragma unroll 4
        for (int k = q; k < splits; k += kRedSub) {
            const float4 v = __ldg(p + (int64_t)k * quads);
            s.x += v.x;
            s.y += v.y;
            s.z += v.z;
            s.w += v.w;
        }
    }
    sub[q][qi] = s;
    __syncthreads();
    if (q != 0 || i >= quads) return;
#pragma unroll
    for (int k = 1; k < kRedSub; ++k) {
        const float4 v = sub[k][qi];
        s.x += v.x;
        s.y += v.y;
        s.z += v.z;
        s.w += v.w;
    }
    const __nv_bfloat162 lo = __floats2bfloat162_rn(s.x, s.y), hi = __floats2bfloat162_rn(s.z, s.w);
    uint2 u;
    u.x = *reinterpret_cast<const unsigned *>(&lo);
    u.y = *reinterpret_cast<const unsigned *>(&hi);
    reinterpret_cast<uint2 *>(out)[i] = u;
}

template <int NT>
cudaError_t launch_xp(XpArgs &a, const void *x, void *state, const void *W, void *xc, __nv_bfloat16 *out,
                      int64_t width, cudaStream_t s) {
    constexpr int kNOut = 8 * NT;
    const uint64_t rs = (uint64_t)width * 2;
    {
        const uint64_t dims[2] = {(uint64_t)width, (uint64_t)kNOut}, strides[1] = {rs};
        const uint32_t box[2] = {64, (uint32_t)kNOut};
        if (!encode_tmap(&a.tm_w, W, 2, 2, dims, strides, box, 128)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[2] = {(uint64_t)width, (uint64_t)a.batch}, strides[1] = {rs};
        const uint32_t box[2] = {(uint32_t)kXpK, (uint32_t)kXpRows}, box_xc[2] = {64, (uint32_t)kXpRows};
        if (!encode_tmap(&a.tm_x, x, 2, 2, dims, strides, box, 0)) return cudaErrorInvalidValue;
        if (!encode_tmap(&a.tm_xc, xc, 2, 2, dims, strides, box_xc, 128)) return cudaErrorInvalidValue;
    }
    {
        const uint64_t dims[3] = {(uint64_t)width, 3, (uint64_t)a.batch}, strides[2] = {rs, 3 * rs};
        const uint32_t box[3] = {(uint32_t)kXpK, 1, (uint32_t)kXpRows};
        if (!encode_tmap(&a.tm_s, state, 2, 3, dims, strides, box, 0)) return cudaErrorInvalidValue;
    }
    const size_t smem = 1024 + 2 * kXpABox + 2 * (size_t)kNOut * 128 + 4 * (size_t)kXpTile + 16;
    auto k = conv_xproj_kernel<NT>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int splits = (int)(width / kXpK);
    const dim3 grid((unsigned)((a.batch + kXpRows - 1) / kXpRows), (unsigned)splits);
    if ((e = launch_pdl(true, k, grid, dim3(kXpThreads), smem, s, a)) != cudaSuccess) return e;
    const int64_t quads = a.batch * kNOut / 4;
    return launch_pdl(true, xproj_reduce_kernel, dim3((unsigned)((quads + kRedQuads - 1) / kRedQuads)),
                      dim3(kRedThreads), 0, s, static_cast<const float *>(a.part), out, quads, splits);
}

}  // namespace

bool conv_xproj_supported(int64_t width, int n_out) {
    if (width <= 0 || width % kXpK != 0 || width / kXpK > 65535) return false;
    switch (n_out) {
        case 40: case 96: case 144: case 176: return true;
        default: return false;
    }
}

size_t conv_xproj_partial_bytes(int64_t batch, int64_t width, int n_out) {
    return (size_t)(width / kXpK) * (size_t)batch * (size_t)n_out * sizeof(float);
}

cudaError_t launch_conv_xproj(const void *x, void *state, const float *w, const float *bias, const void *W,
                              void *xc, void *out, int64_t batch, int64_t width, int n_out, float *part,
                              StatusBlock *status, cudaStream_t s) {
    if (batch == 0) return cudaSuccess;
    XpArgs a;
    memset(&a, 0, sizeof(a));
    a.cw = w;
    a.cb = bias;
    a.part = part;
    a.status = status;
    a.batch = batch;
    __nv_bfloat16 *o = static_cast<__nv_bfloat16 *>(out);
    switch (n_out) {
        case 40: return launch_xp<5>(a, x, state, W, xc, o, width, s);      // tiny test decoder (dt_rank 8)
        case 96: return launch_xp<12>(a, x, state, W, xc, o, width, s);     // d_model 1024 (dt_rank 64)
        case 144: return launch_xp<18>(a, x, state, W, xc, o, width, s);    // d_model 1792 (dt_rank 112)
        case 176: return launch_xp<22>(a, x, state, W, xc, o, width, s);    // d_model 2304 (dt_rank 144)
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace mbscan
