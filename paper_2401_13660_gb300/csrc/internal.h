// Internal launcher interface between the C ABI (mbscan_api.cu) and the
// kernels. Plain C++ structs of device pointers and sizes; no torch types.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mbscan {

// Layout of the workspace status block (first bytes of `ws`).
struct StatusBlock {
    int code;        // 0 = ok, else an mb_status value
    int pad;
    long long detail;  // error-specific (first bad stream, ...), -1 when unset
};
constexpr size_t kStatusBytes = 256;

// One selective-scan problem, validated by the API layer.
struct ScanParams {
    int64_t batch, seqlen, d_inner;  // d_state is fixed to 16
    const void *x, *z, *dt, *B, *C;
    int64_t bc_stride;   // elements between consecutive (b, t) rows of B and C (>= 16)
    const float *A, *D, *dt_bias, *h0;
    void *y;
    float *h_out;      // prefill: h_last (may be null); verify: h_all; step: state
    StatusBlock *status;
    float *h_ckpt;     // prefill with checkpoints: state before every kCkptSteps-step chunk
    // Fused low-rank Delta projection (Eq. 3): when dt_low is set (dt is then
    // null), dt[b, t, d] = sum_k dt_low[b, t, k] * W_dt[d, k], k < dt_rank.
    const void *dt_low;        // [batch, seqlen, dt_rank], rows dt_low_stride elements apart (bf16)
    const void *W_dt;          // [d_inner, dt_rank] (bf16)
    int64_t dt_rank, dt_low_stride;
    // Resume (verify after a bifurcation): when accept is set, row b starts
    // from h0[b] (zeros if null) for accept[b] == 0, else from
    // h_prev_all[b, accept[b] - 1] ([batch, k_prev, d_inner, 16]).
    const float *h_prev_all;
    const int32_t *accept;
    int64_t k_prev;
    // Time split of a prefill over nseg segments of L (1: not split): seg_h,
    // seg_p [batch, nseg, d_inner, 16] hold each segment's end state from a
    // zero start and the product of its decays (scratch in the workspace).
    int64_t nseg;
    float *seg_h, *seg_p;
};

constexpr int kRankTile = 64;    // dt_rank elements per 128-byte swizzled TMA box
constexpr int kMaxRank = 256;

constexpr int kDState = 16;
constexpr int kCkptSteps = 16;   // steps between the state checkpoints of the training forward

// Encode a tiled TMA tensor map over `base` (bf16 when elem_bytes == 2, else
// fp32): dims innermost first, strides[i] = byte stride of dimension i + 1,
// box = tile extent per dimension. Out-of-range elements load as zeros.
// swizzle: 0 (rows stored as they are), 64 or 128: rows of the box (that
// many bytes) stored with that swizzle, 16-byte chunk j of row i at chunk
// j ^ (i % 8) for 128 (destination 1024-byte aligned), j ^ ((i / 2) % 4) for
// 64 (destination 512-byte aligned).
bool encode_tmap(CUtensorMap *m, const void *base, int elem_bytes, int rank, const uint64_t *dims,
                 const uint64_t *strides, const uint32_t *box, int swizzle = 0);

constexpr long long kMaxWaitCycles = 4000000000LL;   // the kernels' wait limit (~2 s at 2 GHz)

// Launchers: return the cudaError_t of the launch.
// Bounded-wait diagnostic (selftest.cu): a wait that runs out after `limit` clocks.
cudaError_t launch_wait_timeout(StatusBlock *sb, long long limit, cudaStream_t s);
cudaError_t launch_prefill(const ScanParams &p, bool bf16, cudaStream_t s);
// Segments a prefill of these sizes is split into when the workspace has room
// (1 when the batch rows and channels alone fill the GPU), and the scratch
// bytes that split needs beyond the status block.
int64_t prefill_segments(const ScanParams &p, bool bf16);
size_t prefill_split_bytes(const ScanParams &p, int64_t nseg);
cudaError_t launch_verify(const ScanParams &p, bool bf16, cudaStream_t s);
// Prefill that also writes p.h_ckpt [batch, ceil(L / kCkptSteps), d_inner, 16].
cudaError_t launch_prefill_ckpt(const ScanParams &p, bool bf16, cudaStream_t s);
// Backward of the layer core (backward.cu).
struct GradParams {
    const float *h_ckpt;          // [batch, nchunks, d_inner, 16] from launch_prefill_ckpt
    const void *dout;             // [batch, L, d_inner], input dtype
    const float *dh_last;         // [batch, d_inner, 16] or null
    void *dx, *dz, *ddt;          // [batch, L, d_inner], input dtype (dz null without a gate)
    float *dB, *dC;               // [batch, L, 16]
    float *dA;                    // [d_inner, 16]
    float *dD, *ddt_bias;         // [d_inner] or null
    float *dh0;                   // [batch, d_inner, 16] or null
};
cudaError_t launch_backward(const ScanParams &p, const GradParams &g, bool bf16, cudaStream_t s);
// Block steps around the scan (block.cu).
cudaError_t launch_rmsnorm(const void *add, float *residual, const float *w, float eps, void *out,
                           int64_t batch, int64_t width, bool bf16, cudaStream_t s);
cudaError_t launch_conv_step(const void *x, void *state, const float *w, const float *bias, void *out,
                             int64_t batch, int64_t width, bool bf16, cudaStream_t s);
// Decode-step convolution fused with the x-projection (xproj.cu): supported
// widths and output widths, the fp32 partial-sum scratch it needs, the launch.
bool conv_xproj_supported(int64_t width, int n_out);
size_t conv_xproj_partial_bytes(int64_t batch, int64_t width, int n_out);
cudaError_t launch_conv_xproj(const void *x, void *state, const float *w, const float *bias, const void *W,
                              void *xc, void *out, int64_t batch, int64_t width, int n_out, float *part,
                              StatusBlock *status, cudaStream_t s);
cudaError_t launch_step(const ScanParams &p, bool bf16, cudaStream_t s);
// One step from the state kept after accept[s] drafted bytes: p.h0 (may be
// null = zeros) when accept[s] == 0, else h_all[s, accept[s]-1]; the new state
// goes to p.h_out (may alias p.h0).
cudaError_t launch_step_resume(const ScanParams &p, bool bf16, const float *h_all,
                               const int32_t *accept, int64_t k, cudaStream_t s);
cudaError_t launch_accept(const void *logits, bool bf16, const uint8_t *drafted, int64_t streams,
                          int64_t k, int beta, int32_t *accept, cudaStream_t s);
cudaError_t launch_rollback(const float *h0, const float *h_all, const int32_t *accept,
                            float *h_out, int64_t batch, int64_t k, int64_t d_inner,
                            StatusBlock *status, cudaStream_t s);

}  // namespace mbscan
