/*
 * mbscan.h - C ABI of the GB300 selective-scan layer core of MambaByte
 * (arXiv 2401.13660).
 *
 * The layer core is the selective SSM of Section 2 (Eq. 1-3), discretised as
 * in the appendix "Discretization and selection" (zero-order hold for A, the
 * Euler rule Bbar = Delta*B that Mamba uses for B), followed by the output
 * and gating rows of Table 6:
 *
 *   Delta_t = softplus(dt[b,t,d] + dt_bias[d])                   (Eq. 3)
 *   h_t[n]  = exp(Delta_t * A[d,n]) * h_{t-1}[n]
 *             + Delta_t * B[b,t,n] * x[b,t,d]                    (Eq. 2)
 *   y[b,t,d] = (sum_n C[b,t,n] * h_t[n] + D[d] * x[b,t,d]) * silu(z[b,t,d])
 *
 * with one fp32 state vector h[b,d,0..N-1] per (batch row, channel). Every
 * (b, d) channel is independent; the recurrence runs over t.
 *
 * Conventions shared by every entry point:
 *  - All tensor pointers are DEVICE pointers (cudaMalloc / torch CUDA
 *    tensors), row-major and contiguous, 16-byte aligned. The caller owns
 *    every buffer; the library allocates nothing.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream). Every call is asynchronous on that stream.
 *  - Argument errors are detected on the host before any launch and return
 *    MB_ERR_INVALID_ARG or MB_ERR_UNSUPPORTED; nothing is launched then.
 *    A failed launch returns MB_ERR_CUDA.
 *  - Outputs must not alias inputs unless stated.
 *  - Supported today: d_state == 16, dtype MB_F32 or MB_BF16,
 *    d_inner % 8 == 0, batch*seqlen*d_inner <= 2^31.
 */
#ifndef MBSCAN_H
#define MBSCAN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MB_OK = 0,
    MB_ERR_INVALID_ARG = 1,  /* null pointer, bad size, misalignment, aliasing */
    MB_ERR_UNSUPPORTED = 2,  /* valid but not implemented (d_state, dtype)     */
    MB_ERR_CUDA = 3,         /* a CUDA runtime call failed                       */
    MB_ERR_TIMEOUT = 4       /* a bounded device-side wait gave up               */
} mb_status;

typedef enum { MB_F32 = 0, MB_BF16 = 1 } mb_dtype;

/*
 * Arguments of one selective-scan problem (Eq. 2-3 and Table 6).
 *   batch    : independent sequences (>= 0)
 *   seqlen   : time steps L (>= 0); 1 for mb_step
 *   d_inner  : channels D = e * d_model (the SSM's input width)
 *   d_state  : N = n_state, state size per channel (16 in MambaByte)
 *   dtype    : element type of x, z, dt, B, C and y (mb_dtype)
 *   x, z, dt : [batch, seqlen, d_inner], dtype. dt is the pre-softplus
 *              timestep (W_Delta W_R x in Eq. 3). z is the gate input; NULL
 *              means no gate (y = C.h + D x).
 *   B, C     : [batch, seqlen, d_state], dtype (W_B x and W_C x in Eq. 3);
 *              row (b, t) starts bc_stride elements after row (b, t-1)
 *   bc_stride: elements between consecutive (b, t) rows of B and of C; 0
 *              means d_state (contiguous). Otherwise >= d_state with
 *              bc_stride * element size a multiple of 16 bytes: B and C may
 *              then be column blocks of one wider row, e.g. of the
 *              [dt_low | B | C] output of a single x-projection GEMM.
 *   A        : [d_inner, d_state] fp32, the diagonal of A per channel
 *   D        : [d_inner] fp32 skip weight; NULL means 0
 *   dt_bias  : [d_inner] fp32 added to dt before softplus; NULL means 0
 *   h0       : [batch, d_inner, d_state] fp32 initial state; NULL means 0
 *   y        : [batch, seqlen, d_inner], dtype, output
 * Fused low-rank Delta projection (Eq. 3: Delta = softplus(W_Delta (W_R x)),
 * W_Delta of size d_inner x r). Leave dt_low NULL to pass dt itself. When
 * dt_low is not NULL, dt must be NULL and the kernels evaluate
 *     dt[b,t,d] = sum_{k < dt_rank} dt_low[b,t,k] * W_dt[d,k]
 * in fp32 on the tensor cores (bf16 operands, fp32 accumulation; dt is never
 * rounded to the input dtype):
 *   dt_low   : [batch, seqlen, dt_rank], dtype (W_R x); row (b, t) starts
 *              dt_low_stride elements after row (b, t-1), e.g. the first
 *              dt_rank columns of the [dt_low | B | C] x-projection output
 *   W_dt     : [d_inner, dt_rank], dtype, contiguous (W_Delta)
 *   dt_rank  : r; supported: dtype MB_BF16, r % 16 == 0, 64 <= r <= 256
 *              (MB_ERR_UNSUPPORTED otherwise)
 *   dt_low_stride: 0 means dt_rank; otherwise >= dt_rank, a multiple of 8
 * Accepted by mb_scan_prefill and mb_scan_verify; mb_step, mb_step_resume,
 * mb_scan_prefill_ckpt and mb_scan_backward return MB_ERR_UNSUPPORTED (they
 * take dt).
 */
typedef struct {
    int64_t batch, seqlen, d_inner, d_state;
    int32_t dtype;
    int32_t bc_stride;
    const void *x, *z, *dt;
    const void *B, *C;
    const float *A;
    const float *D;
    const float *dt_bias;
    const float *h0;
    void *y;
    const void *dt_low;
    const void *W_dt;
    int32_t dt_rank;
    int32_t dt_low_stride;
} mb_scan_args;

/* Bytes of device workspace to pass with `args`: a 256-byte status block
 * (written by bounded device-side waits), plus, when the batch rows and
 * channels of a long span fill less than half of the GPU, scratch that lets
 * mb_scan_prefill split the span over L (two passes: per-segment summaries,
 * then the scan of every segment from its folded start state; Section 2's
 * associative operator). Any workspace of at least 256 bytes is accepted: a
 * smaller one than this runs such spans unsplit. The caller allocates it
 * (256-byte aligned) and may reuse it across calls on one stream; calls that
 * overlap on the GPU need distinct workspaces. Returns 0 for invalid
 * arguments. */
size_t mb_workspace_size(const mb_scan_args *args);

/*
 * Prefill / training-forward scan (Section 2 "parallel scans": the whole span
 * is available at once). Runs the layer core over all `seqlen` steps of every
 * channel, writes y and, if h_last != NULL, the final state
 * h_last[batch, d_inner, d_state] fp32 (the state MambaByte caches to resume
 * generation). h_last may alias h0.
 *   ws, ws_bytes : workspace of at least 256 bytes (mb_workspace_size(args)
 *                  for the split of long few-channel spans); its status block
 *                  (first 256 bytes) must start zeroed once after allocation
 *                  and is left zeroed by every successful call.
 */
mb_status mb_scan_prefill(const mb_scan_args *args, float *h_last, void *ws, size_t ws_bytes,
                          void *stream);

/*
 * Speculative-decoding verify (Section 3 "Speculative decoding through
 * subword drafting" and Algorithm 1): resume from the cached verifier state
 * h0 and scan the k = args->seqlen drafted bytes of each stream in one call,
 * recording every per-position state:
 *   h_all[b, j, d, n] = state after drafted byte j (j = 0..k-1), fp32,
 *   shape [batch, k, d_inner, d_state]; y as in prefill.
 * h_all must not alias h0.
 */
mb_status mb_scan_verify(const mb_scan_args *args, float *h_all, void *ws, size_t ws_bytes,
                         void *stream);

/*
 * Verify that resumes each stream from the state kept at the previous
 * bifurcation, with no rollback copy in between (Algorithm 1: when the
 * corrector loop adds no byte, the next round starts from h_c, the state
 * after the accepted drafted bytes). Stream s starts from
 *   args->h0[s] (zeros if NULL)      if accept[s] == 0
 *   h_all_prev[s, accept[s]-1]       if 1 <= accept[s] <= k_prev
 * and is then scanned exactly as by mb_scan_verify (y, h_all).
 *   h_all_prev : [batch, k_prev, d_inner, d_state] fp32, the previous
 *                verify's per-position states (must not overlap h_all or y)
 *   accept     : [batch] int32 on the device
 *   ws         : required; an accept count outside [0, k_prev] is recorded
 *                there (read it with mb_check) and that stream's y and h_all
 *                are left untouched.
 */
mb_status mb_scan_verify_resume(const mb_scan_args *args, const float *h_all_prev, const int32_t *accept,
                                int64_t k_prev, float *h_all, void *ws, size_t ws_bytes, void *stream);

/*
 * Rollback at the bifurcation (Algorithm 1: the verifier resumes from the
 * state after the accepted drafted bytes). For every stream s,
 *   h_out[s] = h0[s]                 if accept[s] == 0
 *            = h_all[s, accept[s]-1] if 1 <= accept[s] <= k
 * h0: [batch, d_inner, d_state] fp32 (NULL = zeros), h_all: [batch, k,
 * d_inner, d_state] fp32, accept: [batch] int32 on the device, h_out:
 * [batch, d_inner, d_state] fp32. h_out may alias h0 (not h_all). An accept
 * count outside [0, k] is a caller error: that stream's h_out is left
 * untouched and the first such stream index is recorded in the status block
 * of `ws` when ws != NULL (read it with mb_check).
 */
mb_status mb_rollback(const float *h0, const float *h_all, const int32_t *accept, float *h_out,
                      int64_t batch, int64_t k, int64_t d_inner, int64_t d_state, void *ws,
                      void *stream);

/*
 * Bifurcation test of speculative decoding (Algorithm 1): how many leading
 * drafted bytes of each stream are among the verifier's top-beta candidates.
 *   logits  : [streams, k, 256], dtype (MB_F32 or MB_BF16); row (s, i) is the
 *             verifier's next-byte score for drafted position i of stream s
 *             (the p_i of Algorithm 1, up to a monotone map)
 *   drafted : [streams, k] uint8, the drafted bytes
 *   beta    : >= 1; rank(b) = 1 + #{v : logit[v] > logit[b]} (ties share the
 *             better rank, a NaN score is never larger); byte i is accepted
 *             when rank <= beta
 *   accept  : [streams] int32 output, the index of the first drafted byte that
 *             is not accepted, or k when all are; this is the accept count
 *             that mb_rollback takes.
 * Device pointers; logits 16-byte aligned.
 */
mb_status mb_accept_topk(const void *logits, int32_t dtype, const uint8_t *drafted, int64_t streams,
                         int64_t k, int32_t beta, int32_t *accept, void *stream);

/*
 * One recurrent decode step (Section 6.3: generation runs the recurrence
 * directly, one byte per call). args->seqlen must be 1; args->h0 is ignored.
 * `state` [batch, d_inner, d_state] fp32 is read and updated in place; y is
 * [batch, 1, d_inner]. Used for the corrector loop of Algorithm 1 and for
 * plain generation.
 *   ws, ws_bytes : workspace (at least 256 bytes, 256-byte aligned, its
 *                  status block zeroed once after allocation) or NULL. The
 *                  kernel's waits for its own TMA copies are bounded; one that
 *                  gives up records MB_ERR_TIMEOUT there (read it with
 *                  mb_check), and the rows it did not reach keep their old
 *                  state. With ws == NULL such a timeout is not reported.
 * Launch overlap: the step kernel is launched with programmatic dependent
 * launch. It waits for the previous kernel on the stream to complete before
 * touching memory, and lets the next kernel launch while it runs. A kernel
 * the caller launches next with programmatic stream serialization must
 * therefore execute griddepcontrol.wait (cudaGridDependencySynchronize)
 * before reading y or state, as CUDA requires for any such launch. Plainly
 * launched work is ordered as usual.
 */
mb_status mb_step(const mb_scan_args *args, float *state, void *ws, size_t ws_bytes, void *stream);

/*
 * Resume after the bifurcation (Algorithm 1): one recurrent decode step for
 * every stream s, starting from the state kept after accept[s] drafted bytes
 * (args->h0[s] when accept[s] == 0, h_all[s, accept[s]-1] when
 * 1 <= accept[s] <= k), writing the new state to state[s]. The result is that
 * of mb_rollback(args->h0, h_all, accept, state, ...) followed by
 * mb_step(args, state), without the rollback's own pass over the state.
 *   args    : as for mb_step (seqlen 1); args->h0 = the cached states
 *             [batch, d_inner, d_state] fp32, NULL = zeros
 *   h_all   : [batch, k, d_inner, d_state] fp32, the per-position states of
 *             the last mb_scan_verify (k >= 1)
 *   accept  : [batch] int32 device array, values in [0, k] (mb_accept_topk)
 *   state   : [batch, d_inner, d_state] fp32 output; may alias args->h0, not
 *             h_all
 *   ws      : workspace (at least 256 bytes, 256-byte aligned) or NULL; an
 *             accept count outside [0, k] is a caller error: that stream's
 *             state and y are left untouched and the first such stream index
 *             is recorded in ws's status block (mb_check).
 * Launched with the same launch overlap as mb_step.
 */
mb_status mb_step_resume(const mb_scan_args *args, const float *h_all, const int32_t *accept,
                         int64_t k, float *state, void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Training path (the paper trains through this scan: Section 2 "parallel
 * scans", Section 4 training setup, L = 8192, bf16 mixed precision).
 * ------------------------------------------------------------------------ */

/* Steps between the state checkpoints that the training forward keeps for
 * the backward (the backward recomputes the states inside each chunk). */
#define MB_CKPT_STEPS 16

/*
 * Training forward: mb_scan_prefill that also writes the state before every
 * MB_CKPT_STEPS-step chunk:
 *   h_ckpt[b, i, d, n] = state before step i * MB_CKPT_STEPS, fp32, shape
 *   [batch, ceil(seqlen / MB_CKPT_STEPS), d_inner, d_state] (h_ckpt[b, 0] is
 *   h0, or zeros). Everything else is as for mb_scan_prefill. h_ckpt must
 *   not overlap any other argument.
 */
mb_status mb_scan_prefill_ckpt(const mb_scan_args *args, float *h_last, float *h_ckpt, void *ws,
                               size_t ws_bytes, void *stream);

/* Gradients written by mb_scan_backward (device pointers, overwritten). */
typedef struct {
    void *dx, *dz, *ddt;   /* [batch, seqlen, d_inner], dtype; dz is required when args->z is
                              not NULL and ignored otherwise */
    float *dB, *dC;        /* [batch, seqlen, d_state] fp32 (sums over channels) */
    float *dA;             /* [d_inner, d_state] fp32 */
    float *dD, *ddt_bias;  /* [d_inner] fp32, or NULL to skip */
    float *dh0;            /* [batch, d_inner, d_state] fp32 (dJ/dh0), or NULL to skip */
} mb_scan_grads;

/*
 * Backward of the layer core: every input gradient of a scalar J given
 *   dout    : dJ/dy [batch, seqlen, d_inner], dtype (y as written by the
 *             forward, i.e. after the gate)
 *   dh_last : dJ/dh_last [batch, d_inner, d_state] fp32, or NULL (= 0)
 * args: the forward's arguments (args->y is not read and may be NULL);
 * h_ckpt: the checkpoints written by mb_scan_prefill_ckpt for the same args.
 * The adjoint recurrence (Eq. 2 transposed), per (b, d) from t = L-1 down to
 * 0 with g = dJ/dh_t:
 *   dy = dout * silu(z), dz = dout * y_t * silu'(z), g += dy C_t,
 *   dC_t += dy h_t, dx_t = dy D + Delta_t g.B_t, dB_t += g Delta_t x_t,
 *   dDelta_t = x_t g.B_t + sum_n g Abar h_{t-1} A, dA += g Abar h_{t-1} Delta_t,
 *   g = Abar g, ddt_t = dDelta_t sigmoid(dt_t + dt_bias), dD += dy x_t,
 *   dt_bias gradient = sum of ddt; dh0 = g after t = 0.
 * Sums over channels (dB, dC) and over batch rows (dA, dD, ddt_bias) are
 * accumulated with fp32 atomics: their rounding order is not fixed. The
 * outputs must not overlap the inputs or each other. ws as for prefill.
 */
mb_status mb_scan_backward(const mb_scan_args *args, const float *h_ckpt, const void *dout,
                           const float *dh_last, const mb_scan_grads *grads, void *ws,
                           size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Element-wise steps of the Mamba block around the scan, for recurrent
 * decoding of a whole MambaByte model (Figure 6; Table 6 "Pre-SSM 1D
 * convolution"). Rows are [batch, width], contiguous, 16-byte aligned;
 * width % 8 == 0.
 * ------------------------------------------------------------------------ */

/*
 * Residual add and RMS normalisation that open a block:
 *   residual[b] += add[b]            (skipped when add == NULL)
 *   out[b] = residual[b] * w / sqrt(mean_j residual[b, j]^2 + eps)
 * residual: fp32 [batch, width], read and written; add, out: dtype
 * [batch, width]; w: fp32 [width]. out must not overlap the
 * other arguments.
 */
mb_status mb_rmsnorm(const void *add, float *residual, const float *w, float eps, void *out,
                     int64_t batch, int64_t width, int32_t dtype, void *stream);

/*
 * One decode step of the causal depthwise convolution (kernel size 4) and its
 * SiLU, the step that feeds the scan's x:
 *   out[b, d] = silu(w[d,0] s[b,0,d] + w[d,1] s[b,1,d] + w[d,2] s[b,2,d]
 *                    + w[d,3] x[b,d] + bias[d])
 * then s[b,0] <- s[b,1], s[b,1] <- s[b,2], s[b,2] <- x[b].
 *   x, out : [batch, width], dtype
 *   state  : [batch, 3, width], dtype, the three previous inputs (oldest
 *            first; zeros at the start of a sequence), read and written
 *   w      : [width, 4] fp32 (w[d, 3] multiplies the current input);
 *   bias   : [width] fp32 or NULL
 * out must not overlap x, state, w or bias.
 */
mb_status mb_conv1d_step(const void *x, void *state, const float *w, const float *bias, void *out,
                         int64_t batch, int64_t width, int32_t dtype, void *stream);

/*
 * The convolution step above fused with the x-projection that follows it
 * (Figure 6; Table 6 "Pre-SSM 1D convolution" and "Delta, B, C from input
 * x"), for decoding a whole model:
 *   xc  = the output of mb_conv1d_step (same arithmetic, window updated the same way)
 *   out[b, n] = sum_d xc[b, d] W[n, d]   ([dt_low | B | C] = xc W^T)
 * with xc rounded to bf16 before the product (as the unfused pair does),
 * products accumulated in fp32 and out rounded to bf16 once. The sum runs
 * in width / 128 fp32 partial sums (one per 128 channels) added in a fixed
 * order, so results are reproducible run to run and differ from one fp32
 * GEMM only by rounding order.
 *   x, xc  : [batch, width] bf16; xc is written
 *   state  : [batch, 3, width] bf16, read and written (as mb_conv1d_step)
 *   w, bias: [width, 4] fp32, [width] fp32 or NULL
 *   W      : [n_out, width] bf16 (rows dt_low, then B, then C)
 *   out    : [batch, n_out] bf16
 *   dtype  : MB_BF16 only (MB_ERR_UNSUPPORTED otherwise)
 *   ws     : 256-byte aligned, ws_bytes >= mb_conv_xproj_workspace_size(
 *            batch, width, n_out): the status block (zeroed once after
 *            allocation, as for mb_scan_prefill), then the partial sums. A wait
 *            for a tile that gives up records MB_ERR_TIMEOUT there.
 * Supported: width % 128 == 0, n_out in {40, 96, 144, 176} (dt_rank + 32
 * for d_state 16 and dt_rank 8, 64, 112, 144); MB_ERR_UNSUPPORTED otherwise.
 * xc, out, state and ws must not overlap one another or the inputs.
 */
size_t mb_conv_xproj_workspace_size(int64_t batch, int64_t width, int32_t n_out);
mb_status mb_conv_xproj(const void *x, void *state, const float *w, const float *bias, const void *W, void *xc,
                        void *out, int64_t batch, int64_t width, int32_t n_out, int32_t dtype, void *ws,
                        size_t ws_bytes, void *stream);

/*
 * Read and clear the status block of a workspace (blocking: waits for
 * `stream`). Returns MB_OK, or the first device-side error recorded by
 * calls on that workspace since the last mb_check. If detail != NULL it
 * receives an error-specific value (e.g. the first bad stream of
 * mb_rollback), else -1.
 */
mb_status mb_check(void *ws, void *stream, int64_t *detail);

/*
 * Diagnostic of the bounded device-side waits (failure detection; an
 * addition of this library, the paper has no counterpart). Every wait inside
 * the kernels (for a TMA stage, a ring slot) gives up after about 2 s of SM
 * clocks, records MB_ERR_TIMEOUT in the workspace status block and returns,
 * so that a stalled copy cannot hang the GPU. This call runs that path on
 * purpose: one warp waits on a barrier nothing arrives on, for wait_cycles SM
 * clocks (1 .. 4e9), then records MB_ERR_TIMEOUT with detail = the clocks it
 * waited. Read it with mb_check; the context stays usable.
 *   ws, ws_bytes : a workspace as for mb_scan_prefill (>= 256 bytes, 256-byte aligned)
 * Returns MB_ERR_INVALID_ARG for a bad workspace or wait_cycles.
 */
mb_status mb_selftest_timeout(void *ws, size_t ws_bytes, int64_t wait_cycles, void *stream);

/*
 * mb_scan_prefill without a caller-provided workspace. (An addition of this
 * library; the paper has no counterpart.)
 *
 * Some callers cannot allocate device memory at the point where they run the
 * scan: code running under an allocator that owns all device memory,
 * real-time paths that must not allocate after start-up, or plugins that are
 * handed only their input and output buffers. This entry point takes the
 * same arguments as mb_scan_prefill but no workspace: its scratch (the
 * 256-byte status block of the bounded device-side waits) is a fixed array
 * inside the library, one per GPU, kept for as long as the library is
 * loaded. It calls no allocator.
 *
 *  - Arguments, layouts and h_last rules are those of mb_scan_prefill.
 *  - The fixed array has room for the status block only (256 bytes), not for
 *    the segment summaries of the time split, so every span runs unsplit:
 *    the result is bit for bit that of mb_scan_prefill given a 256-byte
 *    workspace. (A single long prompt therefore takes the unsplit kernel's
 *    time; mb_scan_prefill with mb_workspace_size(args) bytes is faster.)
 *  - The first call on each GPU looks up the array's device address with
 *    that GPU current and keeps it for the life of the process; make that
 *    first call before any stream capture, and do not call this entry point
 *    again on a device after resetting it (cudaDeviceReset).
 *  - Every call clears the array on `stream` before the launch. All calls on
 *    one GPU share the one array, so calls that may run at the same time on
 *    the GPU (different streams without ordering) race on it; order them.
 *  - A device-side timeout is recorded in that internal array; it cannot be
 *    read back through mb_check (use mb_scan_prefill with a workspace when
 *    the status matters).
 */
mb_status mb_scan_prefill_noalloc(const mb_scan_args *args, float *h_last, void *stream);

/* Human-readable name of a status code (static string). */
const char *mb_status_string(mb_status s);

/* Library version, e.g. "mbscan 0.1.0 sm_103a". */
const char *mb_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MBSCAN_H */
