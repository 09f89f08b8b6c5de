// C ABI of the selective-scan layer core: host-side validation, then one
// kernel launch per call on the caller's stream. Declarations and the
// contract of every entry point are in include/mbscan.h.
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <mutex>

#include "../../include/mbscan.h"
#include "internal.h"

using mbscan::ScanParams;
using mbscan::StatusBlock;

namespace {

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Range {
    uintptr_t lo, hi;
};
Range range_of(const void *p, int64_t bytes) {   // a null pointer is an empty range
    uintptr_t a = reinterpret_cast<uintptr_t>(p);
    return Range{a, p ? a + (uintptr_t)(bytes > 0 ? bytes : 0) : a};
}
bool overlap(Range a, Range b) { return a.lo < b.hi && b.lo < a.hi && a.lo != a.hi && b.lo != b.hi; }

// Products of sizes must stay far from int64 overflow and inside the
// 32-bit element counts the kernels assume for token tensors.
constexpr int64_t kMaxTokens = (int64_t)1 << 31;

// Bytes spanned by B (or C): rows bc_stride elements apart.
int64_t bc_bytes(const mb_scan_args *a) {
    const int64_t rows = a->batch * a->seqlen;
    if (rows <= 0) return 0;
    const int64_t es = a->dtype == MB_BF16 ? 2 : 4;
    const int64_t stride = a->bc_stride ? a->bc_stride : a->d_state;
    return ((rows - 1) * stride + a->d_state) * es;
}

// Bytes spanned by dt_low (fused Delta projection): rows dt_low_stride apart.
int64_t dtl_bytes(const mb_scan_args *a) {
    const int64_t rows = a->batch * a->seqlen;
    if (!a->dt_low || rows <= 0) return 0;
    const int64_t stride = a->dt_low_stride ? a->dt_low_stride : a->dt_rank;
    return ((rows - 1) * stride + a->dt_rank) * 2;
}
int64_t wdt_bytes(const mb_scan_args *a) { return a->dt_low ? a->d_inner * a->dt_rank * 2 : 0; }

// The fused Delta projection's arguments (dt_low set); MB_OK when dt_low is null.
mb_status check_fused(const mb_scan_args *a) {
    if (!a->dt_low) return MB_OK;
    if (a->dt) return MB_ERR_INVALID_ARG;
    if (a->dt_rank <= 0 || a->dt_low_stride < 0) return MB_ERR_INVALID_ARG;
    if (a->dtype != MB_BF16 || a->dt_rank % 16 != 0 || a->dt_rank < mbscan::kRankTile ||
        a->dt_rank > mbscan::kMaxRank)
        return MB_ERR_UNSUPPORTED;
    if (a->dt_low_stride != 0 && (a->dt_low_stride < a->dt_rank || a->dt_low_stride % 8 != 0))
        return MB_ERR_INVALID_ARG;
    if (a->batch * a->d_inner > 0 && !a->W_dt) return MB_ERR_INVALID_ARG;
    if (!aligned16(a->dt_low) || (a->W_dt && !aligned16(a->W_dt))) return MB_ERR_INVALID_ARG;
    return MB_OK;
}

// Validate the common part of a scan problem; `need_seqlen1` for mb_step.
mb_status check_args(const mb_scan_args *a, bool need_seqlen1, bool need_y = true) {
    if (a == nullptr) return MB_ERR_INVALID_ARG;
    if (a->batch < 0 || a->seqlen < 0 || a->d_inner < 0 || a->d_state < 0) return MB_ERR_INVALID_ARG;
    if (a->dtype != MB_F32 && a->dtype != MB_BF16) return MB_ERR_INVALID_ARG;
    if (need_seqlen1 && a->seqlen != 1) return MB_ERR_INVALID_ARG;
    if (a->d_state != mbscan::kDState) return MB_ERR_UNSUPPORTED;
    if (a->bc_stride != 0 && (a->bc_stride < a->d_state ||
                              (a->bc_stride * (a->dtype == MB_BF16 ? 2 : 4)) % 16 != 0))
        return MB_ERR_INVALID_ARG;
    if (a->d_inner % 8 != 0) return MB_ERR_UNSUPPORTED;
    if (a->batch > kMaxTokens || a->seqlen > kMaxTokens || a->d_inner > kMaxTokens)
        return MB_ERR_INVALID_ARG;
    if (mb_status f = check_fused(a); f != MB_OK) return f;
    const int64_t chans = a->batch * a->d_inner;
    if (a->seqlen > 0 && chans > kMaxTokens / a->seqlen) return MB_ERR_INVALID_ARG;
    if (chans > kMaxTokens / mbscan::kDState) return MB_ERR_INVALID_ARG;
    const bool any_tokens = a->batch * a->seqlen * a->d_inner > 0;
    const bool any_chan = chans > 0;
    if (any_tokens && (!a->x || !(a->dt || a->dt_low) || !a->B || !a->C || (need_y && !a->y)))
        return MB_ERR_INVALID_ARG;
    if (any_chan && !a->A) return MB_ERR_INVALID_ARG;
    const void *ptrs[] = {a->x, a->z, a->dt, a->B, a->C, a->A, a->D, a->dt_bias, a->h0, a->y};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return MB_ERR_INVALID_ARG;
    // y must not overlap any input.
    const int64_t es = a->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = a->batch * a->seqlen * a->d_inner * es;
    const int64_t bc = bc_bytes(a);
    const Range ry = range_of(a->y, tok);
    const Range ins[] = {range_of(a->x, tok), range_of(a->z, tok), range_of(a->dt, tok),
                         range_of(a->B, bc), range_of(a->C, bc),
                         range_of(a->A, a->d_inner * a->d_state * 4),
                         range_of(a->D, a->d_inner * 4), range_of(a->dt_bias, a->d_inner * 4),
                         range_of(a->h0, chans * a->d_state * 4),
                         range_of(a->dt_low, dtl_bytes(a)), range_of(a->W_dt, wdt_bytes(a))};
    for (const Range &r : ins)
        if (overlap(ry, r)) return MB_ERR_INVALID_ARG;
    return MB_OK;
}

ScanParams to_params(const mb_scan_args *a, float *h_out, StatusBlock *status) {
    ScanParams p;
    p.batch = a->batch;
    p.seqlen = a->seqlen;
    p.d_inner = a->d_inner;
    p.x = a->x; p.z = a->z; p.dt = a->dt; p.B = a->B; p.C = a->C;
    p.bc_stride = a->bc_stride ? a->bc_stride : a->d_state;
    p.A = a->A; p.D = a->D; p.dt_bias = a->dt_bias; p.h0 = a->h0;
    p.y = a->y;
    p.h_out = h_out;
    p.status = status;
    p.h_ckpt = nullptr;
    p.dt_low = a->dt_low;
    p.W_dt = a->W_dt;
    p.dt_rank = a->dt_low ? a->dt_rank : 0;
    p.dt_low_stride = a->dt_low ? (a->dt_low_stride ? a->dt_low_stride : a->dt_rank) : 0;
    p.h_prev_all = nullptr;
    p.accept = nullptr;
    p.k_prev = 0;
    p.nseg = 1;
    p.seg_h = p.seg_p = nullptr;
    return p;
}

// The status block must fit; a larger workspace (mb_workspace_size) only
// lets mb_scan_prefill split long few-channel spans.
mb_status check_ws(const mb_scan_args *a, void *ws, size_t ws_bytes) {
    if (mb_workspace_size(a) == 0) return MB_OK;
    if (ws == nullptr || ws_bytes < mbscan::kStatusBytes) return MB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return MB_ERR_INVALID_ARG;
    return MB_OK;
}

// Long spans with few channels are split over L when the workspace holds the
// segment summaries (after the status block); else they run unsplit.
mb_status setup_split(const mb_scan_args *args, ScanParams &p, const float *h_last, void *ws, size_t ws_bytes) {
    const bool bf16 = args->dtype == MB_BF16;
    const int64_t nseg = mbscan::prefill_segments(p, bf16);
    const size_t split = mbscan::prefill_split_bytes(p, nseg);
    if (nseg < 2 || ws_bytes < mbscan::kStatusBytes + split) return MB_OK;
    const int64_t es = bf16 ? 2 : 4;
    const int64_t tok = args->batch * args->seqlen * args->d_inner * es;
    const int64_t sbytes = args->batch * args->d_inner * args->d_state * 4;
    const Range rs = range_of(static_cast<char *>(ws) + mbscan::kStatusBytes, (int64_t)split);
    const Range others[] = {range_of(args->x, tok), range_of(args->z, tok), range_of(args->dt, tok),
                            range_of(args->y, tok), range_of(args->B, bc_bytes(args)),
                            range_of(args->C, bc_bytes(args)), range_of(args->h0, sbytes), range_of(h_last, sbytes),
                            range_of(args->A, args->d_inner * args->d_state * 4),
                            range_of(args->D, args->d_inner * 4), range_of(args->dt_bias, args->d_inner * 4)};
    for (const Range &r : others)
        if (overlap(rs, r)) return MB_ERR_INVALID_ARG;
    p.nseg = nseg;
    p.seg_h = reinterpret_cast<float *>(static_cast<char *>(ws) + mbscan::kStatusBytes);
    p.seg_p = p.seg_h + split / (2 * sizeof(float));
    return MB_OK;
}

mb_status from_cuda(cudaError_t e) { return e == cudaSuccess ? MB_OK : MB_ERR_CUDA; }

// The prefill's rules for h_last (shared by mb_scan_prefill and
// mb_scan_prefill_noalloc): 16-byte aligned; it may be exactly h0 (in-place
// resume) but must not partially overlap h0, nor overlap y or any input that
// the kernel still reads while it writes h_last.
mb_status check_h_last(const mb_scan_args *args, const float *h_last) {
    if (!h_last) return MB_OK;
    if (!aligned16(h_last)) return MB_ERR_INVALID_ARG;
    const int64_t sbytes = args->batch * args->d_inner * args->d_state * 4;
    const Range rh = range_of(h_last, sbytes);
    if (args->h0 != h_last && overlap(rh, range_of(args->h0, sbytes))) return MB_ERR_INVALID_ARG;
    const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = args->batch * args->seqlen * args->d_inner * es;
    const int64_t bc = bc_bytes(args);
    const Range others[] = {range_of(args->y, tok), range_of(args->x, tok), range_of(args->dt, tok),
                            range_of(args->z, tok), range_of(args->B, bc), range_of(args->C, bc),
                            range_of(args->A, args->d_inner * args->d_state * 4),
                            range_of(args->D, args->d_inner * 4), range_of(args->dt_bias, args->d_inner * 4),
                            range_of(args->dt_low, dtl_bytes(args)), range_of(args->W_dt, wdt_bytes(args))};
    for (const Range &r : others)
        if (overlap(rh, r)) return MB_ERR_INVALID_ARG;
    return MB_OK;
}

}  // namespace

extern "C" {

size_t mb_workspace_size(const mb_scan_args *args) {
    if (check_args(args, false, false) != MB_OK) return 0;
    const ScanParams p = to_params(args, nullptr, nullptr);
    const bool bf16 = args->dtype == MB_BF16;
    return mbscan::kStatusBytes + mbscan::prefill_split_bytes(p, mbscan::prefill_segments(p, bf16));
}

mb_status mb_scan_prefill(const mb_scan_args *args, float *h_last, void *ws, size_t ws_bytes,
                          void *stream) {
    mb_status st = check_args(args, false);
    if (st != MB_OK) return st;
    if ((st = check_ws(args, ws, ws_bytes)) != MB_OK) return st;
    if ((st = check_h_last(args, h_last)) != MB_OK) return st;
    if (args->batch * args->d_inner == 0) return MB_OK;
    ScanParams p = to_params(args, h_last, static_cast<StatusBlock *>(ws));
    const bool bf16 = args->dtype == MB_BF16;
    if ((st = setup_split(args, p, h_last, ws, ws_bytes)) != MB_OK) return st;
    return from_cuda(mbscan::launch_prefill(p, bf16, (cudaStream_t)stream));
}

mb_status mb_scan_verify(const mb_scan_args *args, float *h_all, void *ws, size_t ws_bytes,
                         void *stream) {
    mb_status st = check_args(args, false);
    if (st != MB_OK) return st;
    if ((st = check_ws(args, ws, ws_bytes)) != MB_OK) return st;
    const int64_t n_all = args->batch * args->seqlen * args->d_inner * args->d_state;
    if (n_all > 0) {
        if (h_all == nullptr || !aligned16(h_all)) return MB_ERR_INVALID_ARG;
        const Range ra = range_of(h_all, n_all * 4);
        const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
        const int64_t tok = args->batch * args->seqlen * args->d_inner * es;
        if (overlap(ra, range_of(args->h0, args->batch * args->d_inner * args->d_state * 4)) ||
            overlap(ra, range_of(args->y, tok)) || overlap(ra, range_of(args->x, tok)) ||
            overlap(ra, range_of(args->dt, tok)) || overlap(ra, range_of(args->z, tok)) ||
            overlap(ra, range_of(args->dt_low, dtl_bytes(args))) ||
            overlap(ra, range_of(args->W_dt, wdt_bytes(args))))
            return MB_ERR_INVALID_ARG;
    }
    if (n_all == 0) return MB_OK;
    ScanParams p = to_params(args, h_all, static_cast<StatusBlock *>(ws));
    return from_cuda(mbscan::launch_verify(p, args->dtype == MB_BF16, (cudaStream_t)stream));
}

mb_status mb_scan_verify_resume(const mb_scan_args *args, const float *h_all_prev, const int32_t *accept,
                                int64_t k_prev, float *h_all, void *ws, size_t ws_bytes, void *stream) {
    mb_status st = check_args(args, false);
    if (st != MB_OK) return st;
    if ((st = check_ws(args, ws, ws_bytes)) != MB_OK) return st;
    if (ws == nullptr) return MB_ERR_INVALID_ARG;   // bad accept counts are reported there
    const int64_t chans = args->batch * args->d_inner;
    if (k_prev < 1 || k_prev > kMaxTokens) return MB_ERR_INVALID_ARG;
    if (chans > 0 && k_prev > kMaxTokens * 16 / (chans * args->d_state)) return MB_ERR_INVALID_ARG;
    const int64_t n_all = chans * args->seqlen * args->d_state;
    if (n_all == 0) return MB_OK;
    if (!h_all || !aligned16(h_all) || !h_all_prev || !aligned16(h_all_prev) || !accept ||
        (reinterpret_cast<uintptr_t>(accept) & 3u))
        return MB_ERR_INVALID_ARG;
    const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = chans * args->seqlen * es;
    const Range ra = range_of(h_all, n_all * 4), ry = range_of(args->y, tok);
    const Range ins[] = {range_of(h_all_prev, chans * k_prev * args->d_state * 4),
                         range_of(accept, args->batch * 4),
                         range_of(args->h0, chans * args->d_state * 4), range_of(args->x, tok),
                         range_of(args->dt, tok), range_of(args->z, tok),
                         range_of(args->dt_low, dtl_bytes(args)), range_of(args->W_dt, wdt_bytes(args))};
    for (const Range &r : ins)
        if (overlap(ra, r) || overlap(ry, r)) return MB_ERR_INVALID_ARG;
    ScanParams p = to_params(args, h_all, static_cast<StatusBlock *>(ws));
    p.h_prev_all = h_all_prev;
    p.accept = accept;
    p.k_prev = k_prev;
    return from_cuda(mbscan::launch_verify(p, args->dtype == MB_BF16, (cudaStream_t)stream));
}

mb_status mb_rollback(const float *h0, const float *h_all, const int32_t *accept, float *h_out,
                      int64_t batch, int64_t k, int64_t d_inner, int64_t d_state, void *ws,
                      void *stream) {
    if (batch < 0 || k < 0 || d_inner < 0 || d_state < 0) return MB_ERR_INVALID_ARG;
    if (d_state != mbscan::kDState) return MB_ERR_UNSUPPORTED;
    if (batch > kMaxTokens || k > kMaxTokens || d_inner > kMaxTokens) return MB_ERR_INVALID_ARG;
    const int64_t per = d_inner * d_state;
    if (batch > 0 && per > 0 && k > 0 && batch * k > kMaxTokens * 16 / per) return MB_ERR_INVALID_ARG;
    if (batch * per == 0) return MB_OK;
    if (!accept || !h_out || (k > 0 && !h_all)) return MB_ERR_INVALID_ARG;
    if (!aligned16(h_out) || (h0 && !aligned16(h0)) || (h_all && !aligned16(h_all)) ||
        (reinterpret_cast<uintptr_t>(accept) & 3u))
        return MB_ERR_INVALID_ARG;
    if (ws && (reinterpret_cast<uintptr_t>(ws) & 255u)) return MB_ERR_INVALID_ARG;
    const Range ro = range_of(h_out, batch * per * 4);
    if (overlap(ro, range_of(h_all, batch * k * per * 4))) return MB_ERR_INVALID_ARG;
    if (h0 && h0 != h_out && overlap(ro, range_of(h0, batch * per * 4))) return MB_ERR_INVALID_ARG;
    if (overlap(ro, range_of(accept, batch * 4))) return MB_ERR_INVALID_ARG;
    return from_cuda(mbscan::launch_rollback(h0, h_all, accept, h_out, batch, k, d_inner,
                                             static_cast<StatusBlock *>(ws), (cudaStream_t)stream));
}

mb_status mb_accept_topk(const void *logits, int32_t dtype, const uint8_t *drafted, int64_t streams,
                         int64_t k, int32_t beta, int32_t *accept, void *stream) {
    if (streams < 0 || k < 0 || beta < 1) return MB_ERR_INVALID_ARG;
    if (dtype != MB_F32 && dtype != MB_BF16) return MB_ERR_INVALID_ARG;
    if (streams > kMaxTokens || k > kMaxTokens || (k > 0 && streams > kMaxTokens / (256 * k)))
        return MB_ERR_INVALID_ARG;
    if (streams == 0) return MB_OK;
    if (!accept || (reinterpret_cast<uintptr_t>(accept) & 3u)) return MB_ERR_INVALID_ARG;
    if (k > 0 && (!logits || !drafted || !aligned16(logits))) return MB_ERR_INVALID_ARG;
    const int64_t es = dtype == MB_BF16 ? 2 : 4;
    const Range ra = range_of(accept, streams * 4);
    if (overlap(ra, range_of(logits, streams * k * 256 * es)) || overlap(ra, range_of(drafted, streams * k)))
        return MB_ERR_INVALID_ARG;
    return from_cuda(mbscan::launch_accept(logits, dtype == MB_BF16, drafted, streams, k, beta, accept,
                                           (cudaStream_t)stream));
}

mb_status mb_step(const mb_scan_args *args, float *state, void *ws, size_t ws_bytes, void *stream) {
    mb_status st = check_args(args, true);
    if (st != MB_OK) return st;
    if (args->dt_low) return MB_ERR_UNSUPPORTED;   // the step kernel takes dt
    const int64_t chans = args->batch * args->d_inner;
    if (chans == 0) return MB_OK;
    if (state == nullptr || !aligned16(state)) return MB_ERR_INVALID_ARG;
    if (ws && ((reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < mbscan::kStatusBytes))
        return MB_ERR_INVALID_ARG;
    const Range rs = range_of(state, chans * args->d_state * 4);
    const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = chans * es;
    const Range others[] = {range_of(args->y, tok), range_of(args->x, tok), range_of(args->z, tok),
                            range_of(args->dt, tok), range_of(args->B, bc_bytes(args)),
                            range_of(args->C, bc_bytes(args)),
                            range_of(args->A, args->d_inner * args->d_state * 4),
                            range_of(args->D, args->d_inner * 4), range_of(args->dt_bias, args->d_inner * 4),
                            range_of(args->dt_low, dtl_bytes(args)), range_of(args->W_dt, wdt_bytes(args)),
                            range_of(ws, ws ? (int64_t)mbscan::kStatusBytes : 0)};
    for (const Range &r : others)
        if (overlap(rs, r)) return MB_ERR_INVALID_ARG;
    if (ws && overlap(range_of(ws, mbscan::kStatusBytes), range_of(args->y, tok))) return MB_ERR_INVALID_ARG;
    ScanParams p = to_params(args, state, static_cast<StatusBlock *>(ws));
    p.h0 = nullptr;
    return from_cuda(mbscan::launch_step(p, args->dtype == MB_BF16, (cudaStream_t)stream));
}

mb_status mb_step_resume(const mb_scan_args *args, const float *h_all, const int32_t *accept,
                         int64_t k, float *state, void *ws, size_t ws_bytes, void *stream) {
    mb_status st = check_args(args, true);
    if (st != MB_OK) return st;
    if (args->dt_low) return MB_ERR_UNSUPPORTED;   // the step kernel takes dt
    const int64_t chans = args->batch * args->d_inner;
    if (k < 1 || k > kMaxTokens) return MB_ERR_INVALID_ARG;
    if (chans > 0 && k > kMaxTokens * 16 / (chans * args->d_state)) return MB_ERR_INVALID_ARG;
    if (chans == 0) return MB_OK;
    if (!state || !aligned16(state) || !h_all || !aligned16(h_all) || !accept ||
        (reinterpret_cast<uintptr_t>(accept) & 3u))
        return MB_ERR_INVALID_ARG;
    if (ws && ((reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < mb_workspace_size(args)))
        return MB_ERR_INVALID_ARG;
    const int64_t per = args->d_inner * args->d_state * 4;
    const Range rs = range_of(state, args->batch * per);
    const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = chans * es;
    const Range others[] = {range_of(args->y, tok), range_of(args->x, tok), range_of(args->z, tok),
                            range_of(args->dt, tok), range_of(args->B, bc_bytes(args)),
                            range_of(args->C, bc_bytes(args)),
                            range_of(args->A, args->d_inner * args->d_state * 4),
                            range_of(h_all, args->batch * k * per), range_of(accept, args->batch * 4),
                            range_of(args->dt_low, dtl_bytes(args)), range_of(args->W_dt, wdt_bytes(args))};
    for (const Range &r : others)
        if (overlap(rs, r)) return MB_ERR_INVALID_ARG;
    if (args->h0 && args->h0 != state && overlap(rs, range_of(args->h0, args->batch * per)))
        return MB_ERR_INVALID_ARG;
    if (overlap(range_of(args->y, tok), range_of(h_all, args->batch * k * per)) ||
        overlap(range_of(args->y, tok), range_of(args->h0, args->batch * per)))
        return MB_ERR_INVALID_ARG;
    ScanParams p = to_params(args, state, static_cast<StatusBlock *>(ws));
    return from_cuda(mbscan::launch_step_resume(p, args->dtype == MB_BF16, h_all, accept, k,
                                                (cudaStream_t)stream));
}

mb_status mb_scan_prefill_ckpt(const mb_scan_args *args, float *h_last, float *h_ckpt, void *ws,
                               size_t ws_bytes, void *stream) {
    mb_status st = check_args(args, false);
    if (st != MB_OK) return st;
    if (args->dt_low) return MB_ERR_UNSUPPORTED;   // the training path takes dt
    if ((st = check_ws(args, ws, ws_bytes)) != MB_OK) return st;
    const int64_t chans = args->batch * args->d_inner;
    const int64_t nchunks = (args->seqlen + mbscan::kCkptSteps - 1) / mbscan::kCkptSteps;
    const int64_t ck_bytes = chans * nchunks * args->d_state * 4;
    if (chans > 0 && nchunks > 0 && (!h_ckpt || !aligned16(h_ckpt))) return MB_ERR_INVALID_ARG;
    if (h_last && !aligned16(h_last)) return MB_ERR_INVALID_ARG;
    const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = chans * args->seqlen * es;
    const int64_t bc = bc_bytes(args);
    const Range rc = range_of(h_ckpt, ck_bytes);
    const Range others[] = {range_of(args->x, tok), range_of(args->z, tok), range_of(args->dt, tok),
                            range_of(args->B, bc), range_of(args->C, bc), range_of(args->y, tok),
                            range_of(args->A, args->d_inner * args->d_state * 4),
                            range_of(args->h0, chans * args->d_state * 4),
                            range_of(h_last, chans * args->d_state * 4), range_of(ws, ws_bytes)};
    for (const Range &r : others)
        if (overlap(rc, r)) return MB_ERR_INVALID_ARG;
    if (h_last && h_last != args->h0 && overlap(range_of(h_last, chans * args->d_state * 4),
                                                range_of(args->h0, chans * args->d_state * 4)))
        return MB_ERR_INVALID_ARG;
    ScanParams p = to_params(args, h_last, static_cast<StatusBlock *>(ws));
    p.h_ckpt = h_ckpt;
    if ((st = setup_split(args, p, h_last, ws, ws_bytes)) != MB_OK) return st;
    if (p.nseg > 1 && overlap(rc, range_of(p.seg_h, (int64_t)mbscan::prefill_split_bytes(p, p.nseg))))
        return MB_ERR_INVALID_ARG;
    return from_cuda(mbscan::launch_prefill_ckpt(p, args->dtype == MB_BF16, (cudaStream_t)stream));
}

mb_status mb_scan_backward(const mb_scan_args *args, const float *h_ckpt, const void *dout,
                           const float *dh_last, const mb_scan_grads *grads, void *ws,
                           size_t ws_bytes, void *stream) {
    mb_status st = check_args(args, false, false);
    if (st != MB_OK) return st;
    if (args->dt_low) return MB_ERR_UNSUPPORTED;   // the training path takes dt
    if (!grads) return MB_ERR_INVALID_ARG;
    if ((st = check_ws(args, ws, ws_bytes)) != MB_OK) return st;
    const int64_t Bn = args->batch, L = args->seqlen, Dn = args->d_inner, N = args->d_state;
    const int64_t chans = Bn * Dn;
    const bool any_tokens = chans * L > 0;
    const mb_scan_grads &g = *grads;
    if (Dn > 0 && (!g.dA || !aligned16(g.dA))) return MB_ERR_INVALID_ARG;
    if (Bn * L > 0 && (!g.dB || !g.dC || !aligned16(g.dB) || !aligned16(g.dC))) return MB_ERR_INVALID_ARG;
    if (any_tokens && (!h_ckpt || !dout || !g.dx || !g.ddt || (args->z && !g.dz)))
        return MB_ERR_INVALID_ARG;
    const void *al[] = {h_ckpt, dout, dh_last, g.dx, g.ddt, args->z ? g.dz : nullptr, g.dD, g.ddt_bias,
                        g.dh0};
    for (const void *q : al)
        if (q && !aligned16(q)) return MB_ERR_INVALID_ARG;
    const int64_t es = args->dtype == MB_BF16 ? 2 : 4;
    const int64_t tok = chans * L * es, bcb = bc_bytes(args), st_b = chans * N * 4;
    const int64_t nchunks = (L + mbscan::kCkptSteps - 1) / mbscan::kCkptSteps;
    // outputs: disjoint from each other and from every input
    const Range outs[] = {range_of(g.dx, any_tokens ? tok : 0), range_of(g.ddt, any_tokens ? tok : 0),
                          range_of(args->z ? g.dz : nullptr, any_tokens ? tok : 0),
                          range_of(g.dB, Bn * L * N * 4), range_of(g.dC, Bn * L * N * 4),
                          range_of(g.dA, Dn * N * 4), range_of(g.dD, Dn * 4), range_of(g.ddt_bias, Dn * 4),
                          range_of(g.dh0, st_b)};
    const Range ins[] = {range_of(args->x, tok), range_of(args->z, tok), range_of(args->dt, tok),
                         range_of(args->B, bcb), range_of(args->C, bcb), range_of(args->A, Dn * N * 4),
                         range_of(args->D, Dn * 4), range_of(args->dt_bias, Dn * 4), range_of(args->h0, st_b),
                         range_of(h_ckpt, chans * nchunks * N * 4), range_of(dout, tok),
                         range_of(dh_last, st_b), range_of(ws, ws_bytes)};
    constexpr int kOuts = sizeof(outs) / sizeof(outs[0]);
    for (int i = 0; i < kOuts; ++i) {
        for (const Range &r : ins)
            if (overlap(outs[i], r)) return MB_ERR_INVALID_ARG;
        for (int j = i + 1; j < kOuts; ++j)
            if (overlap(outs[i], outs[j])) return MB_ERR_INVALID_ARG;
    }
    ScanParams p = to_params(args, nullptr, static_cast<StatusBlock *>(ws));
    mbscan::GradParams gp;
    gp.h_ckpt = h_ckpt;
    gp.dout = dout;
    gp.dh_last = dh_last;
    gp.dx = g.dx;
    gp.dz = args->z ? g.dz : nullptr;
    gp.ddt = g.ddt;
    gp.dB = g.dB;
    gp.dC = g.dC;
    gp.dA = g.dA;
    gp.dD = g.dD;
    gp.ddt_bias = g.ddt_bias;
    gp.dh0 = g.dh0;
    return from_cuda(mbscan::launch_backward(p, gp, args->dtype == MB_BF16, (cudaStream_t)stream));
}

mb_status mb_rmsnorm(const void *add, float *residual, const float *w, float eps, void *out,
                     int64_t batch, int64_t width, int32_t dtype, void *stream) {
    if (batch < 0 || width < 0 || batch > kMaxTokens || width > kMaxTokens) return MB_ERR_INVALID_ARG;
    if (width % 8 != 0) return MB_ERR_UNSUPPORTED;
    if (batch > 0 && width > 0 && batch > kMaxTokens / width) return MB_ERR_INVALID_ARG;
    if (dtype != MB_F32 && dtype != MB_BF16) return MB_ERR_INVALID_ARG;
    if (batch * width == 0) return MB_OK;
    if (!(eps >= 0.f)) return MB_ERR_INVALID_ARG;
    if (!residual || !w || !out || !aligned16(residual) || !aligned16(w) || !aligned16(out) ||
        (add && !aligned16(add)))
        return MB_ERR_INVALID_ARG;
    const int64_t es = dtype == MB_BF16 ? 2 : 4;
    const Range ro = range_of(out, batch * width * es);
    if (overlap(ro, range_of(residual, batch * width * 4)) || overlap(ro, range_of(w, width * 4)) ||
        overlap(ro, range_of(add, batch * width * es)) ||
        overlap(range_of(residual, batch * width * 4), range_of(add, batch * width * es)))
        return MB_ERR_INVALID_ARG;
    return from_cuda(mbscan::launch_rmsnorm(add, residual, w, eps, out, batch, width, dtype == MB_BF16,
                                            (cudaStream_t)stream));
}

mb_status mb_conv1d_step(const void *x, void *state, const float *w, const float *bias, void *out,
                         int64_t batch, int64_t width, int32_t dtype, void *stream) {
    if (batch < 0 || width < 0 || batch > kMaxTokens || width > kMaxTokens) return MB_ERR_INVALID_ARG;
    if (width % 8 != 0) return MB_ERR_UNSUPPORTED;
    if (dtype != MB_F32 && dtype != MB_BF16) return MB_ERR_INVALID_ARG;
    if (batch * width == 0) return MB_OK;
    if (batch > kMaxTokens / width) return MB_ERR_INVALID_ARG;
    if (!x || !state || !w || !out || !aligned16(x) || !aligned16(state) || !aligned16(w) ||
        !aligned16(out) || (bias && !aligned16(bias)))
        return MB_ERR_INVALID_ARG;
    const int64_t es = dtype == MB_BF16 ? 2 : 4;
    const Range ro = range_of(out, batch * width * es), rs = range_of(state, batch * 3 * width * es);
    const Range rx = range_of(x, batch * width * es);
    if (overlap(ro, rx) || overlap(ro, rs) || overlap(rs, rx) || overlap(ro, range_of(w, width * 16)) ||
        overlap(ro, range_of(bias, width * 4)))
        return MB_ERR_INVALID_ARG;
    return from_cuda(mbscan::launch_conv_step(x, state, w, bias, out, batch, width, dtype == MB_BF16,
                                              (cudaStream_t)stream));
}

size_t mb_conv_xproj_workspace_size(int64_t batch, int64_t width, int32_t n_out) {
    if (batch < 0 || batch > kMaxTokens || !mbscan::conv_xproj_supported(width, n_out)) return 0;
    return mbscan::kStatusBytes + mbscan::conv_xproj_partial_bytes(batch, width, n_out);
}

mb_status mb_conv_xproj(const void *x, void *state, const float *w, const float *bias, const void *W, void *xc,
                        void *out, int64_t batch, int64_t width, int32_t n_out, int32_t dtype, void *ws,
                        size_t ws_bytes, void *stream) {
    if (batch < 0 || width < 0 || batch > kMaxTokens || width > kMaxTokens) return MB_ERR_INVALID_ARG;
    if (!mbscan::conv_xproj_supported(width, n_out)) return MB_ERR_UNSUPPORTED;
    if (batch > kMaxTokens / width) return MB_ERR_INVALID_ARG;
    if (batch == 0) return MB_OK;
    if (dtype != MB_BF16) return MB_ERR_UNSUPPORTED;
    if (!x || !state || !w || !W || !xc || !out || !ws) return MB_ERR_INVALID_ARG;
    const void *al[] = {x, state, w, bias, W, xc, out};
    for (const void *q : al)
        if (q && !aligned16(q)) return MB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < mb_conv_xproj_workspace_size(batch, width, n_out))
        return MB_ERR_INVALID_ARG;
    const int64_t tok = batch * width * 2;
    const Range rx = range_of(x, tok), rs = range_of(state, 3 * tok), rxc = range_of(xc, tok),
                ro = range_of(out, batch * n_out * 2), rw = range_of(W, (int64_t)n_out * width * 2),
                rcw = range_of(w, width * 16), rcb = range_of(bias, width * 4),
                rws = range_of(ws, (int64_t)mb_conv_xproj_workspace_size(batch, width, n_out));
    // the written ranges (the first four: xc, out, the window, the scratch) overlap nothing else
    const Range all[] = {rxc, ro, rs, rws, rx, rw, rcw, rcb};
    for (int i = 0; i < 4; ++i)
        for (int j = 0; j < 8; ++j)
            if (j != i && overlap(all[i], all[j])) return MB_ERR_INVALID_ARG;
    StatusBlock *sb = static_cast<StatusBlock *>(ws);
    float *part = reinterpret_cast<float *>(static_cast<char *>(ws) + mbscan::kStatusBytes);
    return from_cuda(mbscan::launch_conv_xproj(x, state, w, bias, W, xc, out, batch, width, n_out, part, sb,
                                               (cudaStream_t)stream));
}

mb_status mb_selftest_timeout(void *ws, size_t ws_bytes, int64_t wait_cycles, void *stream) {
    if (ws == nullptr || ws_bytes < mbscan::kStatusBytes || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return MB_ERR_INVALID_ARG;
    if (wait_cycles < 1 || wait_cycles > mbscan::kMaxWaitCycles) return MB_ERR_INVALID_ARG;
    return from_cuda(mbscan::launch_wait_timeout(static_cast<StatusBlock *>(ws), (long long)wait_cycles,
                                                 (cudaStream_t)stream));
}

mb_status mb_check(void *ws, void *stream, int64_t *detail) {
    if (detail) *detail = -1;
    if (ws == nullptr) return MB_ERR_INVALID_ARG;
    StatusBlock host;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemcpyAsync(&host, ws, sizeof(host), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return MB_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MB_ERR_CUDA;
    if (host.code == MB_OK) return MB_OK;
    if (cudaMemsetAsync(ws, 0, sizeof(StatusBlock), s) != cudaSuccess) return MB_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MB_ERR_CUDA;
    if (detail) *detail = host.detail;
    return (mb_status)host.code;
}

const char *mb_status_string(mb_status s) {
    switch (s) {
        case MB_OK: return "MB_OK";
        case MB_ERR_INVALID_ARG: return "MB_ERR_INVALID_ARG";
        case MB_ERR_UNSUPPORTED: return "MB_ERR_UNSUPPORTED";
        case MB_ERR_CUDA: return "MB_ERR_CUDA";
        case MB_ERR_TIMEOUT: return "MB_ERR_TIMEOUT";
    }
    return "MB_UNKNOWN_STATUS";
}

const char *mb_version(void) { return "mbscan 0.1.0 sm_103a"; }

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free prefill (mb_scan_prefill_noalloc).
//
// The prefill kernel needs a small block of device scratch: the status block
// that its bounded waits write. Normally the caller provides it as `ws`. For
// callers that may not allocate device memory, this file owns one fixed
// scratch array per device instead: a file-scope __device__ array of
// kNoAllocScratchBytes (the 256-byte status block, nothing more). Host code
// must never hand the array's name to a kernel (on the host it is only a
// stand-in symbol); its device address is looked up once per device with
// cudaGetSymbolAddress while that device is current, and that address is what
// the kernel receives. The array lives for as long as the library is loaded
// on the device and keeps the previous call's contents, so every call clears
// it first on its stream. The array holds no room for the segment summaries
// of the time split, so every span runs unsplit: exactly what mb_scan_prefill
// does when its workspace is 256 bytes.
namespace {

constexpr size_t kNoAllocScratchBytes = mbscan::kStatusBytes;
constexpr int kNoAllocMaxDevices = 64;

}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

std::mutex g_noalloc_mutex;
void *g_noalloc_addr[kNoAllocMaxDevices];   // device address of the array, per device

// Device address of g_noalloc_scratch on the current device, looked up on
// the first call for that device and kept for the life of the process (the
// primary context of that device is assumed to live as long).
mb_status noalloc_scratch(void **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return MB_ERR_CUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return MB_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (g_noalloc_addr[dev] == nullptr) {
        void *addr = nullptr;
        if (cudaGetSymbolAddress(&addr, g_noalloc_scratch) != cudaSuccess || addr == nullptr)
            return MB_ERR_CUDA;
        g_noalloc_addr[dev] = addr;
    }
    *out = g_noalloc_addr[dev];
    return MB_OK;
}

}  // namespace

extern "C" mb_status mb_scan_prefill_noalloc(const mb_scan_args *args, float *h_last, void *stream) {
    mb_status st = check_args(args, false);
    if (st != MB_OK) return st;
    if ((st = check_h_last(args, h_last)) != MB_OK) return st;
    if (args->batch * args->d_inner == 0) return MB_OK;
    void *scratch = nullptr;
    if ((st = noalloc_scratch(&scratch)) != MB_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemsetAsync(scratch, 0, kNoAllocScratchBytes, s) != cudaSuccess) return MB_ERR_CUDA;
    // p.nseg stays 1 (to_params): the span runs unsplit
    ScanParams p = to_params(args, h_last, static_cast<StatusBlock *>(scratch));
    return from_cuda(mbscan::launch_prefill(p, args->dtype == MB_BF16, s));
}
