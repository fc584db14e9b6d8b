// C ABI of libdoloss (declared in include/doloss.h): argument validation,
// workspace layout and the launch sequence of each entry point.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>
#include <cstring>

#include <nvtx3/nvToolsExt.h>

#include "dol_internal.cuh"
#include "doloss.h"

namespace {

using dol::Problem;

// An NVTX range around each entry point (a no-op unless a profiler attaches).
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

do_status check_sizes(int64_t T, int32_t E, int32_t k, int32_t L, Problem *p) {
    if (T < 1 || E < 1 || k < 1 || k > E || L < 1) return DO_ERR_INVALID_ARG;
    if (E > 1024 || L > 65535) return DO_ERR_UNSUPPORTED;
    if ((int64_t)(E - 1) * T > (int64_t)INT_MAX) return DO_ERR_UNSUPPORTED;
    p->T = T;
    p->E = E;
    p->k = k;
    p->L = L;
    p->W = (T + 31) / 32;
    return DO_OK;
}

do_status from_cuda(cudaError_t e) { return e == cudaSuccess ? DO_OK : DO_ERR_CUDA; }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Device buffer of do_forward_backward_host, carved in this order.
struct HostBufLayout {
    size_t logits, bits, counts, D, loss, dlogits, ws, total;
};

// Routing outputs of one call (Sec. 3.1.1): ids and combine are required,
// the dispatch arrays may each be null.
struct RouteArgs {
    int32_t *ids;
    float *combine;
    int32_t *offsets, *rows, *pos;
};

// The router's inputs when the logits are computed in the fused path
// (do_router_forward_backward): bf16 X [L][T][H] and W [L][E][H].
struct RouterIn {
    const void *X;
    const void *Wr;
    int H;
};

// Checks shared by the entry points that write routing outputs: the row and
// token indices of the dispatch arrays are int32.
do_status check_route(const Problem &p, const RouteArgs &r) {
    if ((int64_t)p.T * p.k > (int64_t)INT_MAX) return DO_ERR_UNSUPPORTED;
    if (!r.ids || !r.combine) return DO_ERR_INVALID_ARG;
    if (!aligned(r.ids, 4) || !aligned(r.combine, 4) || (r.offsets && !aligned(r.offsets, 4)) ||
        (r.rows && !aligned(r.rows, 4)) || (r.pos && !aligned(r.pos, 4)))
        return DO_ERR_INVALID_ARG;
    return DO_OK;
}

// The vector stores of the fast selection kernel want 16-byte aligned rows.
bool route_fast_ok(const RouteArgs *r) {
    return !r || (aligned(r->ids, 16) && aligned(r->combine, 16));
}

// Workspace of do_routing: [status word | pad to 256 B | signatures [L][E][W] |
// dispatch scratch (route_scratch_ints)].
size_t routing_bits_bytes(const Problem &p) {
    return round_up(sizeof(uint32_t) * (size_t)p.L * p.E * p.W, 256);
}

size_t routing_ws_bytes(const Problem &p) {
    return dol::kWsHeader + routing_bits_bytes(p) +
           round_up(sizeof(int) * (size_t)dol::route_scratch_ints(p), 256);
}

HostBufLayout host_layout(const Problem &p) {
    HostBufLayout b;
    size_t off = 0;
    const size_t te = (size_t)p.L * (size_t)p.T * (size_t)p.E;
    b.logits = off; off = round_up(off + sizeof(float) * te, 256);
    b.bits = off;   off = round_up(off + sizeof(uint32_t) * (size_t)p.L * p.E * p.W, 256);
    b.counts = off; off = round_up(off + sizeof(int32_t) * (size_t)p.L * p.E, 256);
    b.D = off;      off = round_up(off + sizeof(int32_t) * (size_t)p.L * p.E * p.E, 256);
    b.loss = off;   off = round_up(off + sizeof(float) * (size_t)p.L + sizeof(int), 256);  // + status
    b.dlogits = off; off = round_up(off + sizeof(float) * te, 256);
    b.ws = off;     off = round_up(off + dol::workspace_bytes_plain(p), 256);
    b.total = off;
    return b;
}

}  // namespace

extern "C" {

do_status do_signatures(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                        uint32_t *bits, int32_t *counts, void *stream) {
    NvtxRange nvtx("do_signatures");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!logits || !bits || !counts) return DO_ERR_INVALID_ARG;
    if (!aligned(logits, 4) || !aligned(bits, 4) || !aligned(counts, 4)) return DO_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    if (dol::signatures_fast_supported(logits, p)) {
        cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int) * (size_t)p.L * p.E, s);
        const dol::ZeroSpans none = {{nullptr, nullptr, nullptr}, {0, 0, 0}};
        if (e == cudaSuccess)
            e = dol::launch_signatures_fast(logits, p, bits, counts, nullptr, nullptr, none, nullptr,
                                            s);
        return from_cuda(e);
    }
    return from_cuda(dol::launch_signatures(logits, p, bits, counts, s));
}

do_status do_pairwise_hamming(const uint32_t *bits, int64_t T, int32_t E, int32_t L, int32_t *D,
                              void *stream) {
    NvtxRange nvtx("do_pairwise_hamming");
    Problem p;
    do_status st = check_sizes(T, E, 1, L, &p);
    if (st != DO_OK) return st;
    if (!bits || !D) return DO_ERR_INVALID_ARG;
    if (!aligned(bits, 4) || !aligned(D, 4)) return DO_ERR_INVALID_ARG;
    return from_cuda(dol::launch_hamming(bits, p, D, (cudaStream_t)stream));
}

do_status do_pairwise_hamming_accumulate(const uint32_t *bits, int64_t T, int32_t E, int32_t L,
                                         int32_t *D, void *stream) {
    NvtxRange nvtx("do_pairwise_hamming_accumulate");
    Problem p;
    do_status st = check_sizes(T, E, 1, L, &p);
    if (st != DO_OK) return st;
    if (!bits || !D) return DO_ERR_INVALID_ARG;
    if (!aligned(bits, 4) || !aligned(D, 4)) return DO_ERR_INVALID_ARG;
    return from_cuda(dol::launch_hamming_accumulate(bits, p, D, (cudaStream_t)stream));
}

do_status do_offdiag_variance(const int64_t *origin_do, int64_t T, int32_t E, int32_t k, int32_t L,
                              double *var, void *stream) {
    NvtxRange nvtx("do_offdiag_variance");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (E < 2 || !origin_do || !var || !aligned(origin_do, 8) || !aligned(var, 8))
        return DO_ERR_INVALID_ARG;
    return from_cuda(dol::launch_offdiag_variance(reinterpret_cast<const long long *>(origin_do), p,
                                                  var, (cudaStream_t)stream));
}

do_status do_accumulate_distances(const int32_t *D, int32_t E, int32_t L, int32_t *D_sum,
                                  void *stream) {
    NvtxRange nvtx("do_accumulate_distances");
    if (!D || !D_sum || E < 1 || L < 1 || !aligned(D, 4) || !aligned(D_sum, 4))
        return DO_ERR_INVALID_ARG;
    if (E > 1024 || L > 65535) return DO_ERR_UNSUPPORTED;
    return from_cuda(dol::launch_add_distances(D, D_sum, (int64_t)L * E * E, (cudaStream_t)stream));
}

do_status do_loss_fwd_bwd(const float *logits, const uint32_t *bits, const int32_t *D, int64_t T,
                          int32_t E, int32_t k, int32_t L, int32_t gate, float d_scale,
                          float grad_scale, float *loss, int64_t *origin_do, float *dlogits,
                          void *workspace, size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_loss_fwd_bwd");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!logits || !bits || !D || !loss) return DO_ERR_INVALID_ARG;
    if (gate != DO_GATE_SIGMOID_NORM && gate != DO_GATE_SOFTMAX) return DO_ERR_INVALID_ARG;
    if (!(d_scale == d_scale) || !(grad_scale == grad_scale)) return DO_ERR_INVALID_ARG;
    if (!aligned(logits, 4) || !aligned(bits, 4) || !aligned(D, 4) || !aligned(loss, 4) ||
        (dlogits && !aligned(dlogits, 4)) || (origin_do && !aligned(origin_do, 8)))
        return DO_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < dol::workspace_bytes_plain(p))
        return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    if (dol::loss_fast_supported(p, logits, D, dlogits) && aligned(bits, 16)) {
        const dol::WsLayout w = dol::ws_layout(p);
        char *ws = static_cast<char *>(workspace);
        int *done = reinterpret_cast<int *>(ws + w.done);
        uint8_t *idx = reinterpret_cast<uint8_t *>(ws + w.idx);
        cudaError_t e = dol::launch_idx_from_bits(bits, p, idx, done, p.L, s);
        if (e == cudaSuccess)
            e = dol::launch_loss_fast(logits, idx, D, nullptr, nullptr, p, gate, d_scale,
                                      grad_scale, loss, reinterpret_cast<long long *>(origin_do),
                                      dlogits, reinterpret_cast<double *>(ws + w.partials), done,
                                      reinterpret_cast<int *>(ws), nullptr, s);
        return from_cuda(e);
    }
    return from_cuda(dol::launch_loss(logits, bits, D, p, gate, d_scale, grad_scale, loss,
                                      reinterpret_cast<long long *>(origin_do), dlogits,
                                      workspace, s));
}

}  // extern "C"

namespace {

// Steps 1-3.  status_out (may be null): on the fused fast path the last loss
// CTA ORs the device status word of this call into it (so that one copy
// returns the loss and the status); *status_done tells whether it did.
do_status forward_backward_impl(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                                int32_t gate, float grad_scale, uint32_t *bits, int32_t *counts,
                                int32_t *D, float *loss, int64_t *origin_do, float *dlogits,
                                void *workspace, size_t workspace_bytes, void *stream,
                                int *status_out, bool *status_done,
                                const RouteArgs *ra = nullptr, const RouterIn *rin = nullptr) {
    if (status_done) *status_done = false;
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!logits || !bits || !counts || !D || !loss) return DO_ERR_INVALID_ARG;
    if (gate != DO_GATE_SIGMOID_NORM && gate != DO_GATE_SOFTMAX) return DO_ERR_INVALID_ARG;
    if (!(grad_scale == grad_scale)) return DO_ERR_INVALID_ARG;
    if (!aligned(logits, 4) || !aligned(bits, 4) || !aligned(counts, 4) || !aligned(D, 4) ||
        !aligned(loss, 4) || (dlogits && !aligned(dlogits, 4)) ||
        (origin_do && !aligned(origin_do, 8)))
        return DO_ERR_INVALID_ARG;
    if (ra && (st = check_route(p, *ra)) != DO_OK) return st;
    const size_t need = ra ? dol::workspace_bytes(p) : dol::workspace_bytes_plain(p);
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < need) return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    const dol::RouteOut route = {ra ? ra->ids : nullptr, ra ? ra->combine : nullptr, gate};
    const bool fast = dol::signatures_fast_supported(logits, p) &&
                      dol::loss_fast_supported(p, logits, D, dlogits) && aligned(bits, 16) &&
                      route_fast_ok(ra);
    // the router GEMM runs only in the fused fast path, without routing outputs
    if (rin && !(fast && !ra && dol::router_supported(p, rin->H, rin->X, rin->Wr, logits)))
        return DO_ERR_UNSUPPORTED;
    if (fast) {
        // signatures (+ per-CTA co-occurrence counts) -> reduction to C -> loss,
        // which builds D = n_i + n_j - 2 c_ij and writes D and the counts
        const dol::WsLayout w = dol::ws_layout(p);
        char *ws = static_cast<char *>(workspace);
        int *done = reinterpret_cast<int *>(ws + w.done);
        uint8_t *idx = reinterpret_cast<uint8_t *>(ws + w.idx);
        uint32_t *parts = reinterpret_cast<uint32_t *>(ws + w.cooc_parts);
        int *n_acc = reinterpret_cast<int *>(ws + w.n_acc);
        // origin_do is summed by the reduction kernel (integer atomics) and
        // status_out ORed by the loss kernel: zero them first
        const dol::ZeroSpans zero = {{done, reinterpret_cast<int *>(origin_do), status_out},
                                     {(int64_t)p.L, origin_do ? 2 * (int64_t)p.L : 0,
                                      status_out ? 1 : 0}};
        int *status = reinterpret_cast<int *>(ws);
        // D <= T here (one window of tokens): the two-piece fp16 split of the
        // tensor-core path is exact when R < 2^23 (checked by loss_mma_supported)
        const bool mma = dol::loss_mma_supported(p, gate, logits, D, dlogits);
        unsigned char *bimg = mma ? reinterpret_cast<unsigned char *>(ws + w.bimg) : nullptr;
        cudaError_t e =
            rin ? dol::launch_router_signatures(rin->X, rin->Wr, rin->H, const_cast<float *>(logits),
                                                p, bits, n_acc, idx, parts, zero, status, s)
            : ra ? dol::launch_signatures_fast_routed(logits, p, bits, n_acc, idx, parts, zero,
                                                      status, route, s)
                 : dol::launch_signatures_fast(logits, p, bits, n_acc, idx, parts, zero, status, s);
        const int P1 = rin ? dol::router_ctas_per_problem(p) : dol::sig_fast_ctas_per_problem(p);
        int *rscratch = reinterpret_cast<int *>(ws + w.route_base);
        if (e == cudaSuccess)
            e = dol::launch_cooc_reduce(parts, P1, n_acc, p, D, counts, bimg,
                                        reinterpret_cast<long long *>(origin_do), s);
        if (e == cudaSuccess) {
            if (mma)
                e = dol::launch_loss_mma(logits, idx, bimg, n_acc, p, 1.0f, grad_scale, loss, dlogits,
                                         reinterpret_cast<double *>(ws + w.partials), done, status,
                                         status_out, s);
            else
                e = dol::launch_loss_fast(logits, idx, D, counts, n_acc, p, gate, 1.0f, grad_scale,
                                          loss, nullptr, dlogits,
                                          reinterpret_cast<double *>(ws + w.partials), done,
                                          status, status_out, s);
        }
        // the dispatch order (from the signatures and ids alone) follows the loss kernel
        if (e == cudaSuccess && ra)
            e = dol::launch_route_dispatch(bits, ra->ids, p, ra->offsets, ra->rows, ra->pos,
                                           rscratch, s);
        if (e == cudaSuccess && status_done) *status_done = status_out != nullptr;
        return from_cuda(e);
    }
    if (!ra && dol::signatures_fast256_supported(logits, p) && aligned(bits, 16) &&
        dol::loss_fast256_supported(p, logits, D, dlogits)) {
        // E = 256: the fast selection (with the chosen experts), the Hamming
        // matrix from the signatures, and the ALU loss kernel with D in
        // shared-memory planes
        const dol::WsLayout w = dol::ws_layout(p);
        char *ws = static_cast<char *>(workspace);
        int *done = reinterpret_cast<int *>(ws + w.done);
        uint8_t *idx = reinterpret_cast<uint8_t *>(ws + w.idx);
        int *status = reinterpret_cast<int *>(ws);
        const dol::ZeroSpans zero = {{done, status_out, nullptr},
                                     {(int64_t)p.L, status_out ? 1 : 0, 0}};
        cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int) * (size_t)p.L * p.E, s);
        if (e == cudaSuccess)
            e = dol::launch_signatures_fast256(logits, p, bits, counts, idx, zero, status, s);
        if (e == cudaSuccess) e = dol::launch_hamming(bits, p, D, s);
        if (e == cudaSuccess)
            e = dol::launch_loss_fast(logits, idx, D, counts, nullptr, p, gate, 1.0f, grad_scale,
                                      loss, reinterpret_cast<long long *>(origin_do), dlogits,
                                      reinterpret_cast<double *>(ws + w.partials), done, status,
                                      status_out, s);
        if (e == cudaSuccess && status_done) *status_done = status_out != nullptr;
        return from_cuda(e);
    }
    cudaError_t e = dol::launch_signatures(logits, p, bits, counts, s, route);
    if (e == cudaSuccess) e = dol::launch_hamming(bits, p, D, s);
    if (e == cudaSuccess)
        e = dol::launch_loss(logits, bits, D, p, gate, 1.0f, grad_scale, loss,
                             reinterpret_cast<long long *>(origin_do), dlogits, workspace, s);
    if (e == cudaSuccess && ra)
        e = dol::launch_route_dispatch(
            bits, ra->ids, p, ra->offsets, ra->rows, ra->pos,
            reinterpret_cast<int *>(static_cast<char *>(workspace) + dol::ws_layout(p).route_base), s);
    return from_cuda(e);
}

}  // namespace

extern "C" {

do_status do_forward_backward(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                              int32_t gate, float grad_scale, uint32_t *bits, int32_t *counts,
                              int32_t *D, float *loss, int64_t *origin_do, float *dlogits,
                              void *workspace, size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_forward_backward");
    return forward_backward_impl(logits, T, E, k, L, gate, grad_scale, bits, counts, D, loss,
                                 origin_do, dlogits, workspace, workspace_bytes, stream, nullptr,
                                 nullptr);
}

do_status do_forward_backward_routed(const float *logits, int64_t T, int32_t E, int32_t k,
                                     int32_t L, int32_t gate, float grad_scale, uint32_t *bits,
                                     int32_t *counts, int32_t *D, float *loss, int64_t *origin_do,
                                     float *dlogits, int32_t *expert_ids, float *combine,
                                     int32_t *expert_offsets, int32_t *dispatch_rows,
                                     int32_t *dispatch_pos, void *workspace,
                                     size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_forward_backward_routed");
    const RouteArgs ra = {expert_ids, combine, expert_offsets, dispatch_rows, dispatch_pos};
    return forward_backward_impl(logits, T, E, k, L, gate, grad_scale, bits, counts, D, loss,
                                 origin_do, dlogits, workspace, workspace_bytes, stream, nullptr,
                                 nullptr, &ra);
}

do_status do_router_forward_backward(const void *X, const void *Wr, int64_t T, int32_t H, int32_t E,
                                     int32_t k, int32_t L, int32_t gate, float grad_scale,
                                     float *logits, uint32_t *bits, int32_t *counts, int32_t *D,
                                     float *loss, int64_t *origin_do, float *dlogits,
                                     void *workspace, size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_router_forward_backward");
    if (!X || !Wr || !logits) return DO_ERR_INVALID_ARG;
    if (H < 1) return DO_ERR_INVALID_ARG;
    const RouterIn rin = {X, Wr, H};
    return forward_backward_impl(logits, T, E, k, L, gate, grad_scale, bits, counts, D, loss,
                                 origin_do, dlogits, workspace, workspace_bytes, stream, nullptr,
                                 nullptr, nullptr, &rin);
}

// The forward and backward halves of the routed step.  The forward half
// leaves in the workspace what the backward half's loss kernel reads (the
// selected indices, the fp16 image of D'), so the two must agree on the path;
// the choice depends only on the logits, bits and D pointers and the shape,
// which both halves receive.
bool split_fast(const Problem &p, const float *logits, const uint32_t *bits, const int *D) {
    return dol::signatures_fast_supported(logits, p) &&
           dol::loss_fast_supported(p, logits, D, nullptr) && aligned(bits, 16);
}

// Whether the forward half writes the fp16 image of D' for the tensor-core
// loss kernel (dlogits is not known there: the logits' alignment stands in).
bool split_mma(const Problem &p, int gate, const float *logits, const int *D) {
    return dol::loss_mma_supported(p, gate, logits, D, logits);
}

do_status do_routed_forward(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                            int32_t gate, uint32_t *bits, int32_t *counts, int32_t *D,
                            int64_t *origin_do, int32_t *expert_ids, float *combine,
                            int32_t *expert_offsets, int32_t *dispatch_rows, int32_t *dispatch_pos,
                            void *workspace, size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_routed_forward");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!logits || !bits || !counts || !D) return DO_ERR_INVALID_ARG;
    if (gate != DO_GATE_SIGMOID_NORM && gate != DO_GATE_SOFTMAX) return DO_ERR_INVALID_ARG;
    if (!aligned(logits, 4) || !aligned(bits, 4) || !aligned(counts, 4) || !aligned(D, 4) ||
        (origin_do && !aligned(origin_do, 8)))
        return DO_ERR_INVALID_ARG;
    // without routing outputs (expert_ids and combine both NULL, and no
    // dispatch arrays) the call is steps 1-2 alone
    const bool routed = expert_ids || combine;
    const RouteArgs ra = {expert_ids, combine, expert_offsets, dispatch_rows, dispatch_pos};
    if (routed && (st = check_route(p, ra)) != DO_OK) return st;
    if (!routed && (expert_offsets || dispatch_rows || dispatch_pos)) return DO_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < dol::workspace_bytes(p))
        return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    char *ws = static_cast<char *>(workspace);
    const dol::WsLayout w = dol::ws_layout(p);
    int *rscratch = reinterpret_cast<int *>(ws + w.route_base);
    const dol::RouteOut route = {expert_ids, combine, gate};
    const RouteArgs *rap = routed ? &ra : nullptr;
    cudaError_t e = cudaSuccess;
    if (split_fast(p, logits, bits, D)) {
        int *done = reinterpret_cast<int *>(ws + w.done);
        uint8_t *idx = reinterpret_cast<uint8_t *>(ws + w.idx);
        uint32_t *parts = reinterpret_cast<uint32_t *>(ws + w.cooc_parts);
        int *n_acc = reinterpret_cast<int *>(ws + w.n_acc);
        int *status = reinterpret_cast<int *>(ws);
        const dol::ZeroSpans zero = {{done, reinterpret_cast<int *>(origin_do), nullptr},
                                     {(int64_t)p.L, origin_do ? 2 * (int64_t)p.L : 0, 0}};
        unsigned char *bimg =
            split_mma(p, gate, logits, D) ? reinterpret_cast<unsigned char *>(ws + w.bimg) : nullptr;
        if (routed && !route_fast_ok(rap))  // unaligned routing outputs: the generic selection
            e = dol::launch_signatures(logits, p, bits, counts, s, route);
        if (e == cudaSuccess)
            e = routed && route_fast_ok(rap)
                    ? dol::launch_signatures_fast_routed(logits, p, bits, n_acc, idx, parts, zero,
                                                         status, route, s)
                    : dol::launch_signatures_fast(logits, p, bits, n_acc, idx, parts, zero, status, s);
        if (e == cudaSuccess)
            e = dol::launch_cooc_reduce(parts, dol::sig_fast_ctas_per_problem(p), n_acc, p, D,
                                        counts, bimg, reinterpret_cast<long long *>(origin_do), s);
        // no loss kernel follows in this call: the dispatch kernels clear the
        // counts accumulator
        if (e == cudaSuccess)
            e = dol::launch_route_dispatch(bits, expert_ids, p, expert_offsets, dispatch_rows,
                                           dispatch_pos, rscratch, s, n_acc);
        return from_cuda(e);
    } else {
        e = routed ? dol::launch_signatures(logits, p, bits, counts, s, route)
                   : dol::launch_signatures(logits, p, bits, counts, s);
        if (e == cudaSuccess) e = dol::launch_hamming(bits, p, D, s);
        if (e == cudaSuccess && origin_do)
            e = dol::launch_origin_do(D, p, reinterpret_cast<long long *>(origin_do), s);
    }
    if (e == cudaSuccess)
        e = dol::launch_route_dispatch(bits, expert_ids, p, expert_offsets, dispatch_rows,
                                       dispatch_pos, rscratch, s);
    return from_cuda(e);
}

do_status do_routed_backward(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                             int32_t gate, float d_scale, float grad_scale, const uint32_t *bits,
                             const int32_t *counts, const int32_t *D, const int32_t *expert_ids,
                             const float *grad_combine, float *loss, float *dlogits,
                             void *workspace, size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_routed_backward");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!logits || !bits || !counts || !D || !loss || !dlogits) return DO_ERR_INVALID_ARG;
    // the routing gradient is optional: expert_ids and grad_combine together
    if (!expert_ids != !grad_combine) return DO_ERR_INVALID_ARG;
    const bool rg = expert_ids != nullptr;
    if (gate != DO_GATE_SIGMOID_NORM && gate != DO_GATE_SOFTMAX) return DO_ERR_INVALID_ARG;
    if (!(grad_scale == grad_scale) || !(d_scale == d_scale)) return DO_ERR_INVALID_ARG;
    if (!aligned(logits, 4) || !aligned(bits, 4) || !aligned(counts, 4) || !aligned(D, 4) ||
        (rg && (!aligned(expert_ids, 4) || !aligned(grad_combine, 4))) || !aligned(loss, 4) ||
        !aligned(dlogits, 4))
        return DO_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < dol::workspace_bytes(p))
        return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    char *ws = static_cast<char *>(workspace);
    const dol::WsLayout w = dol::ws_layout(p);
    int *status = reinterpret_cast<int *>(ws);
    int *done = reinterpret_cast<int *>(ws + w.done);
    uint8_t *idx = reinterpret_cast<uint8_t *>(ws + w.idx);
    int *n_acc = reinterpret_cast<int *>(ws + w.n_acc);
    double *partials = reinterpret_cast<double *>(ws + w.partials);
    // d_scale = 1: D is the forward half's own matrix, whose fp16 image the
    // forward half left for the tensor-core kernel; otherwise D is a matrix
    // summed over ranks or micro-batches (Eq. global_do), read as given.
    const bool local = d_scale == 1.0f;
    cudaError_t e;
    if (!local && split_fast(p, logits, bits, D) && aligned(dlogits, 16) &&
        dol::loss_mma_supported(p, gate, logits, D, dlogits, true) &&
        (!rg || (aligned(expert_ids, 16) && aligned(grad_combine, 16)))) {
        // a given matrix: its image of D' is built here, with a flag per
        // problem saying whether the two fp16 pieces hold it exactly; the
        // tensor-core kernel takes the exact problems (routing gradient in its
        // epilogue), the ALU kernel and the routing-gradient kernel the others
        unsigned char *bimg = reinterpret_cast<unsigned char *>(ws + w.bimg);
        int *img_ok = reinterpret_cast<int *>(ws + w.img_ok);
        e = dol::launch_dprime_image(D, p, bimg, img_ok, s);
        if (e == cudaSuccess)
            e = dol::launch_loss_mma(logits, idx, bimg, nullptr, p, d_scale, grad_scale, loss,
                                     dlogits, partials, done, status, nullptr, s, expert_ids,
                                     grad_combine, img_ok);
        if (e == cudaSuccess)
            e = dol::launch_loss_fast(logits, idx, D, nullptr, nullptr, p, gate, d_scale,
                                      grad_scale, loss, nullptr, dlogits, partials, done, status,
                                      nullptr, s, img_ok);
        if (e == cudaSuccess && rg)
            e = dol::launch_route_backward(logits, expert_ids, grad_combine, p.T * p.L, E, k, gate,
                                           1, dlogits, status, s, img_ok, p.T);
        return from_cuda(e);
    }
    if (split_fast(p, logits, bits, D) && aligned(dlogits, 16)) {
        if (local && split_mma(p, gate, logits, D) &&
            dol::loss_mma_supported(p, gate, logits, D, dlogits) &&
            (!rg || (aligned(expert_ids, 16) && aligned(grad_combine, 16)))) {
            // the routing gradient is added in the loss kernel's epilogue
            return from_cuda(dol::launch_loss_mma(
                logits, idx, reinterpret_cast<unsigned char *>(ws + w.bimg), n_acc, p, 1.0f,
                grad_scale, loss, dlogits, partials, done, status, nullptr, s, expert_ids,
                grad_combine));
        }
        // the row sums of D come from the counts only for the local matrix
        e = dol::launch_loss_fast(logits, idx, D, local ? counts : nullptr, n_acc, p, gate,
                                  d_scale, grad_scale, loss, nullptr, dlogits, partials, done,
                                  status, nullptr, s);
    } else {
        e = dol::launch_loss(logits, bits, D, p, gate, d_scale, grad_scale, loss, nullptr, dlogits,
                             workspace, s);
    }
    // elsewhere the routing gradient is added by its own kernel
    if (e == cudaSuccess && rg)
        e = dol::launch_route_backward(logits, expert_ids, grad_combine, p.T * p.L, E, k, gate, 1,
                                       dlogits, status, s);
    return from_cuda(e);
}

do_status do_routing(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L, int32_t gate,
                     int32_t *expert_ids, float *combine, int32_t *counts,
                     int32_t *expert_offsets, int32_t *dispatch_rows, int32_t *dispatch_pos,
                     void *workspace, size_t workspace_bytes, void *stream) {
    NvtxRange nvtx("do_routing");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (gate != DO_GATE_SIGMOID_NORM && gate != DO_GATE_SOFTMAX) return DO_ERR_INVALID_ARG;
    const RouteArgs ra = {expert_ids, combine, expert_offsets, dispatch_rows, dispatch_pos};
    if ((st = check_route(p, ra)) != DO_OK) return st;
    if (!logits || !counts || !aligned(logits, 4) || !aligned(counts, 4)) return DO_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < routing_ws_bytes(p))
        return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    char *ws = static_cast<char *>(workspace);
    uint32_t *bits = reinterpret_cast<uint32_t *>(ws + dol::kWsHeader);
    const dol::RouteOut route = {expert_ids, combine, gate};
    cudaError_t e;
    int *rscratch = reinterpret_cast<int *>(ws + dol::kWsHeader + routing_bits_bytes(p));
    if (dol::signatures_fast_supported(logits, p) && route_fast_ok(&ra)) {
        // the selection kernel writes no counts: the dispatch scan takes them
        // from the signatures' popcounts (no memset between the kernels)
        const dol::ZeroSpans none = {{nullptr, nullptr, nullptr}, {0, 0, 0}};
        e = dol::launch_signatures_fast_routed(logits, p, bits, nullptr, nullptr, nullptr, none,
                                               reinterpret_cast<int *>(ws), route, s);
        if (e == cudaSuccess)
            e = dol::launch_route_dispatch(bits, expert_ids, p, expert_offsets, dispatch_rows,
                                           dispatch_pos, rscratch, s, nullptr, counts);
        return from_cuda(e);
    }
    e = dol::launch_signatures(logits, p, bits, counts, s, route);
    if (e == cudaSuccess)
        e = dol::launch_route_dispatch(bits, expert_ids, p, expert_offsets, dispatch_rows,
                                       dispatch_pos, rscratch, s);
    return from_cuda(e);
}

do_status do_route_backward(const float *logits, const int32_t *expert_ids,
                            const float *grad_combine, int64_t T, int32_t E, int32_t k, int32_t L,
                            int32_t gate, int32_t accumulate, float *dlogits,
                            int32_t *status_flags, void *stream) {
    NvtxRange nvtx("do_route_backward");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (gate != DO_GATE_SIGMOID_NORM && gate != DO_GATE_SOFTMAX) return DO_ERR_INVALID_ARG;
    if (accumulate != 0 && accumulate != 1) return DO_ERR_INVALID_ARG;
    if (!logits || !expert_ids || !grad_combine || !dlogits) return DO_ERR_INVALID_ARG;
    if (!aligned(logits, 4) || !aligned(expert_ids, 4) || !aligned(grad_combine, 4) ||
        !aligned(dlogits, 4) || (status_flags && !aligned(status_flags, 4)))
        return DO_ERR_INVALID_ARG;
    return from_cuda(dol::launch_route_backward(logits, expert_ids, grad_combine, p.T * p.L, E, k,
                                                gate, accumulate, dlogits, status_flags,
                                                (cudaStream_t)stream));
}

size_t do_routing_workspace_size(int64_t T, int32_t E, int32_t k, int32_t L) {
    Problem p;
    if (check_sizes(T, E, k, L, &p) != DO_OK) return 0;
    return routing_ws_bytes(p);
}

size_t do_workspace_size(int64_t T, int32_t E, int32_t k, int32_t L) {
    Problem p;
    if (check_sizes(T, E, k, L, &p) != DO_OK) return 0;
    return dol::workspace_bytes_plain(p);
}

size_t do_routed_workspace_size(int64_t T, int32_t E, int32_t k, int32_t L) {
    Problem p;
    if (check_sizes(T, E, k, L, &p) != DO_OK) return 0;
    return dol::workspace_bytes(p);
}

do_status do_device_status(void *workspace, void *stream) {
    if (!workspace || !aligned(workspace, 256)) return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    int flags = 0;
    cudaError_t e = cudaMemcpyAsync(&flags, workspace, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(workspace, 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return DO_ERR_CUDA;
    if (flags & dol::kDevTimeout) return DO_ERR_TIMEOUT;
    if (flags & dol::kDevOverflow) return DO_ERR_OVERFLOW;
    if (flags & dol::kDevBadId) return DO_ERR_INVALID_ARG;
    return DO_OK;
}

size_t do_host_buffer_size(int64_t T, int32_t E, int32_t k, int32_t L) {
    Problem p;
    if (check_sizes(T, E, k, L, &p) != DO_OK) return 0;
    return host_layout(p).total;
}

do_status do_forward_backward_host(const float *h_logits, int64_t T, int32_t E, int32_t k,
                                   int32_t L, int32_t gate, float grad_scale, float *h_loss,
                                   float *h_dlogits, int32_t *h_counts, int32_t *h_D,
                                   void *device_buffer, size_t device_buffer_bytes, void *stream) {
    NvtxRange nvtx("do_forward_backward_host");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!h_logits || !h_loss) return DO_ERR_INVALID_ARG;
    const HostBufLayout b = host_layout(p);
    if (!device_buffer || !aligned(device_buffer, 256) || device_buffer_bytes < b.total)
        return DO_ERR_WORKSPACE;
    char *base = static_cast<char *>(device_buffer);
    float *d_logits = reinterpret_cast<float *>(base + b.logits);
    uint32_t *d_bits = reinterpret_cast<uint32_t *>(base + b.bits);
    int32_t *d_counts = reinterpret_cast<int32_t *>(base + b.counts);
    int32_t *d_D = reinterpret_cast<int32_t *>(base + b.D);
    float *d_loss = reinterpret_cast<float *>(base + b.loss);
    // the gradient is always computed (into the device buffer); it is copied to
    // the host only when h_dlogits is given
    float *d_dlogits = reinterpret_cast<float *>(base + b.dlogits);
    void *ws = base + b.ws;
    cudaStream_t s = (cudaStream_t)stream;
    const size_t te = sizeof(float) * (size_t)p.L * p.T * p.E;

    // A cleared status word, so that the check below sees this call only.
    cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(d_logits, h_logits, te, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return DO_ERR_CUDA;
    // the status word of this call lands right after the loss (fused path)
    int *d_status = reinterpret_cast<int *>(d_loss + p.L);
    bool status_done = false;
    st = forward_backward_impl(d_logits, T, E, k, L, gate, grad_scale, d_bits, d_counts, d_D,
                               d_loss, nullptr, d_dlogits, ws, dol::workspace_bytes_plain(p), stream,
                               d_status, &status_done);
    if (st != DO_OK) return st;
    if (status_done && !h_dlogits && !h_counts && !h_D) {
        // one copy: the loss and the status word behind it
        struct {
            float v[64];
            int pad;
        } small;
        const size_t n = sizeof(float) * p.L + sizeof(int);
        if (p.L <= 63) {
            e = cudaMemcpyAsync(&small, d_loss, n, cudaMemcpyDeviceToHost, s);
            if (e == cudaSuccess) e = cudaStreamSynchronize(s);
            if (e != cudaSuccess) return DO_ERR_CUDA;
            std::memcpy(h_loss, small.v, sizeof(float) * p.L);
            int flags = 0;
            std::memcpy(&flags, reinterpret_cast<const char *>(&small) + sizeof(float) * p.L,
                        sizeof(int));
            if (flags & dol::kDevTimeout) return DO_ERR_TIMEOUT;
            if (flags & dol::kDevOverflow) return DO_ERR_OVERFLOW;
            return DO_OK;
        }
    }
    e = cudaMemcpyAsync(h_loss, d_loss, sizeof(float) * p.L, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && h_dlogits)
        e = cudaMemcpyAsync(h_dlogits, d_dlogits, te, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && h_counts)
        e = cudaMemcpyAsync(h_counts, d_counts, sizeof(int32_t) * (size_t)p.L * p.E,
                            cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && h_D)
        e = cudaMemcpyAsync(h_D, d_D, sizeof(int32_t) * (size_t)p.L * p.E * p.E,
                            cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return DO_ERR_CUDA;
    return do_device_status(ws, stream);
}

do_status do_forward_backward_host_async(const float *h_logits, int64_t T, int32_t E, int32_t k,
                                         int32_t L, int32_t gate, float grad_scale,
                                         void *h_result, void *device_buffer,
                                         size_t device_buffer_bytes, void *stream) {
    NvtxRange nvtx("do_forward_backward_host_async");
    Problem p;
    do_status st = check_sizes(T, E, k, L, &p);
    if (st != DO_OK) return st;
    if (!h_logits || !h_result || !aligned(h_result, 4)) return DO_ERR_INVALID_ARG;
    const HostBufLayout b = host_layout(p);
    if (!device_buffer || !aligned(device_buffer, 256) || device_buffer_bytes < b.total)
        return DO_ERR_WORKSPACE;
    char *base = static_cast<char *>(device_buffer);
    float *d_logits = reinterpret_cast<float *>(base + b.logits);
    float *d_loss = reinterpret_cast<float *>(base + b.loss);
    int *d_status = reinterpret_cast<int *>(d_loss + p.L);
    void *ws = base + b.ws;
    cudaStream_t s = (cudaStream_t)stream;
    const size_t te = sizeof(float) * (size_t)p.L * p.T * p.E;
    // a cleared status word: the result of this call reports this call only
    cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(d_logits, h_logits, te, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return DO_ERR_CUDA;
    bool status_done = false;
    st = forward_backward_impl(d_logits, T, E, k, L, gate, grad_scale,
                               reinterpret_cast<uint32_t *>(base + b.bits),
                               reinterpret_cast<int32_t *>(base + b.counts),
                               reinterpret_cast<int32_t *>(base + b.D), d_loss, nullptr,
                               reinterpret_cast<float *>(base + b.dlogits), ws,
                               dol::workspace_bytes_plain(p), stream, d_status, &status_done);
    if (st != DO_OK) return st;
    // outside the fused path the status word stays in the workspace: put it
    // behind the losses, so that one copy returns both
    if (!status_done) e = cudaMemcpyAsync(d_status, ws, sizeof(int), cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h_result, d_loss, sizeof(float) * p.L + sizeof(int),
                            cudaMemcpyDeviceToHost, s);
    return from_cuda(e);
}

const char *do_status_string(int32_t status) {
    switch (status) {
        case DO_OK: return "ok";
        case DO_ERR_INVALID_ARG: return "invalid argument (null pointer, size or alignment)";
        case DO_ERR_UNSUPPORTED: return "valid arguments outside this build's limits";
        case DO_ERR_CUDA: return "a CUDA runtime call or kernel launch failed";
        case DO_ERR_TIMEOUT: return "a bounded device wait ran out";
        case DO_ERR_OVERFLOW: return "a row sum of the Hamming matrix does not fit int32";
        case DO_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        default: return "unknown status";
    }
}

}  // extern "C"
