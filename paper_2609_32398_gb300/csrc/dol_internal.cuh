// Internal declarations shared by the kernels and the C ABI of libdoloss.
// Nothing here is part of the public interface (include/doloss.h is).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <atomic>

namespace dol {

constexpr unsigned kFull = 0xffffffffu;

// Bits of the device status word kept at the start of the workspace.
constexpr int kDevOverflow = 1;  // a row sum of D did not fit int32
constexpr int kDevTimeout = 2;   // a bounded device wait ran out
constexpr int kDevBadId = 4;     // an expert id given to a backward call was outside [0, E)

// Workspace layout: [status word | pad to 256 B | fp64 loss partials [L][P]].
constexpr size_t kWsHeader = 256;

// Problem description handed from the C ABI to the launchers.
struct Problem {
    int64_t T;    // tokens per problem (the paper's m)
    int E;        // experts (n)
    int k;        // experts selected per token (K)
    int L;        // independent problems in the batch
    int64_t W;    // 32-bit words per signature, ceil(T/32)
};

// Routing outputs written by the selection pass (Sec. 3.1.1); ids == nullptr
// means none.  Both arrays are [L][T][k], one row per token, the chosen
// experts in selection order (largest logit first, equal logits lower index
// first) with their re-normalized weights.
struct RouteOut {
    int *ids;
    float *combine;
    int gate;  // 0 sigmoid-norm, 1 softmax
};

// Raises kernel Kern's dynamic shared-memory limit to `bytes` on the current
// device.  The attribute belongs to the device's context, so it is set once
// per device (devices 0..63), not once per process.
template <auto Kern>
inline cudaError_t ensure_smem_limit(size_t bytes) {
    static std::atomic<unsigned long long> done{0ull};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = dev < 64 ? 1ull << dev : 0ull;
    if (bit && (done.load() & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(Kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) done.fetch_or(bit);
    return e;
}

// Up to three int ranges that a kernel clears for the kernels after it.
struct ZeroSpans {
    int *p[3];
    int64_t n[3];
};

// Workspace of the loss step, carved from the caller's buffer:
//   [0, 256)        device status word (kDevOverflow | kDevTimeout | kDevBadId bits)
//   done            [L] int, per-problem count of finished loss CTAs
//   partials        [L][max CTAs per problem] fp64 sums of A_t
//   idx             [L][T][k] uint8, the selected experts of every token
//   cooc_parts      [L][P1][triangle words] uint32, per-CTA co-occurrence counts
//   n_acc           [L][E] int32, counts summed by the signatures CTAs (kept at
//                   zero between calls: the loss kernel clears it after use)
//   bimg            [L][kBImageBytes], the fp16 image of D' (E = 128 only)
//   img_ok          [L] int32, 1 where the image of a given (summed) D is exact
//   route_base      route_scratch_ints int32, scratch of the dispatch order
struct WsLayout {
    size_t done, partials, idx, cooc_parts, n_acc, bimg, img_ok, route_base, total;
    int max_parts;  // partial slots per problem
};
// Signatures CTAs per problem on the fast path: min(SMs, kMaxSigCtas) / L.
constexpr int kMaxSigCtas = 256;
int max_sig_ctas_per_problem(const Problem &p);
WsLayout ws_layout(const Problem &p);
inline size_t workspace_bytes(const Problem &p) { return ws_layout(p).total; }
// What a call without routing outputs needs: the layout up to the routing scratch.
inline size_t workspace_bytes_plain(const Problem &p) { return ws_layout(p).route_base; }

// Number of generic loss-kernel CTAs per problem; fixes the partial-sum
// layout and therefore the reduction order.
int loss_blocks_per_problem(const Problem &p);

// Launchers (return the first CUDA error, cudaSuccess otherwise).
// route.ids != nullptr: the routing outputs are written too.
cudaError_t launch_signatures(const float *logits, const Problem &p, uint32_t *bits,
                              int *counts, cudaStream_t s,
                              const RouteOut &route = RouteOut{nullptr, nullptr, 0});
cudaError_t launch_hamming(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s);
// The fast selection at E = 256 (k in {1, 2, 4, 8}, 16-byte aligned logits):
// signatures and counts (counts zero on entry), no co-occurrence; idx (may be
// null) the chosen experts of every token; zero: ranges cleared for the
// kernels after it; status (may be null): the device status word.
bool signatures_fast256_supported(const float *logits, const Problem &p);
cudaError_t launch_signatures_fast256(const float *logits, const Problem &p, uint32_t *bits,
                                      int *counts, uint8_t *idx, const ZeroSpans &zero,
                                      int *status, cudaStream_t s);
cudaError_t launch_add_distances(const int *D, int *D_sum, int64_t n, cudaStream_t s);
cudaError_t launch_hamming_accumulate(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s);
cudaError_t launch_origin_do(const int *D, const Problem &p, long long *origin_do, cudaStream_t s);
// var [L] (fp64) = the variance of the off-diagonal entries of each problem's
// local Hamming matrix from its origin_do (App. C.1).
cudaError_t launch_offdiag_variance(const long long *origin_do, const Problem &p, double *var,
                                    cudaStream_t s);
cudaError_t launch_loss(const float *logits, const uint32_t *bits, const int *D,
                        const Problem &p, int gate, float d_scale, float grad_scale,
                        float *loss, long long *origin_do, float *dlogits, void *workspace,
                        cudaStream_t s);

// Fast paths (E in {32, 64, 128}, k in {1, 2, 4, 8}, 16-byte aligned rows).
bool signatures_fast_supported(const float *logits, const Problem &p);
cudaError_t launch_signatures_fast(const float *logits, const Problem &p, uint32_t *bits,
                                   int *counts, uint8_t *idx, uint32_t *cooc, const ZeroSpans &zero,
                                   int *status, cudaStream_t s);
// The same kernel with the routing outputs (ids and combine 16-byte aligned).
cudaError_t launch_signatures_fast_routed(const float *logits, const Problem &p, uint32_t *bits,
                                          int *counts, uint8_t *idx, uint32_t *cooc,
                                          const ZeroSpans &zero, int *status,
                                          const RouteOut &route, cudaStream_t s);
// Dispatch order of the routed (token, choice) pairs from the signatures and
// the chosen ids alone: offsets [L][E+1], rows [L][T k], pos [L][T][k] (each
// may be null).  scratch: route_scratch_ints(p) ints.  Launched as
// programmatic dependents of the previous kernel on `s`.
int64_t route_chunks(const Problem &p);
int64_t route_scratch_ints(const Problem &p);
// Backward of the combine weights to the logits over `rows` token rows
// (route_bwd.cu); status bit 2 for an id outside [0, E).  skip (with
// accumulate only; may be null): [rows / layer_rows] flags, the rows of a
// problem whose flag is nonzero are left alone.
cudaError_t launch_route_backward(const float *z, const int32_t *ids, const float *g, int64_t rows,
                                  int32_t E, int32_t k, int32_t gate, int32_t accumulate,
                                  float *dz, int32_t *status_flags, cudaStream_t s,
                                  const int *skip = nullptr, int64_t layer_rows = 0);

// n_zero (may be null): an [L][E] accumulator cleared once the kernels before
// these have finished (the scan kernel does it after its dependency wait).
// counts_out (may be null): n_e = |F_e| from the scan's popcounts.
cudaError_t launch_route_dispatch(const uint32_t *bits, const int *ids, const Problem &p,
                                  int *offsets, int *rows, int *pos, int *scratch,
                                  cudaStream_t s, int *n_zero = nullptr,
                                  int *counts_out = nullptr);
// Router-side fusion (E = 128, k in {1,2,4,8}, H a multiple of 64, 16-byte
// aligned X, W and logits): logits = X W^T on the tensor cores with the
// fused path's signature step in the epilogue (bits, selected indices,
// per-CTA co-occurrence triangles, counts accumulated into `counts`).
bool router_supported(const Problem &p, int H, const void *X, const void *Wr, const float *logits);
int router_ctas_per_problem(const Problem &p);
cudaError_t launch_router_signatures(const void *X, const void *Wr, int H, float *logits,
                                     const Problem &p, uint32_t *bits, int *counts, uint8_t *idx,
                                     uint32_t *cooc, const ZeroSpans &zero, int *status,
                                     cudaStream_t s);
bool loss_fast_supported(const Problem &p, const float *logits, const int *D, const float *dlogits);
// The E = 256 variant: counts given (D of the same tokens), T < 2^24.
bool loss_fast256_supported(const Problem &p, const float *logits, const int *D,
                            const float *dlogits);
cudaError_t launch_idx_from_bits(const uint32_t *bits, const Problem &p, uint8_t *idx, int *zero_ptr,
                                 int zero_n, cudaStream_t s);
// counts: when given, R_i = (E - 2k) n_i + T k (D local to these tokens) and
// n_zero ([L][E], may be null) is cleared once D is read; otherwise R_i is a
// column sum of D.
// Tensor-core loss path (E = 128, sigmoid-norm gate, k in {1,2,4,8}, T <= 2^22).
bool loss_mma_supported(const Problem &p, int gate, const float *logits, const int *D,
                        const float *dlogits, bool image_checked = false);
int loss_mma_ctas_per_problem(const Problem &p);
// bimg: the fp16 image of D' written by launch_cooc_reduce for these tokens
// (which also gives origin_do on this path).
cudaError_t launch_loss_mma(const float *logits, const uint8_t *idx, const unsigned char *bimg,
                            int *n_zero, const Problem &p, float d_scale, float grad_scale,
                            float *loss, float *dlogits, double *partials, int *done, int *status,
                            int *status_out, cudaStream_t s, const int *rg_ids = nullptr,
                            const float *rg_g = nullptr, const int *img_ok = nullptr);
cudaError_t launch_loss_fast(const float *logits, const uint8_t *idx, const int *D,
                             const int *counts, int *n_zero, const Problem &p, int gate,
                             float d_scale, float grad_scale, float *loss, long long *origin_do,
                             float *dlogits, double *partials, int *done, int *status,
                             int *status_out, cudaStream_t s, const int *img_ok = nullptr);

// Co-occurrence counts c_ab (a <= b) of one CTA are kept as a triangle whose
// row a holds columns (a & ~3) .. E-1, so that every row starts 16-byte
// aligned.  Offset of row a: sum over a' < a of (E - 4 floor(a'/4)).
template <int E>
__host__ __device__ constexpr int cooc_row_offset(int a) {
    return a * E - 8 * (a / 4) * (a / 4 - 1) - 4 * (a % 4) * (a / 4);
}

// The matrix D' of the tensor-core loss kernel (E = 128): D'_ab = D_ab off the
// diagonal, D'_aa = -R_a, stored as two fp16 pieces D' = 2048 hi + lo, both
// exact: off the diagonal (0 <= D <= 2^16) hi = D >> 11 and lo = D & 2047; on
// the diagonal (0 <= R < 2^23) -R = 2048 (-a) + (-b) with a = 2 round(R / 4096)
// even and |b| <= 2048.  The image is the shared-memory operand B of that
// kernel: rows n = 0..127 hold hi of column n, rows 128 + n lo, K-major with
// 128-byte swizzle (two K atoms of 64 columns, 256 rows of 128 bytes each).
constexpr int kBImageBytes = 2 * 256 * 128;
__host__ __device__ __forceinline__ uint32_t sw128_k16_offset(int row, int k, int rows) {
    const int atom = k >> 6, kc = k & 63;
    return (uint32_t)(atom * rows * 128 + row * 128 + ((((kc >> 3) ^ (row & 7))) << 4) + (kc & 7) * 2);
}
__host__ __device__ __forceinline__ void dprime_pieces(bool diag, int v, int *hi, int *lo) {
    if (diag) {  // v = R
        const int a2 = 2 * ((v + 2048) >> 12);
        *hi = -a2;
        *lo = -(v - 2048 * a2);
    } else {     // v = D
        *hi = v >> 11;
        *lo = v & 2047;
    }
}

// Writes the two fp16 pieces of D'_{n,k} (dprime_pieces) into the image at
// row n (hi) and row 128 + n (lo), column k.
__device__ __forceinline__ void put_dprime(unsigned char *img, int n, int k, bool diag, int v) {
    int h, l;
    dprime_pieces(diag, v, &h, &l);
    *reinterpret_cast<__half *>(img + sw128_k16_offset(n, k, 256)) = __int2half_rn(h);
    *reinterpret_cast<__half *>(img + sw128_k16_offset(128 + n, k, 256)) = __int2half_rn(l);
}

int sig_fast_ctas_per_problem(const Problem &p);
size_t cooc_partial_words(int E);
// bimg ([L][kBImageBytes], E = 128 only, may be null): the fp16 image of D'
// for the tensor-core loss kernel, written alongside D.  origin_do (may be
// null) must be zero on entry: sum_{a != b} D_ab^2 is added to it.
cudaError_t launch_cooc_reduce(const uint32_t *partials, int P1, const int *n_acc, const Problem &p,
                               int *D, int *counts, unsigned char *bimg, long long *origin_do,
                               cudaStream_t s);
// The image of D' from a given [L][128][128] matrix D (summed over ranks or
// micro-batches), and img_ok [L] = 1 where its two fp16 pieces are exact.
cudaError_t launch_dprime_image(const int *D, const Problem &p, unsigned char *bimg, int *img_ok,
                                cudaStream_t s);

// ---------------------------------------------------------------- device helpers

// p advanced to the next multiple of A bytes of the shared window.  The offset
// is added to p itself (no round trip through an integer), so the compiler
// keeps every access through the result in the shared state space instead of
// turning it into a generic access.
template <uint32_t A>
__device__ __forceinline__ unsigned char *smem_align(unsigned char *p) {
    const uint32_t off = static_cast<uint32_t>(__cvta_generic_to_shared(p));
    return p + ((A - (off & (A - 1u))) & (A - 1u));
}

__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

// Sum of x[0..n) in a fixed order by the first nthreads (a power of two) of a block:
// thread i adds x[i], x[i + nthreads], ... in turn, then a fixed tree joins
// the thread sums.  The result (valid in thread 0) does not depend on timing.
// red must hold nthreads doubles.  Called by every thread of the block.
__device__ __forceinline__ double block_sum_fixed(const double *x, int64_t n, double *red,
                                                  int nthreads) {
    double s = 0.0;
    if ((int)threadIdx.x < nthreads) {
        for (int64_t i = threadIdx.x; i < n; i += nthreads) s += __ldcg(x + i);
        red[threadIdx.x] = s;
    }
    __syncthreads();
    for (int o = nthreads / 2; o > 0; o >>= 1) {
        if ((int)threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    return red[0];
}

// Sum of x[0..n) by one full warp in a fixed order: lane l adds x[l],
// x[l + 32], ... in turn, then a fixed butterfly joins the lane sums.  The
// result (in every lane) does not depend on timing.
__device__ __forceinline__ double warp_sum_fixed(const double *x, int64_t n) {
    const int lane = threadIdx.x & 31;
    double s = 0.0;
    for (int64_t i = lane; i < n; i += 32) s += __ldcg(x + i);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
    return s;
}

// Weight of a chosen expert before the re-normalization over the chosen set
// (Sec. 3.1.1), for a token whose first chosen logit (the largest) is v0:
//   softmax        exp(v - v0)                       (= p_v / p_v0)
//   sigmoid-norm   sigmoid(v)                        if v0 >= 0
//                  exp(v - v0) (1 + e^v0) / (1 + e^v) if v0 < 0 (= s_v / s_v0)
// The dense normaliser cancels in the ratio.  The two sigmoid forms are equal
// in exact arithmetic; the second keeps every chosen weight away from
// underflow when all chosen logits are very negative.
__device__ __forceinline__ float route_raw_weight(float v, float v0, int gate) {
    if (gate == 1) return expf(v - v0);
    if (v0 >= 0.0f) return 1.0f / (1.0f + expf(-v));
    return expf(v - v0) * ((1.0f + expf(v0)) / (1.0f + expf(v)));
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

}  // namespace dol
