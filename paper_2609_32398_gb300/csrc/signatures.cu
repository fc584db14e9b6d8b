// Step 1: Top-K routing packed into binary load signatures, with counts.
//   f_it = 1(i in Top-K(x_t))   (Sec. 3.1.1, Eq. 1)
//   n_i  = ||F_i||_1            (App. C.3)
// Top-K is taken on the raw fp32 logits; equal values go to the lower expert
// index.  A warp owns 32 consecutive tokens, i.e. one 32-bit word of every
// signature, so no two warps ever write the same word.  With routing outputs
// the kernel also writes each token's chosen experts in selection order and
// their weights re-normalized over the chosen set (Sec. 3.1.1).
#include <climits>
#include <cmath>

#include "dol_internal.cuh"

namespace dol {
namespace {

constexpr int kSigThreads = 256;

// Generic path, any 1 <= k <= E <= 1024.  Lanes hold experts i = lane + 32 r
// (r < R); every token takes k rounds of a warp-wide argmax under the order
// (value descending, index ascending).
template <int R>
__global__ void __launch_bounds__(kSigThreads)
sig_generic_kernel(const float *__restrict__ logits, int64_t T, int E, int k, int64_t W,
                   uint32_t *__restrict__ bits, int *__restrict__ counts, RouteOut route) {
    __shared__ int s_cnt[32 * R];
    const int layer = blockIdx.y;
    const float *z = logits + (int64_t)layer * T * E;
    uint32_t *b = bits + (int64_t)layer * E * W;
    for (int i = threadIdx.x; i < 32 * R; i += blockDim.x) s_cnt[i] = 0;
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    int cnt[R];
#pragma unroll
    for (int r = 0; r < R; ++r) cnt[r] = 0;

    for (int64_t w = (int64_t)blockIdx.x * nwarps + warp; w < W; w += (int64_t)gridDim.x * nwarps) {
        uint32_t word[R];
#pragma unroll
        for (int r = 0; r < R; ++r) word[r] = 0u;
        const int64_t t0 = w * 32;
        const int nt = (int)min64(32, T - t0);
        for (int tt = 0; tt < nt; ++tt) {
            const float *zt = z + (t0 + tt) * E;
            // routing outputs of this token: ids in selection order, and the
            // chosen logits parked in combine until the weights replace them
            const int64_t roff = ((int64_t)layer * T + t0 + tt) * k;
            float v[R];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int i = lane + 32 * r;
                v[r] = (i < E) ? __ldg(zt + i) : 0.0f;
            }
            uint32_t sel = 0u;  // bit r: expert lane + 32 r is selected
            for (int q = 0; q < k; ++q) {
                float bv = 0.0f;
                int bi = INT_MAX;  // INT_MAX: no candidate in this lane
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int i = lane + 32 * r;
                    const bool ok = (i < E) && !((sel >> r) & 1u);
                    if (ok && (bi == INT_MAX || v[r] > bv)) { bv = v[r]; bi = i; }
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const float ov = __shfl_xor_sync(kFull, bv, o);
                    const int oi = __shfl_xor_sync(kFull, bi, o);
                    const bool take = oi != INT_MAX &&
                                      (bi == INT_MAX || ov > bv || (ov == bv && oi < bi));
                    if (take) { bv = ov; bi = oi; }
                }
                if ((bi & 31) == lane) sel |= 1u << (bi >> 5);
                if (route.ids && lane == 0) {
                    route.ids[roff + q] = bi;
                    route.combine[roff + q] = bv;
                }
            }
            if (route.ids) {
                // w_q = u_q / sum u over the chosen set (u: route_raw_weight);
                // the lane-strided sum and the butterfly fix the order
                __syncwarp();
                float *ct = route.combine + roff;
                const float v0 = ct[0];
                float part = 0.0f;
                for (int q = lane; q < k; q += 32) part += route_raw_weight(ct[q], v0, route.gate);
                const float sum = warp_sum(part);
                __syncwarp();
                for (int q = lane; q < k; q += 32) ct[q] = route_raw_weight(ct[q], v0, route.gate) / sum;
            }
#pragma unroll
            for (int r = 0; r < R; ++r) word[r] |= ((sel >> r) & 1u) << tt;
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int i = lane + 32 * r;
            if (i < E) {
                b[(int64_t)i * W + w] = word[r];
                cnt[r] += __popc(word[r]);
            }
        }
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int i = lane + 32 * r;
        if (i < E && cnt[r]) atomicAdd(&s_cnt[i], cnt[r]);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < E; i += blockDim.x)
        if (s_cnt[i]) atomicAdd(&counts[(int64_t)layer * E + i], s_cnt[i]);
}

template <int R>
cudaError_t run_generic(const float *logits, const Problem &p, uint32_t *bits, int *counts,
                        const RouteOut &route, cudaStream_t s) {
    const int warps = kSigThreads / 32;
    int64_t blocks = (p.W + warps - 1) / warps;
    const int64_t cap = (p.L >= 1024) ? 1 : (2048 / p.L);
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    dim3 grid((unsigned)blocks, (unsigned)p.L);
    sig_generic_kernel<R><<<grid, kSigThreads, 0, s>>>(logits, p.T, p.E, p.k, p.W, bits, counts,
                                                             route);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_signatures(const float *logits, const Problem &p, uint32_t *bits, int *counts,
                              cudaStream_t s, const RouteOut &route) {
    cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int) * (size_t)p.L * p.E, s);
    if (e != cudaSuccess) return e;
    if (!route.ids && signatures_fast256_supported(logits, p)) {
        const ZeroSpans none = {{nullptr, nullptr, nullptr}, {0, 0, 0}};
        return launch_signatures_fast256(logits, p, bits, counts, nullptr, none, nullptr, s);
    }
    const int r = (p.E + 31) / 32;
    if (r <= 1) return run_generic<1>(logits, p, bits, counts, route, s);
    if (r <= 2) return run_generic<2>(logits, p, bits, counts, route, s);
    if (r <= 4) return run_generic<4>(logits, p, bits, counts, route, s);
    if (r <= 8) return run_generic<8>(logits, p, bits, counts, route, s);
    if (r <= 16) return run_generic<16>(logits, p, bits, counts, route, s);
    return run_generic<32>(logits, p, bits, counts, route, s);
}

}  // namespace dol
