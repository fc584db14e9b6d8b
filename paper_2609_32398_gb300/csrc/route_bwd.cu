// Backward of the routing combine weights (Sec. 3.1.1): the chosen experts'
// probabilities re-normalized to sum to one, w_tq = p_{e_q,t} / sum_q' p_{e_q',t},
// differentiated with the selection held fixed.  With g_tq the upstream
// gradient of w_tq and dot_t = sum_q g_tq w_tq, for a chosen expert l
//   sigmoid-norm: dz_tl = w_tl (1 - s_tl) (g_tl - dot_t)   (w = s / sum of the chosen s)
//   softmax:      dz_tl = w_tl (g_tl - dot_t)             (w = softmax of the chosen z)
// and zero for the experts not chosen (the dense normaliser of p cancels).
//
// One group of G = pow2ceil(min(k, 32)) lanes per token row, 32/G rows per
// warp pass, so that the row's sums are G-lane butterfly shuffles.  Only the
// k chosen logits are read (gathers); the weights are recomputed from them as
// the forward selection kernel does (the largest chosen logit v0 as the
// shift), so nothing of the forward pass has to be kept.  Rows of all
// problems are independent and the kernels run over the L*T rows as one flat
// range.  With k <= 32 a lane holds one choice of kU rows at once (all loads
// of a pass in flight together); beyond that it loops over the choices
// q = j, j+G, ... of one row.
//
// DRAM moves whole lines: the gathers bring in most of each 512-byte logits
// row at E = 128, k = 8 (measured: about 530 bytes per row with the ids and
// the gradient).  Staging full rows in shared memory with 16-byte async
// copies, and writing dlogits back from there as whole lines, moved the same
// bytes more slowly (fewer warps resident per SM), so the gathers stay.
#include <algorithm>
#include <atomic>

#include "dol_internal.cuh"

namespace dol {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float group_sum(float v, int G) {
    for (int o = G >> 1; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

__device__ __forceinline__ float group_max(float v, int G) {
    for (int o = G >> 1; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

// accumulate = 0: the rows are overwritten (zeros, then the chosen entries);
// accumulate = 1: the chosen entries are added in place (RED.ADD; one
// contribution per entry when the ids of a row are distinct, hence the same
// sum every run).  skip (accumulate only, may be null): rows r of problems
// r / layer_rows whose flag is nonzero are left alone (their gradient was
// added by the tensor-core loss kernel).
__global__ void __launch_bounds__(kThreads)
route_backward_kernel(const float *__restrict__ z, const int32_t *__restrict__ ids,
                      const float *__restrict__ g, int64_t rows, int32_t E, int32_t k, int32_t G,
                      int32_t gate, int32_t accumulate, float *__restrict__ dz,
                      int32_t *status_flags, const int *__restrict__ skip, int64_t layer_rows) {
    const int lane = threadIdx.x & 31;
    const int per_pass = 32 / G;
    const int j = lane & (G - 1);
    const int64_t warp = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
    const bool vec4 = (E & 3) == 0 && (reinterpret_cast<uintptr_t>(dz) & 15) == 0;
    int bad = 0;
    for (int64_t base = warp * per_pass; base < rows; base += nwarps * per_pass) {
        const int64_t r = base + lane / G;
        const bool live = r < rows && !(skip && __ldg(skip + r / layer_rows) != 0);
        const float *zr = z + (live ? r : 0) * (int64_t)E;
        const int32_t *ir = ids + (live ? r : 0) * (int64_t)k;
        const float *gr = g + (live ? r : 0) * (int64_t)k;
        // pass 1: the shift v0 = the largest chosen logit of the row
        float v0 = -INFINITY;
        for (int q = j; q < k; q += G) {
            if (!live) break;
            const int e = __ldg(ir + q);
            if ((unsigned)e < (unsigned)E) v0 = fmaxf(v0, __ldg(zr + e));
        }
        v0 = group_max(v0, G);
        // pass 2: sum of the raw weights and of g times them
        float sraw = 0.0f, sgraw = 0.0f;
        for (int q = j; q < k; q += G) {
            if (!live) break;
            const int e = __ldg(ir + q);
            if ((unsigned)e >= (unsigned)E) { bad = 1; continue; }
            const float raw = route_raw_weight(__ldg(zr + e), v0, gate);
            sraw += raw;
            sgraw += __ldg(gr + q) * raw;
        }
        sraw = group_sum(sraw, G);
        sgraw = group_sum(sgraw, G);
        const float inv = 1.0f / sraw;
        const float dot = sgraw * inv;
        if (!accumulate) {
            // zero the rows of this pass: consecutive rows, one contiguous span
            const int64_t nrows = min((int64_t)per_pass, rows - base);
            float *span = dz + base * (int64_t)E;
            const int64_t n = nrows * (int64_t)E;
            if (vec4) {
                float4 *s4 = reinterpret_cast<float4 *>(span);
                for (int64_t i = lane; i < n / 4; i += 32) s4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            } else {
                for (int64_t i = lane; i < n; i += 32) span[i] = 0.0f;
            }
            __syncwarp();
        }
        for (int q = j; q < k; q += G) {
            if (!live) break;
            const int e = __ldg(ir + q);
            if ((unsigned)e >= (unsigned)E) continue;
            const float v = __ldg(zr + e);
            float d = route_raw_weight(v, v0, gate) * inv * (__ldg(gr + q) - dot);
            if (gate == 0) d *= 1.0f / (1.0f + expf(v));   // 1 - sigmoid(v)
            float *dst = dz + r * (int64_t)E + e;
            if (accumulate) atomicAdd(dst, d);
            else *dst = d;
        }
        __syncwarp();
    }
    if (bad && status_flags) atomicOr(status_flags, 4);
}

// k <= 32: one choice per lane, and each lane group takes kU rows of the
// warp's span at once, so that every load of a pass is issued before the
// first is used (the ids and gradients together, then the kU gathers): two
// memory round trips per pass.  The warp's span is kU * (32 / G) consecutive
// rows; in the overwrite mode it is zeroed while the loads are in flight.
template <int kU>
__global__ void __launch_bounds__(kThreads)
route_backward_small_k(const float *__restrict__ z, const int32_t *__restrict__ ids,
                       const float *__restrict__ g, int64_t rows, int32_t E, int32_t k,
                       int32_t G, int32_t gate, int32_t accumulate, float *__restrict__ dz,
                       int32_t *status_flags, const int *__restrict__ skip, int64_t layer_rows) {
    const int lane = threadIdx.x & 31;
    const int per_pass = 32 / G;
    const int j = lane & (G - 1);
    const int grp = lane / G;
    const bool has_q = j < k;
    const int64_t span_rows = (int64_t)kU * per_pass;
    const int64_t warp = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
    const bool vec4 = (E & 3) == 0 && (reinterpret_cast<uintptr_t>(dz) & 15) == 0;
    int bad = 0;
    for (int64_t base = warp * span_rows; base < rows; base += nwarps * span_rows) {
        int e[kU];
        float gq[kU], v[kU];
        unsigned present = 0;   // bit u: this lane holds a choice of a row in range
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int64_t r = base + (int64_t)u * per_pass + grp;
            const bool on = has_q && r < rows && !(skip && __ldg(skip + r / layer_rows) != 0);
            present |= on ? 1u << u : 0u;
            e[u] = on ? __ldg(ids + r * k + j) : 0;
            gq[u] = on ? __ldg(g + r * k + j) : 0.0f;
        }
        if (!accumulate) {
            const int64_t n = min(span_rows, rows - base) * (int64_t)E;
            float *span = dz + base * (int64_t)E;
            if (vec4) {
                float4 *s4 = reinterpret_cast<float4 *>(span);
                for (int64_t i = lane; i < n / 4; i += 32) s4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            } else {
                for (int64_t i = lane; i < n; i += 32) span[i] = 0.0f;
            }
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int64_t r = base + (int64_t)u * per_pass + grp;
            if (!((present >> u) & 1u)) e[u] = -1;
            const bool ok = (unsigned)e[u] < (unsigned)E;
            if (((present >> u) & 1u) && !ok) bad = 1;
            v[u] = ok ? __ldg(z + r * (int64_t)E + e[u]) : -INFINITY;
        }
        float v0[kU], raw[kU], sr[kU], sg[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) v0[u] = group_max(v[u], G);
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const bool ok = (unsigned)e[u] < (unsigned)E;
            raw[u] = ok ? route_raw_weight(v[u], v0[u], gate) : 0.0f;
            sr[u] = group_sum(raw[u], G);
            sg[u] = group_sum(gq[u] * raw[u], G);
        }
        if (!accumulate) __syncwarp();
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            if ((unsigned)e[u] >= (unsigned)E) continue;
            const int64_t r = base + (int64_t)u * per_pass + grp;
            const float inv = 1.0f / sr[u];
            float d = raw[u] * inv * (gq[u] - sg[u] * inv);
            if (gate == 0) d *= 1.0f / (1.0f + expf(v[u]));   // 1 - sigmoid(v)
            float *dst = dz + r * (int64_t)E + e[u];
            if (accumulate) atomicAdd(dst, d);
            else *dst = d;
        }
        __syncwarp();
    }
    if (bad && status_flags) atomicOr(status_flags, 4);
}

}  // namespace

namespace {

// Grid of a grid-stride kernel: the warps it needs, capped at the blocks
// resident on the device at once (computed once per device and kernel; the
// kernel's dynamic shared memory is fixed).
template <auto Kern>
cudaError_t grid_for(size_t smem, int64_t warps, int *blocks) {
    static std::atomic<int> cap_of[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int cap = dev < 64 ? cap_of[dev].load() : 0;
    if (cap == 0) {
        int sms = 0, per_sm = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess && smem > 48 * 1024) e = ensure_smem_limit<Kern>(smem);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, Kern, kThreads, smem);
        if (e != cudaSuccess) return e;
        cap = sms * std::max(1, per_sm);
        if (dev < 64) cap_of[dev].store(cap);
    }
    const int64_t want = (warps * 32 + kThreads - 1) / kThreads;
    *blocks = (int)std::max<int64_t>(1, std::min<int64_t>(want, cap));
    return cudaSuccess;
}

}  // namespace

cudaError_t launch_route_backward(const float *z, const int32_t *ids, const float *g, int64_t rows,
                                  int32_t E, int32_t k, int32_t gate, int32_t accumulate,
                                  float *dz, int32_t *status_flags, cudaStream_t s,
                                  const int *skip, int64_t layer_rows) {
    constexpr int kU = 4;
    if (skip && (!accumulate || layer_rows < 1)) return cudaErrorInvalidValue;
    int G = 1;
    while (G < k && G < 32) G <<= 1;
    const int64_t per_warp = (k <= 32 ? kU : 1) * (int64_t)(32 / G);
    const int64_t warps = (rows + per_warp - 1) / per_warp;
    int blocks = 0;
    cudaError_t e = k <= 32 ? grid_for<route_backward_small_k<kU>>(0, warps, &blocks)
                            : grid_for<route_backward_kernel>(0, warps, &blocks);
    if (e != cudaSuccess) return e;
    if (k <= 32)
        route_backward_small_k<kU><<<blocks, kThreads, 0, s>>>(
            z, ids, g, rows, E, k, G, gate, accumulate, dz, status_flags, skip, layer_rows);
    else
        route_backward_kernel<<<blocks, kThreads, 0, s>>>(z, ids, g, rows, E, k, G, gate,
                                                          accumulate, dz, status_flags, skip,
                                                          layer_rows);
    return cudaGetLastError();
}

}  // namespace dol
