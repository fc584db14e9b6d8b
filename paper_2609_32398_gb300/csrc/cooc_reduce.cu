// Reduction of the per-CTA co-occurrence triangles of the fused path.
//   c_ab = sum_t f_at f_bt, c_aa = n_a, and the Hamming distance
//   D_ab = n_a + n_b - 2 c_ab                                   (App. C.3)
// The counts n_a were already summed (one atomic per expert and CTA) by the
// signatures kernel.  A CTA owns 32 consecutive triangle words; its 32 warps
// each sum a strided subset of the partials with independent loads, and the
// 32 warp sums are added in a fixed order, so D is an exact integer result
// independent of scheduling.  The kernel writes both halves of the symmetric
// D and the counts.
#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kRedWarps = 32;
constexpr int kRedThreads = kRedWarps * 32;

template <int E>
__global__ void __launch_bounds__(kRedThreads)
cooc_reduce_kernel(const uint32_t *__restrict__ partials, int P1, const int *__restrict__ n_acc,
                   int *__restrict__ D, int *__restrict__ counts) {
    constexpr int kWords = cooc_row_offset<E>(E);
    __shared__ uint32_t s_sum[kRedWarps][33];
    const int e = threadIdx.x & 31, wp = threadIdx.x >> 5;
    const int word = blockIdx.x * 32 + e;
    const int layer = blockIdx.y;
    pdl_wait();
    pdl_trigger();
    uint32_t acc[4] = {0u, 0u, 0u, 0u};
    if (word < kWords) {
        const uint32_t *base = partials + (size_t)layer * P1 * kWords + word;
        for (int p0 = wp; p0 < P1; p0 += 4 * kRedWarps) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int p = p0 + u * kRedWarps;
                if (p < P1) acc[u] += __ldg(base + (size_t)p * kWords);
            }
        }
    }
    s_sum[wp][e] = acc[0] + acc[1] + acc[2] + acc[3];
    __syncthreads();
    if (wp != 0 || word >= kWords) return;
    uint32_t c = 0;
#pragma unroll
    for (int q = 0; q < kRedWarps; ++q) c += s_sum[q][e];
    // word -> (a, b): the row whose offset range holds it
    int lo = 0, hi = E - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (cooc_row_offset<E>(mid) <= word) lo = mid;
        else hi = mid - 1;
    }
    const int a = lo;
    const int b = (a & ~3) + (word - cooc_row_offset<E>(a));
    if (b < a) return;  // alignment padding of row a
    const int *nl = n_acc + (size_t)layer * E;
    int *Dl = D + (size_t)layer * E * E;
    if (a == b) {
        Dl[a * E + a] = 0;
        counts[(size_t)layer * E + a] = (int)c;
    } else {
        const int d = nl[a] + nl[b] - 2 * (int)c;
        Dl[a * E + b] = d;
        Dl[b * E + a] = d;
    }
}

template <int E>
cudaError_t run_reduce(const uint32_t *partials, int P1, const int *n_acc, const Problem &p, int *D,
                       int *counts, cudaStream_t s) {
    constexpr int kWords = cooc_row_offset<E>(E);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((kWords + 31) / 32, (unsigned)p.L);
    cfg.blockDim = dim3(kRedThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, cooc_reduce_kernel<E>, partials, P1, n_acc, D, counts);
}

}  // namespace

cudaError_t launch_cooc_reduce(const uint32_t *partials, int P1, const int *n_acc, const Problem &p,
                               int *D, int *counts, cudaStream_t s) {
    if (p.E == 32) return run_reduce<32>(partials, P1, n_acc, p, D, counts, s);
    if (p.E == 64) return run_reduce<64>(partials, P1, n_acc, p, D, counts, s);
    if (p.E == 128) return run_reduce<128>(partials, P1, n_acc, p, D, counts, s);
    return cudaErrorInvalidValue;
}

}  // namespace dol
