// Routing outputs (Sec. 3.1.1): the router keeps, of each token's normalized
// probabilities, only the K chosen ones and re-normalizes them; these weigh
// the chosen experts' outputs.  The selection pass that builds the signatures
// writes the chosen experts and those weights (the kRoute instantiations of
// the kernel in sig_fast.cuh, or the generic kernel); this file launches them
// and holds the dispatch kernel, which puts the routed (token, choice) pairs
// in expert order:
//   offsets[e] = n_0 + ... + n_{e-1}, offsets[E] = T k
//   rows[offsets[e] + r] = the r-th token (ascending) routed to expert e
//   pos[t][q] = the row of the pair (t, q), so rows[pos[t][q]] = t.
// The rank of token t among expert e's tokens is the number of set bits of
// the signature F_e before position t: a prefix count over the signature
// words, so the order is exact and independent of scheduling.
#include "sig_fast.cuh"

namespace dol {
namespace {

constexpr int kDispThreads = 512;
constexpr int kDispWarps = kDispThreads / 32;

// One CTA per (expert, problem).  It sums the counts of the experts before
// its own for the offset, then walks the expert's signature words in passes of
// kDispThreads consecutive words: a block-wide exclusive scan of the words'
// population counts gives every word its first row, and the word's set bits
// (its tokens, ascending) take the rows after it.
__global__ void __launch_bounds__(kDispThreads)
route_dispatch_kernel(const uint32_t *__restrict__ bits, const int *__restrict__ counts,
                      const int *__restrict__ ids, int64_t T, int E, int k, int64_t W,
                      int *__restrict__ offsets, int *__restrict__ rows, int *__restrict__ pos) {
    __shared__ int s_warp[kDispWarps];
    __shared__ int s_base;
    const int e = blockIdx.x, layer = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, wp = tid >> 5;
    // the signatures, counts and ids come from the kernels before this one
    pdl_wait();
    const int *cl = counts + (size_t)layer * E;
    int part = 0;
    for (int i = tid; i < e; i += kDispThreads) part += cl[i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(kFull, part, o);
    if (lane == 0) s_warp[wp] = part;
    __syncthreads();
    if (tid == 0) {
        int b = 0;
        for (int q = 0; q < kDispWarps; ++q) b += s_warp[q];
        s_base = b;
        if (offsets) {
            offsets[(size_t)layer * (E + 1) + e] = b;
            if (e == E - 1) offsets[(size_t)layer * (E + 1) + E] = b + cl[e];
        }
    }
    __syncthreads();
    if (!rows && !pos) return;
    const int64_t Tk = T * k;
    int run = s_base;  // first row of this pass
    const uint32_t *be = bits + ((size_t)layer * E + e) * W;
    const int *il = ids + (size_t)layer * T * k;
    int *rl = rows ? rows + (size_t)layer * T * k : nullptr;
    int *pl = pos ? pos + (size_t)layer * T * k : nullptr;
    for (int64_t w0 = 0; w0 < W; w0 += kDispThreads) {
        const int64_t w = w0 + tid;
        uint32_t b = w < W ? __ldg(be + w) : 0u;
        const int c = __popc(b);
        int x = c;  // inclusive scan inside the warp
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, x, o);
            if (lane >= o) x += y;
        }
        __syncthreads();  // the previous pass has read s_warp
        if (lane == 31) s_warp[wp] = x;
        __syncthreads();
        int before = 0, total = 0;
#pragma unroll
        for (int q = 0; q < kDispWarps; ++q) {
            const int v = s_warp[q];
            before += q < wp ? v : 0;
            total += v;
        }
        int r = run + before + x - c;
        while (b) {
            const int bit = __ffs(b) - 1;
            b &= b - 1;
            const int64_t t = 32 * w + bit;
            // bits past T are zero and the rows of expert e end at offsets[e+1]
            // when the signatures and counts come from one complete selection;
            // after an aborted one (a timed-out wait, reported in the status
            // word) they may not: never index outside the arrays
            if (t >= T || r < 0 || r >= Tk) break;
            if (rl) rl[r] = (int)t;
            if (pl) {
                const int *it = il + t * k;
                for (int q = 0; q < k; ++q)
                    if (__ldg(it + q) == e) {
                        pl[t * k + q] = r;
                        break;
                    }
            }
            ++r;
        }
        run += total;
    }
}

}  // namespace

cudaError_t launch_signatures_fast_routed(const float *logits, const Problem &p, uint32_t *bits,
                                          int *counts, uint8_t *idx, uint32_t *cooc,
                                          const ZeroSpans &zero, int *status,
                                          const RouteOut &route, cudaStream_t s) {
    CUtensorMap map;
    if (!encode_tensor_map_2d_f32(&map, logits, (uint64_t)p.L * p.T, (uint64_t)p.E, 32))
        return cudaErrorInvalidValue;
    if (p.E == 32) return dispatch_mode<32, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    if (p.E == 64) return dispatch_mode<64, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    return dispatch_mode<128, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
}

cudaError_t launch_route_dispatch(const uint32_t *bits, const int *counts, const int *ids,
                                  const Problem &p, int *offsets, int *rows, int *pos,
                                  cudaStream_t s) {
    if (!offsets && !rows && !pos) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)p.E, (unsigned)p.L);
    cfg.blockDim = dim3(kDispThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, route_dispatch_kernel, bits, counts, ids, p.T, p.E, p.k, p.W,
                              offsets, rows, pos);
}

}  // namespace dol
