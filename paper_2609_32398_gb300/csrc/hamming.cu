// Step 2: the detached Hamming matrix of the load signatures.
//   G_ij = ||F_i - F_j||_1 = sum over words of popc(F_i[w] XOR F_j[w])
//   (Sec. 3.1.3, Eq. gij_cij; App. C.3: n_i = ||F_i||_1)
// A CTA owns an 8 x 8 block of expert pairs on or above the diagonal and all
// the signature words, so every entry of D has one writer: no atomics and no
// clearing beforehand.  Its 256 threads split the words 64 ways (a
// contiguous slice each) and hold 4 x 4 pairs in registers (a quarter of the
// block), so every 16-byte load of a row feeds four pairs; the 64 slices'
// partial sums are added in shared memory in a fixed order.
#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kHB = 8;        // experts per block side
constexpr int kHSlices = 64;  // word slices per block
constexpr int kHThreads = kHSlices * 4;

__device__ __forceinline__ uint4 load_w4(const uint32_t *row, int64_t w, int64_t w_end, bool vec) {
    if (!row) return make_uint4(0u, 0u, 0u, 0u);
    if (vec && w + 4 <= w_end) return __ldg(reinterpret_cast<const uint4 *>(row + w));
    uint32_t q[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) q[i] = (w + i < w_end) ? __ldg(row + w + i) : 0u;
    return make_uint4(q[0], q[1], q[2], q[3]);
}

__device__ __forceinline__ int popc_xor4(uint4 a, uint4 b) {
    return __popc(a.x ^ b.x) + __popc(a.y ^ b.y) + __popc(a.z ^ b.z) + __popc(a.w ^ b.w);
}

// accumulate: D (and counts, when given) += the result; else D = the result
// (and counts = n).
__global__ void __launch_bounds__(kHThreads)
hamming_kernel(const uint32_t *__restrict__ bits, int E, int64_t W, int nside, int *__restrict__ D,
               int *__restrict__ counts, int accumulate, int vec) {
    __shared__ int s_part[kHSlices][kHB * kHB];
    __shared__ int s_cnt[kHSlices][kHB];
    // upper-triangle block index -> (bi, bj), bi <= bj
    int t = blockIdx.x, bi = 0;
    while (t >= nside - bi) {
        t -= nside - bi;
        ++bi;
    }
    const int bj = bi + t;
    const int layer = blockIdx.z;
    const uint32_t *bl = bits + (int64_t)layer * E * W;
    const int sl = threadIdx.x >> 2, sb = threadIdx.x & 3;
    const int ri0 = 4 * (sb >> 1), cj0 = 4 * (sb & 1);  // this thread's 4 rows and 4 columns
    // words of this slice: a multiple of 4 per slice
    const int64_t per = ((W + kHSlices - 1) / kHSlices + 3) / 4 * 4;
    const int64_t w0 = (int64_t)sl * per, w1 = min64(W, w0 + per);
    const uint32_t *ra[4], *rb[4];
#pragma unroll
    for (int x = 0; x < 4; ++x) {
        const int i = kHB * bi + ri0 + x, j = kHB * bj + cj0 + x;
        ra[x] = i < E ? bl + (int64_t)i * W : nullptr;
        rb[x] = j < E ? bl + (int64_t)j * W : nullptr;
    }
    const bool diag_counts = counts && bi == bj && sb == 0;  // rows 0..3 ...
    const bool diag_counts2 = counts && bi == bj && sb == 3; // ... and rows 4..7 of a diagonal block
    pdl_wait();
    pdl_trigger();
    int acc[4][4];
#pragma unroll
    for (int x = 0; x < 4; ++x)
#pragma unroll
        for (int y = 0; y < 4; ++y) acc[x][y] = 0;
    int cnt[4] = {0, 0, 0, 0};
    for (int64_t w = w0; w < w1; w += 4) {
        uint4 a[4], b[4];
#pragma unroll
        for (int x = 0; x < 4; ++x) {
            a[x] = load_w4(ra[x], w, w1, vec);
            b[x] = load_w4(rb[x], w, w1, vec);
        }
#pragma unroll
        for (int x = 0; x < 4; ++x)
#pragma unroll
            for (int y = 0; y < 4; ++y) acc[x][y] += popc_xor4(a[x], b[y]);
        if (diag_counts || diag_counts2) {
#pragma unroll
            for (int x = 0; x < 4; ++x)
                cnt[x] += __popc(a[x].x) + __popc(a[x].y) + __popc(a[x].z) + __popc(a[x].w);
        }
    }
#pragma unroll
    for (int x = 0; x < 4; ++x)
#pragma unroll
        for (int y = 0; y < 4; ++y) s_part[sl][(ri0 + x) * kHB + cj0 + y] = acc[x][y];
    if (diag_counts || diag_counts2)
#pragma unroll
        for (int x = 0; x < 4; ++x) s_cnt[sl][ri0 + x] = cnt[x];
    __syncthreads();
    // the 64 pairs of the block, each the fixed-order sum over the slices
    if (threadIdx.x < kHB * kHB) {
        const int ii = threadIdx.x / kHB, jj = threadIdx.x % kHB;
        const int i = kHB * bi + ii, j = kHB * bj + jj;
        if (i < E && j < E && (bi != bj || ii < jj)) {
            int d = 0;
            for (int v = 0; v < kHSlices; ++v) d += s_part[v][threadIdx.x];
            int *Dl = D + (int64_t)layer * E * E;
            if (accumulate) {
                Dl[(int64_t)i * E + j] += d;
                Dl[(int64_t)j * E + i] += d;
            } else {
                Dl[(int64_t)i * E + j] = d;
                Dl[(int64_t)j * E + i] = d;
            }
        }
        if (bi == bj && ii == jj && i < E) {
            if (!accumulate) D[(int64_t)layer * E * E + (int64_t)i * E + i] = 0;
            if (counts) {
                int n = 0;
                for (int v = 0; v < kHSlices; ++v) n += s_cnt[v][ii];
                int *dst = counts + (int64_t)layer * E + i;
                *dst = accumulate ? *dst + n : n;
            }
        }
    }
}

cudaError_t run_hamming(const uint32_t *bits, const Problem &p, int *D, int *counts, int accumulate,
                        cudaStream_t s) {
    const int nside = (p.E + kHB - 1) / kHB;
    const int nblocks = nside * (nside + 1) / 2;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)nblocks, 1u, (unsigned)p.L);
    cfg.blockDim = dim3(kHThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const int vec = (p.W % 4 == 0) && (reinterpret_cast<uintptr_t>(bits) % 16 == 0);
    return cudaLaunchKernelEx(&cfg, hamming_kernel, bits, p.E, p.W, nside, D, counts, accumulate, vec);
}

}  // namespace

// D (and counts, when given) += the Hamming matrix of bits (and the counts).
cudaError_t launch_hamming_accumulate(const uint32_t *bits, const Problem &p, int *D, int *counts,
                                      cudaStream_t s) {
    return run_hamming(bits, p, D, counts, 1, s);
}

cudaError_t launch_hamming(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s) {
    return run_hamming(bits, p, D, nullptr, 0, s);
}

// D_sum += D over n int32 entries (the Hamming matrices of the micro-batches
// of a window add up, Eq. global_do); a grid-stride loop of 16-byte rows
// where both are aligned.
__global__ void __launch_bounds__(256)
add_distances_kernel(const int *__restrict__ D, int *__restrict__ D_sum, int64_t n, int vec) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (vec) {
        const int4 *a = reinterpret_cast<const int4 *>(D);
        int4 *b = reinterpret_cast<int4 *>(D_sum);
        for (int64_t i = t; i < n / 4; i += stride) {
            const int4 x = __ldg(a + i);
            int4 y = b[i];
            y.x += x.x; y.y += x.y; y.z += x.z; y.w += x.w;
            b[i] = y;
        }
        for (int64_t i = (n / 4) * 4 + t; i < n; i += stride) D_sum[i] += __ldg(D + i);
    } else {
        for (int64_t i = t; i < n; i += stride) D_sum[i] += __ldg(D + i);
    }
}

cudaError_t launch_add_distances(const int *D, int *D_sum, int64_t n, cudaStream_t s) {
    const int vec = (reinterpret_cast<uintptr_t>(D) % 16 == 0 &&
                     reinterpret_cast<uintptr_t>(D_sum) % 16 == 0) ? 1 : 0;
    const int64_t want = ((vec ? (n + 3) / 4 : n) + 255) / 256;
    const int blocks = (int)(want < 1 ? 1 : (want > 1024 ? 1024 : want));
    add_distances_kernel<<<blocks, 256, 0, s>>>(D, D_sum, n, vec);
    return cudaGetLastError();
}

}  // namespace dol
