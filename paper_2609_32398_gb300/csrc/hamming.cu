// Step 2: the detached Hamming matrix of the load signatures.
//   G_ij = ||F_i - F_j||_1 = sum over words of popc(F_i[w] XOR F_j[w])
//   (Sec. 3.1.3, Eq. gij_cij)
// A CTA owns a 16 x 16 tile of expert pairs on or above the diagonal and a
// chunk of signature words; it stages both row blocks of the chunk in shared
// memory and adds its exact integer partial sums into D (zeroed beforehand),
// so the result does not depend on the order in which chunks finish.  On the
// diagonal tiles the threads of pairs (i, i) count the set bits of F_i
// instead, which gives the per-expert counts n_i = ||F_i||_1 (App. C.3).
#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kTile = 16;            // experts per tile side
constexpr int kPass = 256;           // words staged per pass
constexpr int kStride = kPass + 4;   // padded row stride (keeps 16-byte loads conflict-free)
constexpr int kHamThreads = kTile * kTile;

__global__ void __launch_bounds__(kHamThreads)
hamming_kernel(const uint32_t *__restrict__ bits, int E, int64_t W, int nside, int64_t chunk_words,
               int *__restrict__ D, int *__restrict__ counts, int vec) {
    __shared__ __align__(16) uint32_t s_a[kTile * kStride];
    __shared__ __align__(16) uint32_t s_b[kTile * kStride];

    // Upper-triangle tile index -> (bi, bj), bi <= bj.
    int t = blockIdx.x, bi = 0;
    while (t >= nside - bi) {
        t -= nside - bi;
        ++bi;
    }
    const int bj = bi + t;
    const int layer = blockIdx.z;
    const uint32_t *bl = bits + (int64_t)layer * E * W;
    const int64_t w_begin = (int64_t)blockIdx.y * chunk_words;
    const int64_t w_end = min64(W, w_begin + chunk_words);
    const int ti = threadIdx.x / kTile, tj = threadIdx.x % kTile;
    const int I = bi * kTile + ti, J = bj * kTile + tj;
    const bool count_row = (bi == bj) && (ti == tj);
    // staging: thread -> (row, 16-byte column) of both row blocks
    const int srow = threadIdx.x >> 4, scol = (threadIdx.x & 15) * 4;
    const int ra = bi * kTile + srow, rb = bj * kTile + srow;

    pdl_wait();
    pdl_trigger();
    int acc = 0;
    for (int64_t w0 = w_begin; w0 < w_end; w0 += kPass) {
        const int nw = (int)min64(kPass, w_end - w0);
        __syncthreads();
#pragma unroll
        for (int c0 = 0; c0 < kPass; c0 += 64) {
            const int c = c0 + scol;
            uint4 va = make_uint4(0u, 0u, 0u, 0u), vb = va;
            if (c < nw) {
                const uint32_t *pa = bl + (int64_t)ra * W + w0 + c;
                const uint32_t *pb = bl + (int64_t)rb * W + w0 + c;
                if (vec && c + 4 <= nw) {
                    if (ra < E) va = __ldg(reinterpret_cast<const uint4 *>(pa));
                    if (rb < E) vb = __ldg(reinterpret_cast<const uint4 *>(pb));
                } else {
                    uint32_t a4[4] = {0u, 0u, 0u, 0u}, b4[4] = {0u, 0u, 0u, 0u};
                    for (int q = 0; q < 4 && c + q < nw; ++q) {
                        if (ra < E) a4[q] = __ldg(pa + q);
                        if (rb < E) b4[q] = __ldg(pb + q);
                    }
                    va = make_uint4(a4[0], a4[1], a4[2], a4[3]);
                    vb = make_uint4(b4[0], b4[1], b4[2], b4[3]);
                }
            }
            *reinterpret_cast<uint4 *>(s_a + srow * kStride + c) = va;
            *reinterpret_cast<uint4 *>(s_b + srow * kStride + c) = vb;
        }
        __syncthreads();
        const uint4 *pa = reinterpret_cast<const uint4 *>(s_a + ti * kStride);
        const uint4 *pb = reinterpret_cast<const uint4 *>(s_b + tj * kStride);
        const int n4 = (nw + 3) >> 2;
        if (count_row) {
            for (int c = 0; c < n4; ++c) {
                const uint4 a = pa[c];
                acc += __popc(a.x) + __popc(a.y) + __popc(a.z) + __popc(a.w);
            }
        } else {
            for (int c = 0; c < n4; ++c) {
                const uint4 a = pa[c], b = pb[c];
                acc += __popc(a.x ^ b.x) + __popc(a.y ^ b.y) + __popc(a.z ^ b.z) + __popc(a.w ^ b.w);
            }
        }
    }
    if (count_row) {
        if (counts && I < E && acc) atomicAdd(counts + (int64_t)layer * E + I, acc);
        return;
    }
    const bool pair = (I < E) && (J < E) && (bi != bj || ti < tj);
    if (pair && acc) {
        int *Dl = D + (int64_t)layer * E * E;
        atomicAdd(Dl + (int64_t)I * E + J, acc);
        atomicAdd(Dl + (int64_t)J * E + I, acc);
    }
}

}  // namespace

// D (and counts, when given) must be zero when the kernel starts; the caller
// either memsets them or has the preceding kernel clear them.
cudaError_t launch_hamming_accumulate(const uint32_t *bits, const Problem &p, int *D, int *counts,
                                      cudaStream_t s) {
    const int nside = (p.E + kTile - 1) / kTile;
    const int ntiles = nside * (nside + 1) / 2;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // Split the words so that one launch fills the GPU about twice.
    int64_t target = (2LL * sms + (int64_t)ntiles * p.L - 1) / ((int64_t)ntiles * p.L);
    if (target < 1) target = 1;
    int64_t max_chunks = (p.W + 63) / 64;
    if (max_chunks < 1) max_chunks = 1;
    const int64_t nchunks = target < max_chunks ? target : max_chunks;
    int64_t chunk = (p.W + nchunks - 1) / nchunks;
    chunk = (chunk + 3) / 4 * 4;
    const int64_t gy = (p.W + chunk - 1) / chunk;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)ntiles, (unsigned)gy, (unsigned)p.L);
    cfg.blockDim = dim3(kHamThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const int vec = (p.W % 4 == 0) && (reinterpret_cast<uintptr_t>(bits) % 16 == 0);
    return cudaLaunchKernelEx(&cfg, hamming_kernel, bits, p.E, p.W, nside, chunk, D, counts, vec);
}

cudaError_t launch_hamming(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(D, 0, sizeof(int) * (size_t)p.L * p.E * p.E, s);
    if (e != cudaSuccess) return e;
    return launch_hamming_accumulate(bits, p, D, nullptr, s);
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
