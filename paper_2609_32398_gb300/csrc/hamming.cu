// Step 2: the detached Hamming matrix of the load signatures.
//   G_ij = ||F_i - F_j||_1 = sum over words of popc(F_i[w] XOR F_j[w])
//   (Sec. 3.1.3, Eq. gij_cij)
// A CTA owns a 16 x 16 tile of expert pairs on or above the diagonal and a
// chunk of signature words; it stages both row blocks of the chunk in shared
// memory and adds its exact integer partial sums into D (zeroed first), so
// the result does not depend on the order in which chunks finish.
#include "dol_internal.cuh"

namespace dol {
namespace {

constexpr int kTile = 16;            // experts per tile side
constexpr int kPass = 256;           // words staged per pass
constexpr int kStride = kPass + 4;   // padded row stride (keeps 16-byte loads conflict-free)
constexpr int kHamThreads = kTile * kTile;

__global__ void __launch_bounds__(kHamThreads)
hamming_kernel(const uint32_t *__restrict__ bits, int E, int64_t W, int nside,
               int64_t chunk_words, int *__restrict__ D) {
    __shared__ __align__(16) uint32_t s_a[kTile * kStride];
    __shared__ __align__(16) uint32_t s_b[kTile * kStride];

    // Upper-triangle tile index -> (bi, bj), bi <= bj.
    int t = blockIdx.x, bi = 0;
    while (t >= nside - bi) { t -= nside - bi; ++bi; }
    const int bj = bi + t;

    const int layer = blockIdx.z;
    const uint32_t *bl = bits + (int64_t)layer * E * W;
    const int64_t w_begin = (int64_t)blockIdx.y * chunk_words;
    const int64_t w_end = min64(W, w_begin + chunk_words);

    const int ti = threadIdx.x / kTile, tj = threadIdx.x % kTile;
    const int I = bi * kTile + ti, J = bj * kTile + tj;
    int acc = 0;

    for (int64_t w0 = w_begin; w0 < w_end; w0 += kPass) {
        const int nw = (int)min64(kPass, w_end - w0);
        const int nw4 = (nw + 3) & ~3;
        __syncthreads();
        for (int idx = threadIdx.x; idx < kTile * nw4; idx += blockDim.x) {
            const int row = idx / nw4, c = idx % nw4;
            const int ra = bi * kTile + row, rb = bj * kTile + row;
            uint32_t va = 0u, vb = 0u;
            if (c < nw) {
                if (ra < E) va = __ldg(bl + (int64_t)ra * W + w0 + c);
                if (rb < E) vb = __ldg(bl + (int64_t)rb * W + w0 + c);
            }
            s_a[row * kStride + c] = va;
            s_b[row * kStride + c] = vb;
        }
        __syncthreads();
        const uint4 *pa = reinterpret_cast<const uint4 *>(s_a + ti * kStride);
        const uint4 *pb = reinterpret_cast<const uint4 *>(s_b + tj * kStride);
        for (int c = 0; c < nw4 / 4; ++c) {
            const uint4 a = pa[c], b = pb[c];
            acc += __popc(a.x ^ b.x) + __popc(a.y ^ b.y) + __popc(a.z ^ b.z) + __popc(a.w ^ b.w);
        }
    }
    const bool pair = (I < E) && (J < E) && (bi != bj || ti < tj);
    if (pair && acc) {
        int *Dl = D + (int64_t)layer * E * E;
        atomicAdd(Dl + (int64_t)I * E + J, acc);
        atomicAdd(Dl + (int64_t)J * E + I, acc);
    }
}

}  // namespace

cudaError_t launch_hamming(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(D, 0, sizeof(int) * (size_t)p.L * p.E * p.E, s);
    if (e != cudaSuccess) return e;
    const int nside = (p.E + kTile - 1) / kTile;
    const int ntiles = nside * (nside + 1) / 2;
    // Split the words so that a launch has a few hundred CTAs.
    int64_t target = 320 / ((int64_t)ntiles * p.L);
    if (target < 1) target = 1;
    int64_t max_chunks = (p.W + 63) / 64;
    if (max_chunks < 1) max_chunks = 1;
    const int64_t nchunks = target < max_chunks ? target : max_chunks;
    const int64_t chunk = (p.W + nchunks - 1) / nchunks;
    const int64_t gy = (p.W + chunk - 1) / chunk;
    dim3 grid((unsigned)ntiles, (unsigned)gy, (unsigned)p.L);
    hamming_kernel<<<grid, kHamThreads, 0, s>>>(bits, p.E, p.W, nside, chunk, D);
    return cudaGetLastError();
}

}  // namespace dol
