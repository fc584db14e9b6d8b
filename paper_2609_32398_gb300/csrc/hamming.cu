// Step 2: the detached Hamming matrix of the load signatures.
//   G_ij = ||F_i - F_j||_1 = sum over words of popc(F_i[w] XOR F_j[w])
//   (Sec. 3.1.3, Eq. gij_cij)
// The experts are cut into blocks of 16.  A pair of blocks (bi <= bj) is one
// unit of 16 x 16 expert pairs, cut into 4 x 4 tiles; 16 threads share a
// tile, each holding the tile's 16 counts in registers.  The signature words
// are cut into stages of 128 words; a unit's rows for one stage (32 rows, 16
// on the diagonal) sit in shared memory, padded to 528 bytes a row, filled
// by asynchronous copies (cp.async, zero-filled past W and past E) in a ring
// of 4 stages, so later stages load while one is counted.  The threads of a
// tile take interleaved 16-byte chunks of a stage; a chunk gives 16 pairs x
// 4 words (XOR + POPC each) from 8 shared-memory loads, so the kernel runs
// at the POPC rate.  The 16 threads of a tile then add their counts with a
// shuffle reduce-scatter, after which each holds one pair's sum.
// The words of a unit may be split across the CTAs of a thread-block cluster
// (one word range each): every CTA leaves its sums in shared memory and the
// entries are added across the cluster through distributed shared memory in
// rank order.  Each entry of D has one writer, so there are no atomics and
// no clearing beforehand, and the integer sums do not depend on the split.
#include <algorithm>
#include <atomic>

#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kHB = 16;                          // experts per block side
constexpr int kHSide = kHB / 4;                  // tiles per block side
constexpr int kHTiles = kHSide * kHSide;
constexpr int kHThreads = 256;
constexpr int kHTpt = kHThreads / kHTiles;       // threads per tile
constexpr int kHStageWords = 128;                // words of a row per stage
constexpr int kHRowWords = kHStageWords + 4;     // padded row (528 bytes)
constexpr int kHRowChunks = kHRowWords / 4;      // 16-byte chunks of a padded row
constexpr int kHChunks = kHStageWords / 4 / kHTpt;  // chunks per stage per thread
constexpr int kHStages = 4;
constexpr int kHRows = 2 * kHB;
constexpr int kHStageU32 = kHRows * kHRowWords;
constexpr size_t kHSmem = sizeof(uint32_t) * (size_t)kHStages * kHStageU32;
constexpr int kHMaxCluster = 8;
static_assert(kHTiles * kHTpt == kHThreads && 32 % kHTpt == 0 && kHTpt == 16,
              "a tile's threads are half a warp and end with one sum each");

template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

// 16 bytes, or zeros when src_bytes == 0
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
                 : "memory");
}

// 4 bytes, or zeros when src_bytes == 0
__device__ __forceinline__ void cp_async4(uint32_t dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
                 : "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" :::
                     "memory");
}

// the 32-bit word at a shared address of CTA `rank` of this cluster
__device__ __forceinline__ uint32_t ld_cluster(uint32_t addr, uint32_t rank) {
    uint32_t remote, v;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(addr), "r"(rank));
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(remote) : "memory");
    return v;
}

// Entry (i, j) of a unit, i of block bi and j of block bj (bi <= bj): both
// halves of D once per unordered pair, and zero on the diagonal.
__device__ __forceinline__ void put_entry(int *Dl, int E, int i, int j, int v, bool accumulate) {
    if (i >= E || j >= E) return;
    if (i < j) {
        if (accumulate) {
            Dl[(int64_t)i * E + j] += v;
            Dl[(int64_t)j * E + i] += v;
        } else {
            Dl[(int64_t)i * E + j] = v;
            Dl[(int64_t)j * E + i] = v;
        }
    } else if (i == j && !accumulate) {
        Dl[(int64_t)i * E + i] = 0;
    }
}

// grid (units x C, L), cluster (C, 1, 1); accumulate: D += the result.
__global__ void __launch_bounds__(kHThreads, 2)
hamming_kernel(const uint32_t *__restrict__ bits, int E, int64_t W, int nside, int C,
               int *__restrict__ D, int accumulate, int vec) {
    extern __shared__ __align__(16) uint32_t h_ring[];
    __shared__ int s_part[kHTiles * 16];
    // upper-triangle unit index -> (bi, bj), bi <= bj
    int u = blockIdx.x / C, bi = 0;
    while (u >= nside - bi) {
        u -= nside - bi;
        ++bi;
    }
    const int bj = bi + u;
    const bool diag = bi == bj;
    const uint32_t rank = C > 1 ? cluster_rank() : 0u;
    const int layer = blockIdx.y;
    const uint32_t *bl = bits + (int64_t)layer * E * W;
    int *Dl = D + (int64_t)layer * E * E;
    // this CTA's stages [s0, s0 + nst)
    const int64_t nst_all = (W + kHStageWords - 1) / kHStageWords;
    const int64_t per = (nst_all + C - 1) / C;
    const int64_t s0 = (int64_t)rank * per;
    const int64_t s1 = min64(nst_all, s0 + per);
    const int nst = s1 > s0 ? (int)(s1 - s0) : 0;
    const int rows = diag ? kHB : kHRows;  // on the diagonal both sides are the same rows

    const int tile = threadIdx.x / kHTpt, q = threadIdx.x % kHTpt;
    const int ti = tile / kHSide, tj = tile % kHSide;
    const bool active = !diag || ti <= tj;
    const int rowA = 4 * ti, rowB = (diag ? 0 : kHB) + 4 * tj;

    pdl_wait();
    pdl_trigger();
    auto issue = [&](int s) {
        const int64_t w0 = (s0 + s) * kHStageWords;
        const uint32_t base = smem_u32(h_ring + (s % kHStages) * kHStageU32);
        for (int item = threadIdx.x; item < rows * 32; item += kHThreads) {
            const int r = item >> 5, c = item & 31;
            const int e = r < kHB ? bi * kHB + r : bj * kHB + r - kHB;
            const int64_t w = w0 + 4 * c;
            const uint32_t dst = base + (uint32_t)(r * kHRowWords + 4 * c) * 4u;
            if (vec) {  // W % 4 == 0: a chunk is all in or all out
                const bool in = e < E && w < W;
                cp_async16(dst, in ? bl + (int64_t)e * W + w : bl, in ? 16u : 0u);
            } else {
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    const bool in = e < E && w + x < W;
                    cp_async4(dst + 4u * x, in ? bl + (int64_t)e * W + w + x : bl, in ? 4u : 0u);
                }
            }
        }
    };

    int v[16];
#pragma unroll
    for (int p = 0; p < 16; ++p) v[p] = 0;
#pragma unroll
    for (int s = 0; s < kHStages - 1; ++s) {
        if (s < nst) issue(s);
        cp_async_commit();
    }
    for (int s = 0; s < nst; ++s) {
        cp_async_wait<kHStages - 2>();
        __syncthreads();  // stage s is in for every thread; slot (s - 1) is free
        if (s + kHStages - 1 < nst) issue(s + kHStages - 1);
        cp_async_commit();
        if (!active) continue;
        const uint4 *st = reinterpret_cast<const uint4 *>(h_ring + (s % kHStages) * kHStageU32);
#pragma unroll
        for (int m = 0; m < kHChunks; ++m) {
            const int c = q + m * kHTpt;
            uint4 a[4], b[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) a[x] = st[(rowA + x) * kHRowChunks + c];
#pragma unroll
            for (int y = 0; y < 4; ++y) b[y] = st[(rowB + y) * kHRowChunks + c];
#pragma unroll
            for (int x = 0; x < 4; ++x)
#pragma unroll
                for (int y = 0; y < 4; ++y) {
                    v[4 * x + y] += __popc(a[x].x ^ b[y].x) + __popc(a[x].y ^ b[y].y) +
                                    __popc(a[x].z ^ b[y].z) + __popc(a[x].w ^ b[y].w);
                }
        }
    }
    // reduce-scatter over the 16 lanes of the tile: after it, lane q holds
    // the sum of entry q (row q / 4, column q % 4 of the tile)
#pragma unroll
    for (int half = 8; half >= 1; half >>= 1) {
        const bool up = (q & half) != 0;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const int send = up ? v[i] : v[i + half];
            const int keep = up ? v[i + half] : v[i];
            v[i] = keep + __shfl_xor_sync(kFull, send, half);
        }
    }
    const int i_of = bi * kHB + rowA + (q >> 2);
    const int j_of = bj * kHB + 4 * tj + (q & 3);
    if (C == 1) {
        if (active) put_entry(Dl, E, i_of, j_of, v[0], accumulate != 0);
        return;
    }
    if (active) s_part[tile * 16 + q] = v[0];
    cluster_sync();
    // CTA `rank` adds, in rank order, the C partial sums of the entries
    // rank * per_e .. (rank + 1) * per_e - 1 of the block
    const int per_e = kHTiles * 16 / C;
    for (int e = (int)rank * per_e + threadIdx.x; e < ((int)rank + 1) * per_e; e += kHThreads) {
        const int tl = e >> 4, idx = e & 15;
        const int eti = tl / kHSide, etj = tl % kHSide;
        if (diag && eti > etj) continue;
        const uint32_t addr = smem_u32(&s_part[e]);
        int sum = 0;
        for (int r = 0; r < C; ++r) sum += (int)ld_cluster(addr, (uint32_t)r);
        put_entry(Dl, E, bi * kHB + 4 * eti + (idx >> 2), bj * kHB + 4 * etj + (idx & 3), sum,
                  accumulate != 0);
    }
    cluster_sync();  // no CTA leaves while another still reads its sums
}

// SMs and resident hamming CTAs per SM on the current device, cached per device.
cudaError_t hamming_slots(int *sms, int *per_sm) {
    static std::atomic<int> cache[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int packed = dev < 64 ? cache[dev].load() : 0;
    if (packed == 0) {
        int n = 0, occ = 0;
        e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess) e = ensure_smem_limit<hamming_kernel>(kHSmem);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, hamming_kernel, kHThreads, kHSmem);
        if (e != cudaSuccess) return e;
        packed = (n << 8) | std::max(1, std::min(occ, 255));
        if (dev < 64) cache[dev].store(packed);
    }
    *sms = packed >> 8;
    *per_sm = packed & 255;
    return cudaSuccess;
}

cudaError_t run_hamming(const uint32_t *bits, const Problem &p, int *D, int accumulate,
                        cudaStream_t s) {
    const int nside = (p.E + kHB - 1) / kHB;
    const int64_t units = (int64_t)nside * (nside + 1) / 2;
    const int64_t nst = (p.W + kHStageWords - 1) / kHStageWords;
    int sms = 0, per_sm = 0;
    cudaError_t e = hamming_slots(&sms, &per_sm);
    if (e != cudaSuccess) return e;
    e = ensure_smem_limit<hamming_kernel>(kHSmem);
    if (e != cudaSuccess) return e;
    // split the words over a cluster while the units leave resident slots idle
    const int64_t slots = (int64_t)sms * per_sm;
    int C = 1;
    while (C < kHMaxCluster && units * p.L * C * 2 <= slots && C * 2 <= nst) C *= 2;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(units * C), (unsigned)p.L);
    cfg.blockDim = dim3(kHThreads);
    cfg.dynamicSmemBytes = kHSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)C;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = C > 1 ? 2 : 1;
    const int vec = (p.W % 4 == 0) && (reinterpret_cast<uintptr_t>(bits) % 16 == 0);
    return cudaLaunchKernelEx(&cfg, hamming_kernel, bits, p.E, p.W, nside, C, D, accumulate, vec);
}

}  // namespace

// D += the Hamming matrix of bits.
cudaError_t launch_hamming_accumulate(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s) {
    return run_hamming(bits, p, D, 1, s);
}

cudaError_t launch_hamming(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s) {
    return run_hamming(bits, p, D, 0, s);
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
