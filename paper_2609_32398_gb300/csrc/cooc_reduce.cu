// Reduction of the per-CTA co-occurrence triangles of the fused path.
//   c_ab = sum_t f_at f_bt, c_aa = n_a, and the Hamming distance
//   D_ab = n_a + n_b - 2 c_ab                                   (App. C.3)
// and, alongside, Eq. origin_do: sum over a != b of D_ab^2 (exact integer
// adds, one per CTA).
// The counts n_a were already summed (one atomic per expert and CTA) by the
// signatures kernel.  A CTA owns 32 consecutive triangle words; its 32 warps
// each sum a strided subset of the partials with independent loads, and the
// 32 warp sums are added in a fixed order, so D is an exact integer result
// independent of scheduling (every load of a warp is issued before any add).
// The kernel writes both halves of the symmetric D and the counts.
#include <cuda_fp16.h>

#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kRedWarps = 32;
constexpr int kRedThreads = kRedWarps * 32;
static_assert(kMaxSigCtas <= 8 * kRedWarps, "a warp adds at most eight partials");

template <int E>
__global__ void __launch_bounds__(kRedThreads)
cooc_reduce_kernel(const uint32_t *__restrict__ partials, int P1, const int *__restrict__ n_acc,
                   int *__restrict__ D, int *__restrict__ counts, unsigned char *__restrict__ bimg,
                   long long *__restrict__ origin_do, long long r_base, int r_mult) {
    constexpr int kWords = cooc_row_offset<E>(E);
    __shared__ uint32_t s_sum[kRedWarps][33];
    __shared__ int s_n[E];  // the counts n_a, read once per CTA while the partials load
    const int e = threadIdx.x & 31, wp = threadIdx.x >> 5;
    const int word = blockIdx.x * 32 + e;
    const int layer = blockIdx.y;
    pdl_wait();
    pdl_trigger();
    if ((int)threadIdx.x < E) s_n[threadIdx.x] = n_acc[(size_t)layer * E + threadIdx.x];
    // every partial this warp adds (P1 <= 8 x 32) is requested at once
    uint32_t v[8];
    const uint32_t *base = partials + (size_t)layer * P1 * kWords + word;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        const int p = wp + u * kRedWarps;
        v[u] = (word < kWords && p < P1) ? __ldg(base + (size_t)p * kWords) : 0u;
    }
    uint32_t acc = 0u;
#pragma unroll
    for (int u = 0; u < 8; ++u) acc += v[u];
    s_sum[wp][e] = acc;
    __syncthreads();
    if (wp != 0) return;
    long long sq = 0;  // this word's part of sum_{a != b} D_ab^2
    if (word < kWords) {
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
        int *Dl = D + (size_t)layer * E * E;
        unsigned char *img = (E == 128 && bimg) ? bimg + (size_t)layer * kBImageBytes : nullptr;
        if (b < a) {
            // alignment padding of row a: nothing to write
        } else if (a == b) {
            Dl[a * E + a] = 0;
            counts[(size_t)layer * E + a] = (int)c;
            // R_a = (E - 2k) n_a + T k (every row of the co-occurrence sums to k n_a)
            if (img) put_dprime(img, a, a, true, (int)(r_base + (long long)r_mult * (long long)c));
        } else {
            const int d = s_n[a] + s_n[b] - 2 * (int)c;
            Dl[a * E + b] = d;
            Dl[b * E + a] = d;
            if (img) {
                put_dprime(img, a, b, false, d);
                put_dprime(img, b, a, false, d);
            }
            sq = 2 * (long long)d * (long long)d;
        }
    }
    if (origin_do) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(kFull, sq, o);
        if (e == 0 && sq)
            atomicAdd(reinterpret_cast<unsigned long long *>(origin_do + layer), (unsigned long long)sq);
    }
}

template <int E>
cudaError_t run_reduce(const uint32_t *partials, int P1, const int *n_acc, const Problem &p, int *D,
                       int *counts, unsigned char *bimg, long long *origin_do, cudaStream_t s) {
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
    const long long r_base = p.T * (long long)p.k;
    const int r_mult = E - 2 * p.k;
    return cudaLaunchKernelEx(&cfg, cooc_reduce_kernel<E>, partials, P1, n_acc, D, counts, bimg,
                              origin_do, r_base, r_mult);
}

// The image of D' from a given matrix D (a matrix summed over ranks or
// micro-batches, Eq. global_do): off the diagonal D_ab, on it -R_a with R_a =
// sum_{b != a} D_ab (D symmetric).  img_ok[layer] = 1 when the two fp16
// pieces are exact for this matrix (0 <= D_ab < 2^22 off the diagonal,
// D_aa = 0, R_a < 2^23), else 0: the tensor-core loss kernel takes the
// problems with 1, the ALU kernel the others.  One CTA per problem; a thread
// builds one 16-byte chunk of row n of each piece (8 consecutive k = a) from
// D[n][a .. a + 7], the 16 threads of row n (a half warp) add R_n with
// shuffles, and the chunks are written whole (the 128-byte swizzle moves
// whole 16-byte chunks).
__global__ void __launch_bounds__(kRedThreads)
dprime_image_kernel(const int *__restrict__ D, unsigned char *__restrict__ bimg,
                    int *__restrict__ img_ok) {
    constexpr int E = 128;
    const int layer = blockIdx.x;
    const int *Dl = D + (size_t)layer * E * E;
    unsigned char *img = bimg + (size_t)layer * kBImageBytes;
    pdl_wait();
    pdl_trigger();
    int ok = 1;
#pragma unroll
    for (int pass = 0; pass < 2; ++pass) {
        const int item = pass * kRedThreads + (int)threadIdx.x;
        const int n = item >> 4, a0 = 8 * (item & 15);
        const int4 v0 = __ldg(reinterpret_cast<const int4 *>(Dl + n * E + a0));
        const int4 v1 = __ldg(reinterpret_cast<const int4 *>(Dl + n * E + a0 + 4));
        const int v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        long long row = 0;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if (a0 + u == n) {
                ok &= v[u] == 0;
            } else {
                ok &= v[u] >= 0 && v[u] < (1 << 22);
                row += v[u];
            }
        }
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) row += __shfl_xor_sync(kFull, row, o);
        ok &= row < (1 << 23);
        uint32_t hw[4], lw[4];
#pragma unroll
        for (int u = 0; u < 8; u += 2) {
            int h0, l0, h1, l1;
            dprime_pieces(a0 + u == n, a0 + u == n ? (int)row : v[u], &h0, &l0);
            dprime_pieces(a0 + u + 1 == n, a0 + u + 1 == n ? (int)row : v[u + 1], &h1, &l1);
            hw[u / 2] = (uint32_t)__half_as_ushort(__int2half_rn(h0)) |
                        ((uint32_t)__half_as_ushort(__int2half_rn(h1)) << 16);
            lw[u / 2] = (uint32_t)__half_as_ushort(__int2half_rn(l0)) |
                        ((uint32_t)__half_as_ushort(__int2half_rn(l1)) << 16);
        }
        *reinterpret_cast<uint4 *>(img + sw128_k16_offset(n, a0, 256)) =
            make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *reinterpret_cast<uint4 *>(img + sw128_k16_offset(128 + n, a0, 256)) =
            make_uint4(lw[0], lw[1], lw[2], lw[3]);
    }
    ok = __syncthreads_and(ok);
    if (threadIdx.x == 0) img_ok[layer] = ok;
}

}  // namespace

cudaError_t launch_cooc_reduce(const uint32_t *partials, int P1, const int *n_acc, const Problem &p,
                               int *D, int *counts, unsigned char *bimg, long long *origin_do,
                               cudaStream_t s) {
    if (p.E == 32) return run_reduce<32>(partials, P1, n_acc, p, D, counts, nullptr, origin_do, s);
    if (p.E == 64) return run_reduce<64>(partials, P1, n_acc, p, D, counts, nullptr, origin_do, s);
    if (p.E == 128) return run_reduce<128>(partials, P1, n_acc, p, D, counts, bimg, origin_do, s);
    return cudaErrorInvalidValue;
}

cudaError_t launch_dprime_image(const int *D, const Problem &p, unsigned char *bimg, int *img_ok,
                                cudaStream_t s) {
    if (p.E != 128) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)p.L);
    cfg.blockDim = dim3(kRedThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, dprime_image_kernel, D, bimg, img_ok);
}

}  // namespace dol
