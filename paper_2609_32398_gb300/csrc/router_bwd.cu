// Backward of the router's linear map (Sec. 4.1: hidden size H to the n = 128
// experts, no bias) for the gradient dz of the logits that the loss step
// writes (dlogits):
//   dW[l][e][h] = sum_t dz[l][t][e] X[l][t][h]     fp32
//   dX[l][t][h] = sum_e dz[l][t][e] W[l][e][h]     bf16 (optional)
// on the tcgen05 tensor cores (kind::f16: bf16 operands, fp32 accumulation).
// dz is rounded to bf16 first (round to nearest even), the usual precision of
// a mixed-precision router backward: both products then read bf16 operands
// at the tensor cores' full rate, and the rounding is covered by the
// documented bound (2^-8 + 2n 2^-24) sum |terms| per entry.
//
// dX = dz W (router_dx_kernel): a CTA owns a slice of 64 nq hidden columns and
// a run of 128-token tiles.  Its slice of W (K = 128 experts x N = 64 nq, the
// B operand, MN-major: hidden columns contiguous) is loaded once; the dz
// tiles (M = 128 tokens x K = 128 experts, K-major) stream through a 3-stage
// ring; eight MMAs of K = 16 per tile go into one of two TMEM accumulators;
// four epilogue warps turn the fp32 accumulator into bf16 rows in a swizzled
// shared tile and store it with TMA.
//
// dW = dz^T X (router_dw_kernel): a CTA owns a slice of 64 nq hidden columns
// and a chunk of the tokens.  Both operands are read as stored, MN-major
// (A = dz [t][e]: experts contiguous; B = X [t][h]: hidden contiguous), in
// 64-token k-tiles through a 4-stage ring; the accumulator (M = 128 experts x
// N = 64 nq) holds the chunk's partial sum, which the epilogue writes out;
// router_dw_reduce_kernel adds the chunks' partials in a fixed order, so dW
// does not depend on scheduling.
//
// Every wait is bounded: a wait that runs out records kDevTimeout in the
// status word at the start of the workspace and the CTA leaves (after its
// copies in flight), which do_device_status reports.
#include <cuda_bf16.h>

#include <climits>
#include <cstdint>

#include "dol_internal.cuh"
#include "doloss.h"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kBE = 128;                 // experts: K of dX, M of dW
constexpr int kBTileM = 128;             // tokens per dX tile
constexpr int kBKt = 64;                 // tokens per dW k-tile
constexpr int kBThreads = 6 * 32;        // producer, MMA issuer, 4 epilogue warps
constexpr int kDxStages = 3;
constexpr int kDwStages = 4;
constexpr int kDwChunksMax = 32;         // token chunks of dW at most (partials in the workspace)
constexpr uint32_t kBox128 = 128 * 128;  // 128 rows x 128 bytes
constexpr uint32_t kBox64 = 64 * 128;    // 64 rows x 128 bytes
constexpr uint32_t kBox32 = 32 * 128;    // 32 rows x 128 bytes

// dX shared memory: W slice [nq][128 x 128 B], dz ring [3][2][128 x 128 B],
// output staging [4 warps][nq][32 x 128 B], barriers.
constexpr uint32_t kDxOffB = 0;
constexpr uint32_t kDxOffA = 4 * kBox128;
constexpr uint32_t kDxOffO = kDxOffA + kDxStages * 2 * kBox128;
constexpr uint32_t kDxOffBar = kDxOffO + 4 * 4 * kBox32;
constexpr uint32_t kDxSmem = kDxOffBar + 16 * 8 + 16 + 1024;
// dW shared memory: ring [4][dz 2 x 64 x 128 B | X nq x 64 x 128 B], barriers.
constexpr uint32_t kDwStage = 2 * kBox64 + 4 * kBox64;
constexpr uint32_t kDwOffBar = kDwStages * kDwStage;
constexpr uint32_t kDwSmem = kDwOffBar + 16 * 8 + 16 + 1024;
static_assert(kDxSmem <= 232448 && kDwSmem <= 232448, "shared memory");

// Shared-memory descriptor of an MN-major bf16 operand in the 128-byte
// swizzled layout: rows of 64 MN-contiguous elements along K, 8-row groups
// 1024 bytes apart (stride byte offset) and consecutive 64-wide MN blocks
// `mn_stride` bytes apart (leading byte offset).
__device__ __forceinline__ uint64_t umma_desc_mn_sw128(uint32_t addr, uint32_t mn_stride) {
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)((mn_stride >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// kind::f16 instruction descriptor: fp32 D, bf16 A and B, M = 128, N = n;
// a_mn / b_mn: the operand is MN-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int n, bool a_mn, bool b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (a_mn ? 1u << 15 : 0u) | (b_mn ? 1u << 16 : 0u) |
           ((uint32_t)(n / 8) << 17) | ((uint32_t)(128 / 16) << 24);
}

__device__ __forceinline__ bool bwait(uint64_t *bar, uint32_t ph, int *status, volatile int *abort) {
    if (*abort) return false;
    if (mbar_wait(bar, ph, status)) return true;
    *abort = 1;
    return false;
}

__global__ void to_bf16_kernel(const float *__restrict__ src, __nv_bfloat16 *__restrict__ dst,
                               int64_t n) {
    const int64_t n4 = n / 4;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        const float4 v = reinterpret_cast<const float4 *>(src)[i];
        __nv_bfloat162 lo = __float22bfloat162_rn(make_float2(v.x, v.y));
        __nv_bfloat162 hi = __float22bfloat162_rn(make_float2(v.z, v.w));
        reinterpret_cast<__nv_bfloat162 *>(dst)[2 * i] = lo;
        reinterpret_cast<__nv_bfloat162 *>(dst)[2 * i + 1] = hi;
    }
    for (int64_t i = 4 * n4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        dst[i] = __float2bfloat16_rn(src[i]);
}

struct DxArgs {
    int64_t T;
    int nq;             // 64-column blocks per CTA slice (1, 2 or 4)
    int tiles_per_cta;  // 128-token tiles per CTA
    int *status;
};

__global__ void __launch_bounds__(kBThreads, 1)
router_dx_kernel(const __grid_constant__ CUtensorMap zmap, const __grid_constant__ CUtensorMap wmap,
                 const __grid_constant__ CUtensorMap omap, const DxArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_align<1024>(smem_raw);
    unsigned char *sB = smem + kDxOffB, *sA = smem + kDxOffA, *sO = smem + kDxOffO;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kDxOffBar);
    uint64_t *a_full = bars, *a_empty = bars + kDxStages, *b_full = bars + 2 * kDxStages;
    uint64_t *acc_full = b_full + 1, *acc_empty = acc_full + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 16);
    volatile int *s_abort = reinterpret_cast<volatile int *>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int layer = blockIdx.z, nq = a.nq, n0 = blockIdx.x * 64 * nq;
    const int ntiles = (int)((a.T + kBTileM - 1) / kBTileM);
    const int tb = blockIdx.y * a.tiles_per_cta;
    const int nt = max(0, min(ntiles, tb + a.tiles_per_cta) - tb);
    if (threadIdx.x == 0) {
        for (int i = 0; i < kDxStages; ++i) {
            mbar_init(&a_full[i], 1);
            mbar_init(&a_empty[i], 1);
        }
        mbar_init(b_full, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 4);
        }
        *s_abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();
    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0 && nt > 0) {
            prefetch_tensormap(&zmap);
            prefetch_tensormap(&wmap);
            mbar_arrive_expect_tx(b_full, (uint32_t)nq * kBox128);
            for (int q = 0; q < nq; ++q) tma_load_3d(sB + q * kBox128, &wmap, n0 + 64 * q, 0, layer, b_full);
            int issued = 0;
            for (int i = 0; i < nt; ++i) {
                const int s = i % kDxStages;
                if (i >= kDxStages && !bwait(&a_empty[s], (uint32_t)((i / kDxStages) - 1) & 1u, a.status, s_abort))
                    break;
                mbar_arrive_expect_tx(&a_full[s], 2 * kBox128);
                for (int b = 0; b < 2; ++b)
                    tma_load_3d(sA + (s * 2 + b) * kBox128, &zmap, 64 * b, (tb + i) * kBTileM, layer, &a_full[s]);
                issued = i + 1;
            }
            // every load completes before the CTA may exit
            mbar_wait(b_full, 0u, a.status);
            for (int i = issued > kDxStages ? issued - kDxStages : 0; i < issued; ++i)
                mbar_wait(&a_full[i % kDxStages], (uint32_t)(i / kDxStages) & 1u, a.status);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0 && nt > 0) {
            const uint32_t idesc = idesc_bf16(64 * nq, false, true);
            const uint32_t sa = smem_u32(sA), sb = smem_u32(sB);
            int issued = 0;
            if (bwait(b_full, 0u, a.status, s_abort)) {
                for (int i = 0; i < nt; ++i) {
                    const int s = i % kDxStages, buf = i & 1;
                    if (!bwait(&a_full[s], (uint32_t)(i / kDxStages) & 1u, a.status, s_abort)) break;
                    if (i >= 2 && !bwait(&acc_empty[buf], (uint32_t)((i >> 1) - 1) & 1u, a.status, s_abort))
                        break;
                    tc_fence_after();
                    const uint32_t d = tmem + (uint32_t)(buf * 256);
#pragma unroll
                    for (int kk = 0; kk < kBE / 16; ++kk) {
                        const uint64_t ad = umma_desc_sw128(sa + (s * 2 + (kk >> 2)) * kBox128 + (kk & 3) * 32);
                        const uint64_t bd = umma_desc_mn_sw128(sb + kk * 16 * 128, kBox128);
                        umma_f16(d, ad, bd, idesc, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(&a_empty[s]);
                    umma_commit(&acc_full[buf]);
                    issued = i + 1;
                }
            }
            // the tensor cores are done with TMEM and shared memory before the CTA ends
            if (issued > 0)
                mbar_wait(&acc_full[(issued - 1) & 1], (uint32_t)((issued - 1) >> 1) & 1u, a.status);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------- epilogue
        const int quad = warp & 3;  // TMEM lanes 32 quad .. (tokens of the tile)
        unsigned char *stage = sO + (size_t)quad * 4 * kBox32;
        for (int i = 0; i < nt; ++i) {
            const int buf = i & 1;
            const bool ok = __all_sync(kFull, bwait(&acc_full[buf], (uint32_t)(i >> 1) & 1u, a.status, s_abort));
            if (!ok) break;
            tc_fence_after();
            if (lane == 0) bulk_wait_read<0>();  // the previous tile's stores have read the staging
            __syncwarp();
            for (int q = 0; q < nq; ++q) {
                uint32_t r0[32], r1[32];
                const uint32_t tl = tmem + ((uint32_t)(32 * quad) << 16) + (uint32_t)(buf * 256 + 64 * q);
                tmem_ld32(tl, r0);
                tmem_ld32(tl + 32, r1);
                tmem_wait_ld();
                unsigned char *row = stage + q * kBox32 + lane * 128;
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    uint32_t w[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int e = 8 * c + 2 * j;
                        const float lo = __uint_as_float(e < 32 ? r0[e] : r1[e - 32]);
                        const float hi = __uint_as_float(e + 1 < 32 ? r0[e + 1] : r1[e + 1 - 32]);
                        __nv_bfloat162 p = __float22bfloat162_rn(make_float2(lo, hi));
                        w[j] = *reinterpret_cast<uint32_t *>(&p);
                    }
                    *reinterpret_cast<uint4 *>(row + ((c ^ (lane & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
            // the accumulator may take the tile after next
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[buf]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                for (int q = 0; q < nq; ++q)
                    tma_store_3d(&omap, stage + q * kBox32, n0 + 64 * q, (tb + i) * kBTileM + 32 * quad, layer);
                bulk_commit_group();
            }
            __syncwarp();
        }
        if (lane == 0) bulk_wait_all<0>();
        __syncwarp();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, 512);
}

struct DwArgs {
    int64_t T;
    int nq;
    int64_t chunk_tokens;  // a multiple of kBKt
    int E;
    int H;
    int L;
    float *partials;       // [chunks][L][E][H]
    int *status;
};

__global__ void __launch_bounds__(kBThreads, 1)
router_dw_kernel(const __grid_constant__ CUtensorMap zmap, const __grid_constant__ CUtensorMap xmap,
                 const DwArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_align<1024>(smem_raw);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kDwOffBar);
    uint64_t *full = bars, *empty = bars + kDwStages, *acc_full = bars + 2 * kDwStages;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 16);
    volatile int *s_abort = reinterpret_cast<volatile int *>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int layer = blockIdx.z, nq = a.nq, n0 = blockIdx.x * 64 * nq, chunk = blockIdx.y;
    const int64_t t0 = (int64_t)chunk * a.chunk_tokens;
    const int64_t t1 = min64(a.T, t0 + a.chunk_tokens);
    const int nk = t1 > t0 ? (int)((t1 - t0 + kBKt - 1) / kBKt) : 0;
    const uint32_t stage_bytes = 2 * kBox64 + (uint32_t)nq * kBox64;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kDwStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(acc_full, 1);
        *s_abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, 256);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();
    bool acc_ok = true;
    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0 && nk > 0) {
            prefetch_tensormap(&zmap);
            prefetch_tensormap(&xmap);
            int issued = 0;
            for (int j = 0; j < nk; ++j) {
                const int s = j % kDwStages;
                if (j >= kDwStages && !bwait(&empty[s], (uint32_t)((j / kDwStages) - 1) & 1u, a.status, s_abort))
                    break;
                unsigned char *st = smem + s * kDwStage;
                const int ty = (int)(t0 + (int64_t)j * kBKt);
                mbar_arrive_expect_tx(&full[s], stage_bytes);
                for (int b = 0; b < 2; ++b) tma_load_3d(st + b * kBox64, &zmap, 64 * b, ty, layer, &full[s]);
                for (int q = 0; q < nq; ++q)
                    tma_load_3d(st + (2 + q) * kBox64, &xmap, n0 + 64 * q, ty, layer, &full[s]);
                issued = j + 1;
            }
            for (int j = issued > kDwStages ? issued - kDwStages : 0; j < issued; ++j)
                mbar_wait(&full[j % kDwStages], (uint32_t)(j / kDwStages) & 1u, a.status);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0 && nk > 0) {
            const uint32_t idesc = idesc_bf16(64 * nq, true, true);
            int issued = 0;
            for (int j = 0; j < nk; ++j) {
                const int s = j % kDwStages;
                if (!bwait(&full[s], (uint32_t)(j / kDwStages) & 1u, a.status, s_abort)) break;
                tc_fence_after();
                const uint32_t st = smem_u32(smem + s * kDwStage);
#pragma unroll
                for (int kk = 0; kk < kBKt / 16; ++kk) {
                    const uint64_t ad = umma_desc_mn_sw128(st + kk * 16 * 128, kBox64);
                    const uint64_t bd = umma_desc_mn_sw128(st + 2 * kBox64 + kk * 16 * 128, kBox64);
                    umma_f16(tmem, ad, bd, idesc, (j > 0 || kk > 0) ? 1u : 0u);
                }
                umma_commit(&empty[s]);
                issued = j + 1;
            }
            umma_commit(acc_full);
            mbar_wait(acc_full, 0u, a.status);
            if (issued < nk) *s_abort = 1;
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------- epilogue
        const int quad = warp & 3;  // TMEM lanes 32 quad ..: experts
        if (nk > 0) acc_ok = __all_sync(kFull, bwait(acc_full, 0u, a.status, s_abort));
        tc_fence_after();
        const int e = 32 * quad + lane;
        float *dst = a.partials + (((size_t)chunk * a.L + layer) * a.E + e) * a.H + n0;
        for (int c = 0; c < 2 * nq; ++c) {
            uint32_t r[32];
            if (nk > 0 && acc_ok) {
                tmem_ld32(tmem + ((uint32_t)(32 * quad) << 16) + (uint32_t)(32 * c), r);
                tmem_wait_ld();
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) r[j] = 0u;
            }
#pragma unroll
            for (int j = 0; j < 32; j += 4)
                *reinterpret_cast<float4 *>(dst + 32 * c + j) =
                    make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, 256);
}

// dW = the chunks' partial sums added in chunk order (float4 lanes).
__global__ void __launch_bounds__(256)
router_dw_reduce_kernel(const float *__restrict__ partials, int chunks, int64_t n, float *__restrict__ dW) {
    const int64_t n4 = n / 4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        float4 acc = __ldg(reinterpret_cast<const float4 *>(partials) + i);
        for (int c = 1; c < chunks; ++c) {
            const float4 v = __ldg(reinterpret_cast<const float4 *>(partials + (size_t)c * n) + i);
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
        reinterpret_cast<float4 *>(dW)[i] = acc;
    }
}

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

int sms_now_bwd() {
    int dev = 0, n = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n;
}

int hidden_blocks(int H) { return (H / 64) % 4 == 0 ? 4 : ((H / 64) % 2 == 0 ? 2 : 1); }

cudaError_t launch_ex(const void *kern, dim3 grid, uint32_t smem, void **args, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kBThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelExC(&cfg, kern, args);
}

}  // namespace
}  // namespace dol

extern "C" {

size_t do_router_backward_workspace_size(int64_t T, int32_t E, int32_t H, int32_t L) {
    if (T < 1 || E < 1 || H < 1 || L < 1) return 0;
    return dol::kWsHeader + dol::round256(sizeof(uint16_t) * (size_t)L * (size_t)T * (size_t)E) +
           dol::round256(sizeof(float) * (size_t)dol::kDwChunksMax * L * (size_t)E * (size_t)H);
}

do_status do_router_backward(const void *X, const void *Wr, const float *dlogits, int64_t T,
                             int32_t H, int32_t E, int32_t L, float *dW, void *dX,
                             void *workspace, size_t workspace_bytes, void *stream) {
    if (T < 1 || E < 1 || H < 1 || L < 1) return DO_ERR_INVALID_ARG;
    if (!X || !Wr || !dlogits || !dW) return DO_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(Wr) |
         reinterpret_cast<uintptr_t>(dlogits) | reinterpret_cast<uintptr_t>(dW) |
         reinterpret_cast<uintptr_t>(dX)) % 16)
        return DO_ERR_INVALID_ARG;
    if (E != dol::kBE || H % 64 != 0 || T > (int64_t)INT_MAX - dol::kBTileM || L > 65535)
        return DO_ERR_UNSUPPORTED;
    const size_t need = do_router_backward_workspace_size(T, E, H, L);
    if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 256 || workspace_bytes < need)
        return DO_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    char *ws = static_cast<char *>(workspace);
    int *status = reinterpret_cast<int *>(ws);
    __nv_bfloat16 *dzb = reinterpret_cast<__nv_bfloat16 *>(ws + dol::kWsHeader);
    float *partials = reinterpret_cast<float *>(
        ws + dol::kWsHeader + dol::round256(sizeof(uint16_t) * (size_t)L * (size_t)T * (size_t)E));
    const int64_t n = (int64_t)L * T * E;
    dol::to_bf16_kernel<<<1024, 256, 0, s>>>(dlogits, dzb, n);
    if (cudaGetLastError() != cudaSuccess) return DO_ERR_CUDA;
    const int nq = dol::hidden_blocks(H);
    const int nslices = H / (64 * nq);
    const int sms = dol::sms_now_bwd();
    CUtensorMap zmap_k, wmap, xmap, zmap_mn, omap;
    // dz [L][T][E] as the K-major A of dX (boxes of 64 experts x 128 tokens)
    // and as the MN-major A of dW (64 experts x 64 tokens); W [L][E][H] and
    // X [L][T][H] as MN-major B operands; dX [L][T][H] stored in 64 x 32 boxes
    if (!dol::encode_tensor_map_3d_bf16(&zmap_k, dzb, (uint64_t)L, (uint64_t)T, (uint64_t)E, 64, 128) ||
        !dol::encode_tensor_map_3d_bf16(&zmap_mn, dzb, (uint64_t)L, (uint64_t)T, (uint64_t)E, 64, 64) ||
        !dol::encode_tensor_map_3d_bf16(&wmap, Wr, (uint64_t)L, (uint64_t)E, (uint64_t)H, 64, 128) ||
        !dol::encode_tensor_map_3d_bf16(&xmap, X, (uint64_t)L, (uint64_t)T, (uint64_t)H, 64, 64))
        return DO_ERR_INVALID_ARG;
    static bool attrs_set[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DO_ERR_CUDA;
    if (dev >= 0 && dev < 64 && !attrs_set[dev]) {
        if (cudaFuncSetAttribute(dol::router_dx_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)dol::kDxSmem) != cudaSuccess ||
            cudaFuncSetAttribute(dol::router_dw_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)dol::kDwSmem) != cudaSuccess)
            return DO_ERR_CUDA;
        attrs_set[dev] = true;
    }
    // dW: chunks of the tokens so that slices x chunks x L fill the GPU once
    int64_t chunks = sms / ((int64_t)nslices * L);
    if (chunks < 1) chunks = 1;
    if (chunks > dol::kDwChunksMax) chunks = dol::kDwChunksMax;
    const int64_t ktiles = (T + dol::kBKt - 1) / dol::kBKt;
    if (chunks > ktiles) chunks = ktiles;
    const int64_t chunk_tokens = (ktiles + chunks - 1) / chunks * dol::kBKt;
    chunks = (T + chunk_tokens - 1) / chunk_tokens;
    dol::DwArgs dwa = {T, nq, chunk_tokens, E, H, L, partials, status};
    void *dw_args[] = {&zmap_mn, &xmap, &dwa};
    if (dol::launch_ex((const void *)dol::router_dw_kernel, dim3(nslices, (unsigned)chunks, L),
                       dol::kDwSmem, dw_args, s) != cudaSuccess)
        return DO_ERR_CUDA;
    const int64_t nw = (int64_t)L * E * H;
    dol::router_dw_reduce_kernel<<<(unsigned)((nw / 4 + 255) / 256 < 4096 ? (nw / 4 + 255) / 256 : 4096), 256, 0, s>>>(
        partials, (int)chunks, nw, dW);
    if (cudaGetLastError() != cudaSuccess) return DO_ERR_CUDA;
    if (dX) {
        if (!dol::encode_tensor_map_3d_bf16(&omap, dX, (uint64_t)L, (uint64_t)T, (uint64_t)H, 64, 32))
            return DO_ERR_INVALID_ARG;
        const int ntiles = (int)((T + dol::kBTileM - 1) / dol::kBTileM);
        int gy = sms / (nslices * L);
        if (gy < 1) gy = 1;
        if (gy > ntiles) gy = ntiles;
        const int per = (ntiles + gy - 1) / gy;
        gy = (ntiles + per - 1) / per;
        dol::DxArgs dxa = {T, nq, per, status};
        void *dx_args[] = {&zmap_k, &wmap, &omap, &dxa};
        if (dol::launch_ex((const void *)dol::router_dx_kernel, dim3(nslices, gy, L), dol::kDxSmem,
                           dx_args, s) != cudaSuccess)
            return DO_ERR_CUDA;
    }
    return DO_OK;
}

}  // extern "C"
