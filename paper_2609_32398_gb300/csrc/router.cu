// Router-side fusion: the router's linear map z = X W^T (bf16 hidden states
// X [L][T][H] and weights W [L][E][H], fp32 accumulation; Sec. 4.1: a linear
// map from the hidden size to the n = 128 experts) on the tcgen05 tensor
// cores, with step 1 of the DO-loss (Top-K, Sec. 3.1.1 Eq. 1; the signatures
// and the per-CTA co-occurrence counts of App. C.3) in the GEMM's epilogue.
// The logits are written once, for the loss kernel, and never read back for
// the selection.
//
// One persistent CTA per SM owns a contiguous, balanced range of 32-token
// signature words (13 or 14 words for T = 65536 on 152 SMs) and walks it in
// pair tiles of up to eight words (two 128-token MMA tiles that share one
// slice of W):
//   warp 0   TMA producer: per 64-wide slice of the hidden size, one X box
//            [32 tokens x 64] per word and one W box [128 experts x 64] (bf16,
//            128-byte swizzle) into a 3-stage ring (48 KB a stage, 32 KB of it
//            X, so each SM keeps 96 KB of X in flight);
//   warp 1   MMA issuer: per stage 2 x 4 tcgen05.mma kind::f16 (bf16, K = 16)
//            into the two accumulators [128 lanes x 128 fp32] of the pair,
//            double-buffered (all 512 TMEM columns);
//   warps 2-5 epilogue, one TMEM lane quarter each (the same 32 rows of both
//            tiles): the logits go TMEM -> registers -> a swizzled shared-memory
//            tile (the signature kernel's layout), out to HBM by TMA stores, and
//            the signature kernel's per-token selection and signature words run
//            on that tile.  The co-occurrence counts go into a shared triangle
//            of 16-bit counters (two per word: the CTA's range is below 65536
//            tokens), written out unpacked at the end; for longer ranges they
//            go straight to the CTA's triangle in global memory as L2
//            reductions.

#include "sig_fast.cuh"

namespace dol {
namespace {

constexpr int kRE = 128;                        // experts = N of the MMA
constexpr int kRTileM = 128;                    // tokens per MMA tile = M
constexpr int kRPairWords = 8;                  // signature words of a pair tile (2 x 128 tokens)
constexpr int kRSlice = 64;                     // hidden columns per stage (128 bytes of bf16)
constexpr int kRStages = 3;
constexpr int kRWordBox = 32 * 128;             // the X box of one signature word (32 rows)
constexpr int kRTileBytes = kRTileM * 128;      // one MMA tile's A slice, or the W slice
constexpr int kRStageBytes = 3 * kRTileBytes;   // X of two tiles + W
constexpr int kREpiWarps = 4;
constexpr int kRThreads = (2 + kREpiWarps) * 32;
constexpr int kRZTileBytes = 32 * kRE * 4;      // one warp's 32 tokens x 128 logits
constexpr int kRTmemCols = 4 * kRE;             // two buffers x two fp32 accumulators
using RC = SigCfg<kRE>;

constexpr size_t kROffZ = (size_t)kRStages * kRStageBytes;
constexpr size_t kROffRowoff = kROffZ + (size_t)kREpiWarps * kRZTileBytes;
constexpr size_t kROffTri = kROffRowoff + (size_t)kRE * 4;          // packed 16-bit counters
constexpr size_t kROffBars = kROffTri + (size_t)(RC::kCoocWords / 2) * 4;
constexpr size_t kRNumBars = 2 * kRStages + 4;
constexpr size_t kROffScal = kROffBars + kRNumBars * 8;
constexpr size_t kRSmem = kROffScal + 16 + 1024;  // + alignment slack of the base

struct RouterArgs {
    int64_t T, W;
    int H;
    int packed;  // 1: 16-bit shared counters (no CTA range above 65535 tokens); 0: L2 reductions
    uint32_t *bits;
    uint8_t *idx;
    uint32_t *cooc;
    int *counts;
    ZeroSpans zero;
    int *status;
};

// Words of the next tile of a range with r words left: pairs of MMA tiles
// (eight words) that share each slice of W, the remainder last.
__device__ __forceinline__ int next_tile_words(int64_t r) {
    return r < kRPairWords ? (int)r : kRPairWords;
}

template <int K>
__global__ void __launch_bounds__(kRThreads, 1)
router_sig_kernel(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap wmap,
                  const __grid_constant__ CUtensorMap zmap, RouterArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_align<1024>(smem_raw);
    unsigned char *ring = smem;
    unsigned char *ztiles = smem + kROffZ;
    int *s_rowoff = reinterpret_cast<int *>(smem + kROffRowoff);
    uint32_t *s_tri = reinterpret_cast<uint32_t *>(smem + kROffTri);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kROffBars);
    uint64_t *full = bars, *empty = bars + kRStages;
    uint64_t *acc_full = bars + 2 * kRStages, *acc_free = acc_full + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + kROffScal);
    volatile int *s_abort = reinterpret_cast<volatile int *>(smem + kROffScal + 4);

    pdl_trigger();
    const int layer = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nkb = a.H / kRSlice;
    // this CTA's signature words [wb, we): an even split of the problem's W words
    const int64_t wb = (int64_t)blockIdx.x * a.W / gridDim.x;
    const int64_t we = (int64_t)(blockIdx.x + 1) * a.W / gridDim.x;
    // this CTA's co-occurrence triangle (the reduction kernel's input)
    uint32_t *tri = a.cooc + ((size_t)layer * gridDim.x + blockIdx.x) * (size_t)RC::kCoocWords;
    // Shared-memory and TMEM set-up touch no global memory: they overlap the
    // end of the previous kernel on the stream.
    for (int e = threadIdx.x; e < kRE; e += kRThreads) s_rowoff[e] = cooc_row_offset<kRE>(e) - (e & ~3);
    if (a.packed)
        for (int i = threadIdx.x; i < RC::kCoocWords / 2; i += kRThreads) s_tri[i] = 0u;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kRStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_free[b], kREpiWarps);
        }
        *s_abort = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&xmap);
        prefetch_tensormap(&wmap);
        prefetch_tensormap(&zmap);
    }
    if (warp == 1) tmem_alloc(tmem_slot, kRTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // The previous kernel on the stream may still read the accumulators that
    // are cleared here (and may have written X): wait for it first.
    pdl_wait();
#pragma unroll
    for (int z = 0; z < 3; ++z)
        for (int64_t i = (int64_t)blockIdx.x * kRThreads + threadIdx.x; i < a.zero.n[z];
             i += (int64_t)gridDim.x * kRThreads)
            a.zero.p[z][i] = 0;
    if (!a.packed) {  // the global triangle starts at zero (ordered by the barrier)
        uint4 *t4 = reinterpret_cast<uint4 *>(tri);
        for (int q = threadIdx.x; q < RC::kCoocWords / 4; q += kRThreads) t4[q] = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int g = 0;
            for (int64_t wt = wb, nw = 0; wt < we && !*s_abort; wt += nw) {
                nw = next_tile_words(we - wt);
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const int s = g % kRStages, r = g / kRStages;
                    if (r > 0 && !mbar_wait(&empty[s], (uint32_t)(r - 1) & 1u, a.status)) *s_abort = 1;
                    if (*s_abort) break;
                    unsigned char *st = ring + (size_t)s * kRStageBytes;
                    // rows of missing words keep stale data: their outputs are not used
                    mbar_arrive_expect_tx(&full[s], (uint32_t)((int)nw * kRWordBox + kRTileBytes));
                    for (int j = 0; j < nw; ++j)
                        tma_load_3d(st + j * kRWordBox, &xmap, kb * kRSlice, (int)(32 * (wt + j)), layer,
                                    &full[s]);
                    tma_load_3d(st + 2 * kRTileBytes, &wmap, kb * kRSlice, 0, layer, &full[s]);
                }
            }
            // every issued load lands before the CTA may exit
            for (int q = g > kRStages ? g - kRStages : 0; q < g; ++q)
                mbar_wait(&full[q % kRStages], (uint32_t)(q / kRStages) & 1u, a.status);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            // kind::f16: fp32 accumulate, bf16 A and B, both K-major, N = 128, M = 128
            const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kRE / 8) << 17) |
                                   ((uint32_t)(kRTileM / 16) << 24);
            const uint32_t ring_u32 = smem_u32(ring);
            int g = 0, i = 0;
            for (int64_t wt = wb, nw = 0; wt < we && !*s_abort; wt += nw, ++i) {
                nw = next_tile_words(we - wt);
                const int buf = i & 1;
                const int halves = nw > 4 ? 2 : 1;  // the second MMA tile has words
                if (i >= 2 && !mbar_wait(&acc_free[buf], (uint32_t)((i >> 1) - 1) & 1u, a.status)) {
                    *s_abort = 1;
                    break;
                }
                tc_fence_after();
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const int s = g % kRStages;
                    if (!mbar_wait(&full[s], (uint32_t)(g / kRStages) & 1u, a.status)) *s_abort = 1;
                    if (*s_abort) break;
                    tc_fence_after();
                    const uint32_t sa = ring_u32 + (uint32_t)(s * kRStageBytes);
                    for (int h = 0; h < halves; ++h) {
                        const uint32_t d_tmem = tmem + (uint32_t)((2 * buf + h) * kRE);
#pragma unroll
                        for (int kk = 0; kk < kRSlice / 16; ++kk)
                            umma_f16(d_tmem, umma_desc_sw128(sa + h * kRTileBytes + kk * 32),
                                     umma_desc_sw128(sa + 2 * kRTileBytes + kk * 32), idesc,
                                     (kb > 0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(&empty[s]);  // the stage is free once these MMAs are done
                }
                if (*s_abort) break;
                umma_commit(&acc_full[buf]);
            }
            // the tensor cores are done with shared memory and TMEM before the
            // CTA moves on (the last commit covers every MMA before it)
            if (g > 0) mbar_wait(&empty[(g - 1) % kRStages], (uint32_t)((g - 1) / kRStages) & 1u, a.status);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int ew = warp - 2, quarter = warp & 3;
        unsigned char *tp = ztiles + (size_t)ew * kRZTileBytes;
        uint32_t cnt[kRE / 32];
#pragma unroll
        for (int r = 0; r < kRE / 32; ++r) cnt[r] = 0u;
        int i = 0;
        for (int64_t wt = wb, nw = 0; wt < we; wt += nw, ++i) {
            nw = next_tile_words(we - wt);
            const int buf = i & 1;
            const bool ok = !*s_abort && mbar_wait(&acc_full[buf], (uint32_t)(i >> 1) & 1u, a.status);
            if (!__all_sync(kFull, ok)) {  // leave together: the warp collectives below
                *s_abort = 1;
                break;
            }
            tc_fence_after();
            for (int h = 0; h < 2; ++h) {
                const int64_t w = wt + 4 * h + quarter;  // this warp's word of tile h
                const bool mine = 4 * h + quarter < nw;
                if (mine) {
                    // the staging tile is free once the previous stores have read it
                    if (lane == 0) bulk_wait_read<0>();
                    __syncwarp();
                    const uint32_t tl =
                        tmem + (uint32_t)((2 * buf + h) * kRE) + ((uint32_t)(quarter * 32) << 16);
#pragma unroll
                    for (int b = 0; b < kRE / 32; ++b) {
                        uint32_t v[32];
                        tmem_ld32(tl + 32 * b, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            *reinterpret_cast<uint4 *>(chunk_ptr(tp, 8 * b + c, lane)) =
                                make_uint4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
                    }
                }
                if (h == 1) {  // both accumulators of the pair have been read
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&acc_free[buf]);
                }
                if (!mine) continue;
                // the logits of these 32 tokens go out while the selection reads them
                fence_proxy_async_smem();
                __syncwarp();
                const int row0 = (int)(32 * w);
                if (lane == 0) {
#pragma unroll
                    for (int b = 0; b < kRE / 32; ++b)
                        tma_store_3d(&zmap, tp + b * 4096, 32 * b, row0, layer);
                    bulk_commit_group();
                }
                const int64_t t = (int64_t)row0 + lane;
                const bool valid = t < a.T;
                int sel[K];
                float val[K];
                select_topk<kRE, K, true>(tp, lane, sel, val);
                if (a.idx && valid) store_idx<K>(a.idx + ((int64_t)layer * a.T + t) * K, sel);
                if (valid) {  // c_ab += 1 for the pairs a < b, 16-bit halves of shared words
                    int so[K];
#pragma unroll
                    for (int q = 0; q < K; ++q) so[q] = sel[q];
#pragma unroll
                    for (int i2 = 1; i2 < K; ++i2)
#pragma unroll
                        for (int j2 = i2; j2 > 0; --j2) {
                            const int lo = min(so[j2 - 1], so[j2]), hi = max(so[j2 - 1], so[j2]);
                            so[j2 - 1] = lo;
                            so[j2] = hi;
                        }
#pragma unroll
                    for (int q1 = 0; q1 < K - 1; ++q1) {
                        const int row = s_rowoff[so[q1]];
#pragma unroll
                        for (int q2 = q1 + 1; q2 < K; ++q2) {
                            const int wi = row + so[q2];
                            if (a.packed) atomicAdd(&s_tri[wi >> 1], 1u << (16 * (wi & 1)));
                            else atomicAdd(&tri[wi], 1u);
                        }
                    }
                }
                emit_words<kRE, K, true>(sel, valid, lane, a.bits + (int64_t)layer * kRE * a.W + w, a.W,
                                         cnt);
            }
        }
        if (lane == 0) bulk_wait_all<0>();  // the last stores are complete before exit
        // counts n_a: on the triangle's diagonal and into the problem's totals
#pragma unroll
        for (int r = 0; r < kRE / 32; ++r)
            if (cnt[r]) {
                const int e = 32 * r + lane;
                const int wi = s_rowoff[e] + e;
                if (a.packed) atomicAdd(&s_tri[wi >> 1], cnt[r] << (16 * (wi & 1)));
                else atomicAdd(&tri[wi], cnt[r]);
                atomicAdd(&a.counts[layer * kRE + e], (int)cnt[r]);
            }
        if (a.packed) {
            // all epilogue warps have counted: the triangle out, unpacked
            asm volatile("bar.sync 1, %0;" ::"n"(kREpiWarps * 32) : "memory");
            for (int q = threadIdx.x - 64; q < RC::kCoocWords / 2; q += kREpiWarps * 32) {
                const uint32_t v = s_tri[q];
                reinterpret_cast<uint2 *>(tri)[q] = make_uint2(v & 0xFFFFu, v >> 16);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, kRTmemCols);
    }
}

template <int K>
cudaError_t run_router(const CUtensorMap &xm, const CUtensorMap &wm, const CUtensorMap &zm,
                       const RouterArgs &a, int ctas, int L, cudaStream_t s) {
    auto kern = router_sig_kernel<K>;
    cudaError_t e = ensure_smem_limit<router_sig_kernel<K>>(kRSmem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)ctas, (unsigned)L);
    cfg.blockDim = dim3(kRThreads);
    cfg.dynamicSmemBytes = kRSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, xm, wm, zm, a);
}

int sm_count_router() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 148;
    return n;
}

}  // namespace

bool router_supported(const Problem &p, int H, const void *X, const void *Wr, const float *logits) {
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    return p.E == kRE && k_ok && H >= kRSlice && H % kRSlice == 0 &&
           reinterpret_cast<uintptr_t>(X) % 16 == 0 && reinterpret_cast<uintptr_t>(Wr) % 16 == 0 &&
           reinterpret_cast<uintptr_t>(logits) % 16 == 0 && p.T <= (int64_t)INT_MAX - kRTileM;
}

int router_ctas_per_problem(const Problem &p) {
    int sms = sm_count_router();
    if (sms > kMaxSigCtas) sms = kMaxSigCtas;
    int64_t gx = sms / p.L;
    if (gx > p.W) gx = p.W;
    if (gx < 1) gx = 1;
    return (int)gx;
}

cudaError_t launch_router_signatures(const void *X, const void *Wr, int H, float *logits,
                                     const Problem &p, uint32_t *bits, int *counts, uint8_t *idx,
                                     uint32_t *cooc, const ZeroSpans &zero, int *status,
                                     cudaStream_t s) {
    CUtensorMap xm, wm, zm;
    if (!encode_tensor_map_3d_bf16(&xm, X, (uint64_t)p.L, (uint64_t)p.T, (uint64_t)H, kRSlice, 32) ||
        !encode_tensor_map_3d_bf16(&wm, Wr, (uint64_t)p.L, (uint64_t)kRE, (uint64_t)H, kRSlice, kRE) ||
        !encode_tensor_map_3d_f32(&zm, logits, (uint64_t)p.L, (uint64_t)p.T, (uint64_t)kRE, 32))
        return cudaErrorInvalidValue;
    RouterArgs a;
    a.T = p.T;
    a.W = p.W;
    a.H = H;
    const int ctas = router_ctas_per_problem(p);
    // 16-bit shared counters hold a CTA's counts while its range is below
    // 65536 tokens; longer ranges add into the CTA's global triangle (L2)
    a.packed = 32 * ((p.W + ctas - 1) / ctas) <= 65535;
    a.bits = bits;
    a.idx = idx;
    a.cooc = cooc;
    a.counts = counts;
    a.zero = zero;
    a.status = status;
    switch (p.k) {
        case 1: return run_router<1>(xm, wm, zm, a, ctas, p.L, s);
        case 2: return run_router<2>(xm, wm, zm, a, ctas, p.L, s);
        case 4: return run_router<4>(xm, wm, zm, a, ctas, p.L, s);
        default: return run_router<8>(xm, wm, zm, a, ctas, p.L, s);
    }
}

}  // namespace dol
