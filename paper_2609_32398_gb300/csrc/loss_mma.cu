// Step 3 on the tensor cores (E = 128, sigmoid-norm gate, k in {1, 2, 4, 8},
// D from the co-occurrence counts of the same tokens): the surrogate DO-loss
// and its gradient (Sec. 3.1.3, Eq. do_loss).
//
// Put D'_ij = D_ij off the diagonal and D'_ii = -R_i, R_i = sum_j D_ij.  The
// k-row gather of D' for token t is then minus the integer weight:
//   V_ti = sum_{j in S_t} D'_ji = -w_ti,   w_ti = f_ti R_i - sum_{j in S_t} D_ji,
// and with F the one-hot rows of the selected experts V = F D' is a matrix
// product.  It is exact on the tensor cores: F is 0/1 in fp16 and D' is cut
// into two fp16 pieces D' = 2048 hi + lo.  Off the diagonal 0 <= D <= T, so
// hi = D >> 11 and lo = D & 2047; on the diagonal -R = 2048 a + b with a even
// (a = -2 round(R / 4096)) and |b| <= 2048.  All pieces are exact in fp16
// while R < 2^23 (R <= (E - 1) T, so T <= 66052), and k-term sums of them
// stay below 2^24, exact in the fp32 accumulators.  With s = sigmoid(z),
// S = sum_i s_i, SV = sum_i s_i V_ti and c = grad_scale d_scale / (m^2 k):
//   A_t = sum_i p_ti w_ti = -SV / S,
//   dz_ti = c/S s_i (1 - s_i) (w_ti - A_t) = s_i (1 - s_i) (c SV / S^2 - c/S V_ti).
//
// The pieces of D' come ready-made from the reduction kernel as the image of
// the shared-memory operand B (dprime_pieces, 64 KB per problem).
//
// A persistent CTA takes a run of 128-token tiles of one problem:
//   warp 0       allocates TMEM; one thread copies B in with one bulk copy and
//                issues the MMAs V(tile) = F(tile) [hi | lo] (M = 128, N = 256,
//                K = 128) into one of two accumulators, committed to an
//                mbarrier per accumulator;
//   warps 1-3    write F of the next tile (K-major, 128-byte swizzle) once
//                the MMA of the previous one has read it;
//   warps 4-19   the epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31 (its
//                32 tokens) and the 32 experts of chunk (w - 4) / 4.  Each owns
//                a 32 x 32 logits box per tile, loaded by TMA two tiles ahead;
//                pass 1 forms s = 1 / (1 + e^-z), S and SV and writes s (1 - s)
//                and V back into the accumulator; the four warps of a
//                token quadrant exchange their (S, SV) through their boxes;
//                pass 2 writes dz into the box in place and a TMA store sends
//                it to dlogits; once the store has read the box it takes the
//                logits of the tile after next.
// Tensor maps are 3-D [L][T][E]: rows past the end of a problem read as zero
// and are dropped on store.
//
// With the routing gradient (kRG, the backward half of the routed step), each
// epilogue thread also adds, for its token, the gradient of the re-normalized
// combine weights (Sec. 3.1.1) w_q = s_q / sum of the chosen s, for the
// upstream gradient g_q of the chosen experts e_q held fixed:
//   dz_{e_q} += w_q (1 - s_q) (g_q - sum_q' g_q' w_q').
// The chosen logits are read from the boxes after pass 1 (each warp those in
// its 64 columns), the two warps of the token swap their partial sums with the
// (S, SV) exchange, and after pass 2 each adds its entries into the dz boxes
// before the TMA store.  The sigmoid is pass 1's: one ex2 and one rcp.
#include <cuda_fp16.h>

#include <climits>

#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kE = 128;
constexpr int kTileM = 128;
constexpr int kEpiWarp0 = 4;                        // warps 4..19: w % 4 = TMEM quadrant
constexpr int kEpiWarps = 16;                       // 4 quadrants x 4 expert chunks
constexpr int kWarps = kEpiWarp0 + kEpiWarps;
constexpr int kThreads = kWarps * 32;
constexpr int kFWarp0 = 1, kFWarps = 3;             // builders of F
constexpr int kFThreads = kFWarps * 32;
constexpr int kBoxBytes = 32 * 128;                 // 32 rows x 32 fp32
constexpr int kAtomA = kTileM * 128;                // one 64-column K atom of F
constexpr int kAtomB = 2 * kE * 128;                // one 64-column K atom of B (256 rows)
constexpr int kZBoxes = 2 * kEpiWarps;              // two tiles of boxes in flight
constexpr int kOffB = 0;
constexpr int kOffA = kOffB + 2 * kAtomB;           // 64 KB
constexpr int kOffZ = kOffA + 2 * kAtomA;           // 96 KB
constexpr int kOffBar = kOffZ + kZBoxes * kBoxBytes;  // 224 KB
constexpr int kNumBars = 2 + 2 + 1 + 1 + kZBoxes;   // mma_done[2], acc_free[2], f_full, b_full, zfull[32]
constexpr int kOffScal = kOffBar + 8 * kNumBars;    // tmem base, abort, last
constexpr int kOffPart = kOffScal + 16;             // [kWarps] fp64
constexpr int kSmemMma = kOffPart + 8 * kWarps + 1024;  // + alignment slack
static_assert(kOffScal % 8 == 0 && kOffPart % 8 == 0, "alignment");
static_assert(2 * kAtomB == kBImageBytes, "B image");
static_assert(kSmemMma <= 232448, "shared memory");
constexpr uint32_t kTmemCols = 512;                 // two 256-column accumulators
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// s = sigmoid(z) and 1 - s, each without cancellation, from e = 2^(-|z| log2 e)
// and one approximate reciprocal (as pass 1 forms s)
__device__ __forceinline__ void sigmoid_pair(float z, float &s, float &oms) {
    const float e = ex2_approx(fabsf(z) * -kLog2e);
    const float r = rcp_approx(1.0f + e);
    s = z >= 0.0f ? r : e * r;
    oms = z >= 0.0f ? e * r : r;
}

__device__ __forceinline__ int atom_add_acq_rel(int *p, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

__device__ __forceinline__ void named_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

struct MmaArgs {
    const float *logits;
    const uint8_t *idx;
    const unsigned char *bimg;  // [L][kBImageBytes]
    int *n_zero;                // may be null
    int64_t T;
    int tiles_per_cta;
    float coef;
    double scale;
    double *partials;
    int *done;
    float *loss;
    int *status;
    int *status_out;  // may be null: the last CTA ORs the status word into it
    // routing gradient (kRG): the chosen experts [L][T][K] and the upstream
    // gradient of their combine weights [L][T][K]
    const int *rg_ids;
    const float *rg_g;
    // a matrix summed over ranks (Eq. global_do): img_ok [L] from the image
    // kernel; a layer whose flag is 0 is left to the ALU kernel (may be null)
    const int *img_ok;
};

// K ints and K floats of one token row (16-, 8- or 4-byte loads)
template <int K>
__device__ __forceinline__ void load_route_row(const int *ids, const float *g, int (&e)[K],
                                               float (&v)[K]) {
    if constexpr (K >= 4) {
#pragma unroll
        for (int q = 0; q < K; q += 4) {
            const int4 a = __ldg(reinterpret_cast<const int4 *>(ids + q));
            const float4 b = __ldg(reinterpret_cast<const float4 *>(g + q));
            e[q] = a.x; e[q + 1] = a.y; e[q + 2] = a.z; e[q + 3] = a.w;
            v[q] = b.x; v[q + 1] = b.y; v[q + 2] = b.z; v[q + 3] = b.w;
        }
    } else if constexpr (K == 2) {
        const int2 a = __ldg(reinterpret_cast<const int2 *>(ids));
        const float2 b = __ldg(reinterpret_cast<const float2 *>(g));
        e[0] = a.x; e[1] = a.y;
        v[0] = b.x; v[1] = b.y;
    } else {
        e[0] = __ldg(ids);
        v[0] = __ldg(g);
    }
}

template <int K>
__device__ __forceinline__ void load_sel(const uint8_t *p, uint32_t (&r)[2]) {
    r[0] = r[1] = 0u;
    if (K == 8) {
        const uint2 v = __ldg(reinterpret_cast<const uint2 *>(p));
        r[0] = v.x;
        r[1] = v.y;
    } else if (K == 4) {
        r[0] = __ldg(reinterpret_cast<const uint32_t *>(p));
    } else if (K == 2) {
        r[0] = __ldg(reinterpret_cast<const uint16_t *>(p));
    } else {
        r[0] = __ldg(p);
    }
}

template <int K, bool kRG>
__global__ void __launch_bounds__(kThreads, 1)
loss_mma_kernel(const __grid_constant__ CUtensorMap zmap, const __grid_constant__ CUtensorMap dzmap,
                const MmaArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_align<1024>(smem_raw);
    unsigned char *sB = smem + kOffB;
    unsigned char *sA = smem + kOffA;
    unsigned char *sZ = smem + kOffZ;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
    uint64_t *mma_done = bars;      // [accumulator]: phase n = n-th MMA into it done
    uint64_t *acc_free = bars + 2;  // [accumulator]: the epilogue has read it
    uint64_t *f_full = bars + 4;    // F of the next tile written
    uint64_t *b_full = bars + 5;    // B copied in
    uint64_t *zfull = bars + 6;     // [set][epilogue warp]: logits box loaded
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + kOffScal);
    volatile int *s_abort = reinterpret_cast<volatile int *>(smem + kOffScal + 4);
    int *s_last = reinterpret_cast<int *>(smem + kOffScal + 8);
    double *s_part = reinterpret_cast<double *>(smem + kOffPart);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int layer = blockIdx.y;
    const int64_t T = a.T;
    const int ntiles_layer = (int)((T + kTileM - 1) / kTileM);
    const int tb = blockIdx.x * a.tiles_per_cta;
    const int te = min(ntiles_layer, tb + a.tiles_per_cta);
    const int nt = te > tb ? te - tb : 0;

    pdl_trigger();  // the next kernel may be scheduled (it waits for this one to finish)
    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&mma_done[i], 1);
            mbar_init(&acc_free[i], kEpiWarps / 2);
        }
        mbar_init(f_full, kFWarps);
        mbar_init(b_full, 1);
        for (int i = 0; i < kZBoxes; ++i) mbar_init(&zfull[i], 1);
        *s_abort = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // epilogue warps: group g = tiles of parity g (accumulator g, box set g);
    // within it quadrant q (tokens 32q ..) and chunk pair p (experts 64p ..)
    const bool epi = warp >= kEpiWarp0;
    const int ew = epi ? warp - kEpiWarp0 : 0;
    const int group = ew >> 3, quad = warp & 3, pair = (ew >> 2) & 1;
    auto box_id = [&](int cc) { return group * kEpiWarps + (2 * pair + cc) * 4 + quad; };
    auto issue_z = [&](int m) {  // tile tb + m (parity = group) into this warp's two boxes
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
            uint64_t *bar = &zfull[box_id(cc)];
            mbar_arrive_expect_tx(bar, kBoxBytes);
            tma_load_3d(sZ + (size_t)box_id(cc) * kBoxBytes, &zmap, 32 * (2 * pair + cc),
                        (tb + m) * kTileM + 32 * quad, layer, bar);
        }
    };
    // The logits are an input of the whole path: each group's first tile is
    // requested before waiting for the previous kernels.
    int z_issued = 0;  // tiles of this group requested (lane 0)
    if (epi && lane == 0) {
        prefetch_tensormap(&zmap);
        prefetch_tensormap(&dzmap);
        if (group < nt) {
            issue_z(group);
            z_issued = 1;
        }
    }

    pdl_wait();  // the image of D', D and the selected experts come from the previous kernels
    if (a.img_ok && __ldg(a.img_ok + layer) == 0) {
        // this problem's matrix does not fit the image (the ALU kernel that
        // follows takes it): wait for the logits requested above, release
        // TMEM and leave
        if (epi && lane == 0 && z_issued) {
            mbar_wait(&zfull[box_id(0)], 0u, a.status);
            mbar_wait(&zfull[box_id(1)], 0u, a.status);
        }
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (warp == 0) tmem_dealloc(tmem, kTmemCols);
        return;
    }

    float tok_sum = 0.0f;  // sum of A_t over this thread's tokens (at most a few tiles)
    if (warp == 0) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            // kind::f16: fp32 accumulate, fp16 A and B, both K-major, N = 256, M = 128
            const uint32_t idesc =
                (1u << 4) | ((uint32_t)(2 * kE / 8) << 17) | ((uint32_t)(kTileM / 16) << 24);
            const uint32_t sA_u32 = smem_u32(sA), sB_u32 = smem_u32(sB);
            mbar_arrive_expect_tx(b_full, kBImageBytes);
            const unsigned char *img = a.bimg + (size_t)layer * kBImageBytes;
#pragma unroll
            for (int q = 0; q < 4; ++q)
                bulk_load(sB + q * (kBImageBytes / 4), img + q * (kBImageBytes / 4), kBImageBytes / 4,
                          b_full);
            const bool have_b = mbar_wait(b_full, 0u, a.status);
            if (!have_b) *s_abort = 1;
            int issued = 0;
            for (int m = 0; m < nt && have_b; ++m) {
                const int buf = m & 1;
                bool ok = mbar_wait(f_full, (uint32_t)m & 1u, a.status);
                if (ok && m >= 2)
                    ok = mbar_wait(&acc_free[buf], (uint32_t)((m >> 1) - 1) & 1u, a.status);
                if (!ok) *s_abort = 1;
                if (*s_abort) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * 2 * kE);
#pragma unroll
                for (int kk = 0; kk < kE / 16; ++kk) {
                    const uint32_t koff = (uint32_t)((kk & 3) * 32);
                    const uint64_t adesc = umma_desc_sw128(sA_u32 + (kk >> 2) * kAtomA + koff);
                    const uint64_t bdesc = umma_desc_sw128(sB_u32 + (kk >> 2) * kAtomB + koff);
                    umma_f16(d_tmem, adesc, bdesc, idesc, kk > 0 ? 1u : 0u);
                }
                umma_commit(&mma_done[buf]);
                issued = m + 1;
            }
            // the tensor cores must be done with TMEM before it is released
            if (issued > 0)
                mbar_wait(&mma_done[(issued - 1) & 1], (uint32_t)((issued - 1) >> 1) & 1u, a.status);
            if (!have_b) mbar_wait(b_full, 0u, a.status);  // no copy may outlive the CTA
        }
        __syncwarp();
    } else if (warp < kEpiWarp0) {
        // ------------------------------------------------------------ F builders
        const int ft = threadIdx.x - kFWarp0 * 32;
        constexpr int kRows = (kTileM + kFThreads - 1) / kFThreads;
        uint32_t sel[kRows][2];
        auto load_rows = [&](int m) {
#pragma unroll
            for (int i = 0; i < kRows; ++i) {
                const int r = ft + i * kFThreads;
                const int64_t t = (int64_t)(tb + m) * kTileM + r;
                sel[i][0] = sel[i][1] = 0u;
                if (r < kTileM && t < T) load_sel<K>(a.idx + ((int64_t)layer * T + t) * K, sel[i]);
            }
        };
        if (nt > 0) load_rows(0);
        // the counts accumulator of the signatures kernel is read (by the
        // reduction): clear it for the next call
        if (a.n_zero && blockIdx.x == 0)
            for (int i = ft; i < kE; i += kFThreads) a.n_zero[(int64_t)layer * kE + i] = 0;
        const __half one = __float2half(1.0f);
        for (int m = 0; m < nt; ++m) {
            // F(m - 1) has been read by its MMA
            bool ok = true;
            if (m >= 1)
                ok = mbar_wait(&mma_done[(m - 1) & 1], (uint32_t)((m - 1) >> 1) & 1u, a.status);
            if (!ok) *s_abort = 1;
            if (*s_abort) break;
#pragma unroll
            for (int i = 0; i < kRows; ++i) {
                const int r = ft + i * kFThreads;
                if (r >= kTileM) break;
#pragma unroll
                for (int at = 0; at < 2; ++at)
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        *reinterpret_cast<uint4 *>(sA + at * kAtomA + r * 128 + ((q ^ (r & 7)) << 4)) =
                            make_uint4(0, 0, 0, 0);
                const int64_t t = (int64_t)(tb + m) * kTileM + r;
                if (t < T) {
#pragma unroll
                    for (int q = 0; q < K; ++q) {
                        const int j = (sel[i][q / 4] >> (8 * (q % 4))) & 0xff;
                        *reinterpret_cast<__half *>(sA + sw128_k16_offset(r, j, kTileM)) = one;
                    }
                }
            }
            if (m + 1 < nt) load_rows(m + 1);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(f_full);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int row = 32 * quad + lane;
        const uint32_t tl0 = tmem + ((uint32_t)(32 * quad) << 16) + (uint32_t)(group * 2 * kE) +
                             (uint32_t)(64 * pair);
        int z_done = 0;  // tiles of this group waited for (lane 0)
        for (int m = group; m < nt; m += 2) {
            const uint32_t ph = (uint32_t)(m >> 1) & 1u;
            bool ok = mbar_wait(&mma_done[group], ph, a.status);
            if (ok) ok = mbar_wait(&zfull[box_id(0)], ph, a.status) && mbar_wait(&zfull[box_id(1)], ph, a.status);
            if (ok) z_done = (m >> 1) + 1;
            if (!ok) *s_abort = 1;
            ok = __all_sync(kFull, ok && !*s_abort);
            tc_fence_after();
            float S = 0.f, SV = 0.f;
            const int64_t tok = (int64_t)(tb + m) * kTileM + row;
            const int64_t rg_off = ((int64_t)layer * T + tok) * K;
            // the routing inputs of this token are brought into L2 now and
            // loaded after pass 1 (registers are full during it)
            if constexpr (kRG) {
                if (ok && tok < T) {
                    asm volatile("prefetch.global.L2 [%0];" ::"l"(a.rg_ids + rg_off));
                    asm volatile("prefetch.global.L2 [%0];" ::"l"(a.rg_g + rg_off));
                }
            }
            if (ok) {
                // pass 1: s, S, SV; s (1 - s) and V back into the accumulator
#pragma unroll 1
                for (int cc = 0; cc < 2; ++cc) {
                    const unsigned char *zrow = sZ + (size_t)box_id(cc) * kBoxBytes + lane * 128;
                    const uint32_t tl = tl0 + 32 * cc;
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        uint32_t hi[8], lo[8];
                        tmem_ld8(tl + 8 * h, hi);
                        tmem_ld8(tl + kE + 8 * h, lo);
                        float z[8];
#pragma unroll
                        for (int q = 0; q < 2; ++q) {
                            const float4 v = *reinterpret_cast<const float4 *>(
                                zrow + (((2 * h + q) ^ (lane & 7)) << 4));
                            z[4 * q] = v.x;
                            z[4 * q + 1] = v.y;
                            z[4 * q + 2] = v.z;
                            z[4 * q + 3] = v.w;
                        }
                        tmem_wait_ld();
                        // s = 1 / (1 + 2^(-z log2 e)), four at a time with one
                        // reciprocal: with y_q = 1 + 2^(-z_q log2 e) and
                        // r = 1 / (y0 y1 y2 y3), 1 / y0 = r y1 (y2 y3) and so
                        // on (the exponent is capped at 30 so the product
                        // stays finite: s >= 2^-30 below z = -20.8, an
                        // absolute error under 1e-9).  The Jacobian entry
                        // s (1 - s) is s - s^2 in one FMA (its absolute error
                        // is an ulp of s, far below the gradient's tolerance
                        // relative to its largest entry).
#pragma unroll
                        for (int g4 = 0; g4 < 2; ++g4) {
                            float y[4];
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                y[q] = 1.0f + ex2_approx(fminf(z[4 * g4 + q] * -kLog2e, 30.0f));
                            const float p01 = y[0] * y[1], p23 = y[2] * y[3];
                            const float r = rcp_approx(p01 * p23);
                            const float r01 = r * p23, r23 = r * p01;
                            const float sq4[4] = {r01 * y[1], r01 * y[0], r23 * y[3], r23 * y[2]};
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const int e = 4 * g4 + q;
                                const float V = fmaf(__uint_as_float(hi[e]), 2048.0f, __uint_as_float(lo[e]));
                                const float s = sq4[q];
                                S += s;
                                SV = fmaf(s, V, SV);
                                hi[e] = __float_as_uint(fmaf(-s, s, s));
                                lo[e] = __float_as_uint(V);
                            }
                        }
                        tmem_st8(tl + 8 * h, hi);
                        tmem_st8(tl + kE + 8 * h, lo);
                    }
                }
                tmem_wait_st();
            }
            // Routing gradient, part 1: over the chosen experts in this warp's
            // 64 columns, read while their logits are still in the boxes (the
            // exchange below overwrites two 16-byte chunks of a row), the sums
            // of their sigmoids and of g times them.  (Unshifted: this kernel
            // already needs sum_i s_i > 0, i.e. the largest logit above about
            // -87, and the chosen experts hold the largest logits.)
            float zq[K];
            float rsr = 0.0f, rsg = 0.0f;
            bool bad_id = false;
            int rid[K];
            float rgv[K];
            if constexpr (kRG) {
                if (ok && tok < T) {
                    load_route_row<K>(a.rg_ids + rg_off, a.rg_g + rg_off, rid, rgv);
                } else {
#pragma unroll
                    for (int q = 0; q < K; ++q) { rid[q] = -1; rgv[q] = 0.0f; }
                }
#pragma unroll
                for (int q = 0; q < K; ++q) {
                    const int e = rid[q];
                    if (tok < T && (unsigned)e >= (unsigned)kE) bad_id = true;
                    const bool mine = (unsigned)e < (unsigned)kE && (e >> 6) == pair;
                    zq[q] = mine ? *reinterpret_cast<const float *>(
                                       sZ + (size_t)(group * kEpiWarps + (e >> 5) * 4 + quad) * kBoxBytes +
                                       lane * 128 + ((((e & 31) >> 2) ^ (lane & 7)) << 4) + 4 * (e & 3))
                                 : -INFINITY;
                    if (mine) {
                        float sq, omq;
                        sigmoid_pair(zq[q], sq, omq);
                        rsr += sq;
                        rsg = fmaf(rgv[q], sq, rsg);
                    }
                }
            }
            // exchange with the other chunk pair of the quadrant through the
            // first 16 bytes of this row of the pair's first box (and the next
            // 16 for the routing gradient)
            unsigned char *myrow = sZ + (size_t)box_id(0) * kBoxBytes + lane * 128;
            float *slot = reinterpret_cast<float *>(myrow + ((lane & 7) << 4));
            slot[0] = S;
            slot[1] = SV;
            slot[2] = ok ? 1.0f : 0.0f;
            if constexpr (kRG) {
                slot[3] = rsr;
                float *slot2 = reinterpret_cast<float *>(myrow + (((lane & 7) ^ 1) << 4));
                slot2[0] = rsg;
            }
            named_sync(1 + 4 * group + quad, 64);
            float St = 0.f, SVt = 0.f;
            bool all_ok = true;
            float psr[2], psg[2];
#pragma unroll
            for (int pp = 0; pp < 2; ++pp) {
                const unsigned char *orow =
                    sZ + (size_t)(group * kEpiWarps + (2 * pp) * 4 + quad) * kBoxBytes + lane * 128;
                const float *o = reinterpret_cast<const float *>(orow + ((lane & 7) << 4));
                St += o[0];
                SVt += o[1];
                all_ok = all_ok && o[2] != 0.0f;
                if constexpr (kRG) {
                    const float *o2 = reinterpret_cast<const float *>(orow + (((lane & 7) ^ 1) << 4));
                    psr[pp] = o[3];
                    psg[pp] = o2[0];
                }
            }
            all_ok = __all_sync(kFull, all_ok);
            if (!all_ok) break;  // the same decision in both warps of the quadrant
            // Routing gradient, part 2: the two halves' sums added in pair
            // order (the same numbers in both warps), then this warp's chosen
            // entries: dz = w (1 - s) (g - dot), w = s / sum of the chosen s.
            float rd[K];
            uint32_t epk[(K + 3) / 4];
            if constexpr (kRG) {
                const float inv = 1.0f / (psr[0] + psr[1]);
                const float dot = (psg[0] + psg[1]) * inv;
#pragma unroll
                for (int q = 0; q < K; ++q) {
                    const bool mine = zq[q] > -INFINITY;
                    float sq = 0.0f, omq = 0.0f;
                    if (mine) sigmoid_pair(zq[q], sq, omq);
                    rd[q] = sq * inv * (rgv[q] - dot) * omq;
                    // this warp's chosen columns, one byte each (0xff: not this warp's)
                    const uint32_t byte = mine ? (uint32_t)rid[q] : 0xffu;
                    if (q % 4 == 0) epk[q / 4] = byte;
                    else epk[q / 4] |= byte << (8 * (q % 4));
                }
                if (bad_id) atomicOr(a.status, kDevBadId);
            }
            named_sync(1 + 4 * group + quad, 64);
            const float cs = a.coef / St;
            const float csA = cs * (SVt / St);
            if (pair == 0 && (int64_t)(tb + m) * kTileM + row < T) tok_sum -= SVt / St;
            // pass 2: dz into the boxes, in place
#pragma unroll 1
            for (int cc = 0; cc < 2; ++cc) {
                unsigned char *zrow = sZ + (size_t)box_id(cc) * kBoxBytes + lane * 128;
                const uint32_t tl = tl0 + 32 * cc;
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    uint32_t jac[8], vv[8];
                    tmem_ld8(tl + 8 * h, jac);
                    tmem_ld8(tl + kE + 8 * h, vv);
                    tmem_wait_ld();
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        float4 o;
                        o.x = __uint_as_float(jac[4 * q]) * fmaf(-cs, __uint_as_float(vv[4 * q]), csA);
                        o.y = __uint_as_float(jac[4 * q + 1]) * fmaf(-cs, __uint_as_float(vv[4 * q + 1]), csA);
                        o.z = __uint_as_float(jac[4 * q + 2]) * fmaf(-cs, __uint_as_float(vv[4 * q + 2]), csA);
                        o.w = __uint_as_float(jac[4 * q + 3]) * fmaf(-cs, __uint_as_float(vv[4 * q + 3]), csA);
                        *reinterpret_cast<float4 *>(zrow + (((2 * h + q) ^ (lane & 7)) << 4)) = o;
                    }
                }
            }
            if constexpr (kRG) {
                // the routing gradient added to this warp's chosen entries
#pragma unroll
                for (int q = 0; q < K; ++q) {
                    const int e = (int)((epk[q / 4] >> (8 * (q % 4))) & 0xffu);
                    if (e == 0xff) continue;
                    float *dst = reinterpret_cast<float *>(
                        sZ + (size_t)box_id((e >> 5) & 1) * kBoxBytes + lane * 128 +
                        ((((e & 31) >> 2) ^ (lane & 7)) << 4) + 4 * (e & 3));
                    *dst += rd[q];
                }
            }
            // the accumulator may take the MMA of tile m + 2
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_free[group]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
#pragma unroll
                for (int cc = 0; cc < 2; ++cc)
                    tma_store_3d(&dzmap, sZ + (size_t)box_id(cc) * kBoxBytes, 32 * (2 * pair + cc),
                                 (tb + m) * kTileM + 32 * quad, layer);
                bulk_commit_group();
                // the boxes take this group's next tile once the stores have read them
                if (m + 2 < nt) {
                    bulk_wait_read<0>();
                    issue_z(m + 2);
                    ++z_issued;
                }
            }
            __syncwarp();
        }
        if (lane == 0) {
            bulk_wait_all<0>();  // dz stores complete
            // loads requested but not consumed (only after a failed wait)
            for (int j = z_done; j < z_issued; ++j) {
                mbar_wait(&zfull[box_id(0)], (uint32_t)j & 1u, a.status);
                mbar_wait(&zfull[box_id(1)], (uint32_t)j & 1u, a.status);
            }
        }
        __syncwarp();
    }

    // TMEM released once every role is done with it
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, kTmemCols);

    // CTA partial in a fixed order: a shuffle tree per warp, then over the
    // warp sums (fp32: at most a few hundred tokens per CTA, pairwise; the
    // CTA partials are added in fp64)
    float tok = tok_sum;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) tok += __shfl_xor_sync(kFull, tok, off);
    float *s_partf = reinterpret_cast<float *>(s_part);
    if (lane == 0) s_partf[warp] = tok;
    __syncthreads();
    if (warp == 0) {
        float vf = lane < kWarps ? s_partf[lane] : 0.0f;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) vf += __shfl_xor_sync(kFull, vf, off);
        const double v = (double)vf;
        if (lane == 0) {
            a.partials[(int64_t)layer * gridDim.x + blockIdx.x] = v;
            // release: the partial is visible to the CTA that sees the last count
            *s_last = (atom_add_acq_rel(&a.done[layer], 1) == (int)gridDim.x - 1);
        }
    }
    __syncthreads();
    if (!*s_last) return;
    __threadfence();
    if (warp == 0) {
        const double sum = warp_sum_fixed(a.partials + (int64_t)layer * gridDim.x, gridDim.x);
        if (lane == 0) {
            a.loss[layer] = (float)(sum * a.scale);
            a.done[layer] = 0;
            if (a.status_out) atomicOr(a.status_out, *reinterpret_cast<volatile int *>(a.status));
        }
    }
}

int sms_now() {
    int dev = 0, n = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n;
}

template <int K, bool kRG>
cudaError_t run_mma(const CUtensorMap &zmap, const CUtensorMap &dzmap, const MmaArgs &args, int gx,
                    int L, cudaStream_t s) {
    cudaError_t e = ensure_smem_limit<loss_mma_kernel<K, kRG>>(kSmemMma);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)gx, (unsigned)L);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemMma;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, loss_mma_kernel<K, kRG>, zmap, dzmap, args);
}

}  // namespace

bool loss_mma_supported(const Problem &p, int gate, const float *logits, const int *D,
                        const float *dlogits, bool image_checked) {
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    auto al = [](const void *q) { return reinterpret_cast<uintptr_t>(q) % 16 == 0; };
    // R_i <= (E - 1) T must stay below 2^23 for the two-piece split of D'
    // (unless the image kernel checks the split of a given matrix)
    const bool t_ok = image_checked || (int64_t)(kE - 1) * p.T < (int64_t)(1 << 23);
    return p.E == kE && gate == 0 && k_ok && dlogits != nullptr && t_ok && al(logits) &&
           al(dlogits) && al(D);
}

int loss_mma_ctas_per_problem(const Problem &p) {
    const int tiles = (int)((p.T + kTileM - 1) / kTileM);
    int gx = sms_now() / p.L;
    if (gx < 1) gx = 1;
    if (gx > tiles) gx = tiles;
    const int per = (tiles + gx - 1) / gx;
    return (tiles + per - 1) / per;
}

cudaError_t launch_loss_mma(const float *logits, const uint8_t *idx, const unsigned char *bimg, int *n_zero, const Problem &p, float d_scale,
                            float grad_scale, float *loss, float *dlogits,
                            double *partials, int *done, int *status, int *status_out,
                            cudaStream_t s, const int *rg_ids, const float *rg_g,
                            const int *img_ok) {
    if (!bimg) return cudaErrorInvalidValue;
    CUtensorMap zmap, dzmap;
    if (!encode_tensor_map_3d_f32(&zmap, logits, (uint64_t)p.L, (uint64_t)p.T, (uint64_t)kE, 32) ||
        !encode_tensor_map_3d_f32(&dzmap, dlogits, (uint64_t)p.L, (uint64_t)p.T, (uint64_t)kE, 32))
        return cudaErrorInvalidValue;
    const int tiles = (int)((p.T + kTileM - 1) / kTileM);
    const int gx = loss_mma_ctas_per_problem(p);
    const double norm = 1.0 / ((double)p.T * (double)p.T * (double)p.k);
    MmaArgs args;
    args.logits = logits;
    args.idx = idx;
    args.bimg = bimg;
    args.n_zero = n_zero;
    args.T = p.T;
    args.tiles_per_cta = (tiles + gx - 1) / gx;
    args.coef = (float)((double)grad_scale * (double)d_scale * norm);
    args.scale = (double)d_scale * norm;
    args.partials = partials;
    args.done = done;
    args.loss = loss;
    args.status = status;
    args.status_out = status_out;
    args.rg_ids = rg_ids;
    args.rg_g = rg_g;
    args.img_ok = img_ok;
    if (rg_ids && rg_g) {
        switch (p.k) {
            case 1: return run_mma<1, true>(zmap, dzmap, args, gx, p.L, s);
            case 2: return run_mma<2, true>(zmap, dzmap, args, gx, p.L, s);
            case 4: return run_mma<4, true>(zmap, dzmap, args, gx, p.L, s);
            default: return run_mma<8, true>(zmap, dzmap, args, gx, p.L, s);
        }
    }
    switch (p.k) {
        case 1: return run_mma<1, false>(zmap, dzmap, args, gx, p.L, s);
        case 2: return run_mma<2, false>(zmap, dzmap, args, gx, p.L, s);
        case 4: return run_mma<4, false>(zmap, dzmap, args, gx, p.L, s);
        default: return run_mma<8, false>(zmap, dzmap, args, gx, p.L, s);
    }
}

}  // namespace dol
