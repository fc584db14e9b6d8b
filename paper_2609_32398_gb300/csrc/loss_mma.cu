// Step 3 on the tensor cores (E = 128, sigmoid-norm gate, k in {1, 2, 4, 8}):
// the surrogate DO-loss and its gradient (Sec. 3.1.3, Eq. do_loss).
//
// With F_t the one-hot rows of the selected experts, G = F D is the k-row
// gather G_ti = sum_{j in S_t} D_ji, and
//   w_ti = f_ti R_i - G_ti,   A_t = (sum_{j in S_t} s_j R_j - sum_i s_i G_ti) / S,
//   dz_ti = c/S s_i (1 - s_i) (w_ti - A_t)
//         = -c/S jac_i (G_ti + A_t)  +  [i in S_t] c/S jac_i R_i,
// with s = sigmoid(z), S = sum_i s_i, jac = s (1 - s), c = grad_scale d_scale/(m^2 k).
// G is computed exactly on the tensor cores: F is 0/1 in fp16 and D (zero
// diagonal, 0 <= D <= 2^22) is split into two fp16 pieces D = 2048 hi + lo,
// both exact (< 2048), with fp32 accumulation of at most k terms each.
//
// A persistent CTA owns a run of 128-token tiles of one problem.  Per tile:
//   1. the four epilogue warps write F (128 x 128 fp16, K-major, 128-byte
//      swizzle) from the selected-expert bytes;
//   2. one thread issues 8 tcgen05.mma (M=128, N=256: hi | lo, K=16 each) into
//      one of two TMEM accumulators, and commits to an mbarrier;
//   3. meanwhile the epilogue of the previous tile runs: thread = token =
//      TMEM lane.  Pass 1 streams the logits in 32 x 32 TMA boxes, forms s, S,
//      sum s G and writes jac and G back into the accumulator columns; pass 2
//      reads them again, writes dz into a swizzled staging box (plus the
//      [i in S_t] term for the k selected experts) and stores it with TMA.
// Tensor maps are 3-D [L][T][E], so boxes past the end of a problem are
// zero-filled on load and dropped on store.
#include <cuda_fp16.h>

#include <climits>

#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kE = 128;
constexpr int kTileM = 128;
constexpr int kEpiWarps = 8;                     // two per TMEM lane quadrant
constexpr int kCtrlWarp = kEpiWarps;
constexpr int kMmaThreads = (kEpiWarps + 1) * 32;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kBoxBytes = 32 * 128;              // 32 rows x 32 fp32
constexpr int kAtomA = kTileM * 128;             // one 64-column K atom of A
constexpr int kAtomB = 2 * kE * 128;             // one 64-column K atom of B (256 rows)
constexpr int kBytesA = 2 * kAtomA;              // 32 KB
constexpr int kBytesB = 2 * kAtomB;              // 64 KB
constexpr int kOffB = 0;
constexpr int kOffA = kOffB + kBytesB;           // one A buffer
constexpr int kOffZ = kOffA + kBytesA;           // [chunk 4][quadrant 4] logits boxes
constexpr int kOffO = kOffZ + 16 * kBoxBytes;    // [warp] dlogits staging box
constexpr int kOffBar = kOffO + kEpiWarps * kBoxBytes;  // mma_done, zfull[16]
constexpr int kOffScal = kOffBar + 8 * (1 + 16);        // tmem base, abort, last
constexpr int kOffR = kOffScal + 16;                    // R_i [E] (64-bit)
constexpr int kOffX = kOffR + 8 * kE;                   // exchange [half 2][token 128][3] fp32
constexpr int kOffPart = kOffX + 2 * kTileM * 3 * 4;    // [kMmaThreads] fp64
constexpr int kSmemMma = kOffPart + 8 * kMmaThreads + 1024;  // + alignment slack
constexpr uint32_t kTmemCols = 512;              // two 256-column accumulators
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float sig_fast(float z) {
    float e, r;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(z * -kLog2e));
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(1.0f + e));
    return r;
}

// Byte offset of element (row, k) of a K-major 128-byte-swizzled fp16 operand
// with `rows` rows: K atoms of 64 columns, 128-byte rows, 16-byte chunks
// XOR-ed with (row mod 8).
__device__ __forceinline__ uint32_t sw128_fp16_offset(int row, int k, int rows) {
    const int atom = k >> 6, kc = k & 63;
    return (uint32_t)(atom * rows * 128 + row * 128 + ((((kc >> 3) ^ (row & 7))) << 4) + (kc & 7) * 2);
}

struct MmaArgs {
    const float *logits;
    const uint8_t *idx;
    const int *D;
    const int *counts;  // may be null: R then comes from the rows of D
    int *n_zero;        // may be null
    int64_t T;
    int tiles_per_cta;
    float coef;
    double scale;
    double *partials;
    int *done;
    float *loss;
    long long *origin_do;
    int *status;
};

template <int K>
__global__ void __launch_bounds__(kMmaThreads, 1)
loss_mma_kernel(const __grid_constant__ CUtensorMap zmap, const __grid_constant__ CUtensorMap dzmap,
                const MmaArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    unsigned char *sB = smem + kOffB;
    unsigned char *sA = smem + kOffA;
    unsigned char *sZ = smem + kOffZ;
    unsigned char *sO = smem + kOffO;
    uint64_t *mma_done = reinterpret_cast<uint64_t *>(smem + kOffBar);      // one phase per tile
    uint64_t *zfull = mma_done + 1;                                          // [chunk][quadrant]
    float *s_x = reinterpret_cast<float *>(smem + kOffX);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + kOffScal);
    volatile int *s_abort = reinterpret_cast<volatile int *>(smem + kOffScal + 4);
    int *s_last = reinterpret_cast<int *>(smem + kOffScal + 8);
    unsigned long long *s_R = reinterpret_cast<unsigned long long *>(smem + kOffR);
    double *s_part = reinterpret_cast<double *>(smem + kOffPart);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int layer = blockIdx.y;
    const int64_t T = a.T;
    const int ntiles_layer = (int)((T + kTileM - 1) / kTileM);
    const int tb = blockIdx.x * a.tiles_per_cta;
    const int te = min(ntiles_layer, tb + a.tiles_per_cta);
    const int nt = te > tb ? te - tb : 0;

    if (threadIdx.x == 0) {
        mbar_init(&mma_done[0], 1);
        for (int i = 0; i < 16; ++i) mbar_init(&zfull[i], 1);
        *s_abort = 0;
        fence_barrier_init();
    }
    if (threadIdx.x < kE) s_R[threadIdx.x] = 0ull;
    if (warp == kCtrlWarp) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // The logits are an input of the whole path: start the first tile's boxes
    // before waiting for the previous kernels.
    // epilogue warp w: TMEM lane quadrant q = w % 4 (tokens 32q..), half h = w / 4
    // (experts 64h .. 64h+63, chunks 2h and 2h+1); it loads and consumes the
    // logits boxes (chunk, q) of its chunks.
    const int quad = warp & 3, half = warp >> 2;
    auto issue_z = [&](int tile, int chunk) {
        uint64_t *bar = &zfull[chunk * 4 + quad];
        mbar_arrive_expect_tx(bar, kBoxBytes);
        tma_load_3d(sZ + (chunk * 4 + quad) * kBoxBytes, &zmap, 32 * chunk,
                    tile * kTileM + 32 * quad, layer, bar);
    };
    if (warp < kEpiWarps && lane == 0 && nt > 0) {
        prefetch_tensormap(&zmap);
        prefetch_tensormap(&dzmap);
        issue_z(tb, 2 * half);
        issue_z(tb, 2 * half + 1);
    }

    pdl_wait();  // D, the counts and the selected experts come from the previous kernels

    // B = [hi rows 0..127 | lo rows 128..255] x K 128, from the rows of D
    // (D symmetric: row n of D is column n); R_i = sum_j D_ij alongside.
    const int *Dl = a.D + (int64_t)layer * kE * kE;
    constexpr int kItems = kE * (kE / 8);  // 16-byte fp16 chunks of one B half
    constexpr int kPer = (kItems + kMmaThreads - 1) / kMmaThreads;
    int4 dv[kPer][2];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {  // all loads first: one round trip
        const int item = threadIdx.x + u * kMmaThreads;
        if (item < kItems) {
            const int n = item >> 4, k0 = (item & 15) * 8;
            dv[u][0] = __ldg(reinterpret_cast<const int4 *>(Dl + n * kE + k0));
            dv[u][1] = __ldg(reinterpret_cast<const int4 *>(Dl + n * kE + k0 + 4));
        }
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
        const int item = threadIdx.x + u * kMmaThreads;
        if (item >= kItems) break;
        const int n = item >> 4, k0 = (item & 15) * 8;
        const int4 v0 = dv[u][0], v1 = dv[u][1];
        const int d[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        __align__(16) __half hi[8], lo[8];
        long long rs = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            hi[q] = __int2half_rn(d[q] >> 11);
            lo[q] = __int2half_rn(d[q] & 2047);
            rs += d[q];
        }
        *reinterpret_cast<uint4 *>(sB + sw128_fp16_offset(n, k0, 2 * kE)) =
            *reinterpret_cast<const uint4 *>(hi);
        *reinterpret_cast<uint4 *>(sB + sw128_fp16_offset(kE + n, k0, 2 * kE)) =
            *reinterpret_cast<const uint4 *>(lo);
        if (!a.counts) atomicAdd(&s_R[n], (unsigned long long)rs);
    }
    if (a.counts && threadIdx.x < kE) {
        const long long nn = a.counts[(int64_t)layer * kE + threadIdx.x];
        s_R[threadIdx.x] = (unsigned long long)((long long)(kE - 2 * K) * nn + T * (long long)K);
        if (a.n_zero && blockIdx.x == 0) a.n_zero[(int64_t)layer * kE + threadIdx.x] = 0;
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (threadIdx.x < kE) {
        const long long r = (long long)s_R[threadIdx.x];
        if (r > INT_MAX || r < 0) atomicOr(a.status, kDevOverflow);
    }

    // kind::f16 instruction descriptor: fp32 accumulate, fp16 A and B, both
    // K-major, N = 256, M = 128.
    const uint32_t idesc = (1u << 4) | ((uint32_t)(2 * kE / 8) << 17) | ((uint32_t)(kTileM / 16) << 24);
    const uint32_t sA_u32 = smem_u32(sA), sB_u32 = smem_u32(sB);

    double tok_sum = 0.0;
    // selected experts of this thread's token (row 32 quad + lane) in the
    // current and the previous tile, and the raw bytes of the next tile
    int js[K], js_prev[K];
    uint32_t jn[2] = {0u, 0u};
    bool valid_prev = false;
    const int row = 32 * quad + lane;
#pragma unroll
    for (int q = 0; q < K; ++q) js[q] = js_prev[q] = 0;
    auto load_idx_raw = [&](int tile, uint32_t (&r)[2]) {
        const int64_t tt = (int64_t)tile * kTileM + row;
        r[0] = r[1] = 0u;
        if (tt < T) {
            const uint8_t *ip = a.idx + ((int64_t)layer * T + tt) * K;
            if (K == 8) {
                const uint2 v = __ldg(reinterpret_cast<const uint2 *>(ip));
                r[0] = v.x;
                r[1] = v.y;
            } else if (K == 4) {
                r[0] = __ldg(reinterpret_cast<const uint32_t *>(ip));
            } else if (K == 2) {
                r[0] = __ldg(reinterpret_cast<const uint16_t *>(ip));
            } else {
                r[0] = __ldg(ip);
            }
        }
    };
    if (warp < kEpiWarps && nt > 0) load_idx_raw(tb, jn);

    for (int it = 0; it <= nt; ++it) {
        bool valid = false;
        if (warp < kEpiWarps) {
            // the MMA of the previous tile is done: A is free, its accumulator full
            if (it >= 1 && !mbar_wait(&mma_done[0], (uint32_t)((it - 1) & 1), a.status)) *s_abort = 1;
            tc_fence_after();
            if (it < nt) {
                valid = (int64_t)(tb + it) * kTileM + row < T;
#pragma unroll
                for (int q = 0; q < K; ++q) js[q] = (jn[q / 4] >> (8 * (q % 4))) & 0xff;
                if (it + 1 < nt) load_idx_raw(tb + it + 1, jn);
                // 1. F of tile it: half h writes K atom h of the token's row
                unsigned char *arow = sA + half * kAtomA + row * 128;
#pragma unroll
                for (int q = 0; q < 8; ++q)  // chunk order rotated by row: conflict-free
                    *reinterpret_cast<uint4 *>(arow + ((q ^ (row & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                if (valid) {
                    const __half one = __float2half(1.0f);
#pragma unroll
                    for (int q = 0; q < K; ++q)
                        if ((js[q] >> 6) == half)
                            *reinterpret_cast<__half *>(sA + sw128_fp16_offset(row, js[q], kTileM)) = one;
                }
                fence_proxy_async_smem();
            }
        }
        tc_fence_before();
        asm volatile("bar.sync 1, %0;" ::"n"(kMmaThreads) : "memory");
        tc_fence_after();
        if (*s_abort) break;
        // 2. the tensor cores: G(it) = F(it) [D_hi | D_lo] into accumulator it & 1
        if (it < nt && warp == kCtrlWarp && lane == 0) {
            const uint32_t d_tmem = tmem + (uint32_t)((it & 1) * 2 * kE);
#pragma unroll
            for (int kk = 0; kk < kE / 16; ++kk) {
                const uint32_t koff = (uint32_t)((kk & 3) * 32);
                const uint64_t adesc = umma_desc_sw128(sA_u32 + (kk >> 2) * kAtomA + koff);
                const uint64_t bdesc = umma_desc_sw128(sB_u32 + (kk >> 2) * kAtomB + koff);
                umma_f16(d_tmem, adesc, bdesc, idesc, kk > 0 ? 1u : 0u);
            }
            umma_commit(&mma_done[0]);
        }
        // 3. epilogue of tile it - 1 on this warp's half of the experts
        if (it >= 1 && warp < kEpiWarps) {
            const int pt = it - 1, pbuf = pt & 1;
            const int ptile = tb + pt;
            bool ok = true;
            const uint32_t tl = tmem + ((uint32_t)(32 * quad) << 16) + (uint32_t)(pbuf * 2 * kE);
            float S0 = 0.f, S1 = 0.f, G0 = 0.f, G1 = 0.f;
            float zsel[K];
#pragma unroll
            for (int q = 0; q < K; ++q) zsel[q] = 0.0f;
            // pass 1
#pragma unroll 1
            for (int cc = 0; cc < 2; ++cc) {
                const int c = 2 * half + cc;
                ok = mbar_wait(&zfull[c * 4 + quad], (uint32_t)pt & 1u, a.status);
                if (!ok) break;
                uint32_t hi[32], lo[32];
                tmem_ld32(tl + 32 * c, hi);
                tmem_ld32(tl + kE + 32 * c, lo);
                const unsigned char *zrow = sZ + (c * 4 + quad) * kBoxBytes + lane * 128;
                float z[32];
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float4 v =
                        *reinterpret_cast<const float4 *>(zrow + ((q ^ (lane & 7)) << 4));
                    z[4 * q] = v.x;
                    z[4 * q + 1] = v.y;
                    z[4 * q + 2] = v.z;
                    z[4 * q + 3] = v.w;
                }
#pragma unroll
                for (int q = 0; q < K; ++q)
                    if ((js_prev[q] >> 5) == c) {
                        const int e = js_prev[q] & 31;
                        zsel[q] = *reinterpret_cast<const float *>(
                            zrow + ((((e >> 2) ^ (lane & 7))) << 4) + (e & 3) * 4);
                    }
                tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 32; e += 2) {
                    const float Ga = fmaf(__uint_as_float(hi[e]), 2048.0f, __uint_as_float(lo[e]));
                    const float Gb =
                        fmaf(__uint_as_float(hi[e + 1]), 2048.0f, __uint_as_float(lo[e + 1]));
                    const float sa = sig_fast(z[e]), sb = sig_fast(z[e + 1]);
                    S0 += sa;
                    S1 += sb;
                    G0 = fmaf(sa, Ga, G0);
                    G1 = fmaf(sb, Gb, G1);
                    hi[e] = __float_as_uint(fmaf(-sa, sa, sa));
                    hi[e + 1] = __float_as_uint(fmaf(-sb, sb, sb));
                    lo[e] = __float_as_uint(Ga);
                    lo[e + 1] = __float_as_uint(Gb);
                }
                tmem_st32(tl + 32 * c, hi);
                tmem_st32(tl + kE + 32 * c, lo);
                // every lane has consumed its row of the box: load the next tile's box
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0 && pt + 1 < nt) issue_z(ptile + 1, c);
            }
            tmem_wait_st();
            // the selected experts in this half: sum s_j R_j, and jac_j R_j for dz
            float SRv = 0.0f, patch[K];
#pragma unroll
            for (int q = 0; q < K; ++q) {
                const bool mine = (js_prev[q] >> 6) == half;
                const float sj = sig_fast(zsel[q]);
                const float rj = (float)(long long)s_R[js_prev[q]];
                SRv += mine ? sj * rj : 0.0f;
                patch[q] = fmaf(-sj, sj, sj) * rj;
            }
            // exchange the half sums of every token; add them in a fixed order
            float *xr = s_x + (half * kTileM + row) * 3;
            xr[0] = S0 + S1;
            xr[1] = G0 + G1;
            xr[2] = SRv;
            asm volatile("bar.sync 2, %0;" ::"n"(kEpiThreads) : "memory");
            const float *x0 = s_x + row * 3, *x1 = s_x + (kTileM + row) * 3;
            const float S = x0[0] + x1[0];
            const float A = ((x0[2] + x1[2]) - (x0[1] + x1[1])) / S;
            const float cs = a.coef / S;
            asm volatile("bar.sync 2, %0;" ::"n"(kEpiThreads) : "memory");
            if (half == 0 && valid_prev && ok) tok_sum += (double)A;
            // pass 2
#pragma unroll 1
            for (int cc = 0; cc < 2 && ok; ++cc) {
                const int c = 2 * half + cc;
                uint32_t jac[32], gg[32];
                tmem_ld32(tl + 32 * c, jac);
                tmem_ld32(tl + kE + 32 * c, gg);
                if (lane == 0) bulk_wait_read<0>();
                __syncwarp();
                tmem_wait_ld();
                unsigned char *orow = sO + warp * kBoxBytes + lane * 128;
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    float4 v;
                    v.x = -cs * __uint_as_float(jac[4 * q]) * (__uint_as_float(gg[4 * q]) + A);
                    v.y = -cs * __uint_as_float(jac[4 * q + 1]) * (__uint_as_float(gg[4 * q + 1]) + A);
                    v.z = -cs * __uint_as_float(jac[4 * q + 2]) * (__uint_as_float(gg[4 * q + 2]) + A);
                    v.w = -cs * __uint_as_float(jac[4 * q + 3]) * (__uint_as_float(gg[4 * q + 3]) + A);
                    *reinterpret_cast<float4 *>(orow + ((q ^ (lane & 7)) << 4)) = v;
                }
#pragma unroll
                for (int q = 0; q < K; ++q) {
                    if (valid_prev && (js_prev[q] >> 5) == c) {
                        const int e = js_prev[q] & 31;
                        float *p = reinterpret_cast<float *>(orow + ((((e >> 2) ^ (lane & 7))) << 4)) + (e & 3);
                        *p += cs * patch[q];
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_3d(&dzmap, sO + warp * kBoxBytes, 32 * c, ptile * kTileM + 32 * quad,
                                 layer);
                    bulk_commit_group();
                }
            }
            if (!ok) *s_abort = 1;
        }
#pragma unroll
        for (int q = 0; q < K; ++q) js_prev[q] = js[q];
        valid_prev = valid;
    }

    // drain: stores complete, TMEM released
    if (warp < kEpiWarps && lane == 0) bulk_wait_all<0>();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == kCtrlWarp) tmem_dealloc(tmem, kTmemCols);

    // CTA partial in a fixed order (fp64 adds are slow on this part: a
    // shuffle tree per warp, then the warp sums), then the last CTA
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) tok_sum += __shfl_xor_sync(kFull, tok_sum, off);
    if (lane == 0) s_part[warp] = tok_sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        double sum = 0.0;
        for (int i = 0; i < kMmaThreads / 32; ++i) sum += s_part[i];
        a.partials[(int64_t)layer * gridDim.x + blockIdx.x] = sum;
        __threadfence();
        *s_last = (atomicAdd(&a.done[layer], 1) == (int)gridDim.x - 1);
    }
    __syncthreads();
    if (!*s_last) return;
    __threadfence();
    {
        const double sum = block_sum_fixed(a.partials + (int64_t)layer * gridDim.x, gridDim.x,
                                           s_part, 256);
        if (threadIdx.x == 0) {
            a.loss[layer] = (float)(sum * a.scale);
            a.done[layer] = 0;
        }
    }
    if (a.origin_do) {
        long long o = 0;
        for (int e = threadIdx.x; e < kE * kE; e += kMmaThreads) {
            if (e / kE != e % kE) {
                const long long d = Dl[e];
                o += d * d;
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) o += __shfl_xor_sync(kFull, o, off);
        __syncthreads();
        long long *s_o = reinterpret_cast<long long *>(s_part);
        if (lane == 0) s_o[warp] = o;
        __syncthreads();
        if (threadIdx.x == 0) {
            long long sum = 0;
            for (int q = 0; q < kMmaThreads / 32; ++q) sum += s_o[q];
            a.origin_do[layer] = sum;
        }
    }
}

int sms_now() {
    int dev = 0, n = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n;
}

template <int K>
cudaError_t run_mma(const CUtensorMap &zmap, const CUtensorMap &dzmap, const MmaArgs &args, int gx,
                    int L, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(loss_mma_kernel<K>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMma);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)gx, (unsigned)L);
    cfg.blockDim = dim3(kMmaThreads);
    cfg.dynamicSmemBytes = kSmemMma;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, loss_mma_kernel<K>, zmap, dzmap, args);
}

}  // namespace

bool loss_mma_supported(const Problem &p, int gate, const float *logits, const int *D,
                        const float *dlogits) {
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    auto al = [](const void *q) { return reinterpret_cast<uintptr_t>(q) % 16 == 0; };
    return p.E == kE && gate == 0 && k_ok && dlogits != nullptr && p.T <= (1 << 22) && al(logits) &&
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

cudaError_t launch_loss_mma(const float *logits, const uint8_t *idx, const int *D, const int *counts,
                            int *n_zero, const Problem &p, float d_scale, float grad_scale,
                            float *loss, long long *origin_do, float *dlogits, double *partials,
                            int *done, int *status, cudaStream_t s) {
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
    args.D = D;
    args.counts = counts;
    args.n_zero = n_zero;
    args.T = p.T;
    args.tiles_per_cta = (tiles + gx - 1) / gx;
    args.coef = (float)((double)grad_scale * (double)d_scale * norm);
    args.scale = (double)d_scale * norm;
    args.partials = partials;
    args.done = done;
    args.loss = loss;
    args.origin_do = origin_do;
    args.status = status;
    switch (p.k) {
        case 1: return run_mma<1>(zmap, dzmap, args, gx, p.L, s);
        case 2: return run_mma<2>(zmap, dzmap, args, gx, p.L, s);
        case 4: return run_mma<4>(zmap, dzmap, args, gx, p.L, s);
        default: return run_mma<8>(zmap, dzmap, args, gx, p.L, s);
    }
}

}  // namespace dol
