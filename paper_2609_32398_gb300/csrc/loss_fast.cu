// Step 3, fast path (E in {32, 64, 128, 256}, k in {1, 2, 4, 8}): the
// surrogate DO-loss and its gradient (Sec. 3.1.3, Eq. do_loss; Eq. global_do
// scaling).
//
// With R_i = sum_j D_ij, put D'_ij = D_ij off the diagonal and D'_ii = -R_i.
// Then for the k experts S_t of token t
//   sum_{j in S_t} D'_ji = sum_{j in S_t} D_ji - f_it R_i = -w_it,
// the integer weight w_it = sum_j D_ij (f_it - f_jt) whose product with
// d_scale/(m^2 k) is dL/dp_it.  One k-row gather of D' per token therefore
// gives every w_it without looking at the signature bits.  D must be
// symmetric (every Hamming matrix and every sum of them is).
//
// R_i is a column sum of D, or -- in the fused path, where D comes from the
// same tokens' co-occurrence counts (D_ij = n_i + n_j - 2 c_ij, App. C.3) --
//   R_i = (E - 2k) n_i + T k      (sum_j c_ij = k n_i, sum_j n_j = T k).
//
// Layout: a CTA stages D' in shared memory, then its warps walk tokens with
// G = E/16 lanes per token; lane g of a token group owns experts
// c*E/4 + 4g .. +3 for c = 0..3, so a group reads 16-byte chunks of the
// logits row and of the D' rows and writes the dlogits row with coalesced
// 16-byte accesses.  The next token group's logits and indices are loaded
// while the current one is computed.  Per token:
//   sigmoid-norm  s = sigmoid(z), A = sum s w / sum s,
//                 dz = c s (1 - s) (w - A) / sum s
//   softmax       e = exp(z - max), A = sum e w / sum e, dz = c e (w - A) / sum e
// with c = grad_scale d_scale / (m^2 k).  A is summed per CTA in fp64 and the
// last CTA of each problem adds the CTA partials in index order.
//
// At E = 256 an int32 D (256 KB) does not fit in shared memory: D is kept
// there as a 16-bit low plane and an 8-bit high plane (192 KB; exact for the
// matrix of the same tokens, whose entries are at most T < 2^24), with zeros
// on the diagonal, and the -R_i of the k chosen experts are added to their
// sums after the gather (R from the counts).  A row chunk of 4 entries is one
// 8-byte and one 4-byte load; the low halves are summed per entry and the
// high bytes in pairs of 16-bit fields, joined after the k rows.  One CTA of
// 512 threads per SM.
#include <climits>

#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kLossFastThreads = 256;
// E = 256: one CTA per SM (the planes of D take 192 KB), with more warps
constexpr int kLossPlaneThreads = 512;
template <int E>
constexpr int loss_fast_threads() { return E == 256 ? kLossPlaneThreads : kLossFastThreads; }
template <int E>
constexpr size_t loss_fast_smem() { return E == 256 ? (size_t)3 * E * E : sizeof(int) * E * E; }

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

// sigmoid(z) = 1 / (1 + 2^(-z log2 e)); for z -> -inf the power is +inf and
// the reciprocal 0, for z -> +inf the power is 0 and the result 1.
__device__ __forceinline__ float sigmoid_fast(float z) {
    return rcp_approx(1.0f + ex2_approx(z * -1.4426950408889634f));
}

template <int K>
__device__ __forceinline__ void load_idx(const uint8_t *p, int (&j)[K]) {
    if (K == 8) {
        const uint2 v = __ldg(reinterpret_cast<const uint2 *>(p));
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            j[q % K] = (v.x >> (8 * q)) & 0xff;
            j[(4 + q) % K] = (v.y >> (8 * q)) & 0xff;
        }
    } else if (K == 4) {
        const uint32_t v = __ldg(reinterpret_cast<const uint32_t *>(p));
#pragma unroll
        for (int q = 0; q < K; ++q) j[q] = (v >> (8 * q)) & 0xff;
    } else if (K == 2) {
        const uint32_t v = __ldg(reinterpret_cast<const uint16_t *>(p));
        j[0] = v & 0xff;
        j[1 % K] = (v >> 8) & 0xff;
    } else {
        j[0] = __ldg(p);
    }
}

struct LossArgs {
    const float *logits;
    const uint8_t *idx;
    const int *D;        // [L][E][E], symmetric
    const int *counts;   // fused path: n_i [L][E] of the same tokens (else null)
    int *n_zero;         // fused path: accumulator [L][E] to clear after use (or null)
    int64_t T;
    int k;
    int tokens_per_cta;
    float coef;
    double scale;
    float *dlogits;
    double *partials;
    int *done;
    float *loss;
    long long *origin_do;
    int *status;
    int *status_out;  // may be null: the last CTA ORs the status word into it
    // layers whose img_ok flag is 1 went to the tensor-core kernel: skipped
    // here (may be null)
    const int *img_ok;
};

template <int E, int K, int kGate, bool kRFromCounts>
__global__ void __launch_bounds__(loss_fast_threads<E>(), E == 256 ? 1 : 3)
loss_fast_kernel(const LossArgs a) {
    constexpr int G = E / 16;    // lanes per token
    constexpr int TPW = 32 / G;  // tokens per warp pass
    constexpr int Q = E / 4;     // expert stride between a lane's chunks
    constexpr bool kPlanes = E == 256;
    constexpr int kWarps = loss_fast_threads<E>() / 32;
    static_assert(!kPlanes || kRFromCounts, "the planes hold the matrix of the same tokens");
    extern __shared__ __align__(128) int sD[];  // [E][E], or the two planes
    uint16_t *sLo = reinterpret_cast<uint16_t *>(sD);             // [E][E] (planes)
    uint8_t *sHi = reinterpret_cast<uint8_t *>(sD) + 2 * E * E;    // [E][E] (planes)
    __shared__ __align__(8) uint64_t bar;
    __shared__ double s_part[kWarps];
    __shared__ long long s_o[kWarps];
    __shared__ long long s_r[E];
    __shared__ int s_last;

    const int layer = blockIdx.y;
    const int P = gridDim.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int grp = lane / G, g = lane % G;
    const int64_t T = a.T;
    const float *zl = a.logits + (int64_t)layer * T * E;
    float *dzl = a.dlogits ? a.dlogits + (int64_t)layer * T * E : nullptr;
    const uint8_t *il = a.idx + (int64_t)layer * T * K;
    const int64_t t_begin = (int64_t)blockIdx.x * a.tokens_per_cta;
    const int64_t t_end = min64(T, t_begin + a.tokens_per_cta);
    const int64_t stride = (int64_t)kWarps * TPW;

    pdl_trigger();  // the next kernel may be scheduled (it waits for this one to finish)
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    // The logits are an input of the whole path, so the first token group's
    // rows can be fetched before the previous kernels have finished.
    int64_t tb = t_begin + (int64_t)warp * TPW;
    float4 zc[4];
    {
        const int64_t t = tb + grp;
        const int64_t tc = (t < t_end) ? t : t_begin;
#pragma unroll
        for (int c = 0; c < 4; ++c)
            zc[c] = __ldg(reinterpret_cast<const float4 *>(zl + tc * E + c * Q + 4 * g));
    }
    __syncthreads();
    pdl_wait();  // D, idx and the cleared counters come from the previous kernels
    if (a.img_ok && __ldg(a.img_ok + layer) != 0) return;
    if (!kPlanes && threadIdx.x == 0) {
        mbar_arrive_expect_tx(&bar, (uint32_t)(sizeof(int) * E * E));
        bulk_load(sD, a.D + (int64_t)layer * E * E, (uint32_t)(sizeof(int) * E * E), &bar);
    }
    if constexpr (kPlanes) {
        // four entries of a row per load: low halves and high bytes, the
        // diagonal zero; an entry outside [0, 2^24) is reported
        const int4 *src = reinterpret_cast<const int4 *>(a.D + (int64_t)layer * E * E);
        int bad = 0;
        for (int q = threadIdx.x; q < E * E / 4; q += blockDim.x) {
            const int4 v = __ldg(src + q);
            const int e0 = 4 * q, i = e0 / E, j0 = e0 % E;
            int x[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                if (j0 + u == i) x[u] = 0;
                bad |= (unsigned)x[u] >= (1u << 24);
            }
            *reinterpret_cast<uint2 *>(sLo + e0) =
                make_uint2(((uint32_t)x[0] & 0xFFFFu) | ((uint32_t)x[1] << 16),
                           ((uint32_t)x[2] & 0xFFFFu) | ((uint32_t)x[3] << 16));
            *reinterpret_cast<uint32_t *>(sHi + e0) =
                (((uint32_t)x[0] >> 16) & 0xFFu) | ((((uint32_t)x[1] >> 16) & 0xFFu) << 8) |
                ((((uint32_t)x[2] >> 16) & 0xFFu) << 16) | ((((uint32_t)x[3] >> 16) & 0xFFu) << 24);
        }
        if (bad) atomicOr(a.status, kDevOverflow);
    }
    int js[K];
    {
        const int64_t t = tb + grp;
        load_idx<K>(il + ((t < t_end) ? t : t_begin) * K, js);
    }
    const bool have_d = kPlanes || mbar_wait(&bar, 0, a.status);
    if (__syncthreads_or(!have_d)) return;

    if (kRFromCounts) {
        if (threadIdx.x < E) {
            const int i = threadIdx.x;
            const long long n = a.counts[(int64_t)layer * E + i];
            const long long r = (long long)(E - 2 * K) * n + T * (long long)K;
            if (r > INT_MAX || r < 0) atomicOr(a.status, kDevOverflow);
            if (kPlanes) s_r[i] = r;
            else sD[i * E + i] = -(int)r;
            if (a.n_zero && blockIdx.x == 0) a.n_zero[(int64_t)layer * E + i] = 0;
        }
    } else {
        // R_i = sum_j D_ji (D symmetric): kPer threads per column, four chains each
        constexpr int kPer = kLossFastThreads / E;  // 2, 4 or 8
        const int i = threadIdx.x % E, part = threadIdx.x / E;
        long long r0 = 0, r1 = 0, r2 = 0, r3 = 0;
        for (int j = part; j < E; j += 4 * kPer) {
            r0 += sD[j * E + i];
            if (j + kPer < E) r1 += sD[(j + kPer) * E + i];
            if (j + 2 * kPer < E) r2 += sD[(j + 2 * kPer) * E + i];
            if (j + 3 * kPer < E) r3 += sD[(j + 3 * kPer) * E + i];
        }
        if (threadIdx.x < E) s_r[threadIdx.x] = 0;
        __syncthreads();
        atomicAdd(reinterpret_cast<unsigned long long *>(&s_r[i]),
                  (unsigned long long)(r0 + r1 + r2 + r3));
        __syncthreads();
        if (threadIdx.x < E) {
            const long long r = s_r[threadIdx.x];
            if (r > INT_MAX || r < 0) atomicOr(a.status, kDevOverflow);
            sD[threadIdx.x * E + threadIdx.x] = -(int)r;
        }
    }
    __syncthreads();

    double tok_sum = 0.0;
    for (; tb < t_end; tb += stride) {
        const int64_t t = tb + grp;
        const bool valid = t < t_end;
        // prefetch the next token group
        const int64_t tn = tb + stride + grp;
        const int64_t tnc = (tn < t_end) ? tn : t_begin;
        float4 zn[4];
        int jn[K];
        if (tb + stride < t_end) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                zn[c] = __ldg(reinterpret_cast<const float4 *>(zl + tnc * E + c * Q + 4 * g));
            load_idx<K>(il + tnc * K, jn);
        }
        int4 acc[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[c] = make_int4(0, 0, 0, 0);
        if constexpr (kPlanes) {
            uint32_t hp[4][2];  // high bytes of entries (0, 2) and (1, 3), 16-bit fields
#pragma unroll
            for (int c = 0; c < 4; ++c) hp[c][0] = hp[c][1] = 0u;
#pragma unroll
            for (int q = 0; q < K; ++q) {
                const int base = js[q] * E + 4 * g;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const uint2 lw = *reinterpret_cast<const uint2 *>(sLo + base + c * Q);
                    const uint32_t hw = *reinterpret_cast<const uint32_t *>(sHi + base + c * Q);
                    acc[c].x += (int)(lw.x & 0xFFFFu);
                    acc[c].y += (int)(lw.x >> 16);
                    acc[c].z += (int)(lw.y & 0xFFFFu);
                    acc[c].w += (int)(lw.y >> 16);
                    hp[c][0] += __byte_perm(hw, 0u, 0x4240);
                    hp[c][1] += __byte_perm(hw, 0u, 0x4341);
                }
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                acc[c].x += (int)((hp[c][0] & 0xFFFFu) << 16);
                acc[c].z += (int)(hp[c][0] & 0xFFFF0000u);
                acc[c].y += (int)((hp[c][1] & 0xFFFFu) << 16);
                acc[c].w += (int)(hp[c][1] & 0xFFFF0000u);
            }
            // the diagonal of D': -R_j in the sum of each chosen expert j
#pragma unroll
            for (int q = 0; q < K; ++q) {
                const int j = js[q];
                if (((j & (Q - 1)) >> 2) != g) continue;
                const int rj = (int)s_r[j];
                const int cj = j / Q, ej = j & 3;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    if (c != cj) continue;
                    acc[c].x -= ej == 0 ? rj : 0;
                    acc[c].y -= ej == 1 ? rj : 0;
                    acc[c].z -= ej == 2 ? rj : 0;
                    acc[c].w -= ej == 3 ? rj : 0;
                }
            }
        } else {
#pragma unroll
            for (int q = 0; q < K; ++q) {
                const int *row = sD + js[q] * E + 4 * g;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int4 d = *reinterpret_cast<const int4 *>(row + c * Q);
                    acc[c].x += d.x;
                    acc[c].y += d.y;
                    acc[c].z += d.z;
                    acc[c].w += d.w;
                }
            }
        }
        float w[16], zz[16], gv[16];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            w[4 * c] = -(float)acc[c].x;
            w[4 * c + 1] = -(float)acc[c].y;
            w[4 * c + 2] = -(float)acc[c].z;
            w[4 * c + 3] = -(float)acc[c].w;
            zz[4 * c] = zc[c].x;
            zz[4 * c + 1] = zc[c].y;
            zz[4 * c + 2] = zc[c].z;
            zz[4 * c + 3] = zc[c].w;
        }
        float den = 0.0f, num = 0.0f;
        if (kGate == 0) {
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                gv[e] = sigmoid_fast(zz[e]);
                den += gv[e];
                num = fmaf(gv[e], w[e], num);
            }
        } else {
            float mx = zz[0];
#pragma unroll
            for (int e = 1; e < 16; ++e) mx = fmaxf(mx, zz[e]);
#pragma unroll
            for (int o = G / 2; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, o));
            const float mxs = mx * 1.4426950408889634f;
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                gv[e] = ex2_approx(fmaf(zz[e], 1.4426950408889634f, -mxs));
                den += gv[e];
                num = fmaf(gv[e], w[e], num);
            }
        }
#pragma unroll
        for (int o = G / 2; o > 0; o >>= 1) {
            den += __shfl_xor_sync(kFull, den, o);
            num += __shfl_xor_sync(kFull, num, o);
        }
        const float inv = 1.0f / den;
        const float A = num * inv;
        if (valid && g == 0) tok_sum += (double)A;
        if (dzl && valid) {
            // dz = c/S * jac * (w - A) = jac * (cs w - cs A)
            const float cs = a.coef * inv;
            const float csA = cs * A;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float4 o;
                float *op = reinterpret_cast<float *>(&o);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float s = gv[4 * c + e];
                    const float jac = (kGate == 0) ? fmaf(-s, s, s) : s;
                    op[e] = jac * fmaf(cs, w[4 * c + e], -csA);
                }
                *reinterpret_cast<float4 *>(dzl + t * E + c * Q + 4 * g) = o;
            }
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) zc[c] = zn[c];
#pragma unroll
        for (int q = 0; q < K; ++q) js[q] = jn[q];
    }
    // CTA partial, in warp and lane order
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tok_sum += __shfl_xor_sync(kFull, tok_sum, o);
    if (lane == 0) s_part[warp] = tok_sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        double sum = 0.0;
        for (int q = 0; q < kWarps; ++q) sum += s_part[q];
        a.partials[(int64_t)layer * P + blockIdx.x] = sum;
        __threadfence();
        s_last = (atomicAdd(&a.done[layer], 1) == P - 1);
    }
    __syncthreads();
    if (!s_last) return;
    // last CTA of this problem: fixed-order sum of the partials, origin_do
    __threadfence();
    if (warp == 0) {
        const double sum = warp_sum_fixed(a.partials + (int64_t)layer * P, P);
        if (lane == 0) {
            a.loss[layer] = (float)(sum * a.scale);
            a.done[layer] = 0;
            if (a.status_out) atomicOr(a.status_out, *reinterpret_cast<volatile int *>(a.status));
        }
    }
    if (a.origin_do) {
        long long o = 0;
        for (int e = threadIdx.x; e < E * E; e += blockDim.x) {
            const int i = e / E, j = e - (e / E) * E;
            if (i != j) {
                const long long d =
                    kPlanes ? (long long)sLo[e] | ((long long)sHi[e] << 16) : (long long)sD[e];
                o += d * d;
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) o += __shfl_xor_sync(kFull, o, off);
        if (lane == 0) s_o[warp] = o;
        __syncthreads();
        if (threadIdx.x == 0) {
            long long sum = 0;
            for (int q = 0; q < kWarps; ++q) sum += s_o[q];
            a.origin_do[layer] = sum;
        }
    }
}

// Selected-expert indices of every token recovered from the signature words
// (for do_loss_fwd_bwd, whose caller passes bits): a warp per 32-token tile
// transposes the E/32 words back to one row per token and lists its set bits.
template <int E, int K>
__global__ void __launch_bounds__(256)
idx_from_bits_kernel(const uint32_t *__restrict__ bits, int64_t T, int64_t W, int64_t ntiles,
                     uint8_t *__restrict__ idx, int *__restrict__ zero_ptr, int zero_n) {
    constexpr int R = E / 32;
    pdl_trigger();
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < zero_n; i += gridDim.x * blockDim.x)
        zero_ptr[i] = 0;
    const int lane = threadIdx.x & 31;
    const int64_t wid = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const uint32_t lo_mask[5] = {0x0000FFFFu, 0x00FF00FFu, 0x0F0F0F0Fu, 0x33333333u, 0x55555555u};
    for (int64_t tile = wid; tile < ntiles; tile += nw) {
        const int64_t layer = tile / W, w = tile - layer * W;
        uint32_t m[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            uint32_t x = __ldg(bits + (layer * E + 32 * r + lane) * W + w);
            // lane = expert column -> lane = token row (the same bit transpose)
#pragma unroll
            for (int s = 0; s < 5; ++s) {
                const int j = 16 >> s;
                const uint32_t lo = lo_mask[s];
                const uint32_t p = __shfl_xor_sync(kFull, x, j);
                x = (lane & j) ? ((x & ~lo) | ((p >> j) & lo)) : ((x & lo) | ((p << j) & ~lo));
            }
            m[r] = x;
        }
        const int64_t t = 32 * w + lane;
        if (t >= T) continue;
        uint8_t out[K];
        int n = 0;
#pragma unroll
        for (int q = 0; q < K; ++q) out[q] = 0;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            uint32_t x = m[r];
            while (x && n < K) {
                const int b = __ffs(x) - 1;
                x &= x - 1;
#pragma unroll
                for (int q = 0; q < K; ++q)
                    if (q == n) out[q] = (uint8_t)(32 * r + b);
                ++n;
            }
        }
        uint8_t *p = idx + (layer * T + t) * K;
#pragma unroll
        for (int q = 0; q < K; ++q) p[q] = out[q];
    }
}

template <int E, int K, bool kRFromCounts>
cudaError_t run_loss_fast(const LossArgs &args, int gate, int P, const Problem &p, cudaStream_t s) {
    const size_t smem = loss_fast_smem<E>();
    cudaError_t e = ensure_smem_limit<loss_fast_kernel<E, K, 0, kRFromCounts>>(smem);
    if (e == cudaSuccess) e = ensure_smem_limit<loss_fast_kernel<E, K, 1, kRFromCounts>>(smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)P, (unsigned)p.L);
    cfg.blockDim = dim3(loss_fast_threads<E>());
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (gate == 0) return cudaLaunchKernelEx(&cfg, loss_fast_kernel<E, K, 0, kRFromCounts>, args);
    return cudaLaunchKernelEx(&cfg, loss_fast_kernel<E, K, 1, kRFromCounts>, args);
}

template <int E, bool kRFromCounts>
cudaError_t dispatch_loss_k(const LossArgs &args, int gate, int P, const Problem &p, cudaStream_t s) {
    switch (p.k) {
        case 1: return run_loss_fast<E, 1, kRFromCounts>(args, gate, P, p, s);
        case 2: return run_loss_fast<E, 2, kRFromCounts>(args, gate, P, p, s);
        case 4: return run_loss_fast<E, 4, kRFromCounts>(args, gate, P, p, s);
        default: return run_loss_fast<E, 8, kRFromCounts>(args, gate, P, p, s);
    }
}

template <int E, int K>
cudaError_t run_idx(const uint32_t *bits, const Problem &p, uint8_t *idx, int *zero_ptr, int zero_n,
                    cudaStream_t s) {
    const int64_t ntiles = (int64_t)p.L * p.W;
    int64_t blocks = (ntiles + 7) / 8;
    if (blocks > 4096) blocks = 4096;
    idx_from_bits_kernel<E, K><<<(unsigned)blocks, 256, 0, s>>>(bits, p.T, p.W, ntiles, idx, zero_ptr,
                                                                zero_n);
    return cudaGetLastError();
}

}  // namespace

bool loss_fast_supported(const Problem &p, const float *logits, const int *D, const float *dlogits) {
    const bool e_ok = p.E == 32 || p.E == 64 || p.E == 128;
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    return e_ok && k_ok && reinterpret_cast<uintptr_t>(logits) % 16 == 0 &&
           reinterpret_cast<uintptr_t>(D) % 16 == 0 &&
           (dlogits == nullptr || reinterpret_cast<uintptr_t>(dlogits) % 16 == 0);
}

// The E = 256 variant (the matrix of the same tokens, with counts): T < 2^24
// keeps every entry of D within the 24 bits of its shared-memory planes.
bool loss_fast256_supported(const Problem &p, const float *logits, const int *D,
                            const float *dlogits) {
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    return p.E == 256 && k_ok && p.T < (int64_t)(1 << 24) &&
           reinterpret_cast<uintptr_t>(logits) % 16 == 0 &&
           reinterpret_cast<uintptr_t>(D) % 16 == 0 &&
           (dlogits == nullptr || reinterpret_cast<uintptr_t>(dlogits) % 16 == 0);
}

// CTAs per problem of the fast loss kernel and the tokens each one takes.
void loss_fast_grid(const Problem &p, int *P, int *tokens_per_cta) {
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // one wave: three CTAs fit on an SM, one at E = 256
    int64_t want = (int64_t)sms * (p.E == 256 ? 1 : 3) / p.L;
    if (want < 1) want = 1;
    int64_t tpc = (p.T + want - 1) / want;
    tpc = (tpc + 31) / 32 * 32;
    if (tpc < 32) tpc = 32;
    *tokens_per_cta = (int)tpc;
    *P = (int)((p.T + tpc - 1) / tpc);
}

cudaError_t launch_idx_from_bits(const uint32_t *bits, const Problem &p, uint8_t *idx, int *zero_ptr,
                                 int zero_n, cudaStream_t s) {
#define DOL_IDX_CASE(EE)                                                          \
    if (p.E == EE) {                                                              \
        switch (p.k) {                                                            \
            case 1: return run_idx<EE, 1>(bits, p, idx, zero_ptr, zero_n, s);     \
            case 2: return run_idx<EE, 2>(bits, p, idx, zero_ptr, zero_n, s);     \
            case 4: return run_idx<EE, 4>(bits, p, idx, zero_ptr, zero_n, s);     \
            default: return run_idx<EE, 8>(bits, p, idx, zero_ptr, zero_n, s);    \
        }                                                                         \
    }
    DOL_IDX_CASE(32)
    DOL_IDX_CASE(64)
    DOL_IDX_CASE(128)
#undef DOL_IDX_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_loss_fast(const float *logits, const uint8_t *idx, const int *D,
                             const int *counts, int *n_zero, const Problem &p, int gate,
                             float d_scale, float grad_scale, float *loss, long long *origin_do,
                             float *dlogits, double *partials, int *done, int *status,
                             int *status_out, cudaStream_t s, const int *img_ok) {
    int P = 1, tpc = 32;
    loss_fast_grid(p, &P, &tpc);
    const double norm = 1.0 / ((double)p.T * (double)p.T * (double)p.k);
    LossArgs args;
    args.logits = logits;
    args.idx = idx;
    args.D = D;
    args.counts = counts;
    args.n_zero = n_zero;
    args.T = p.T;
    args.k = p.k;
    args.tokens_per_cta = tpc;
    args.coef = (float)((double)grad_scale * (double)d_scale * norm);
    args.scale = (double)d_scale * norm;
    args.dlogits = dlogits;
    args.partials = partials;
    args.done = done;
    args.loss = loss;
    args.origin_do = origin_do;
    args.status = status;
    args.status_out = status_out;
    args.img_ok = img_ok;
    if (counts) {
        if (p.E == 32) return dispatch_loss_k<32, true>(args, gate, P, p, s);
        if (p.E == 64) return dispatch_loss_k<64, true>(args, gate, P, p, s);
        if (p.E == 256) return dispatch_loss_k<256, true>(args, gate, P, p, s);
        return dispatch_loss_k<128, true>(args, gate, P, p, s);
    }
    if (p.E == 256) return cudaErrorInvalidValue;  // the planes need the counts' R
    if (p.E == 32) return dispatch_loss_k<32, false>(args, gate, P, p, s);
    if (p.E == 64) return dispatch_loss_k<64, false>(args, gate, P, p, s);
    return dispatch_loss_k<128, false>(args, gate, P, p, s);
}

}  // namespace dol
