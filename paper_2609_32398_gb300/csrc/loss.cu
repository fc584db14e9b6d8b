// Step 3: the surrogate DO-loss and its gradient to the router logits.
//
// Eq. do_loss (Sec. 3.1.3) with G = d_scale * D detached (Eq. global_do):
//   L = 1/(m^2 k) sum_i sum_j G_ij C_ij,   C_ij = sum_t p_it (f_it - f_jt).
// Summing over j first turns the double sum into one integer weight per
// token and expert:
//   sum_j G_ij (f_it - f_jt) = d_scale * w_it,
//   w_it = f_it R_i - sum_{j in S_t} D_ij,   R_i = sum_j D_ij,
// so L = d_scale/(m^2 k) sum_t A_t with A_t = sum_i p_it w_it, and
// dL/dp_it = d_scale w_it / (m^2 k).  Through the gate (S = sum_i s_it):
//   sigmoid-norm  dz_lt = c s_lt (1 - s_lt) / S (w_lt - A_t)
//   softmax       dz_lt = c p_lt (w_lt - A_t)
// with c = grad_scale * d_scale / (m^2 k).  w is exact in int32; A_t is
// accumulated in fp32 inside a token and in fp64 across tokens, in a fixed
// order.  The k-row gather of D reads rows of D, which relies on D being
// symmetric (every Hamming matrix, and every sum of them, is).
#include <climits>

#include "dol_internal.cuh"

namespace dol {
namespace {

constexpr int kLossThreads = 256;
constexpr int kLossWarps = kLossThreads / 32;
constexpr size_t kSmemDLimit = 200 * 1024;

__device__ __forceinline__ float sigmoid_f(float z) {
    // exp of at most 80 keeps 1 + e finite, so the fast divide stays exact enough
    const float e = __expf(-fmaxf(z, -80.0f));
    return __fdividef(1.0f, 1.0f + e);
}

template <int R, bool kSmemD, int kGate>
__global__ void __launch_bounds__(kLossThreads)
loss_generic_kernel(const float *__restrict__ logits, const uint32_t *__restrict__ bits,
                    const int *__restrict__ Dg, int64_t T, int E, int64_t W, float coef,
                    float *__restrict__ dlogits, double *__restrict__ partials, int P,
                    int *__restrict__ status) {
    extern __shared__ __align__(16) int smem[];
    __shared__ double s_part[kLossWarps];
    int *sD = smem;
    int *sR = smem + (kSmemD ? E * E : 0);

    const int layer = blockIdx.y;
    const int *Dl = Dg + (int64_t)layer * E * E;
    const float *z = logits + (int64_t)layer * T * E;
    float *dz = dlogits ? dlogits + (int64_t)layer * T * E : nullptr;
    const uint32_t *bl = bits + (int64_t)layer * E * W;

    if (kSmemD)
        for (int idx = threadIdx.x; idx < E * E; idx += blockDim.x) sD[idx] = __ldg(Dl + idx);
    __syncthreads();
    const int *Dsrc = kSmemD ? sD : Dl;
    for (int i = threadIdx.x; i < E; i += blockDim.x) {
        long long acc = 0;
        for (int j = 0; j < E; ++j) acc += Dsrc[(int64_t)i * E + j];
        if (acc > INT_MAX || acc < 0) atomicOr(status, kDevOverflow);
        sR[i] = (int)acc;
    }
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    int Ri[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int i = lane + 32 * r;
        Ri[r] = (i < E) ? sR[i] : 0;
    }
    double tok_sum = 0.0;  // sum of A_t over this warp's tokens (meaningful in lane 0)

    for (int64_t w = (int64_t)blockIdx.x * kLossWarps + warp; w < W;
         w += (int64_t)P * kLossWarps) {
        uint32_t bw[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int i = lane + 32 * r;
            bw[r] = (i < E) ? __ldg(bl + (int64_t)i * W + w) : 0u;
        }
        const int64_t t0 = w * 32;
        const int nt = (int)min64(32, T - t0);
        for (int tt = 0; tt < nt; ++tt) {
            const int64_t t = t0 + tt;
            const float *zt = z + t * E;
            int acc[R];
#pragma unroll
            for (int r = 0; r < R; ++r) acc[r] = 0;
            // sum_{j in S_t} D_ji for this lane's experts i
#pragma unroll
            for (int rr = 0; rr < R; ++rr) {
                unsigned m = __ballot_sync(kFull, (bw[rr] >> tt) & 1u);
                while (m) {
                    const int j = 32 * rr + __ffs(m) - 1;
                    m &= m - 1;
                    const int *row = Dsrc + (int64_t)j * E;
#pragma unroll
                    for (int r = 0; r < R; ++r) {
                        const int i = lane + 32 * r;
                        if (i < E) acc[r] += row[i];
                    }
                }
            }
            float zr[R], wr[R], g[R];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int i = lane + 32 * r;
                const bool f = (bw[r] >> tt) & 1u;
                wr[r] = (float)(f ? Ri[r] - acc[r] : -acc[r]);
                zr[r] = (i < E) ? __ldg(zt + i) : 0.0f;
            }
            float num = 0.0f, den = 0.0f;
            if (kGate == 0) {  // sigmoid-norm
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int i = lane + 32 * r;
                    g[r] = (i < E) ? sigmoid_f(zr[r]) : 0.0f;
                    den += g[r];
                    num += g[r] * wr[r];
                }
            } else {  // softmax
                float mx = -INFINITY;
#pragma unroll
                for (int r = 0; r < R; ++r)
                    if (lane + 32 * r < E) mx = fmaxf(mx, zr[r]);
                mx = warp_max(mx);
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int i = lane + 32 * r;
                    g[r] = (i < E) ? __expf(zr[r] - mx) : 0.0f;
                    den += g[r];
                    num += g[r] * wr[r];
                }
            }
            den = warp_sum(den);
            num = warp_sum(num);
            const float inv = 1.0f / den;
            const float A = num * inv;
            tok_sum += (double)A;
            if (dz) {
                const float cs = coef * inv;
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int i = lane + 32 * r;
                    if (i < E) {
                        const float jac = (kGate == 0) ? g[r] * (1.0f - g[r]) : g[r];
                        dz[t * E + i] = cs * jac * (wr[r] - A);
                    }
                }
            }
        }
    }
    if (lane == 0) s_part[warp] = tok_sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        double s = 0.0;
        for (int q = 0; q < kLossWarps; ++q) s += s_part[q];
        partials[(int64_t)layer * P + blockIdx.x] = s;
    }
}

// loss[l] = d_scale/(m^2 k) * sum of the partials in block order; origin_do[l]
// = sum_{i != j} D_ij^2 (Eq. origin_do), exact in int64.
__global__ void __launch_bounds__(256)
loss_finalize_kernel(const double *__restrict__ partials, int P, const int *__restrict__ Dg, int E,
                     double scale, float *__restrict__ loss, long long *__restrict__ origin_do) {
    __shared__ long long s_red[256];
    __shared__ double s_dred[256];
    const int layer = blockIdx.x;
    {
        const double s = block_sum_fixed(partials + (int64_t)layer * P, P, s_dred, 256);
        if (threadIdx.x == 0) loss[layer] = (float)(s * scale);
    }
    if (origin_do) {
        const int *Dl = Dg + (int64_t)layer * E * E;
        long long acc = 0;
        for (int64_t idx = threadIdx.x; idx < (int64_t)E * E; idx += blockDim.x) {
            const int i = (int)(idx / E), j = (int)(idx % E);
            if (i != j) {
                const long long d = Dl[idx];
                acc += d * d;
            }
        }
        s_red[threadIdx.x] = acc;
        __syncthreads();
        for (int o = blockDim.x / 2; o > 0; o >>= 1) {
            if (threadIdx.x < o) s_red[threadIdx.x] += s_red[threadIdx.x + o];
            __syncthreads();
        }
        if (threadIdx.x == 0) origin_do[layer] = s_red[0];
    }
}

// origin_do alone (Eq. origin_do), one CTA per problem, exact in int64.
__global__ void __launch_bounds__(256)
origin_do_kernel(const int *__restrict__ Dg, int E, long long *__restrict__ origin_do) {
    __shared__ long long s_red[256];
    const int *Dl = Dg + (int64_t)blockIdx.x * E * E;
    long long acc = 0;
    for (int64_t idx = threadIdx.x; idx < (int64_t)E * E; idx += blockDim.x) {
        const int i = (int)(idx / E), j = (int)(idx % E);
        if (i != j) {
            const long long d = Dl[idx];
            acc += d * d;
        }
    }
    s_red[threadIdx.x] = acc;
    __syncthreads();
    for (int o = blockDim.x / 2; o > 0; o >>= 1) {
        if (threadIdx.x < o) s_red[threadIdx.x] += s_red[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) origin_do[blockIdx.x] = s_red[0];
}

template <int R, bool kSmemD, int kGate>
cudaError_t run_loss(const float *logits, const uint32_t *bits, const int *D, const Problem &p,
                     float coef, float *dlogits, double *partials, int P, int *status,
                     cudaStream_t s) {
    const size_t smem = sizeof(int) * ((kSmemD ? (size_t)p.E * p.E : 0) + (size_t)p.E);
    auto kern = loss_generic_kernel<R, kSmemD, kGate>;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
    }
    dim3 grid((unsigned)P, (unsigned)p.L);
    kern<<<grid, kLossThreads, smem, s>>>(logits, bits, D, p.T, p.E, p.W, coef, dlogits, partials,
                                          P, status);
    return cudaGetLastError();
}

template <int R>
cudaError_t dispatch_gate(const float *logits, const uint32_t *bits, const int *D, const Problem &p,
                          int gate, float coef, float *dlogits, double *partials, int P,
                          int *status, cudaStream_t s) {
    const bool smem_d = sizeof(int) * ((size_t)p.E * p.E + p.E) <= kSmemDLimit;
    if (gate == 0)
        return smem_d ? run_loss<R, true, 0>(logits, bits, D, p, coef, dlogits, partials, P, status, s)
                      : run_loss<R, false, 0>(logits, bits, D, p, coef, dlogits, partials, P, status, s);
    return smem_d ? run_loss<R, true, 1>(logits, bits, D, p, coef, dlogits, partials, P, status, s)
                  : run_loss<R, false, 1>(logits, bits, D, p, coef, dlogits, partials, P, status, s);
}

}  // namespace

int loss_blocks_per_problem(const Problem &p) {
    int64_t blocks = (p.W + kLossWarps - 1) / kLossWarps;
    int64_t cap = 1024 / p.L;
    if (cap < 1) cap = 1;
    if (blocks > cap) blocks = cap;
    return (int)(blocks < 1 ? 1 : blocks);
}

WsLayout ws_layout(const Problem &p) {
    auto up = [](size_t x) { return (x + 255) / 256 * 256; };
    WsLayout w;
    const int64_t fast_parts = p.W;  // the fast kernel gives every CTA at least 32 tokens
    const int64_t gen_parts = loss_blocks_per_problem(p);
    w.max_parts = (int)(fast_parts > gen_parts ? fast_parts : gen_parts);
    const bool fast_k = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    const bool fast_e = p.E == 32 || p.E == 64 || p.E == 128;
    w.done = kWsHeader;
    w.partials = up(w.done + sizeof(int) * (size_t)p.L);
    w.idx = up(w.partials + sizeof(double) * (size_t)p.L * (size_t)w.max_parts);
    w.cooc_parts = up(w.idx + (fast_k ? (size_t)p.L * (size_t)p.T * (size_t)p.k : 0));
    const size_t parts = (fast_k && fast_e) ? sizeof(uint32_t) * (size_t)p.L *
                                                  (size_t)max_sig_ctas_per_problem(p) *
                                                  cooc_partial_words(p.E)
                                            : 0;
    w.n_acc = up(w.cooc_parts + parts);
    w.bimg = up(w.n_acc + ((fast_k && fast_e) ? sizeof(int) * (size_t)p.L * p.E : 0));
    // the dispatch order of a routed call may run beside the loss kernel: its
    // scratch has a region of its own
    w.img_ok = up(w.bimg + ((fast_k && p.E == 128) ? (size_t)kBImageBytes * (size_t)p.L : 0));
    w.route_base = up(w.img_ok + ((fast_k && p.E == 128) ? sizeof(int) * (size_t)p.L : 0));
    w.total = up(w.route_base + sizeof(int) * (size_t)route_scratch_ints(p));
    return w;
}

int max_sig_ctas_per_problem(const Problem &p) {
    int64_t gx = kMaxSigCtas / p.L;
    if (gx > p.W) gx = p.W;
    return (int)(gx < 1 ? 1 : gx);
}

cudaError_t launch_loss(const float *logits, const uint32_t *bits, const int *D, const Problem &p,
                        int gate, float d_scale, float grad_scale, float *loss,
                        long long *origin_do, float *dlogits, void *workspace, cudaStream_t s) {
    int *status = reinterpret_cast<int *>(workspace);
    double *partials =
        reinterpret_cast<double *>(static_cast<char *>(workspace) + ws_layout(p).partials);
    const int P = loss_blocks_per_problem(p);
    const double norm = 1.0 / ((double)p.T * (double)p.T * (double)p.k);
    const float coef = (float)((double)grad_scale * (double)d_scale * norm);
    const int r = (p.E + 31) / 32;
    cudaError_t e;
    if (r <= 1) e = dispatch_gate<1>(logits, bits, D, p, gate, coef, dlogits, partials, P, status, s);
    else if (r <= 2) e = dispatch_gate<2>(logits, bits, D, p, gate, coef, dlogits, partials, P, status, s);
    else if (r <= 4) e = dispatch_gate<4>(logits, bits, D, p, gate, coef, dlogits, partials, P, status, s);
    else if (r <= 8) e = dispatch_gate<8>(logits, bits, D, p, gate, coef, dlogits, partials, P, status, s);
    else if (r <= 16) e = dispatch_gate<16>(logits, bits, D, p, gate, coef, dlogits, partials, P, status, s);
    else e = dispatch_gate<32>(logits, bits, D, p, gate, coef, dlogits, partials, P, status, s);
    if (e != cudaSuccess) return e;
    loss_finalize_kernel<<<p.L, 256, 0, s>>>(partials, P, D, p.E, (double)d_scale * norm, loss,
                                             origin_do);
    return cudaGetLastError();
}

// Variance of the E (E - 1) off-diagonal distances of a local window from
// Eq. origin_do (their sum of squares) and Eq. zero_sum (their sum is
// 2 T k (E - k)): var = origin_do / (E (E - 1)) - mean^2 (App. C.1).  One
// thread per problem, fp64.
__global__ void offdiag_variance_kernel(const long long *__restrict__ origin_do, int64_t T, int E,
                                        int k, int L, double *__restrict__ var) {
    const int l = blockIdx.x * blockDim.x + threadIdx.x;
    if (l >= L) return;
    const double n = (double)E * (double)(E - 1);
    const double mean = 2.0 * (double)T * (double)k * (double)(E - k) / n;
    var[l] = (double)origin_do[l] / n - mean * mean;
}

cudaError_t launch_offdiag_variance(const long long *origin_do, const Problem &p, double *var,
                                    cudaStream_t s) {
    offdiag_variance_kernel<<<(p.L + 255) / 256, 256, 0, s>>>(origin_do, p.T, p.E, p.k, p.L, var);
    return cudaGetLastError();
}

cudaError_t launch_origin_do(const int *D, const Problem &p, long long *origin_do, cudaStream_t s) {
    origin_do_kernel<<<p.L, 256, 0, s>>>(D, p.E, origin_do);
    return cudaGetLastError();
}

}  // namespace dol
