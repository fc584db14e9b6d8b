// Consumers of the per-expert token counts n_e (App. C.3) on the
// expert-parallel side of training:
//  * MaxVio (App. E): with L_r the tokens of the experts that reside on rank
//    r and tau = (1/|R|) sum_r L_r the ideal load,
//      MaxVio = max_r |L_r / tau - 1|,
//    one CTA per problem (MoE layer) on the device, straight from the counts
//    the signature kernels leave there;
//  * the Replica Expert Mechanism's global-batch replica allocation (Sec. 3.2,
//    Eq. benefit_score; App. B.1, Algorithm rem_allocation), a short greedy
//    loop over |R| D placements that runs on the host, as the paper's
//    controller does at each global-batch boundary.
#include <cmath>
#include <cstdint>
#include <vector>

#include "dol_internal.cuh"
#include "doloss.h"

namespace dol {
namespace {

constexpr int kMaxVioThreads = 256;
constexpr int kDevBadRank = 4;  // an expert_rank entry outside [0, R)

__global__ void __launch_bounds__(kMaxVioThreads)
maxvio_kernel(const int *__restrict__ counts, const int *__restrict__ expert_rank, int E, int R,
              long long *__restrict__ rank_loads, double *__restrict__ maxvio,
              int *__restrict__ status) {
    extern __shared__ unsigned long long s_load[];  // [R]
    __shared__ long long s_part[kMaxVioThreads / 32];
    __shared__ double s_max[kMaxVioThreads / 32];
    const int layer = blockIdx.x, tid = threadIdx.x, lane = tid & 31, wp = tid >> 5;
    for (int r = tid; r < R; r += kMaxVioThreads) s_load[r] = 0ull;
    __syncthreads();
    // L_r = sum of n_e over the experts on rank r (integer adds: the order of
    // the shared-memory atomics does not change the sums)
    const int *cl = counts + (size_t)layer * E;
    for (int e = tid; e < E; e += kMaxVioThreads) {
        const int r = __ldg(expert_rank + e);
        if ((unsigned)r >= (unsigned)R) {
            if (status) atomicOr(status, kDevBadRank);
            continue;
        }
        atomicAdd(&s_load[r], (unsigned long long)(long long)__ldg(cl + e));
    }
    __syncthreads();
    long long part = 0;
    for (int r = tid; r < R; r += kMaxVioThreads) {
        const long long v = (long long)s_load[r];
        part += v;
        if (rank_loads) rank_loads[(size_t)layer * R + r] = v;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(kFull, part, o);
    if (lane == 0) s_part[wp] = part;
    __syncthreads();
    long long total = 0;
#pragma unroll
    for (int q = 0; q < kMaxVioThreads / 32; ++q) total += s_part[q];
    // tau in double from the exact integer total; a batch without tokens has
    // no violation
    const double tau = (double)total / (double)R;
    double m = 0.0;
    if (total != 0)
        for (int r = tid; r < R; r += kMaxVioThreads)
            m = fmax(m, fabs((double)(long long)s_load[r] / tau - 1.0));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmax(m, __shfl_xor_sync(kFull, m, o));
    if (lane == 0) s_max[wp] = m;
    __syncthreads();
    if (tid == 0) {
        double mm = 0.0;
        for (int q = 0; q < kMaxVioThreads / 32; ++q) mm = fmax(mm, s_max[q]);
        maxvio[layer] = mm;
    }
}

// Eq. benefit_score: tokens the receiving rank (load lr) can take over from
// the sending rank (load ls) for an expert with remaining volume te.
double benefit_score(double te, double ls, double lr, double tau) {
    if (lr < tau && ls > tau) return std::fmin(std::fmin(tau - lr, te), ls - tau);
    if (lr >= tau && ls > lr) return std::fmin(std::floor((ls - lr) / 2.0), te);
    return -1.0;
}

}  // namespace
}  // namespace dol

extern "C" {

do_status do_maxvio(const int32_t *counts, const int32_t *expert_rank, int32_t E, int32_t R,
                    int32_t L, int64_t *rank_loads, double *maxvio, int32_t *status_flags,
                    void *stream) {
    if (E < 1 || R < 1 || L < 1) return DO_ERR_INVALID_ARG;
    if (E > (1 << 20) || R > 4096 || L > (1 << 24)) return DO_ERR_UNSUPPORTED;
    if (!counts || !expert_rank || !maxvio) return DO_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(counts) | reinterpret_cast<uintptr_t>(expert_rank)) % 4 ||
        reinterpret_cast<uintptr_t>(maxvio) % 8 ||
        (rank_loads && reinterpret_cast<uintptr_t>(rank_loads) % 8) ||
        (status_flags && reinterpret_cast<uintptr_t>(status_flags) % 4))
        return DO_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    dol::maxvio_kernel<<<(unsigned)L, dol::kMaxVioThreads, sizeof(unsigned long long) * (size_t)R, s>>>(
        counts, expert_rank, E, R, reinterpret_cast<long long *>(rank_loads), maxvio, status_flags);
    return cudaGetLastError() == cudaSuccess ? DO_OK : DO_ERR_CUDA;
}

do_status do_rem_allocate(const double *loads, const double *expert_tokens,
                          const int32_t *expert_rank, int32_t R, int32_t E, int32_t D,
                          int32_t *placed_expert, int32_t *placed_sender,
                          int32_t *placed_receiver, double *placed_tokens, int32_t *n_placed,
                          double *loads_out) {
    if (R < 1 || E < 1 || D < 0) return DO_ERR_INVALID_ARG;
    if ((int64_t)R * E > (int64_t)1 << 26 || (int64_t)R * D > (int64_t)1 << 26)
        return DO_ERR_UNSUPPORTED;
    if (!loads || !expert_tokens || !expert_rank || !n_placed || !loads_out) return DO_ERR_INVALID_ARG;
    if (D > 0 && (!placed_expert || !placed_sender || !placed_receiver || !placed_tokens))
        return DO_ERR_INVALID_ARG;
    for (int32_t e = 0; e < E; ++e)
        if (expert_rank[e] < 0 || expert_rank[e] >= R) return DO_ERR_INVALID_ARG;
    std::vector<double> L(loads, loads + R), T(expert_tokens, expert_tokens + E);
    double sum = 0.0;
    for (int32_t r = 0; r < R; ++r) sum += L[r];
    const double tau = sum / (double)R;  // fixed for the whole allocation
    std::vector<int32_t> used(R, 0);                        // replicas placed on each rank
    std::vector<char> has((size_t)R * E, 0);                 // has[r][e]: e already on r
    int32_t n = 0;
    for (;;) {
        // receiver: the least-loaded rank with a free slot (lowest index on ties)
        int32_t rr = -1;
        for (int32_t r = 0; r < R; ++r)
            if (used[r] < D && (rr < 0 || L[r] < L[rr])) rr = r;
        if (rr < 0) break;
        // the (expert, sender) pair of largest score; an expert is sent from its
        // home rank (lowest expert index on ties)
        int32_t best_e = -1;
        double best = 0.0;
        for (int32_t e = 0; e < E; ++e) {
            const int32_t rs = expert_rank[e];
            if (rs == rr || has[(size_t)rr * E + e]) continue;
            const double sc = dol::benefit_score(T[e], L[rs], L[rr], tau);
            if (best_e < 0 || sc > best) {
                best = sc;
                best_e = e;
            }
        }
        if (best_e < 0 || !(best > 0.0)) break;
        const int32_t rs = expert_rank[best_e];
        placed_expert[n] = best_e;
        placed_sender[n] = rs;
        placed_receiver[n] = rr;
        placed_tokens[n] = best;
        ++n;
        ++used[rr];
        has[(size_t)rr * E + best_e] = 1;
        L[rr] += best;
        L[rs] -= best;
        T[best_e] -= best;
    }
    *n_placed = n;
    for (int32_t r = 0; r < R; ++r) loads_out[r] = L[r];
    return DO_OK;
}

}  // extern "C"
