// Internal declarations shared by the kernels and the C ABI of libdoloss.
// Nothing here is part of the public interface (include/doloss.h is).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace dol {

constexpr unsigned kFull = 0xffffffffu;

// Bits of the device status word kept at the start of the workspace.
constexpr int kDevOverflow = 1;  // a row sum of D did not fit int32
constexpr int kDevTimeout = 2;   // a bounded device wait ran out

// Workspace layout: [status word | pad to 256 B | fp64 loss partials [L][P]].
constexpr size_t kWsHeader = 256;

// Problem description handed from the C ABI to the launchers.
struct Problem {
    int64_t T;    // tokens per problem (the paper's m)
    int E;        // experts (n)
    int k;        // experts selected per token (K)
    int L;        // independent problems in the batch
    int64_t W;    // 32-bit words per signature, ceil(T/32)
};

// Up to three int ranges that a kernel clears for the kernels after it.
struct ZeroSpans {
    int *p[3];
    int64_t n[3];
};

// Workspace of the loss step, carved from the caller's buffer:
//   [0, 256)        device status word (kDevOverflow | kDevTimeout bits)
//   done            [L] int, per-problem count of finished loss CTAs
//   partials        [L][max CTAs per problem] fp64 sums of A_t
//   idx             [L][T][k] uint8, the selected experts of every token
struct WsLayout {
    size_t done, partials, idx, total;
    int max_parts;  // partial slots per problem
};
WsLayout ws_layout(const Problem &p);
inline size_t workspace_bytes(const Problem &p) { return ws_layout(p).total; }

// Number of generic loss-kernel CTAs per problem; fixes the partial-sum
// layout and therefore the reduction order.
int loss_blocks_per_problem(const Problem &p);

// Launchers (return the first CUDA error, cudaSuccess otherwise).
cudaError_t launch_signatures(const float *logits, const Problem &p, uint32_t *bits,
                              int *counts, cudaStream_t s);
cudaError_t launch_hamming(const uint32_t *bits, const Problem &p, int *D, cudaStream_t s);
cudaError_t launch_hamming_accumulate(const uint32_t *bits, const Problem &p, int *D, int *counts,
                                      cudaStream_t s);
cudaError_t launch_loss(const float *logits, const uint32_t *bits, const int *D,
                        const Problem &p, int gate, float d_scale, float grad_scale,
                        float *loss, long long *origin_do, float *dlogits, void *workspace,
                        cudaStream_t s);

// Fast paths (E in {32, 64, 128}, k in {1, 2, 4, 8}, 16-byte aligned rows).
bool signatures_fast_supported(const float *logits, const Problem &p);
cudaError_t launch_signatures_fast(const float *logits, const Problem &p, uint32_t *bits,
                                   int *counts, uint8_t *idx, const ZeroSpans &zero, int *status,
                                   cudaStream_t s);
bool loss_fast_supported(const Problem &p, const float *logits, const int *D, const float *dlogits);
cudaError_t launch_idx_from_bits(const uint32_t *bits, const Problem &p, uint8_t *idx, int *zero_ptr,
                                 int zero_n, cudaStream_t s);
cudaError_t launch_loss_fast(const float *logits, const uint8_t *idx, const int *D, const Problem &p,
                             int gate, float d_scale, float grad_scale, float *loss,
                             long long *origin_do, float *dlogits, double *partials, int *done,
                             int *status, cudaStream_t s);

// ---------------------------------------------------------------- device helpers

__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

}  // namespace dol
