// Step 1, fast path: the launchers of the Top-K signature kernel (the kernel
// itself is in sig_fast.cuh) without routing outputs.
#include "sig_fast.cuh"

namespace dol {
namespace {

int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 148;
    return n;
}

}  // namespace

int sig_fast_ctas_per_problem(const Problem &p) {
    int sms = sm_count();
    if (sms > kMaxSigCtas) sms = kMaxSigCtas;
    int64_t gx = sms / p.L;
    if (gx > p.W) gx = p.W;
    if (gx < 1) gx = 1;
    return (int)gx;
}

size_t cooc_partial_words(int E) {
    return E == 32 ? SigCfg<32>::kCoocWords : E == 64 ? SigCfg<64>::kCoocWords : SigCfg<128>::kCoocWords;
}

bool signatures_fast_supported(const float *logits, const Problem &p) {
    const bool e_ok = p.E == 32 || p.E == 64 || p.E == 128;
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    return e_ok && k_ok && (reinterpret_cast<uintptr_t>(logits) % 16 == 0) &&
           (int64_t)p.L * p.T + 32 < (int64_t)INT_MAX;
}

cudaError_t launch_signatures_fast(const float *logits, const Problem &p, uint32_t *bits,
                                   int *counts, uint8_t *idx, uint32_t *cooc, const ZeroSpans &zero,
                                   int *status, cudaStream_t s) {
    CUtensorMap map;
    if (!encode_tensor_map_2d_f32(&map, logits, (uint64_t)p.L * p.T, (uint64_t)p.E, 32))
        return cudaErrorInvalidValue;
    const RouteOut none = {nullptr, nullptr, 0};
    if (p.E == 32) return dispatch_mode<32, false>(map, p, bits, counts, idx, cooc, zero, status, none, s);
    if (p.E == 64) return dispatch_mode<64, false>(map, p, bits, counts, idx, cooc, zero, status, none, s);
    return dispatch_mode<128, false>(map, p, bits, counts, idx, cooc, zero, status, none, s);
}

bool signatures_fast256_supported(const float *logits, const Problem &p) {
    const bool k_ok = p.k == 1 || p.k == 2 || p.k == 4 || p.k == 8;
    return p.E == 256 && k_ok && (reinterpret_cast<uintptr_t>(logits) % 16 == 0) &&
           (int64_t)p.L * p.T + 32 < (int64_t)INT_MAX;
}

cudaError_t launch_signatures_fast256(const float *logits, const Problem &p, uint32_t *bits,
                                      int *counts, uint8_t *idx, const ZeroSpans &zero,
                                      int *status, cudaStream_t s) {
    CUtensorMap map;
    if (!encode_tensor_map_2d_f32(&map, logits, (uint64_t)p.L * p.T, (uint64_t)p.E, 32))
        return cudaErrorInvalidValue;
    const RouteOut none = {nullptr, nullptr, 0};
    return dispatch_k<256, true, false, false>(map, p, bits, counts, idx, nullptr, zero, status,
                                               none, s);
}

}  // namespace dol
