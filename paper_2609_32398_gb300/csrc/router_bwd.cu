// Backward of the router's linear map (Sec. 4.1: hidden size H to the E
// experts, no bias) for the gradient dz of the logits that the loss step
// writes (dlogits):
//   dW[l][e][h] = sum_t dz[l][t][e] X[l][t][h]     fp32
//   dX[l][t][h] = sum_e dz[l][t][e] W[l][e][h]     bf16 (optional)
// Both are plain matrix products with the reduction index outermost in
// memory.  This file's kernel rounds dz to bf16 (round to nearest even); the
// products run in cuBLAS with bf16 inputs and fp32 accumulation.  cuBLAS is
// opened at run time, so the library has no link-time dependency on it; the
// entry point reports DO_ERR_UNSUPPORTED where it cannot be opened.
#include <cuda_bf16.h>
#include <cublas_api.h>
#include <dlfcn.h>

#include <cstdint>
#include <mutex>

#include "dol_internal.cuh"
#include "doloss.h"

namespace dol {
namespace {

constexpr size_t kCublasWorkspace = (size_t)32 << 20;

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

using CreateFn = cublasStatus_t (*)(cublasHandle_t *);
using SetStreamFn = cublasStatus_t (*)(cublasHandle_t, cudaStream_t);
using SetWorkspaceFn = cublasStatus_t (*)(cublasHandle_t, void *, size_t);
using GemmFn = cublasStatus_t (*)(cublasHandle_t, cublasOperation_t, cublasOperation_t, int, int,
                                  int, const void *, const void *, cudaDataType, int, long long,
                                  const void *, cudaDataType, int, long long, const void *, void *,
                                  cudaDataType, int, long long, int, cublasComputeType_t,
                                  cublasGemmAlgo_t);

struct Cublas {
    bool ok = false;
    CreateFn create = nullptr;
    SetStreamFn set_stream = nullptr;
    SetWorkspaceFn set_workspace = nullptr;
    GemmFn gemm = nullptr;
    cublasHandle_t handle[64] = {};
    std::mutex mu;
};

Cublas &cublas() {
    static Cublas c;
    static std::once_flag once;
    std::call_once(once, [] {
        const char *names[] = {"libcublas.so.13", "libcublas.so", "/usr/local/cuda/lib64/libcublas.so.13"};
        void *h = nullptr;
        for (const char *n : names)
            if ((h = dlopen(n, RTLD_NOW | RTLD_GLOBAL)) != nullptr) break;
        if (!h) return;
        c.create = reinterpret_cast<CreateFn>(dlsym(h, "cublasCreate_v2"));
        c.set_stream = reinterpret_cast<SetStreamFn>(dlsym(h, "cublasSetStream_v2"));
        c.set_workspace = reinterpret_cast<SetWorkspaceFn>(dlsym(h, "cublasSetWorkspace_v2"));
        c.gemm = reinterpret_cast<GemmFn>(dlsym(h, "cublasGemmStridedBatchedEx"));
        c.ok = c.create && c.set_stream && c.set_workspace && c.gemm;
    });
    return c;
}

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace
}  // namespace dol

extern "C" {

size_t do_router_backward_workspace_size(int64_t T, int32_t E, int32_t H, int32_t L) {
    if (T < 1 || E < 1 || H < 1 || L < 1) return 0;
    return dol::round256(sizeof(uint16_t) * (size_t)L * (size_t)T * (size_t)E) + dol::kCublasWorkspace;
}

do_status do_router_backward(const void *X, const void *Wr, const float *dlogits, int64_t T,
                             int32_t H, int32_t E, int32_t L, float *dW, void *dX,
                             void *workspace, size_t workspace_bytes, void *stream) {
    if (T < 1 || E < 1 || H < 1 || L < 1) return DO_ERR_INVALID_ARG;
    if (T > (int64_t)INT32_MAX || (int64_t)E * H > (int64_t)INT32_MAX) return DO_ERR_UNSUPPORTED;
    if (!X || !Wr || !dlogits || !dW) return DO_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(Wr) |
         reinterpret_cast<uintptr_t>(dlogits) | reinterpret_cast<uintptr_t>(dW) |
         reinterpret_cast<uintptr_t>(dX)) % 16)
        return DO_ERR_INVALID_ARG;
    const size_t need = do_router_backward_workspace_size(T, E, H, L);
    if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 256 || workspace_bytes < need)
        return DO_ERR_WORKSPACE;
    dol::Cublas &cb = dol::cublas();
    if (!cb.ok) return DO_ERR_UNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return DO_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    char *ws = static_cast<char *>(workspace);
    __nv_bfloat16 *dzb = reinterpret_cast<__nv_bfloat16 *>(ws);
    void *cws = ws + dol::round256(sizeof(uint16_t) * (size_t)L * (size_t)T * (size_t)E);
    const int64_t n = (int64_t)L * T * E;
    dol::to_bf16_kernel<<<1024, 256, 0, s>>>(dlogits, dzb, n);
    if (cudaGetLastError() != cudaSuccess) return DO_ERR_CUDA;
    std::lock_guard<std::mutex> lock(cb.mu);  // the handle's stream and workspace are per call
    if (!cb.handle[dev] && cb.create(&cb.handle[dev]) != CUBLAS_STATUS_SUCCESS) {
        cb.handle[dev] = nullptr;
        return DO_ERR_CUDA;
    }
    cublasHandle_t h = cb.handle[dev];
    if (cb.set_stream(h, s) != CUBLAS_STATUS_SUCCESS ||
        cb.set_workspace(h, cws, dol::kCublasWorkspace) != CUBLAS_STATUS_SUCCESS)
        return DO_ERR_CUDA;
    const float one = 1.0f, zero = 0.0f;
    const int t = (int)T;
    // Column-major views: X [T][H] is (H x T), dz [T][E] is (E x T), W [E][H]
    // is (H x E).  dW^T (H x E) = X^T dz = (H x T)(E x T)^T; it is dW [E][H].
    cublasStatus_t st = cb.gemm(h, CUBLAS_OP_N, CUBLAS_OP_T, H, E, t, &one, X, CUDA_R_16BF, H,
                                (long long)T * H, dzb, CUDA_R_16BF, E, (long long)T * E, &zero, dW,
                                CUDA_R_32F, H, (long long)E * H, L, CUBLAS_COMPUTE_32F,
                                CUBLAS_GEMM_DEFAULT);
    if (st != CUBLAS_STATUS_SUCCESS) return DO_ERR_CUDA;
    if (dX) {
        // dX^T (H x T) = W^T dz^T = (H x E)(E x T); it is dX [T][H].
        st = cb.gemm(h, CUBLAS_OP_N, CUBLAS_OP_N, H, t, E, &one, Wr, CUDA_R_16BF, H,
                     (long long)E * H, dzb, CUDA_R_16BF, E, (long long)T * E, &zero, dX,
                     CUDA_R_16BF, H, (long long)T * H, L, CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT);
        if (st != CUBLAS_STATUS_SUCCESS) return DO_ERR_CUDA;
    }
    return DO_OK;
}

}  // extern "C"
