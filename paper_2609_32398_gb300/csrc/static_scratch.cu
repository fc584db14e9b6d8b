// do_forward_backward_static (declared in include/doloss.h): the fused path
// of do_forward_backward with its workspace taken from a fixed device array
// inside libdoloss instead of from the caller.
//
// It serves callers that cannot allocate device memory at call time: a plain C
// host that embeds the library without any device allocator of its own, or a
// serving process that hands all spare HBM to its own pool at start-up and
// forbids cudaMalloc afterwards (an allocation there would fail or fragment
// the pool).  Nothing here calls cudaMalloc, cudaFree or an allocating library.
//
// The scratch is one array per device (one per CUDA context), so calls that
// overlap in time — on two streams, or from two host threads — share it and
// race; such callers must serialize their calls on one stream.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <mutex>

#include "dol_internal.cuh"
#include "doloss.h"

namespace {

constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[DO_STATIC_SCRATCH_BYTES];

// The driver's current-context queries, reached through the runtime (the
// library links no -lcuda).
struct CtxFns {
    PFN_cuCtxGetCurrent_v4000 current = nullptr;
    PFN_cuCtxGetId_v12000 id = nullptr;
};

const CtxFns &ctx_fns() {
    static CtxFns f;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            f.current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            f.id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
    });
    return f;
}

// Identifier of the current context (unique for the life of the process,
// never reused), 0 if none is current or the query is unavailable.
unsigned long long current_ctx_id() {
    const CtxFns &f = ctx_fns();
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (f.current && f.id && f.current(&ctx) == CUDA_SUCCESS && ctx && f.id(ctx, &id) == CUDA_SUCCESS)
        return id;
    return 0;
}

std::mutex g_mu;
struct Cached {
    unsigned long long ctx;
    void *ptr;
};
Cached g_cache[kMaxDevices] = {};

// Device address of the scratch array in the current context.  In host code
// the name g_scratch stands for a host-side shadow, not a device address, so
// the address is looked up with cudaGetSymbolAddress, with the device current.
// The lookup is cached per device and keyed by the context's identifier: a
// context created after cudaDeviceReset (or after the primary context was
// released) holds a new copy of the module, and its first call looks up the
// address again.  The first call in a context therefore does this set-up; it
// should come before any stream capture begins.
do_status scratch_on_current_device(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DO_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return DO_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    const unsigned long long ctx = current_ctx_id();
    if (ctx != 0 && g_cache[dev].ctx == ctx && g_cache[dev].ptr) {
        *out = g_cache[dev].ptr;
        return DO_OK;
    }
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) return DO_ERR_CUDA;
    // the lookup makes the device's primary context current if none was
    g_cache[dev].ctx = ctx != 0 ? ctx : current_ctx_id();
    g_cache[dev].ptr = p;
    *out = p;
    return DO_OK;
}

}  // namespace

extern "C" do_status do_forward_backward_static(const float *logits, int64_t T, int32_t E,
                                                int32_t k, int32_t L, int32_t gate,
                                                float grad_scale, uint32_t *bits, int32_t *counts,
                                                int32_t *D, float *loss, int64_t *origin_do,
                                                float *dlogits, int32_t *status_flags,
                                                void *stream) {
    // the sizes are checked by do_workspace_size (0 = invalid) before anything else
    if (do_workspace_size(T, E, k, L) == 0) {
        if (T < 1 || E < 1 || k < 1 || k > E || L < 1) return DO_ERR_INVALID_ARG;
        return DO_ERR_UNSUPPORTED;
    }
    dol::Problem p;
    p.T = T;
    p.E = E;
    p.k = k;
    p.L = L;
    p.W = (T + 31) / 32;
    // no routing outputs here: the layout up to the routing scratch
    if (dol::workspace_bytes_plain(p) > DO_STATIC_SCRATCH_BYTES) return DO_ERR_WORKSPACE;
    if (!logits || !bits || !counts || !D || !loss) return DO_ERR_INVALID_ARG;
    if (status_flags && reinterpret_cast<uintptr_t>(status_flags) % 4 != 0)
        return DO_ERR_INVALID_ARG;
    void *ws = nullptr;
    do_status st = scratch_on_current_device(&ws);
    if (st != DO_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // What must be zero when a call starts: the status word and the done
    // counters (the first 256-byte-aligned span) and the counts accumulator
    // [n_acc, bimg).  The kernels leave them zero after a complete call;
    // clearing them here also recovers from a call that gave up on a wait.
    // Everything else in the array is written before it is read (the image
    // of D' at bimg by the reduction kernel, every entry of it).
    const dol::WsLayout w = dol::ws_layout(p);
    char *base = static_cast<char *>(ws);
    if (cudaMemsetAsync(base, 0, w.partials, s) != cudaSuccess) return DO_ERR_CUDA;
    if (w.bimg > w.n_acc && cudaMemsetAsync(base + w.n_acc, 0, w.bimg - w.n_acc, s) != cudaSuccess)
        return DO_ERR_CUDA;
    st = do_forward_backward(logits, T, E, k, L, gate, grad_scale, bits, counts, D, loss, origin_do,
                             dlogits, ws, DO_STATIC_SCRATCH_BYTES, stream);
    if (st != DO_OK) return st;
    if (status_flags &&
        cudaMemcpyAsync(status_flags, base, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) !=
            cudaSuccess)
        return DO_ERR_CUDA;
    return DO_OK;
}
