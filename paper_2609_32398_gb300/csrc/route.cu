// Routing outputs (Sec. 3.1.1): the router keeps, of each token's normalized
// probabilities, only the K chosen ones and re-normalizes them; these weigh
// the chosen experts' outputs.  The selection pass that builds the signatures
// writes the chosen experts and those weights (the kRoute instantiations of
// the kernel in sig_fast.cuh, or the generic kernel); this file launches them
// and holds the two dispatch kernels, which put the routed (token, choice)
// pairs in expert order:
//   offsets[e] = n_0 + ... + n_{e-1}, offsets[E] = T k
//   rows[offsets[e] + r] = the r-th token (ascending) routed to expert e
//   pos[t][q] = the row of the pair (t, q), so rows[pos[t][q]] = t.
// The rank of token t among expert e's tokens is the number of set bits of
// the signature F_e before position t: a prefix count over the signature
// words, so the order is exact and independent of scheduling.
#include "sig_fast.cuh"

namespace dol {
namespace {

constexpr int kScanThreads = 256;
constexpr int kScanWarps = kScanThreads / 32;
constexpr int kScatterThreads = 256;
constexpr int kMaxChunkWords = 32;
constexpr int kBatch = 8;  // independent global loads a scatter thread keeps in flight

// Kernel 1, one CTA per (expert e, problem): n_e and, for every chunk of
// C = 2^lc signature words, the first row of e's tokens in that chunk counted
// from the start of e's rows:
//   chunk_base[c] = set bits of F_e in chunks 0 .. c-1,   totals[e] = n_e.
// A thread sums its chunk's population counts; a block-wide exclusive scan
// over the chunks of a pass (kScanThreads chunks) and the running total of
// the passes before it give the bases.  Only the signatures are read, so the
// dispatch order can be built as soon as the selection is done.
__global__ void __launch_bounds__(kScanThreads)
route_scan_kernel(const uint32_t *__restrict__ bits, int E, int64_t W, int lc, int64_t nchunks,
                  int *__restrict__ chunk_base, int *__restrict__ totals, int *__restrict__ n_zero,
                  int *__restrict__ counts_out) {
    __shared__ int s_warp[kScanWarps];
    const int e = blockIdx.x, layer = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, wp = tid >> 5;
    const int C = 1 << lc;
    const uint32_t *be = bits + ((size_t)layer * E + e) * W;
    // population count of chunk c of F_e, its loads all in flight at once
    auto chunk_count = [&](int64_t c) {
        uint32_t v[kMaxChunkWords];
        const int64_t wa = c << lc;
#pragma unroll
        for (int j = 0; j < kMaxChunkWords; ++j)
            v[j] = (c < nchunks && j < C && wa + j < W) ? __ldg(be + wa + j) : 0u;
        int n = 0;
#pragma unroll
        for (int j = 0; j < kMaxChunkWords; ++j) n += __popc(v[j]);
        return n;
    };
    // the signatures come from the kernel before this one
    pdl_wait();
    pdl_trigger();
    // an accumulator the kernels before this one have read, cleared for the next call
    if (n_zero && tid == 0) n_zero[(size_t)layer * E + e] = 0;
    int run = 0;
    int *cb = chunk_base + ((size_t)layer * E + e) * nchunks;
    for (int64_t c0 = 0; c0 < nchunks; c0 += kScanThreads) {
        const int64_t c = c0 + tid;
        const int n = chunk_count(c);
        int x = n;  // inclusive scan inside the warp
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, x, o);
            if (lane >= o) x += y;
        }
        __syncthreads();  // s_warp is free again
        if (lane == 31) s_warp[wp] = x;
        __syncthreads();
        int before = 0, total = 0;
#pragma unroll
        for (int q = 0; q < kScanWarps; ++q) {
            const int v = s_warp[q];
            before += q < wp ? v : 0;
            total += v;
        }
        if (c < nchunks) cb[c] = run + before + x - n;
        run += total;
    }
    if (tid == 0) {
        totals[(size_t)layer * E + e] = run;
        if (counts_out) counts_out[(size_t)layer * E + e] = run;   // n_e = |F_e|
    }
}

// Kernel 2, one CTA per (chunk of C = 2^lc signature words = 32 C tokens,
// problem): the chunk's words of every expert and their exclusive prefix
// counts inside the chunk go to shared memory.  Then
//   rows: a thread per (expert e, word) writes the word's tokens, ascending,
//         from row chunk_base[e][c] + (set bits of F_e in the chunk before
//         the word) on (runs of consecutive rows per expert);
//   pos:  the routed pairs (t, q) of the chunk are read from ids in order and
//         each gets r = chunk_base[e][c] + (set bits of F_e in the chunk
//         before t), written to pos[t][q] in order.
// Indices inside a problem fit int32 (T k <= INT32_MAX); lk = log2 k when k
// is a power of two (the pair index is then split by a shift), else -1.
__global__ void __launch_bounds__(kScatterThreads)
route_scatter_kernel(const uint32_t *__restrict__ bits, const int *__restrict__ ids,
                     const int *__restrict__ chunk_base, const int *__restrict__ totals, int T,
                     int E, int k, int lk, int64_t W, int lc, int64_t nchunks,
                     int *__restrict__ offsets, int *__restrict__ rows, int *__restrict__ pos) {
    extern __shared__ int smem_i[];
    const int C = 1 << lc, EC = E << lc;
    uint32_t *s_bits = reinterpret_cast<uint32_t *>(smem_i);  // [E][C]
    int *s_pre = smem_i + EC;                                 // [E][C]
    int *s_cb = s_pre + EC;                                   // [E]
    const int64_t c = blockIdx.x;
    const int layer = blockIdx.y;
    const int tid = threadIdx.x;
    pdl_wait();
    const int64_t w0 = c << lc;
    const int nw = (int)min64(C, W - w0);
    const int Tk = T * k;
    const int i0 = (int)(32 * w0) * k, i1 = (int)min64(T, 32 * (w0 + nw)) * k;
    const int *il = ids + (size_t)layer * Tk;
    // this thread's experts' totals and chunk bases (at most four consecutive
    // experts per thread, E <= 1024), loaded with everything else up front so
    // that the kernel waits for one round trip of loads, not three
    const int per = (E + kScatterThreads - 1) / kScatterThreads;
    int tot_v[4], cb_v[4];
    {
        const int *tl = totals + (size_t)layer * E;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e = tid * per + j;
            const bool on = j < per && e < E;
            tot_v[j] = on ? __ldg(tl + e) : 0;
            cb_v[j] = on ? __ldg(chunk_base + ((size_t)layer * E + e) * nchunks + c) : 0;
        }
    }
    // the first batch of this thread's expert ids: loaded before the barriers
    // below, so that its latency overlaps the shared-memory set-up
    int ev[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
        const int i = i0 + tid + u * kScatterThreads;
        ev[u] = (pos && i < i1) ? __ldg(il + i) : -1;
    }
    const uint32_t *bl = bits + (size_t)layer * E * W;
    for (int m0 = tid; m0 < EC; m0 += kScatterThreads * kBatch) {
        uint32_t v[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int i = m0 + u * kScatterThreads;
            const int e = i >> lc, j = i & (C - 1);
            v[u] = (i < EC && j < nw) ? __ldg(bl + (size_t)e * W + w0 + j) : 0u;
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int i = m0 + u * kScatterThreads;
            if (i < EC) s_bits[i] = v[u];
        }
    }
    // first row of every expert: an exclusive scan of the totals (E <= 1024,
    // at most four consecutive experts per thread)
    {
        __shared__ int s_wsum[kScatterThreads / 32];
        const int lane = tid & 31, wp = tid >> 5;
        int loc[4], sum = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            loc[j] = sum;
            sum += tot_v[j];
        }
        int x = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) s_wsum[wp] = x;
        __syncthreads();
        int before = 0, all = 0;
#pragma unroll
        for (int q = 0; q < kScatterThreads / 32; ++q) {
            before += q < wp ? s_wsum[q] : 0;
            all += s_wsum[q];
        }
        const int excl = before + x - sum;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e = tid * per + j;
            if (j < per && e < E) {
                s_cb[e] = excl + loc[j] + cb_v[j];
                if (offsets && c == 0) offsets[(size_t)layer * (E + 1) + e] = excl + loc[j];
            }
        }
        if (offsets && c == 0 && tid == 0) offsets[(size_t)layer * (E + 1) + E] = all;
    }
    __syncthreads();
    if (!rows && !pos) return;
    for (int e = tid; e < E; e += kScatterThreads) {
        int acc = 0;
        for (int j = 0; j < C; ++j) {
            s_pre[(e << lc) + j] = acc;
            acc += __popc(s_bits[(e << lc) + j]);
        }
    }
    __syncthreads();
    if (rows) {
        int *rl = rows + (size_t)layer * Tk;
        for (int i = tid; i < EC; i += kScatterThreads) {
            uint32_t b = s_bits[i];
            int r = s_cb[i >> lc] + s_pre[i];
            const int tb = (int)(32 * (w0 + (i & (C - 1))));
            while (b) {
                const int bit = __ffs(b) - 1;
                b &= b - 1;
                // bits past T are zero and the rows of an expert end before the
                // next expert's when the signatures and counts come from one
                // complete selection; after an aborted one (a timed-out wait,
                // reported in the status word) they may not: stay in bounds
                if (r >= 0 && r < Tk) rl[r] = tb + bit;
                ++r;
            }
        }
    }
    if (!pos) return;
    int *pl = pos + (size_t)layer * Tk;
    for (int ib = i0 + tid; ib < i1; ib += kScatterThreads * kBatch) {
        if (ib != i0 + tid) {
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int i = ib + u * kScatterThreads;
                ev[u] = i < i1 ? __ldg(il + i) : -1;
            }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int i = ib + u * kScatterThreads;
            const int e = ev[u];
            // ids from an aborted selection may hold anything: stay in bounds
            if (i >= i1 || (unsigned)e >= (unsigned)E) continue;
            const int t = lk >= 0 ? (i >> lk) : i / k;
            const int sj = (e << lc) + (t >> 5) - (int)w0;
            pl[i] = s_cb[e] + s_pre[sj] + __popc(s_bits[sj] & ((1u << (t & 31)) - 1u));
        }
    }
}

}  // namespace

cudaError_t launch_signatures_fast_routed(const float *logits, const Problem &p, uint32_t *bits,
                                          int *counts, uint8_t *idx, uint32_t *cooc,
                                          const ZeroSpans &zero, int *status,
                                          const RouteOut &route, cudaStream_t s) {
    CUtensorMap map;
    if (!encode_tensor_map_2d_f32(&map, logits, (uint64_t)p.L * p.T, (uint64_t)p.E, 32))
        return cudaErrorInvalidValue;
    if (p.E == 32) return dispatch_mode<32, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    if (p.E == 64) return dispatch_mode<64, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    return dispatch_mode<128, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
}

// Signature words per dispatch chunk: a power of two with about 2048 routed
// pairs per chunk (32 C k), at most kMaxChunkWords, and the chunk's words of
// all experts (E C) within 4096 words of shared memory.
int route_chunk_words(const Problem &p) {
    int lim = 64 / p.k;
    if (lim > kMaxChunkWords) lim = kMaxChunkWords;
    if (lim > 4096 / p.E) lim = 4096 / p.E;
    int c = 1;
    while (2 * c <= lim) c *= 2;
    return c;
}

int64_t route_chunks(const Problem &p) {
    const int C = route_chunk_words(p);
    return (p.W + C - 1) / C;
}

cudaError_t launch_route_dispatch(const uint32_t *bits, const int *ids, const Problem &p,
                                  int *offsets, int *rows, int *pos, int *scratch,
                                  cudaStream_t s, int *n_zero, int *counts_out) {
    if (!offsets && !rows && !pos && !counts_out)
        return n_zero ? cudaMemsetAsync(n_zero, 0, sizeof(int) * (size_t)p.L * p.E, s) : cudaSuccess;
    const int C = route_chunk_words(p);
    int lc = 0;
    while ((1 << lc) < C) ++lc;
    const int64_t nchunks = route_chunks(p);
    int *chunk_base = scratch;
    int *totals = scratch + (size_t)p.L * p.E * nchunks;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)p.E, (unsigned)p.L);
    cfg.blockDim = dim3(kScanThreads);
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, route_scan_kernel, bits, p.E, p.W, lc, nchunks,
                                       chunk_base, totals, n_zero, counts_out);
    if (e != cudaSuccess) return e;
    if (!offsets && !rows && !pos) return cudaSuccess;
    cfg.gridDim = dim3((unsigned)nchunks, (unsigned)p.L);
    cfg.blockDim = dim3(kScatterThreads);
    cfg.dynamicSmemBytes = sizeof(int) * (size_t)(2 * p.E * C + p.E);
    const int lk = (p.k & (p.k - 1)) == 0 ? __builtin_ctz((unsigned)p.k) : -1;
    return cudaLaunchKernelEx(&cfg, route_scatter_kernel, bits, ids, (const int *)chunk_base,
                              (const int *)totals, (int)p.T, p.E, p.k, lk, p.W, lc, nchunks,
                              offsets, rows, pos);
}

int64_t route_scratch_ints(const Problem &p) { return (int64_t)p.L * p.E * (route_chunks(p) + 1); }

}  // namespace dol
