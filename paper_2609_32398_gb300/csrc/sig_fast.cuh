// Step 1, fast path (E in {32, 64, 128, 256}, k in {1, 2, 4, 8}, 16-byte
// aligned logits; at E = 256 without the co-occurrence counts): Top-K
// signatures (Sec. 3.1.1, Eq. 1) with one token per lane.
//
// A persistent CTA per SM owns a contiguous range of 32-token tiles.  One
// producer warp streams each tile [32 tokens x E] into a ring of shared
// memory slots with 2-D TMA loads (32 x 32 fp32 boxes, 128-byte swizzle, so
// a lane reading its own row is bank-conflict free); eight consumer warps
// take the tiles in turn, each lane selecting the Top-K of its token:
//   1. the row is cut into NG groups of GS consecutive experts and each
//      group's maximum is kept in registers;
//   2. K times: a tournament over the group maxima (ties to the lower group)
//      picks a group, the first element equal to its maximum is selected
//      (lowest index among equal values), overwritten with -inf in shared
//      memory, and the group maximum is recomputed.
// Each lane sets its token's bit in the words of its K chosen experts with
// shared-memory atomic ORs into a per-warp scratch of E words, from which
// lane c stores the words of experts c, c + 32, ... (the router kernel, whose
// shared memory is full, builds the same words by 32x32 bit transposes).
// The k selected indices of every token are also written (one byte each) for
// the loss kernel, and the CTAs zero the accumulators of the next kernels.
// The routing instantiations (kRoute) also write, per token, the chosen
// experts in selection order and their re-normalized combine weights
// (Sec. 3.1.1) from the logits the extraction already holds.
//
// This header holds the kernel template; sig_fast.cu instantiates the plain
// variants and route.cu the routing ones (two translation units, compiled in
// parallel).
#pragma once

#include <climits>

#include "dol_internal.cuh"
#include "tma.cuh"

namespace dol {
namespace {

constexpr int kConsumers = 8;
constexpr int kFastThreads = (kConsumers + 1) * 32;
constexpr int kBoxBytes = 32 * 128;  // 32 rows x 32 fp32

template <int E>
struct SigCfg {
    static constexpr int kBoxes = E / 32;
    static constexpr int kTileBytes = kBoxes * kBoxBytes;
    static constexpr int kSlots = (E == 256) ? 6 : (E == 128) ? 11 : 16;
    static constexpr int GS = (E >= 128) ? E / 16 : 4;  // experts per group
    static constexpr int NG = E / GS;                    // groups per row
    // co-occurrence counters: row a holds columns (a & ~3) .. E-1 (E <= 128;
    // at E = 256 the kernel runs without them)
    static constexpr int kCoocWords = E <= 128 ? cooc_row_offset<E>(E) : 0;
    static constexpr size_t kSmem = (size_t)kSlots * kTileBytes + 1024 + 2 * kSlots * 8 +
                                    kSlots * 4 + 32 + (size_t)kCoocWords * 4 + E * 4 +
                                    (size_t)kConsumers * E * 4;
};


// Transpose a 32x32 bit matrix held one row per lane (bit c of lane t is
// element (t, c)); on return lane c holds column c (bit t = element (t, c)).
__device__ __forceinline__ uint32_t transpose32(uint32_t x, int lane) {
    const uint32_t lo_mask[5] = {0x0000FFFFu, 0x00FF00FFu, 0x0F0F0F0Fu, 0x33333333u, 0x55555555u};
#pragma unroll
    for (int s = 0; s < 5; ++s) {
        const int j = 16 >> s;
        const uint32_t lo = lo_mask[s];
        const uint32_t p = __shfl_xor_sync(kFull, x, j);
        x = (lane & j) ? ((x & ~lo) | ((p >> j) & lo)) : ((x & lo) | ((p << j) & ~lo));
    }
    return x;
}

// Byte address of float4 chunk e4 of this lane's row inside a swizzled tile.
__device__ __forceinline__ unsigned char *chunk_ptr(unsigned char *tile, int e4, int lane) {
    return tile + (e4 >> 3) * kBoxBytes + lane * 128 + ((((e4 & 7) ^ (lane & 7))) << 4);
}

template <int K>
__device__ __forceinline__ void store_idx(uint8_t *p, const int (&sel)[K]) {
    if (K == 8) {
        uint2 v;
        v.x = (uint32_t)sel[0] | ((uint32_t)sel[1 % K] << 8) | ((uint32_t)sel[2 % K] << 16) |
              ((uint32_t)sel[3 % K] << 24);
        v.y = (uint32_t)sel[4 % K] | ((uint32_t)sel[5 % K] << 8) | ((uint32_t)sel[6 % K] << 16) |
              ((uint32_t)sel[7 % K] << 24);
        *reinterpret_cast<uint2 *>(p) = v;
    } else if (K == 4) {
        *reinterpret_cast<uint32_t *>(p) = (uint32_t)sel[0] | ((uint32_t)sel[1 % K] << 8) |
                                           ((uint32_t)sel[2 % K] << 16) |
                                           ((uint32_t)sel[3 % K] << 24);
    } else if (K == 2) {
        *reinterpret_cast<uint16_t *>(p) = (uint16_t)((uint32_t)sel[0] | ((uint32_t)sel[1 % K] << 8));
    } else {
        *p = (uint8_t)sel[0];
    }
}

// Chosen experts and their re-normalized weights of one token (kRoute):
// w_q = u_q / sum_q' u_q', u from route_raw_weight, summed in selection order.
template <int K>
__device__ __forceinline__ void store_route(const RouteOut &r, int64_t off, const int (&sel)[K],
                                            const float (&val)[K]) {
    float w[K];
    float sum = 0.0f;
#pragma unroll
    for (int q = 0; q < K; ++q) {
        w[q] = route_raw_weight(val[q], val[0], r.gate);
        sum += w[q];
    }
#pragma unroll
    for (int q = 0; q < K; ++q) w[q] = w[q] / sum;
    if constexpr (K >= 4) {
#pragma unroll
        for (int q = 0; q < K; q += 4) {
            *reinterpret_cast<int4 *>(r.ids + off + q) = make_int4(sel[q], sel[q + 1], sel[q + 2], sel[q + 3]);
            *reinterpret_cast<float4 *>(r.combine + off + q) = make_float4(w[q], w[q + 1], w[q + 2], w[q + 3]);
        }
    } else if constexpr (K == 2) {
        *reinterpret_cast<int2 *>(r.ids + off) = make_int2(sel[0], sel[1]);
        *reinterpret_cast<float2 *>(r.combine + off) = make_float2(w[0], w[1]);
    } else {
        r.ids[off] = sel[0];
        r.combine[off] = w[0];
    }
}

// Top-K of the token held by this lane in a swizzled 32-token tile (the layout
// of chunk_ptr): the row is cut into NG groups of GS experts whose maxima are
// kept in registers; K times a tournament over the group maxima (ties to the
// lower group) picks a group, the first element equal to its maximum is chosen
// (lowest index among equal values), overwritten with -inf in the tile, and
// the group maximum recomputed.  sel: the chosen experts in selection order;
// val: their logits.
// kMask: chosen experts are excluded through a per-lane bit mask instead of
// -inf writes, so the tile is only read (it may be in flight to HBM meanwhile).
template <int E, int K, bool kMask = false>
__device__ __forceinline__ void select_topk(unsigned char *tp, int lane, int (&sel)[K],
                                            float (&val)[K]) {
    constexpr int GS = SigCfg<E>::GS, NG = SigCfg<E>::NG, GS4 = GS / 4;
    uint32_t chosen[E / 32];
#pragma unroll
    for (int r = 0; r < E / 32; ++r) chosen[r] = 0u;
    float g[NG];
#pragma unroll
    for (int gi = 0; gi < NG; ++gi) {
        float m = -INFINITY;
#pragma unroll
        for (int c = 0; c < GS4; ++c) {
            const float4 v = *reinterpret_cast<const float4 *>(chunk_ptr(tp, gi * GS4 + c, lane));
            m = fmaxf(m, fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)));
        }
        g[gi] = m;
    }
#pragma unroll
    for (int qk = 0; qk < K; ++qk) {
        float tv[NG];
        int ti[NG];
#pragma unroll
        for (int j = 0; j < NG / 2; ++j) {
            const bool right = g[2 * j + 1] > g[2 * j];
            tv[j] = right ? g[2 * j + 1] : g[2 * j];
            ti[j] = right ? 2 * j + 1 : 2 * j;
        }
#pragma unroll
        for (int nn = NG / 2; nn > 1; nn >>= 1) {
#pragma unroll
            for (int j = 0; j < nn / 2; ++j) {
                const bool right = tv[2 * j + 1] > tv[2 * j];
                tv[j] = right ? tv[2 * j + 1] : tv[2 * j];
                ti[j] = right ? ti[2 * j + 1] : ti[2 * j];
            }
        }
        const float bv = tv[0];
        const int bi = ti[0];
        float x[GS];
#pragma unroll
        for (int c = 0; c < GS4; ++c) {
            const float4 v = *reinterpret_cast<const float4 *>(chunk_ptr(tp, bi * GS4 + c, lane));
            x[4 * c] = v.x;
            x[4 * c + 1] = v.y;
            x[4 * c + 2] = v.z;
            x[4 * c + 3] = v.w;
        }
        if (kMask) {  // the experts of this group chosen before
            uint32_t word = 0u;
#pragma unroll
            for (int r = 0; r < E / 32; ++r) word = ((bi * GS) >> 5) == r ? chosen[r] : word;
            const uint32_t gm = (word >> ((bi * GS) & 31)) & ((1u << GS) - 1u);
#pragma unroll
            for (int j = 0; j < GS; ++j) x[j] = ((gm >> j) & 1u) ? -INFINITY : x[j];
        }
        int p = GS - 1;
#pragma unroll
        for (int j = GS - 1; j >= 0; --j)
            if (x[j] == bv) p = j;
        float m2 = -INFINITY;
#pragma unroll
        for (int j = 0; j < GS; ++j) m2 = fmaxf(m2, j == p ? -INFINITY : x[j]);
        const int e = bi * GS + p;
        if (kMask) {
#pragma unroll
            for (int r = 0; r < E / 32; ++r) chosen[r] |= (e >> 5) == r ? 1u << (e & 31) : 0u;
        } else {
            reinterpret_cast<float *>(chunk_ptr(tp, e >> 2, lane))[e & 3] = -INFINITY;
        }
#pragma unroll
        for (int gi = 0; gi < NG; ++gi) g[gi] = (gi == bi) ? m2 : g[gi];
        sel[qk] = e;
        val[qk] = bv;
    }
}

// Batcher's odd-even merge sort of K indices (K in {1, 2, 4, 8}) in registers.
template <int K>
__device__ __forceinline__ void sort_small(int (&so)[K]) {
    auto cx = [&](int i, int j) {
        const int lo = min(so[i], so[j]), hi = max(so[i], so[j]);
        so[i] = lo;
        so[j] = hi;
    };
    if constexpr (K == 2) {
        cx(0, 1);
    } else if constexpr (K == 4) {
        cx(0, 1); cx(2, 3); cx(0, 2); cx(1, 3); cx(1, 2);
    } else if constexpr (K == 8) {
        cx(0, 1); cx(2, 3); cx(4, 5); cx(6, 7);
        cx(0, 2); cx(1, 3); cx(4, 6); cx(5, 7);
        cx(1, 2); cx(5, 6);
        cx(0, 4); cx(1, 5); cx(2, 6); cx(3, 7);
        cx(2, 4); cx(3, 5);
        cx(1, 2); cx(3, 4); cx(5, 6);
    }
}

// c_ab += 1 for every pair a < b of one token's chosen experts, in a
// shared-memory triangle whose row a starts at s_rowoff[a] (the counts on the
// diagonal come from the signature words).
template <int K>
__device__ __forceinline__ void cooc_add(uint32_t *s_cooc, const int *s_rowoff, const int (&sel)[K]) {
    int so[K];
#pragma unroll
    for (int q = 0; q < K; ++q) so[q] = sel[q];
    sort_small<K>(so);
#pragma unroll
    for (int q1 = 0; q1 < K - 1; ++q1) {
        uint32_t *row = s_cooc + s_rowoff[so[q1]];
#pragma unroll
        for (int q2 = q1 + 1; q2 < K; ++q2) atomicAdd(row + so[q2], 1u);
    }
}

// The signature words of the warp's 32 tokens (lane = token): a bit per chosen
// expert, turned into one word per expert by 32x32 bit transposes; lane c
// stores the word of expert 32 r + c at words[(32 r + c) W].  With kCount,
// cnt[r] accumulates the word's population count.
template <int E, int K, bool kCount>
__device__ __forceinline__ void emit_words(const int (&sel)[K], bool valid, int lane,
                                           uint32_t *words, int64_t W, uint32_t (&cnt)[E / 32]) {
    constexpr int R = E / 32;
    uint32_t m[R];
#pragma unroll
    for (int r = 0; r < R; ++r) m[r] = 0u;
#pragma unroll
    for (int qk = 0; qk < K; ++qk) {
        const uint32_t bit = 1u << (sel[qk] & 31);
        const int rq = sel[qk] >> 5;
#pragma unroll
        for (int r = 0; r < R; ++r) m[r] |= (rq == r) ? bit : 0u;
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const uint32_t word = transpose32(valid ? m[r] : 0u, lane);
        words[(int64_t)(32 * r + lane) * W] = word;
        if (kCount) cnt[r] += __popc(word);
    }
}

// The signature words of the warp's 32 tokens (lane = token) through the
// warp's scratch s_w [E] (zero on entry and on return): every lane ORs its bit
// into the words of its chosen experts, then lane c stores the words of
// experts 32 r + c at words[(32 r + c) W].  With kCount, cnt[r] accumulates
// the word's population count.
template <int E, int K, bool kCount>
__device__ __forceinline__ void emit_words_or(const int (&sel)[K], bool valid, int lane, uint32_t *s_w,
                                              uint32_t *words, int64_t W, uint32_t (&cnt)[E / 32]) {
    if (valid) {
        const uint32_t bit = 1u << lane;
#pragma unroll
        for (int q = 0; q < K; ++q) atomicOr(s_w + sel[q], bit);
    }
    __syncwarp();
#pragma unroll
    for (int r = 0; r < E / 32; ++r) {
        const uint32_t word = s_w[32 * r + lane];
        s_w[32 * r + lane] = 0u;
        words[(int64_t)(32 * r + lane) * W] = word;
        if (kCount) cnt[r] += __popc(word);
    }
    __syncwarp();
}

template <int E, int K, bool kCounts, bool kCooc, bool kRoute>
__global__ void __launch_bounds__(kFastThreads, 1)
sig_fast_kernel(const __grid_constant__ CUtensorMap tmap, int64_t T, int64_t W,
                uint32_t *__restrict__ bits, int *__restrict__ counts, uint8_t *__restrict__ idx,
                uint32_t *__restrict__ cooc, ZeroSpans zero, int *__restrict__ status,
                RouteOut route) {
    using C = SigCfg<E>;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_align<1024>(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + (size_t)C::kSlots * C::kTileBytes);
    uint64_t *empty = full + C::kSlots;
    // slot_round[s] = the round of slot s the producer has started to load.
    // A consumer waits for it before testing the slot's phase parity: the
    // consumers of consecutive rounds of one slot are different warps, and a
    // parity test alone cannot tell round r + 1 from round r - 1.
    volatile int *slot_round = reinterpret_cast<volatile int *>(empty + C::kSlots);
    volatile int *s_abort = slot_round + C::kSlots;
    uint32_t *s_cooc = reinterpret_cast<uint32_t *>(
        smem_align<16>(reinterpret_cast<unsigned char *>(const_cast<int *>(s_abort + 1))));
    int *s_rowoff = reinterpret_cast<int *>(s_cooc + C::kCoocWords);
    uint32_t *s_wsc = reinterpret_cast<uint32_t *>(s_rowoff + E);  // [consumer warp][E]

    pdl_trigger();
    // this CTA: layer blockIdx.y, a contiguous range of its 32-token tiles
    const int64_t layer = blockIdx.y;
    const int64_t per = (W + gridDim.x - 1) / gridDim.x;
    const int64_t tb = (int64_t)blockIdx.x * per;
    const int64_t te = min64(W, tb + per);
    const int n = te > tb ? (int)(te - tb) : 0;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // Shared-memory set-up first: it touches no global memory, so it overlaps
    // the end of the previous kernel on the stream.
    for (int i = threadIdx.x; i < kConsumers * E; i += blockDim.x) s_wsc[i] = 0u;
    if (kCooc) {
        for (int i = threadIdx.x; i < C::kCoocWords; i += blockDim.x) s_cooc[i] = 0u;
        for (int a = threadIdx.x; a < E; a += blockDim.x) s_rowoff[a] = cooc_row_offset<E>(a) - (a & ~3);
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kSlots; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
            slot_round[s] = -1;
        }
        *s_abort = 0;
        fence_barrier_init();
    }
    if (warp == kConsumers && lane == 0) prefetch_tensormap(&tmap);
    __syncthreads();
    // Launched as a programmatic dependent of whatever ran before on the
    // stream: wait for it before touching global memory (it may have written
    // the logits, or still read the accumulators cleared below).
    pdl_wait();
#pragma unroll
    for (int z = 0; z < 3; ++z)
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < zero.n[z];
             i += (int64_t)gridDim.x * blockDim.x)
            zero.p[z][i] = 0;

    if (warp == kConsumers) {  // producer
        if (lane == 0 && n > 0) {
            int issued = 0;
            for (int q = 0; q < n; ++q) {
                const int s = q % C::kSlots, round = q / C::kSlots;
                if (round > 0 && !mbar_wait(&empty[s], (round - 1) & 1, status)) {
                    *s_abort = 1;
                    break;
                }
                if (*s_abort) break;
                const int64_t w = tb + q;
                const int y = (int)(layer * T + 32 * w);
                slot_round[s] = round;
                mbar_arrive_expect_tx(&full[s], C::kTileBytes);
#pragma unroll
                for (int b = 0; b < C::kBoxes; ++b)
                    tma_load_2d(smem + (size_t)s * C::kTileBytes + b * kBoxBytes, &tmap, b * 32, y,
                                &full[s]);
                issued = q + 1;
            }
            // Every issued load completes before the CTA may exit.
            for (int q = issued > C::kSlots ? issued - C::kSlots : 0; q < issued; ++q)
                mbar_wait(&full[q % C::kSlots], (q / C::kSlots) & 1, status);
        }
        return;
    }

    // consumers
    constexpr int R = E / 32;
    uint32_t cnt[R];
#pragma unroll
    for (int r = 0; r < R; ++r) cnt[r] = 0u;

    for (int q = warp; q < n; q += kConsumers) {
        if (__any_sync(kFull, *s_abort)) break;
        const int s = q % C::kSlots, round = q / C::kSlots;
        bool started = slot_round[s] >= round;
        if (!started) {
            const unsigned long long t0 = global_ns();
            while (!(started = slot_round[s] >= round) && !*s_abort) {
                __nanosleep(64);
                if (global_ns() - t0 > kWaitLimitNs) {
                    if (status) atomicOr(status, kDevTimeout);
                    *s_abort = 1;
                    break;
                }
            }
        }
        const bool ok = started && mbar_wait(&full[s], round & 1, status);
        if (!__all_sync(kFull, ok)) {  // leave together: the warp shuffles below
            *s_abort = 1;
            break;
        }
        const int64_t w = tb + q;
        const int64_t t = 32 * w + lane;
        const bool valid = t < T;
        unsigned char *tp = smem + (size_t)s * C::kTileBytes;

        int sel[K];
        float val[K];  // the chosen logits (kRoute)
        select_topk<E, K>(tp, lane, sel, val);
        // the tile is no longer read: hand the slot back to the producer
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[s]);

        if (idx && valid) store_idx<K>(idx + (layer * T + t) * K, sel);
        if (kRoute && valid) store_route<K>(route, (layer * T + t) * K, sel, val);
        if (kCooc && valid) cooc_add<K>(s_cooc, s_rowoff, sel);
        emit_words_or<E, K, kCounts || kCooc>(sel, valid, lane, s_wsc + warp * E,
                                             bits + layer * E * W + w, W, cnt);
    }
    if (kCounts) {
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (cnt[r]) atomicAdd(&counts[layer * E + 32 * r + lane], (int)cnt[r]);
    }
    if (kCooc) {  // counts n_a on the triangle's diagonal
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (cnt[r]) atomicAdd(&s_cooc[s_rowoff[32 * r + lane] + 32 * r + lane], cnt[r]);
    }
    if (kCooc) {
        // all consumer warps have counted: store this CTA's triangle for the
        // reduction kernel
        asm volatile("bar.sync 1, %0;" ::"n"(kConsumers * 32) : "memory");
        uint4 *dst = reinterpret_cast<uint4 *>(cooc + ((size_t)layer * gridDim.x + blockIdx.x) *
                                                          (size_t)C::kCoocWords);
        const uint4 *src = reinterpret_cast<const uint4 *>(s_cooc);
        for (int i = threadIdx.x; i < C::kCoocWords / 4; i += kConsumers * 32) dst[i] = src[i];
        // the diagonal holds this CTA's counts n_a: add them to the layer's totals
        // (counts points at the workspace accumulator on this path)
        for (int a = threadIdx.x; a < E; a += kConsumers * 32) {
            const uint32_t na = s_cooc[s_rowoff[a] + a];
            if (na) atomicAdd(&counts[layer * E + a], (int)na);
        }
    }
}

template <int E, int K, bool kCounts, bool kCooc, bool kRoute>
cudaError_t run_fast(const CUtensorMap &map, const Problem &p, uint32_t *bits, int *counts,
                     uint8_t *idx, uint32_t *cooc, const ZeroSpans &zero, int *status,
                     const RouteOut &route, cudaStream_t s) {
    using C = SigCfg<E>;
    auto kern = sig_fast_kernel<E, K, kCounts, kCooc, kRoute>;
    cudaError_t e = ensure_smem_limit<sig_fast_kernel<E, K, kCounts, kCooc, kRoute>>(C::kSmem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)sig_fast_ctas_per_problem(p), (unsigned)p.L);
    cfg.blockDim = dim3(kFastThreads);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, map, p.T, p.W, bits, counts, idx, cooc, zero,
                              status, route);
}

template <int E, bool kCounts, bool kCooc, bool kRoute>
cudaError_t dispatch_k(const CUtensorMap &map, const Problem &p, uint32_t *bits, int *counts,
                       uint8_t *idx, uint32_t *cooc, const ZeroSpans &zero, int *status,
                       const RouteOut &route, cudaStream_t s) {
    switch (p.k) {
        case 1: return run_fast<E, 1, kCounts, kCooc, kRoute>(map, p, bits, counts, idx, cooc, zero, status, route, s);
        case 2: return run_fast<E, 2, kCounts, kCooc, kRoute>(map, p, bits, counts, idx, cooc, zero, status, route, s);
        case 4: return run_fast<E, 4, kCounts, kCooc, kRoute>(map, p, bits, counts, idx, cooc, zero, status, route, s);
        default: return run_fast<E, 8, kCounts, kCooc, kRoute>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    }
}

template <int E, bool kRoute>
cudaError_t dispatch_mode(const CUtensorMap &map, const Problem &p, uint32_t *bits, int *counts,
                          uint8_t *idx, uint32_t *cooc, const ZeroSpans &zero, int *status,
                          const RouteOut &route, cudaStream_t s) {
    // split entry point: counts, no co-occurrence; fused path: co-occurrence;
    // routing outputs alone: neither (the dispatch scan counts)
    if constexpr (kRoute) {
        if (!cooc && !counts)
            return dispatch_k<E, false, false, true>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    }
    if (cooc) return dispatch_k<E, false, true, kRoute>(map, p, bits, counts, idx, cooc, zero, status, route, s);
    return dispatch_k<E, true, false, kRoute>(map, p, bits, counts, idx, cooc, zero, status, route, s);
}

}  // namespace
}  // namespace dol
