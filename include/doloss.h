/*
 * doloss.h -- C ABI of the GB300 DO-loss library (libdoloss.so).
 *
 * The Distributional Orthogonalization loss of "Function Over Form:
 * Distributional Orthogonalization in Mixture-of-Experts with Replica Expert
 * Mechanism" on one GPU, as four steps:
 *   1. Top-K routing of T tokens over E experts, packed into binary load
 *      signatures with per-expert counts               (Sec. 3.1.1, Eq. 1)
 *   2. the all-pairs Hamming matrix of the signatures  (Sec. 3.1.3, Eq. gij_cij)
 *   3. the surrogate loss and its gradient to the router logits
 *                                                       (Sec. 3.1.3, Eq. do_loss)
 *   4. Eq. origin_do, the sum of squared distances, as a diagnostic.
 * and around them: the router's outputs (do_routing) and their backward
 * (do_route_backward), the routed step in the forward and backward halves of
 * a training step (do_routed_forward, do_routed_backward; also the per-rank
 * step of Global-DO, with do_accumulate_distances for accumulation windows),
 * the router's linear map fused with step 1 and its backward
 * (do_router_forward_backward, do_router_backward), and the consumers of the
 * counts (do_maxvio, do_rem_allocate).
 *
 * Notation: E experts (the paper's n), k selected per token (K), T tokens in
 * the signature window (m), L independent problems batched in one call (for
 * example the MoE layers of a model), W = ceil(T/32).
 *
 * Conventions shared by every entry point:
 *  - Every array argument is a DEVICE pointer owned by the caller, except in
 *    do_forward_backward_host(_async), whose h_* arguments are host pointers,
 *    and do_rem_allocate, a host function.  The library allocates nothing and
 *    keeps no state between calls, with one stated exception:
 *    do_forward_backward_static (a fixed scratch array per device).  do_routed_backward
 *    reads what do_routed_forward left in the caller's workspace.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *    stream).  Calls are asynchronous on it, except do_device_status and
 *    do_forward_backward_host, which synchronize it.
 *  - Arguments are validated before anything is launched; a rejected call
 *    returns DO_ERR_INVALID_ARG or DO_ERR_UNSUPPORTED and touches no memory.
 *    A failed launch returns DO_ERR_CUDA.  Conditions only the device can see
 *    (a Hamming row sum that does not fit int32, a device wait that ran out,
 *    an expert id out of range given to do_routed_backward) are recorded in
 *    the workspace and reported by do_device_status.
 *  - Layouts are dense and row-major:
 *      logits, dlogits  [L][T][E] fp32 (token-major: one row per token)
 *      bits             [L][E][W] uint32; bit (t mod 32) of word t/32 of row i
 *                       is f_it; bits of positions t >= T are zero
 *      counts           [L][E]    int32, n_i = ||F_i||_1
 *      D                [L][E][E] int32, D_ij = ||F_i - F_j||_1 (symmetric,
 *                       zero diagonal)
 *      loss             [L] fp32; origin_do [L] int64
 *  - Logits must be finite.  Top-K is taken on the raw logits: larger value
 *    first, equal values in favour of the lower expert index (the gates are
 *    monotone, so this is the Top-K of the gated scores).
 *  - Limits: 1 <= k <= E <= 1024, T >= 1, L >= 1, (E-1)*T < 2^31.  float
 *    arrays need 4-byte alignment (16-byte alignment and E % 4 == 0 select
 *    the vectorised kernels); uint32/int32 arrays 4-byte, int64 8-byte.
 *  - Results are deterministic: bits, counts, D and origin_do are exact
 *    integers; loss and dlogits are bitwise reproducible run to run (fixed
 *    reduction order; the one floating-point atomic, do_route_backward's
 *    accumulate mode, adds once to each entry).
 */
#ifndef DOLOSS_H
#define DOLOSS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DO_OK = 0,
    DO_ERR_INVALID_ARG = 1,  /* null pointer, bad size or alignment          */
    DO_ERR_UNSUPPORTED = 2,  /* valid but outside this build's limits        */
    DO_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed         */
    DO_ERR_TIMEOUT = 4,      /* a bounded device wait ran out                */
    DO_ERR_OVERFLOW = 5,     /* a row sum of D does not fit int32            */
    DO_ERR_WORKSPACE = 6     /* workspace missing or smaller than required   */
} do_status;

typedef enum {
    DO_GATE_SIGMOID_NORM = 0, /* s = sigmoid(z), p = s / sum(s)  (Sec. 3.1.1, App. A) */
    DO_GATE_SOFTMAX = 1       /* p = softmax(z)                                        */
} do_gate;

/* Step 1 (Sec. 3.1.1, Eq. 1: f_it = 1(i in Top-K(x_t))).
 * Reads logits [L][T][E]; writes the load signatures bits [L][E][W] and the
 * per-expert token counts [L][E] (written, not accumulated). */
do_status do_signatures(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                        uint32_t *bits, int32_t *counts, void *stream);

/* Step 2 (Sec. 3.1.3, Eq. gij_cij: G_ij = ||F_i - F_j||_1).
 * Reads bits [L][E][W] (4-byte aligned; the bits past T in the last word
 * zero, as do_signatures writes them); writes D [L][E][E], the exact number
 * of tokens on which experts i and j disagree, every entry once (no
 * clearing needed).  Uses thread-block clusters of up to 8 CTAs. */
do_status do_pairwise_hamming(const uint32_t *bits, int64_t T, int32_t E, int32_t L,
                              int32_t *D, void *stream);

/* D += the Hamming matrix of bits (exact integer adds).  Sums the distance
 * matrices of several token windows, e.g. the micro-batches of one gradient
 * accumulation window (App. batch ablation: the effective batch of G is
 * micro-batch x ranks x accumulation steps); G is additive over disjoint
 * token windows.  D must hold the running sum (zero before the first
 * window); the caller keeps every row sum within int32. */
do_status do_pairwise_hamming_accumulate(const uint32_t *bits, int64_t T, int32_t E, int32_t L,
                                         int32_t *D, void *stream);

/* The variance of the E (E - 1) off-diagonal distances of each problem's
 * local Hamming matrix, the dispersion that Eq. origin_do measures (App. C.1):
 * with Eq. zero_sum their mean is 2 T k (E - k) / (E (E - 1)), so
 *   var[l] = origin_do[l] / (E (E - 1)) - mean^2    (fp64),
 * without reading D.  origin_do [L] int64 as the fused calls write it (a
 * window of T tokens with k experts each; not a matrix summed over ranks);
 * var [L] fp64.  Needs E >= 2.  Asynchronous on `stream`. */
do_status do_offdiag_variance(const int64_t *origin_do, int64_t T, int32_t E, int32_t k, int32_t L,
                              double *var, void *stream);

/* D_sum += D for [L][E][E] int32 Hamming matrices (device): the matrices of
 * the micro-batches of an accumulation window add up before the loss
 * (Eq. global_do).  Integer, exact while each sum stays within int32 (the
 * window's tokens below 2^31).  Asynchronous on `stream`. */
do_status do_accumulate_distances(const int32_t *D, int32_t E, int32_t L, int32_t *D_sum,
                                  void *stream);

/* Step 3 (Sec. 3.1.3, Eq. do_loss; Sec. 3.1.4, Eq. global_do):
 *   L_DO = 1/(T^2 k) sum_i sum_j G_ij C_ij,  C_ij = sum_t p_it (f_it - f_jt),
 * with G = d_scale * D held constant (detached) and p the dense router
 * probability of `gate`.  d_scale is 1 for a local matrix, or 1/|replicas|
 * when D is the sum of the replicas' matrices (Global-DO).
 * Writes loss [L] (unscaled by grad_scale), origin_do [L] = sum_{i!=j} D_ij^2
 * (Eq. origin_do; may be NULL) and dlogits [L][T][E] = grad_scale * dL/dz
 * (may be NULL for a forward-only call).  bits must hold the selection that
 * produced the token rows of logits; D may come from any source whose row
 * sums fit int32.  workspace: do_workspace_size(T, E, k, L) bytes of device
 * memory, 256-byte aligned and zero-filled before its first use (cudaMemset);
 * every call leaves it ready for the next one.  A workspace serves one call
 * at a time; after a call fails or do_device_status reports an error, zero it
 * again before reusing it. */
do_status do_loss_fwd_bwd(const float *logits, const uint32_t *bits, const int32_t *D,
                          int64_t T, int32_t E, int32_t k, int32_t L, int32_t gate,
                          float d_scale, float grad_scale, float *loss, int64_t *origin_do,
                          float *dlogits, void *workspace, size_t workspace_bytes,
                          void *stream);

/* Steps 1-3 in one call on a local window (d_scale = 1): logits in; bits,
 * counts, D, loss, origin_do (may be NULL) and dlogits (may be NULL) out.
 * With E = 128, the sigmoid-normalised gate, k in {1, 2, 4, 8}, T <= 66052
 * and dlogits given, the gradient pass computes V = F D' on the tensor cores
 * (F the one-hot selections, D' = D with -R on the diagonal); elsewhere it
 * gathers rows of D' on the ALU (as do_loss_fwd_bwd always does; at E = 256,
 * k in {1, 2, 4, 8}, T < 2^24 and 16-byte aligned logits, D and dlogits with
 * D held in 24-bit shared-memory planes).  The two agree within the stated
 * tolerances. */
do_status do_forward_backward(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                              int32_t gate, float grad_scale, uint32_t *bits, int32_t *counts,
                              int32_t *D, float *loss, int64_t *origin_do, float *dlogits,
                              void *workspace, size_t workspace_bytes, void *stream);

/* Routing outputs of the router (Sec. 3.1.1: of a token's normalized
 * probabilities only the K chosen ones are kept, re-normalized to sum to
 * one; they weigh the chosen experts' outputs), from the selection of step 1:
 *   expert_ids     [L][T][k] int32, the chosen experts of each token in
 *                  selection order (largest logit first, equal logits lower
 *                  index first)
 *   combine        [L][T][k] fp32, w_tq = p_{e_q,t} / sum_q' p_{e_q',t}
 *                  (sigmoid-norm: s_e / sum of the chosen s; softmax: the
 *                  softmax of the chosen logits)
 *   counts         [L][E] int32, n_e (as do_signatures)
 *   expert_offsets [L][E+1] int32, offsets[e] = n_0 + ... + n_{e-1},
 *                  offsets[E] = T k
 *   dispatch_rows  [L][T*k] int32, the routed (token, choice) pairs grouped
 *                  by expert in expert order, tokens ascending inside an
 *                  expert: row r holds its token id
 *   dispatch_pos   [L][T][k] int32, the row of the pair (t, q), so that
 *                  dispatch_rows[pos] = t
 * expert_ids, combine and counts are required; each dispatch array may be
 * NULL.  All are exact integers except combine, which is fp32 (a few ulp of
 * the exact ratio); all are identical run to run.  Needs T k <= INT32_MAX
 * (DO_ERR_UNSUPPORTED otherwise).  16-byte aligned logits, expert_ids and
 * combine with E in {32, 64, 128} and k in {1, 2, 4, 8} take the fast
 * selection kernel.  workspace: do_routing_workspace_size(T, E, k, L) bytes
 * of device memory, 256-byte aligned, zero-filled before its first use (it
 * holds the device status word, read by do_device_status, and the
 * signatures).  Asynchronous on `stream`. */
do_status do_routing(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L, int32_t gate,
                     int32_t *expert_ids, float *combine, int32_t *counts,
                     int32_t *expert_offsets, int32_t *dispatch_rows, int32_t *dispatch_pos,
                     void *workspace, size_t workspace_bytes, void *stream);

size_t do_routing_workspace_size(int64_t T, int32_t E, int32_t k, int32_t L);

/* The routed step split at the point where a training step splits it: the
 * forward half runs when the router's outputs are needed, the backward half
 * once the gradient of the combine weights has come back from the experts.
 *
 * do_routed_forward: steps 1-2 and the routing outputs from one selection
 * pass -- bits, counts, D, origin_do (may be NULL) as do_forward_backward
 * writes them, and expert_ids, combine and the dispatch arrays as do_routing
 * writes them (the dispatch arrays may be NULL; with expert_ids and combine
 * both NULL, and no dispatch arrays, the call is steps 1-2 alone).  No loss
 * and no gradient.
 *
 * do_routed_backward: step 3 on the same tokens plus the routing gradient:
 *   loss     [L] fp32, L_DO as do_loss_fwd_bwd computes it with D and d_scale
 *   dlogits  [L][T][E] fp32, overwritten with grad_scale * dL_DO/dz plus
 *            the gradient of the combine weights for grad_combine [L][T][k]
 *            (fp32) with the selection expert_ids [L][T][k] held fixed, as
 *            do_route_backward computes it (grad_scale does not apply to it;
 *            expert_ids and grad_combine both NULL: no routing gradient)
 * logits, bits and counts are those of the forward half, expert_ids the ids
 * it wrote.  With d_scale = 1, D is the forward half's matrix; otherwise D
 * is a matrix summed over data-parallel ranks or micro-batches that include
 * these tokens (Eq. global_do, d_scale = 1 / their number) and m stays T.
 * With E = 128, the sigmoid-normalised gate, k in {1, 2, 4, 8} and 16-byte
 * aligned logits, D, bits, dlogits, expert_ids and grad_combine, the
 * tensor-core loss kernel runs and adds the routing gradient in its
 * epilogue: with d_scale = 1 (and T <= 66052) from the image of D' the
 * forward half left; otherwise a kernel first builds the image of the given
 * matrix and checks, per problem, that its two fp16 pieces hold it exactly
 * (0 <= D_ij < 2^22 off the diagonal, D_ii = 0, row sums below 2^23), and
 * the problems that fail the check go to the ALU loss kernel and the
 * routing-gradient kernel instead.  Elsewhere the ALU loss kernels run and a
 * second kernel adds the routing gradient.  The result agrees with
 * do_loss_fwd_bwd's dlogits plus do_route_backward's within the sum of their
 * tolerances.
 *
 * Both take the same workspace (do_routed_workspace_size bytes, 256-byte
 * aligned, zero-filled before its first use): the forward half leaves in it
 * the selected experts and the image of D that the backward half reads, so a
 * backward call uses the workspace of the forward call on the same logits,
 * with no other call on that workspace in between.  The backward half may be
 * repeated.  An expert id outside [0, E) is left out and recorded in the
 * status word (do_device_status then returns DO_ERR_INVALID_ARG).
 * Asynchronous on `stream`. */
do_status do_routed_forward(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                            int32_t gate, uint32_t *bits, int32_t *counts, int32_t *D,
                            int64_t *origin_do, int32_t *expert_ids, float *combine,
                            int32_t *expert_offsets, int32_t *dispatch_rows, int32_t *dispatch_pos,
                            void *workspace, size_t workspace_bytes, void *stream);
do_status do_routed_backward(const float *logits, int64_t T, int32_t E, int32_t k, int32_t L,
                             int32_t gate, float d_scale, float grad_scale, const uint32_t *bits,
                             const int32_t *counts, const int32_t *D, const int32_t *expert_ids,
                             const float *grad_combine, float *loss, float *dlogits,
                             void *workspace, size_t workspace_bytes, void *stream);

/* Backward of the combine weights of do_routing (Sec. 3.1.1) to the logits,
 * the selection held fixed.  With g = grad_combine, dot_t = sum_q g_tq w_tq
 * and l = expert_ids[t][q] a chosen expert:
 *   sigmoid-norm: dlogits[t][l] = w_tl (1 - sigmoid(z_tl)) (g_tq - dot_t)
 *   softmax:      dlogits[t][l] = w_tl (g_tq - dot_t)
 * and 0 for the experts not chosen (the dense normaliser of p cancels).
 *   logits        [L][T][E] fp32 device, the router logits of the forward pass
 *   expert_ids    [L][T][k] int32 device, the chosen experts (as do_routing
 *                 writes them; the ids of a token must be distinct, repeated
 *                 ids leave the values at those entries unspecified)
 *   grad_combine  [L][T][k] fp32 device, the gradient of combine
 *   dlogits       [L][T][E] fp32 device: accumulate = 0 overwrites every
 *                 entry; accumulate = 1 adds the gradient to the chosen
 *                 entries only and leaves the rest as they are (so that the
 *                 call can follow do_forward_backward on the same buffer)
 * The weights are recomputed in fp32 from the chosen logits (shifted by the
 * largest one) as do_routing computes them; each result is within a few ulp
 * of w_tl (|g_tq| + sum_q' |g_tq'| w_tq') times the gate factor.  The result
 * is identical run to run.  status_flags (device int32, may be NULL): bit 2
 * (value 4) is ORed in when an expert_ids entry lies outside [0, E) (that
 * choice is then left out).  4-byte aligned pointers.  Asynchronous on
 * `stream`. */
do_status do_route_backward(const float *logits, const int32_t *expert_ids,
                            const float *grad_combine, int64_t T, int32_t E, int32_t k, int32_t L,
                            int32_t gate, int32_t accumulate, float *dlogits,
                            int32_t *status_flags, void *stream);

/* do_forward_backward that also writes the routing outputs of do_routing
 * (expert_ids, combine required; expert_offsets, dispatch_rows, dispatch_pos
 * may each be NULL) from the same selection pass over the logits, so the
 * logits are read once for both the loss and the dispatch.  workspace:
 * do_routed_workspace_size(T, E, k, L) bytes (do_forward_backward's plus the
 * dispatch scratch), prepared as for do_forward_backward. */
do_status do_forward_backward_routed(const float *logits, int64_t T, int32_t E, int32_t k,
                                     int32_t L, int32_t gate, float grad_scale, uint32_t *bits,
                                     int32_t *counts, int32_t *D, float *loss, int64_t *origin_do,
                                     float *dlogits, int32_t *expert_ids, float *combine,
                                     int32_t *expert_offsets, int32_t *dispatch_rows,
                                     int32_t *dispatch_pos, void *workspace,
                                     size_t workspace_bytes, void *stream);

/* Router-side fusion: the logits come from the router's linear map (Sec. 4.1:
 * hidden size H to the E experts, no bias), computed here on the tensor cores
 * from bf16 inputs with fp32 accumulation,
 *   logits[l][t][e] = sum_h X[l][t][h] W[l][e][h],
 * with step 1 (Top-K, signatures, co-occurrence counts) done on each tile of
 * logits while it is still on chip; the logits are written to `logits`
 * ([L][T][E] fp32, an output here) for the loss step, and everything else is
 * as do_forward_backward.  X [L][T][H] and W [L][E][H] are bf16 (uint16 bit
 * patterns), 16-byte aligned.  Supported: E = 128, k in {1, 2, 4, 8}, H a
 * multiple of 64, logits 16-byte aligned and the conditions of the fused
 * path of do_forward_backward (16-byte aligned bits and dlogits given);
 * otherwise DO_ERR_UNSUPPORTED.  Same workspace as do_forward_backward.  The
 * selection is taken on the fp32 logits this call writes. */
do_status do_router_forward_backward(const void *X, const void *Wr, int64_t T, int32_t H, int32_t E,
                                     int32_t k, int32_t L, int32_t gate, float grad_scale,
                                     float *logits, uint32_t *bits, int32_t *counts, int32_t *D,
                                     float *loss, int64_t *origin_do, float *dlogits,
                                     void *workspace, size_t workspace_bytes, void *stream);

/* Backward of the router's linear map for the gradient dz = dlogits
 * ([L][T][E] fp32, as written by do_router_forward_backward):
 *   dW [L][E][H] fp32,  dW[l][e][h] = sum_t dz[l][t][e] X[l][t][h]
 *   dX [L][T][H] bf16,  dX[l][t][h] = sum_e dz[l][t][e] W[l][e][h]  (may be NULL)
 * X, W bf16 as in do_router_forward_backward; all arrays 16-byte aligned.
 * E = 128 and H a multiple of 64 (DO_ERR_UNSUPPORTED otherwise).  dz is
 * rounded to bf16 (nearest even) and both products run on the tensor cores
 * (bf16 operands, fp32 accumulation; X, W and dz read as stored); dW is the
 * sum of per-chunk partial products over the tokens, added in a fixed order,
 * so results are identical run to run.  workspace:
 * do_router_backward_workspace_size bytes of device memory, 256-byte
 * aligned and zero-filled before its first use (its status word, read by
 * do_device_status; then the bf16 copy of dz and the partial sums).
 * Asynchronous on `stream`. */
do_status do_router_backward(const void *X, const void *Wr, const float *dlogits, int64_t T,
                             int32_t H, int32_t E, int32_t L, float *dW, void *dX,
                             void *workspace, size_t workspace_bytes, void *stream);

size_t do_router_backward_workspace_size(int64_t T, int32_t E, int32_t H, int32_t L);

/* Device workspace, in bytes, that do_loss_fwd_bwd, do_forward_backward and
 * do_router_forward_backward need for these sizes (0 if the sizes are
 * invalid); do_forward_backward_routed, do_routed_forward and
 * do_routed_backward need do_routed_workspace_size. */
size_t do_workspace_size(int64_t T, int32_t E, int32_t k, int32_t L);
size_t do_routed_workspace_size(int64_t T, int32_t E, int32_t k, int32_t L);

/* Synchronizes `stream`, then reads and clears the device-side status that
 * the previous calls with this workspace recorded: DO_OK, DO_ERR_OVERFLOW,
 * DO_ERR_TIMEOUT (outputs of the failing call are then undefined) or, after
 * do_routed_backward, DO_ERR_INVALID_ARG for an expert id outside [0, E). */
do_status do_device_status(void *workspace, void *stream);

/* Host-to-host convenience over do_forward_backward: copies h_logits [L][T][E]
 * to the device, runs steps 1-3 (the gradient included: it stays in
 * device_buffer), and copies loss [L] into h_loss and, when given, dlogits
 * into h_dlogits [L][T][E], counts into h_counts [L][E] and D into
 * h_D [L][E][E].  All device memory comes from `device_buffer`
 * (do_host_buffer_size(T, E, k, L) bytes, 256-byte aligned, zero-filled
 * before its first use, as the workspace above).  Synchronous:
 * returns after the results are in host memory and the device status has been
 * checked.  Pinned host memory gives the full copy bandwidth. */
do_status do_forward_backward_host(const float *h_logits, int64_t T, int32_t E, int32_t k,
                                   int32_t L, int32_t gate, float grad_scale, float *h_loss,
                                   float *h_dlogits, int32_t *h_counts, int32_t *h_D,
                                   void *device_buffer, size_t device_buffer_bytes,
                                   void *stream);

size_t do_host_buffer_size(int64_t T, int32_t E, int32_t k, int32_t L);

/* do_forward_backward_host without the wait, for pipelines that keep the host
 * link busy: enqueues on `stream` the copy of h_logits to the device, steps
 * 1-3 and one copy back of the result into h_result (host memory, pinned for
 * the copies to overlap): bytes [0, 4L) the losses (fp32), bytes [4L, 4L+4)
 * the int32 device status word of this call (bit 0: a Hamming row sum did
 * not fit int32; bit 1: a bounded wait ran out; 0: success).  Returns once
 * the work is enqueued; h_logits must stay unchanged and h_result unread
 * until `stream` has reached that point.  device_buffer as for
 * do_forward_backward_host; calls that share one device_buffer must be
 * ordered on one stream. */
do_status do_forward_backward_host_async(const float *h_logits, int64_t T, int32_t E, int32_t k,
                                         int32_t L, int32_t gate, float grad_scale,
                                         void *h_result, void *device_buffer,
                                         size_t device_buffer_bytes, void *stream);

/* Largest workspace, in bytes, that do_forward_backward_static can hold. */
#define DO_STATIC_SCRATCH_BYTES ((size_t)16 << 20)

/* do_forward_backward for callers that cannot allocate device memory (an
 * embedding C host without a device allocator, or a process that has handed
 * its spare HBM to its own pool).  The paper has no counterpart: it is an
 * interface variant of steps 1-3, with the same arguments and results as
 * do_forward_backward except that the workspace is a fixed 16 MiB array
 * inside the library, one per device.
 *  - Sizes whose do_workspace_size exceeds DO_STATIC_SCRATCH_BYTES are
 *    rejected with DO_ERR_WORKSPACE before anything is launched (for
 *    E = 128, k = 8, L = 1 that is T above about 0.97 million tokens).
 *  - Unlike the other entry points it keeps state: the first call in a CUDA
 *    context (with its device current) looks up the array's device address
 *    and caches it for that context (a context created later, e.g. after
 *    cudaDeviceReset, looks it up again); make that first call before any
 *    stream capture begins.  Every call clears the parts that must start at
 *    zero with cudaMemsetAsync on `stream`; the array keeps the rest of the
 *    last call's contents.
 *  - status_flags (device int32, may be NULL) receives the device status
 *    word of this call, copied on `stream`: bit 0 = a Hamming row sum did
 *    not fit int32, bit 1 = a bounded device wait ran out.
 *  - All calls share one array per device: calls that overlap in time (on
 *    two streams or from two threads) race.  Serialize them on one stream.
 *  - Allocates nothing (no cudaMalloc, no allocating library). */
do_status do_forward_backward_static(const float *logits, int64_t T, int32_t E, int32_t k,
                                     int32_t L, int32_t gate, float grad_scale, uint32_t *bits,
                                     int32_t *counts, int32_t *D, float *loss, int64_t *origin_do,
                                     float *dlogits, int32_t *status_flags, void *stream);

/* Self-test of the failure path shared by every device wait: launches one
 * thread that waits on an mbarrier which nothing completes.  Its bounded wait
 * gives up after about one second and records the time-out in the status word
 * of `workspace` (do_workspace_size bytes, as for the other entry points), so
 * that do_device_status then returns DO_ERR_TIMEOUT; nothing traps or faults
 * and the context stays usable.  Asynchronous on `stream`. */
do_status do_selftest_wait_limit(void *workspace, void *stream);

/* MaxVio (App. E) of each problem's counts: with expert_rank [E] (device
 * int32) the rank that holds each expert, L_r = sum of counts[l][e] over the
 * experts on rank r and tau = (1/R) sum_r L_r,
 *   maxvio[l] = max_r |L_r / tau - 1|   (0 when the problem has no tokens).
 * counts [L][E] device int32 (as written by do_signatures, do_routing or
 * do_forward_backward); rank_loads [L][R] device int64 (may be NULL) receives
 * L_r; maxvio [L] device double.  L_r and tau are exact (integer sums), and
 * the result is the double-precision evaluation of the formula.  status_flags
 * (device int32, may be NULL): bit 2 (value 4) is ORed in when an expert_rank
 * entry lies outside [0, R) (that expert is then left out).  R <= 4096.
 * Asynchronous on `stream`. */
do_status do_maxvio(const int32_t *counts, const int32_t *expert_rank, int32_t E, int32_t R,
                    int32_t L, int64_t *rank_loads, double *maxvio, int32_t *status_flags,
                    void *stream);

/* Global-batch replica allocation of the Replica Expert Mechanism (Sec. 3.2,
 * Eq. benefit_score; App. B.1, Algorithm rem_allocation).  Host function: all
 * pointers are host memory, and it returns when done.
 *   loads [R]          historical rank loads L_r (e.g. moving averages of
 *                      do_maxvio's rank_loads)
 *   expert_tokens [E]  token volume T_e of each expert
 *   expert_rank [E]    home rank of each expert, in [0, R)
 *   D                  replica slots per rank
 * tau = (1/R) sum_r L_r is fixed at the start.  Repeatedly: the receiver is
 * the least-loaded rank with a free slot (lowest index on ties); among the
 * experts not on it and not yet replicated there, sent from their home rank
 * r_s, the one of largest Benefit Score S(e, r_s, r_r, tau) (lowest index on
 * ties) is placed with Delta = S tokens, and L_r_r += Delta, L_r_s -= Delta,
 * T_e -= Delta.  It stops when every rank is full or the best score is not
 * positive.  Writes the placements in order to placed_expert, placed_sender,
 * placed_receiver and placed_tokens (capacity R*D each; may be NULL when
 * D = 0), their number to *n_placed and the updated loads to loads_out [R].
 * DO_ERR_INVALID_ARG for an expert_rank entry outside [0, R). */
do_status do_rem_allocate(const double *loads, const double *expert_tokens,
                          const int32_t *expert_rank, int32_t R, int32_t E, int32_t D,
                          int32_t *placed_expert, int32_t *placed_sender,
                          int32_t *placed_receiver, double *placed_tokens, int32_t *n_placed,
                          double *loads_out);

/* A static description of a status code. */
const char *do_status_string(int32_t status);

#ifdef __cplusplus
}
#endif

#endif /* DOLOSS_H */
