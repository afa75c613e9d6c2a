/*
 * efsparse.h — C ABI of the error-feedback (EF) gradient-sparsification step
 * of "Rethinking gradient sparsification as total error minimization"
 * (Sahu et al., NeurIPS 2021, arXiv:2108.00951).
 *
 * One call performs, for one worker i at one iteration t, the compression
 * part of the distributed EF-SGD loop (Algorithm 1):
 *
 *     a       = e + gamma * g              (Algorithm 1, corrected update p_{i,t})
 *     C(a)    = sum_{j in S(a)} a[j] u_j   (Sec. 4.2: a deterministic sparsifier
 *                                           keeps the coordinates of a support S)
 *     e      <- a - C(a)                   (Algorithm 1, error update)
 *
 * and emits C(a) as (uint32 index, fp32 value) pairs in ascending index order.
 * The support S is either
 *   - the hard-threshold support S_lambda(a) = { j : |a[j]| >= lambda }
 *     (Sec. 1 and Sec. 4.2), the paper's proposed sparsifier, or
 *   - the Top-k support, the k largest-magnitude coordinates (Lemma 2), the
 *     baseline the paper compares against.
 * sparse_aggregate() then sums n workers' sparse vectors into one dense vector
 * (Algorithm 1, exchange-and-average step; the 1/n factor is left to the caller).
 *
 * Conventions shared by every entry point:
 *   - All array pointers are DEVICE pointers (CUDA global memory) unless stated
 *     otherwise. The caller allocates and owns every input and output buffer.
 *   - Every call is asynchronous on `stream` (NULL = the legacy default stream).
 *     No call synchronises with the host, except the one-time growth of the
 *     library's internal workspace (see "Workspace" below). Outputs are valid
 *     once the stream has been synchronised.
 *   - Argument checks happen on the host before any launch; a failing check
 *     returns EF_ERR_INVALID_ARG and launches nothing.
 *   - A CUDA runtime failure (launch or allocation) returns EF_ERR_CUDA or
 *     EF_ERR_NO_MEMORY.
 *   - Errors found on the device (a bounded wait that ran out, malformed sparse
 *     input) are latched in a per-stream device status word and reported by
 *     ef_check_status(); they never fault, trap or hang the GPU.
 *   - No C++ exception crosses this ABI.
 *
 * Numerical contract (identical to the CPU oracle, bit for bit):
 *   - a[j] is ONE fused multiply-add, fmaf(gamma, g[j], e[j]), rounded once to
 *     nearest-even; subnormals are kept (no flush to zero).
 *   - A coordinate with a[j] == +-0 is never sent (sending it changes nothing
 *     and the paper's data volume counts non-zeros, Sec. 6 "average density").
 *   - The residual of a sent coordinate is +0.0f; of an unsent one it is a[j].
 *     Hence a == C(a) + e' holds exactly for every finite a.
 *   - NaN (the paper is silent on it): never satisfies |a| >= lambda (not
 *     sent by hard-threshold); in the Top-k order every NaN is one magnitude,
 *     above +inf, so NaNs tie and the lowest indices win. A NaN carries no
 *     value and its encoding is not part of the result (CUDA arithmetic writes
 *     the quiet NaN 0x7fffffff for every NaN it produces).
 *   - Top-k ties go to the lowest index; exactly k pairs are emitted.
 *
 * Workspace: the library keeps one grow-only device workspace per (device,
 * stream) pair (scan tile status, histograms, candidate buffers, offsets).
 * Growing it synchronises `stream` once. Its size follows the largest d seen
 * on that stream: about 8 bytes per coordinate of pair staging (the size of
 * the outputs: 1.1 GB at d = 138 M) plus, once Top-k has run, 3 x 8 bytes per
 * candidate slot (min(d, max(2^20, d/16)) slots), plus 8 bytes per 4096
 * coordinates and about 260 KB of fixed state, and one 4-byte word of mapped
 * pinned host memory (the density hint of the hard-threshold step's kernel
 * choice, written by the device). Memory is therefore bounded by
 * (number of streams used) x that size; ef_workspace_release() frees all
 * workspaces of the current device (for example after a phase that used
 * extra streams), and ef_hard_threshold_noalloc needs none. Calls on
 * DIFFERENT streams never share a workspace and may run concurrently; calls
 * on the same stream are ordered by the stream.
 *
 * Concurrency: below 4096 tiles (16,777,216 coordinates) the streaming
 * kernel's CTAs wait (bounded) only for lower-numbered CTAs of the same
 * launch, which the device dispatches first; kernels that wait on every CTA
 * of their grid (the Top-k select, the layer-wise select with teams) are
 * cooperative launches. If kernels on other streams or other processes (MPS)
 * hold SMs long enough that a CTA cannot start within the bound (2 s), the
 * call fails with EF_ERR_TIMEOUT (reported by ef_check_status); it never
 * hangs and never returns a wrong result. From 4096 tiles on, the streaming
 * kernel's CTAs claim groups of tiles in the order they start, and the
 * one-tile-per-CTA path (misaligned g or e, ef_hard_threshold_noalloc) takes
 * its tiles the same way: neither needs co-residency.
 */
#ifndef EFSPARSE_H
#define EFSPARSE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream handle; the same type as cudaStream_t (struct CUstream_st*). */
typedef struct CUstream_st* ef_stream_t;

/* Storage type of a gradient passed through the _ex entry points. */
typedef enum { EF_GRAD_F32 = 0, EF_GRAD_BF16 = 1 } ef_grad_type;

typedef enum {
  EF_OK = 0,
  EF_ERR_INVALID_ARG = 1, /* host-side argument check failed; nothing launched */
  EF_ERR_CUDA = 2,        /* a CUDA runtime call or kernel launch failed */
  EF_ERR_TIMEOUT = 3,     /* a bounded device-side wait ran out (latched) */
  EF_ERR_BAD_INPUT = 4,   /* malformed sparse input detected on the device (latched) */
  EF_ERR_NO_MEMORY = 5    /* workspace allocation failed */
} ef_status;

/*
 * ef_hard_threshold — EF accumulate + hard-threshold sparsifier + compaction
 * + residual, fused in one pass over the d coordinates.
 *
 * Defines: Algorithm 1 (p = e + gamma g; error update e <- p - Delta) with the
 * hard-threshold sparsifier C_lambda, S_lambda(x) = { j : |x[j]| >= lambda }
 * (Sec. 1; Sec. 4.2). The threshold is applied to a itself: lambda here equals
 * gamma * lambda_paper of Algorithm 1's Delta = gamma C(p / gamma) (Remark 1),
 * and the value sent is a[j] unchanged.
 *
 *   g          [in]  fp32[d], the stochastic gradient g_{i,t}. 4-byte aligned.
 *   e          [in/out] fp32[d], the error memory e_{i,t}; overwritten with
 *                    e_{i,t+1} = a - C(a). 4-byte aligned; 16-byte alignment of
 *                    both g and e selects the vectorised path.
 *   gamma      step size; must be finite.
 *   lambda     threshold; must be >= 0 and not NaN (+inf sends only +-inf).
 *   d          number of coordinates, 0 <= d <= 2^32 - 1.
 *   idx_out    [out] uint32[capacity >= d]; idx_out[0..count) = the sent
 *                    coordinates, strictly ascending.
 *   val_out    [out] fp32[capacity >= d]; val_out[p] = a[idx_out[p]].
 *   count_out  [out] one uint32 in device memory: the number of pairs
 *                    (= ||C(a)||_0, the per-iteration k_t of Sec. 6).
 *   Outputs must not overlap g or e. Entries of idx_out/val_out at positions
 *   >= count are left untouched.
 */
ef_status ef_hard_threshold(const float* g, float* e, float gamma, float lambda,
                            uint64_t d, uint32_t* idx_out, float* val_out,
                            uint32_t* count_out, ef_stream_t stream);

/*
 * ef_hard_threshold_bf16 — as ef_hard_threshold, with the gradient stored as
 * bfloat16 bit patterns (uint16_t[d], 2-byte aligned; 8-byte alignment of g
 * and 16-byte alignment of e select the vectorised path). Each g[j] is widened
 * exactly to fp32 (its 16 bits become the high half of the fp32 word) before
 * the same fused multiply-add; all other semantics are identical.
 */
ef_status ef_hard_threshold_bf16(const uint16_t* g, float* e, float gamma,
                                 float lambda, uint64_t d, uint32_t* idx_out,
                                 float* val_out, uint32_t* count_out,
                                 ef_stream_t stream);

/*
 * ef_topk — EF accumulate + Top-k sparsifier + compaction + residual.
 *
 * Defines: Algorithm 1 with C = Top-k, the k largest-magnitude coordinates of a
 * (Lemma 1 / Lemma 2: the minimiser of ||a - C(a)||^2 over supports of size
 * k). The paper assumes distinct magnitudes (Sec. 4.3); ties here go to the
 * lowest index, and exactly k pairs are always emitted (zero-magnitude
 * coordinates fill a short support, lowest index first).
 *
 *   g, e, gamma, d   as for ef_hard_threshold.
 *   k          number of coordinates to send, 0 <= k <= d.
 *   idx_out    [out] uint32[capacity >= k], strictly ascending.
 *   val_out    [out] fp32[capacity >= k], val_out[p] = a[idx_out[p]].
 *   count_out  [out] one uint32 in device memory; always equals k.
 *   During the call e temporarily holds a; on completion it holds a - C(a).
 */
ef_status ef_topk(const float* g, float* e, float gamma, uint64_t k, uint64_t d,
                  uint32_t* idx_out, float* val_out, uint32_t* count_out,
                  ef_stream_t stream);

/* ef_topk_bf16 — ef_topk with a bfloat16 gradient, widened as in
 * ef_hard_threshold_bf16. */
ef_status ef_topk_bf16(const uint16_t* g, float* e, float gamma, uint64_t k,
                       uint64_t d, uint32_t* idx_out, float* val_out,
                       uint32_t* count_out, ef_stream_t stream);

/*
 * ef_topk_layerwise — EF accumulate + layer-wise Top-k + compaction + residual.
 *
 * Defines: Algorithm 1 with C = Top-k applied to each tensor of the model on
 * its own (the experiments of Sec. 6 compress layer by layer, with k_t a
 * fraction of each layer; the Appendix section on layer-wise compression).
 * The d coordinates form n_seg consecutive segments,
 * segment s = [seg_end[s-1], seg_end[s]) (seg_end[-1] = 0), and segment s
 * sends its seg_k[s] largest-magnitude coordinates with the ef_topk rules
 * (ties to the lowest index, NaN above +inf, exactly seg_k[s] pairs). The
 * hard-threshold sparsifier acts per coordinate, so it needs no layer-wise
 * variant: ef_hard_threshold already gives it.
 *
 *   g, e, gamma, d   as for ef_topk.
 *   n_seg      number of segments, 1 <= n_seg < 2^31.
 *   seg_end    HOST array of n_seg uint64: the segments' exclusive ends,
 *              non-decreasing, seg_end[n_seg-1] == d (empty segments allowed).
 *   seg_k      HOST array of n_seg uint64: pairs sent by each segment,
 *              0 <= seg_k[s] <= seg_end[s] - seg_end[s-1].
 *   idx_out    [out] uint32[capacity >= K], K = sum of seg_k; segment s fills
 *              positions [seg_k[0] + ... + seg_k[s-1], ... + seg_k[s]) in
 *              ascending index, so the whole list is strictly ascending.
 *   val_out    [out] fp32[capacity >= K], val_out[p] = a[idx_out[p]].
 *   count_out  [out] one uint32 in device memory; always equals K.
 *   The library copies the segment table to the device when it differs from
 *   the previous call's on this stream (so a fixed table costs nothing after
 *   the first call); growing that copy synchronises the stream once. Both
 *   host arrays may be reused as soon as the call returns.
 */
ef_status ef_topk_layerwise(const float* g, float* e, float gamma, uint32_t n_seg,
                            const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                            uint32_t* idx_out, float* val_out, uint32_t* count_out,
                            ef_stream_t stream);

/* ef_topk_layerwise_bf16 — ef_topk_layerwise with a bfloat16 gradient,
 * widened as in ef_hard_threshold_bf16. */
ef_status ef_topk_layerwise_bf16(const uint16_t* g, float* e, float gamma, uint32_t n_seg,
                                 const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                                 uint32_t* idx_out, float* val_out, uint32_t* count_out,
                                 ef_stream_t stream);

/*
 * ef_hard_threshold_ex, ef_topk_ex, ef_topk_layerwise_ex — the same steps as
 * ef_hard_threshold[_bf16], ef_topk[_bf16] and ef_topk_layerwise[_bf16]
 * (identical outputs), with the gradient's storage type as an argument and
 * one optional output:
 *
 *   g_type      EF_GRAD_F32 (g is float[d]) or EF_GRAD_BF16 (uint16_t[d]).
 *   err_sq_out  [out, optional] one double in device memory, 8-byte aligned,
 *               or NULL: the squared error norm of this step,
 *               ||e_{t+1}||^2 = sum_j e'_j^2. Summed over the iterations it
 *               is the total error of Sec. 1 (the term that alone carries
 *               the effect of compression in the EF convergence bound).
 *
 * Precision (the paper fixes none): squares are accumulated with fmaf in fp32
 * in groups of at most 256 terms whose partial sums see at most 13 roundings,
 * and the groups are added in float-float arithmetic (about 44 bits) in a
 * fixed order. The result is within 1e-6 of the exact sum, relatively
 * (nonnegative terms), plus the squares below the fp32 range
 * (|e'_j| < 2^-75), which contribute 0; a sum beyond the fp32 range
 * (|e'_j| >= 2^64 suffices) makes it +inf. It is bit-for-bit reproducible for a given device and input.
 * The streaming kernels add it as they go; steps whose g or e are not
 * 16-byte aligned compute it with one more pass over e'. After a step that
 * failed on the device (a latched timeout) it holds a NaN.
 */
ef_status ef_hard_threshold_ex(const void* g, ef_grad_type g_type, float* e, float gamma,
                               float lambda, uint64_t d, uint32_t* idx_out, float* val_out,
                               uint32_t* count_out, double* err_sq_out, ef_stream_t stream);
ef_status ef_topk_ex(const void* g, ef_grad_type g_type, float* e, float gamma, uint64_t k,
                     uint64_t d, uint32_t* idx_out, float* val_out, uint32_t* count_out,
                     double* err_sq_out, ef_stream_t stream);
ef_status ef_topk_layerwise_ex(const void* g, ef_grad_type g_type, float* e, float gamma,
                               uint32_t n_seg, const uint64_t* seg_end, const uint64_t* seg_k,
                               uint64_t d, uint32_t* idx_out, float* val_out,
                               uint32_t* count_out, double* err_sq_out, ef_stream_t stream);

/*
 * ef_scaled_round_ex — EF accumulate + scaled integer rounding + residual:
 * another absolute compressor behind the same error-feedback step.
 *
 * Defines: Algorithm 1 with C = scaled integer rounding, which Sec. 5 names an
 * absolute compressor (any rounding with error bounded by eps is one, with
 * kappa^2 = d eps^2; the scaled integer rounding of in-network aggregation in
 * particular). With a_j = fmaf(gamma, g_j, e_j):
 *     q_j    = a_j 2^scale_log2 rounded to the nearest integer, ties to even (int32),
 *     C(a)_j = q_j 2^-scale_log2,
 *     e'_j   = a_j - C(a)_j   (exact: a == C(a) + e' bit for bit; |e'_j| <= 2^(-scale_log2-1)).
 * A coordinate whose a_j 2^scale_log2 has magnitude at least 2^31 (or is NaN)
 * is not sent: q_j = 0 and e'_j = a_j; such coordinates are counted.
 *
 *   g, g_type, e, gamma, d, err_sq_out   as for ef_hard_threshold_ex.
 *   scale_log2 the scale exponent m, -100 <= m <= 100 (grid spacing 2^-m).
 *   q_out      [out] int32[d], the dense integer message (4-byte aligned;
 *              16-byte alignment of g, e and q_out selects vector access).
 *   unsent_out [out] one uint32 in device memory: the coordinates not sent.
 * One pass: 16 bytes per coordinate (14 with a bf16 gradient).
 */
ef_status ef_scaled_round_ex(const void* g, ef_grad_type g_type, float* e, float gamma,
                             int32_t scale_log2, uint64_t d, int32_t* q_out,
                             uint32_t* unsent_out, double* err_sq_out, ef_stream_t stream);

/*
 * int_aggregate — exchange of n workers' scaled-integer messages: the
 * integer sum S_j = sum_i q[i][j] is exact (64-bit, so independent of the
 * order), then dense_out[j] = S_j rounded once to fp32, times 2^-scale_log2.
 *
 *   n          1 <= n <= 256.
 *   q          HOST array of n DEVICE pointers to int32[d] messages.
 *   d, scale_log2   as for ef_scaled_round_ex.
 *   dense_out  [out] fp32[d], not overlapping any message.
 */
ef_status int_aggregate(uint32_t n, const int32_t* const* q, uint64_t d, int32_t scale_log2,
                        float* dense_out, ef_stream_t stream);

/*
 * sparse_aggregate — decompress and sum n workers' sparse vectors.
 *
 * Defines: Algorithm 1's exchange step, Delta_bar = (1/n) sum_i Delta_{i,t},
 * without the 1/n factor (the caller scales; exact for power-of-two n):
 *
 *     dense_out[j] = sum over i = 0..n-1 with j in S_i of val[i][p_i(j)],
 *
 * accumulated in fp32 in ascending worker order starting from +0.0f, so the
 * result is bit-for-bit deterministic. Coordinates no worker sent are +0.0f.
 *
 *   n          number of workers, 1 <= n <= 256.
 *   idx        HOST array of n DEVICE pointers; idx[i][0..counts[i]) must be
 *              strictly ascending and < d (the form ef_hard_threshold and
 *              ef_topk produce).
 *   val        HOST array of n DEVICE pointers to fp32 values.
 *   counts     DEVICE array of n uint32 pair counts; counts[i] must not exceed
 *              the allocated length of idx[i] and val[i].
 *   d          length of the dense output, d <= 2^32 - 1.
 *   dense_out  [out] fp32[d], fully overwritten.
 * An index outside [0, d) or an unsorted list never causes an out-of-bounds
 * access: the offending pair is skipped and EF_ERR_BAD_INPUT is latched.
 */
ef_status sparse_aggregate(uint32_t n, const uint32_t* const* idx,
                           const float* const* val, const uint32_t* counts,
                           uint64_t d, float* dense_out, ef_stream_t stream);

/*
 * sparse_aggregate_apply — the exchange step followed by the model update,
 * in one pass: the worker-ordered sum of sparse_aggregate is never written
 * to memory.
 *
 * Defines: with s[j] the sum of sparse_aggregate and Delta'[j] = alpha * s[j]
 * (rounded once; alpha = 1/n gives Algorithm 1's mean Delta_bar),
 *   m == NULL:  x[j] <- x[j] - Delta'[j]
 *               (Algorithm 1's model update x_{t+1} = x_t - Delta_bar_t);
 *   m != NULL:  m[j] <- fmaf(momentum, m[j], Delta'[j]),
 *               x[j] <- fmaf(-lr, Delta'[j] + m[j], x[j]), the sum rounded once
 *               (the Appendix's distributed EF SGD with momentum by gradient
 *               compression: m <- lambda m + Delta', x <- x - gamma (Delta' + m),
 *               the EF strategy of the paper's experiments).
 * The paper does not fix the rounding of these updates; these single
 * roundings are the library's definition, bit-identical with the oracle.
 *
 *   n, idx, val, counts, d   as for sparse_aggregate.
 *   alpha      scale of the sum, finite.
 *   x          [in/out] fp32[d], the model parameters (DEVICE pointer, 4-byte
 *              aligned; 16-byte alignment of x and m selects vector access).
 *   m          [in/out] fp32[d], the momentum state, or NULL for Algorithm 1.
 *   momentum   momentum factor (lambda of the Appendix algorithm), finite.
 *   lr         learning rate (gamma of the Appendix algorithm), finite.
 * x and m must not overlap each other or any idx/val list. Malformed lists
 * behave as in sparse_aggregate (pair skipped, EF_ERR_BAD_INPUT latched).
 */
ef_status sparse_aggregate_apply(uint32_t n, const uint32_t* const* idx,
                                 const float* const* val, const uint32_t* counts,
                                 uint64_t d, float alpha, float* x, float* m,
                                 float momentum, float lr, ef_stream_t stream);

/*
 * Tile index of a sparse message (an implementation device; the paper's
 * messages are the (index, value) lists alone). The coordinates [0, d) are cut
 * into T = ceil(d / EF_TILE) tiles of EF_TILE coordinates; a message's tile
 * index is uint32[T + 1] with
 *     tiles[t] = the number of its pairs with index < EF_TILE * t, t < T,
 *     tiles[T] = its count.
 * The aggregation works tile by tile and otherwise finds these positions by a
 * binary search of every list at every tile boundary (one more kernel, whose
 * chains of dependent loads make it latency-bound); the hard-threshold kernel
 * knows them as it places the pairs and writes them for T + 1 words. A worker
 * can send the tile index with its message (4 (T + 1) bytes against 8 bytes per
 * pair).
 *
 * ef_hard_threshold_tiled — ef_hard_threshold_ex (identical outputs) that also
 * writes the message's tile index.
 *   tiles_out  [out] uint32[ceil(d / EF_TILE) + 1], 4-byte aligned, device,
 *              not overlapping any other argument; required (non-NULL).
 *
 * sparse_aggregate_tiled, sparse_aggregate_apply_tiled — sparse_aggregate and
 * sparse_aggregate_apply (identical outputs for well-formed input) given the
 * lists' tile indexes.
 *   tiles      HOST array of n DEVICE pointers; tiles[i] is list i's tile index
 *              (uint32[ceil(d / EF_TILE) + 1], 4-byte aligned).
 * A tile index that does not match its list never causes an out-of-bounds
 * access: every position is clamped to [0, counts[i]], and a pair read for a
 * tile it does not belong to is skipped and latches EF_ERR_BAD_INPUT.
 */
#define EF_TILE 4096
ef_status ef_hard_threshold_tiled(const void* g, ef_grad_type g_type, float* e, float gamma,
                                  float lambda, uint64_t d, uint32_t* idx_out, float* val_out,
                                  uint32_t* count_out, uint32_t* tiles_out, double* err_sq_out,
                                  ef_stream_t stream);
ef_status sparse_aggregate_tiled(uint32_t n, const uint32_t* const* idx,
                                 const float* const* val, const uint32_t* const* tiles,
                                 const uint32_t* counts, uint64_t d, float* dense_out,
                                 ef_stream_t stream);
ef_status sparse_aggregate_apply_tiled(uint32_t n, const uint32_t* const* idx,
                                       const float* const* val, const uint32_t* const* tiles,
                                       const uint32_t* counts, uint64_t d, float alpha,
                                       float* x, float* m, float momentum, float lr,
                                       ef_stream_t stream);

/*
 * ef_hard_threshold_noalloc — ef_hard_threshold for callers that cannot
 * allocate device memory. (An implementation convenience; the paper has no
 * counterpart.)
 *
 * The other entry points grow a per-stream workspace with cudaMalloc, which
 * also synchronises the stream once. Some callers cannot allow that: their
 * device memory is owned entirely by their own allocator or a framework's
 * caching pool, they run under a fixed device-memory budget, or they sit in a
 * loop that must never block in cudaMalloc/cudaFree. This entry point computes
 * exactly the same result as ef_hard_threshold (same arguments, same bits)
 * with a fixed scratch array that is part of the library image; it calls no
 * cudaMalloc, cudaFree or allocating library routine.
 *
 *   g, e, gamma, lambda, idx_out, val_out, count_out   as for ef_hard_threshold
 *                (fp32 gradient only).
 *   d          0 <= d <= 268,435,456 (2^28); larger d returns
 *              EF_ERR_INVALID_ARG and launches nothing.
 *   status_out [out, optional] one uint32 in device memory, or NULL: after
 *              the call it holds the device-side error bits of this call
 *              (0 = success; nonzero = a bounded wait ran out or an output
 *              position overflowed). ef_check_status() does not see them.
 *              It must not overlap g, e, idx_out, val_out or count_out
 *              (EF_ERR_INVALID_ARG otherwise, nothing launched).
 *
 * The scratch (512 KiB + 256 bytes) is held on every device that loads the
 * library until the process exits. The first call on a device looks up the
 * scratch's device address; make that first call before any stream capture.
 * All calls on one device share the scratch: calls that overlap on the GPU
 * (on different streams, or from host threads without ordering between them)
 * race and must not be made. The scratch keeps the last call's contents;
 * each call clears what must start at zero. The test hook
 * ef_test_set_lookback_fault applies to this entry too. Testing aid: the
 * environment variable EF_NOALLOC_FIRST_EPOCH, read at a device's first call,
 * starts the per-call tag count there (it wraps at 2^30 - 1).
 */
ef_status ef_hard_threshold_noalloc(const float* g, float* e, float gamma, float lambda,
                                    uint64_t d, uint32_t* idx_out, float* val_out,
                                    uint32_t* count_out, uint32_t* status_out,
                                    ef_stream_t stream);

/*
 * ef_check_status — synchronise `stream`, then return and clear the device-side
 * error latched by earlier calls on that stream (EF_OK if none).
 */
ef_status ef_check_status(ef_stream_t stream);

/* ef_status_string — static, human-readable name of a status code. */
const char* ef_status_string(ef_status status);

/*
 * ef_workspace_release — synchronise the device and free every workspace the
 * library holds on the current device. Later calls re-create them.
 */
ef_status ef_workspace_release(void);

/*
 * ef_kernel_launches — number of kernels this library has launched in this
 * process (all devices, all streams). For accounting in benchmarks.
 */
uint64_t ef_kernel_launches(void);

/*
 * ef_test_set_lookback_fault — test hook for the bounded waits of the
 * ordered-compaction scan. When withheld_tile >= 0, the next compaction
 * launches on any stream make that tile never publish its count, so its
 * successors' waits run out after about spin_limit_us microseconds; they then
 * latch EF_ERR_TIMEOUT, skip their pair writes and finish. withheld_tile < 0
 * restores normal operation (the default). Never needed in production.
 */
void ef_test_set_lookback_fault(int64_t withheld_tile, uint32_t spin_limit_us);

/*
 * ef_test_set_stream_kernel — test hook choosing the streaming kernel of the
 * hard-threshold step and of the Top-k and layer-wise Top-k candidate passes
 * (16-byte aligned g and e): 0 (the default) by size (claimed groups of tiles
 * with look-back from 4096 tiles, 16,777,216 coordinates, on; static chunks
 * below; for the hard-threshold step, a shallower ring with larger pair
 * buffers once an earlier call on the same stream sent at least 1/12 of its
 * coordinates), 1 static chunks, 2 claimed groups, 3 claimed groups with the
 * shallower ring (hard-threshold; the candidate passes treat 3 as 2). Any
 * other value means 0. The results are the same whichever kernel runs; the
 * hook lets tests run each on small inputs. Process-wide; never needed in
 * production.
 */
void ef_test_set_stream_kernel(int mode);

#ifdef __cplusplus
}
#endif

#endif /* EFSPARSE_H */
