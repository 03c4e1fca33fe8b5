/*
 * pro_router.h — C ABI of the GB300 data path of Pro-Router's token-aware
 * verifier (arXiv 2608.28726, Section 3.1).
 *
 * The verifier reads, for every generated token t, the small model's logit row
 * x_t over the vocabulary (V entries) and reduces it to the per-token features
 * of Eq. 3:
 *     l_t   = log p_t(y_t)            the emitted token's log-probability
 *     m_t   = max_v p_t(v)            maximum probability
 *     h_t   = -H_t^K,  H_t^K = -sum_{v in top-K} p_t(v) log p_t(v),  K = 20
 *     rho_t = t / T                   position fraction (t is 1-based)
 * with p_t = softmax(x_t).  The data path also reports the probability margin
 * p(i1) - p(i2) between the first two tokens, the full-vocabulary entropy H,
 * log-sum-exp and the two top indices.  Per request (a ragged run of T rows)
 * the features are pooled, scored by a linear scorer and thresholded: a
 * request ships when its confidence is >= tau (Section 3.1, the ship rule
 * "p >= tau"); otherwise it escalates to the large model.
 *
 * Conventions shared by every call
 *   - Pointers named as device buffers are caller-owned CUDA device memory on
 *     the context's device; the library never frees them.  The library
 *     allocates only inside a context (pr_ctx_create) and, for
 *     pr_route_host, a staging area held by the context.
 *   - Calls are asynchronous on the caller's CUDA stream (`stream` is a
 *     cudaStream_t; NULL is the legacy default stream) unless stated.
 *   - Argument and launch problems return a pr_status; problems in the data
 *     (non-finite rows, bad token ids, bad offsets) never trap: they set the
 *     PR_FLAG_* bits in the per-row / per-request flag outputs and in the
 *     context's flag word (pr_ctx_flags).
 *   - Logits are row-major [n_rows][row_stride] elements, bf16 or fp32;
 *     only the first `vocab` entries of a row count.  Any element alignment is
 *     accepted; rows whose start is 16-byte aligned (base pointer and
 *     row_stride * element size multiples of 16) take the vector path.
 *   - Token ids are int32 (V < 2^31); request offsets are int64 CSR: request r
 *     owns rows [offsets[r], offsets[r+1]).
 *   - Features are written as PR_NFEAT floats per row, in the order of the
 *     PR_F_* slot names; pooled aggregates as PR_NAGG floats per request in
 *     the order of the PR_A_* slot names.
 *   - A row with NaN or +inf, or with no finite entry, has NaN features and
 *     top indices -1 (PR_FLAG_NONFINITE); -inf is a masked token with p = 0.
 *     A request with such a row, or with an out-of-range token id, has NaN
 *     aggregates and score and does not ship.  An empty request (T = 0) has
 *     NaN aggregates, score 0 and does not ship (PR_FLAG_EMPTY_REQ).
 *   - All floating-point accumulation is fp32.
 */
#ifndef PRO_ROUTER_H
#define PRO_ROUTER_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PR_OK = 0,
  PR_ERR_INVALID_ARG = -1, /* a null, negative, out-of-range or misaligned argument */
  PR_ERR_UNSUPPORTED = -2, /* a device or mode this library cannot run */
  PR_ERR_CUDA = -3,        /* a CUDA runtime call failed; see pr_last_cuda_error */
  PR_ERR_NO_MEMORY = -4    /* a context allocation failed */
} pr_status;

typedef enum { PR_DTYPE_F32 = 0, PR_DTYPE_BF16 = 1 } pr_dtype;

/* flag bits written on the device (never a trap) */
#define PR_FLAG_NONFINITE 1u   /* NaN or +inf in the row, or no finite entry */
#define PR_FLAG_BAD_CHOSEN 2u  /* emitted token id outside [0, vocab): l = NaN */
#define PR_FLAG_EMPTY_REQ 4u   /* request with T = 0 */
#define PR_FLAG_BAD_OFFSETS 8u /* offsets not monotone / outside the row range */
#define PR_FLAG_BAD_SLOT 16u   /* decode slot id outside [0, n_slots) */
#define PR_FLAG_TIMEOUT 32u    /* a bounded device-side wait ran out: that call's outputs are
                                  not valid (context flag word only) */

/* per-row feature record, PR_NFEAT floats */
#define PR_NFEAT 8
#define PR_F_LOGP 0   /* l = log p(y)              (Eq. 3) */
#define PR_F_MAXP 1   /* m = max_v p(v)            (Eq. 3) */
#define PR_F_MARGIN 2 /* p(i1) - p(i2) */
#define PR_F_ENT 3    /* H = -sum_v p log p        (full vocabulary) */
#define PR_F_TOPK 4   /* h = -H^K                  (Eq. 3, K = topk) */
#define PR_F_RHO 5    /* rho = t / T               (Eq. 3) */
#define PR_F_LSE 6    /* log sum_v exp(x_v) */
#define PR_F_X1 7     /* x_{i1}, the largest logit */

/* per-request pooled aggregates, PR_NAGG floats: mean / min over t */
#define PR_NAGG 11
#define PR_A_MEAN_LOGP 0
#define PR_A_MIN_LOGP 1
#define PR_A_MEAN_MAXP 2
#define PR_A_MIN_MAXP 3
#define PR_A_MEAN_MARGIN 4
#define PR_A_MIN_MARGIN 5
#define PR_A_MEAN_NEGENT 6 /* mean of -H */
#define PR_A_MIN_NEGENT 7  /* min of -H */
#define PR_A_MEAN_TOPK 8   /* mean of h */
#define PR_A_MIN_TOPK 9    /* min of h */
#define PR_A_MEAN_RHO 10   /* (T + 1) / (2T) */

#define PR_MAX_TOPK 32 /* largest K accepted (the paper uses K = 20) */

/* options (pr_ctx_set_option) */
#define PR_OPT_TOPK 0        /* K of the top-K entropy for pr_route / pr_decode_step; default 20 */
#define PR_OPT_TOPK_RENORM 1 /* 0 (default): raw p over the top K; 1: renormalised over the top K */
#define PR_OPT_SPLIT 2       /* CTAs per row (thread-block cluster): 0 = automatic, or 1, 2, 4, 8;
                                1 runs the persistent kernel (rows of more than 2^16 tiles of
                                1,024 x 16 bytes take one CTA per row instead) */
#define PR_OPT_OVERLAP 3     /* 1: a call may start while the previous kernel on its stream is
                                still running (programmatic dependent launch): it reads its
                                inputs at once and waits for that kernel before writing
                                anything.  Only for callers whose inputs are complete before
                                the preceding kernel starts (e.g. back-to-back verifier calls
                                on resident logits).  Default 0. */
#define PR_OPT_TIMING 4      /* 1: the calls after the verifier's (pr_head_score,
                                pr_quantile_score, pr_selective_metrics, pr_lmhead_features)
                                record a CUDA event after each kernel, for
                                pr_ctx_kernel_times; the kernels then no longer overlap one
                                another.  Default 0. */

typedef struct pr_ctx pr_ctx;

/* ---- context -------------------------------------------------------------- */

/*
 * Create a context on CUDA device `device`.  It owns the workspace of the
 * fused and incremental calls: per-row records for up to `max_rows` rows of
 * one routed batch (pr_route's global row index, row_base + local row, must
 * stay below it), per-request completion counters for up to `max_requests`
 * requests, and `max_requests` decode slots (pr_decode_step).  Everything is
 * zeroed.  Synchronous.  Returns PR_ERR_INVALID_ARG for a null `ctx`, a
 * negative size or a bad device, PR_ERR_NO_MEMORY if an allocation fails.
 */
pr_status pr_ctx_create(pr_ctx** ctx, int device, int64_t max_rows, int32_t max_requests);

/* Free the context and its workspace (synchronises the device first). */
pr_status pr_ctx_destroy(pr_ctx* ctx);

/* Zero counters, decode slots and the flag word, on `stream`.  Needed only
 * after a call that was given inconsistent offsets, slots or row ranges. */
pr_status pr_ctx_reset(pr_ctx* ctx, void* stream);

/* Set an option (PR_OPT_*).  Takes effect for calls issued afterwards. */
pr_status pr_ctx_set_option(pr_ctx* ctx, int32_t option, int32_t value);

/*
 * OR of every flag bit any call on this context has raised since the last
 * clear.  Synchronises `stream`.  With `clear` != 0 the word is zeroed.
 */
pr_status pr_ctx_flags(pr_ctx* ctx, void* stream, int32_t clear, uint32_t* flags);

/*
 * The same word without a stream: waits for all work on the context's device
 * (cudaDeviceSynchronize), then stores in *flags the OR of every flag bit the
 * context's calls have raised since the last clear or reset, leaving the word
 * as it is.  For callers that issue work on several streams and want one
 * check at the end of a batch.
 */
pr_status pr_last_error(pr_ctx* ctx, uint32_t* flags);

/*
 * Per-kernel device times (milliseconds, launch order) of the last call made
 * with PR_OPT_TIMING = 1: for pr_head_score the embedding, the first QKV
 * projection, then per layer the attention and the row-local block, then the
 * pool; for pr_selective_metrics the key transform, per radix pass the
 * histogram, digit scan and scatter, then the label prefix, the tile scan,
 * the metrics (with labels) and the final reduction.  Waits for the call's last event.  Writes min(count, cap) values to
 * `ms` and the count to *n (0 if no timed call was made).
 */
pr_status pr_ctx_kernel_times(pr_ctx* ctx, float* ms, int32_t cap, int32_t* n);

/* ---- the three verifier calls ----------------------------------------------- */

/*
 * Per-token features (Eq. 3) of n_rows logit rows.
 *   logits     device, [n_rows][row_stride] elements of type `dt`
 *   vocab      V, 1 <= V <= row_stride, V < 2^31
 *   chosen     device int32 [n_rows], the emitted token y_t of each row
 *   topk       K in [1, PR_MAX_TOPK] (the paper's K = 20)
 *   offsets    device int64 [n_req + 1] or NULL; with offsets the position
 *              fraction rho = t/T is filled in, without it rho = 0
 *   feat       device float [n_rows][PR_NFEAT]           (output)
 *   top2       device int32 [n_rows][2] = {i1, i2}: the first two tokens in
 *              the order (value descending, index ascending); i2 = -1 if V = 1
 *   row_flags  device uint32 [n_rows]                     (output)
 * Every row is read once from device memory.  Uses the context's PR_OPT_SPLIT
 * and PR_OPT_TOPK_RENORM options.
 */
pr_status pr_token_features(pr_ctx* ctx, const void* logits, pr_dtype dt, int64_t n_rows,
                            int64_t vocab, int64_t row_stride, const int32_t* chosen,
                            int32_t topk, const int64_t* offsets, int32_t n_req, float* feat,
                            int32_t* top2, uint32_t* row_flags, void* stream);

/*
 * Pool per-row features into per-request aggregates, score and threshold
 * (Section 3.1: mean pool, sigmoid score, ship iff score >= tau).
 *   feat       device float [n_rows][PR_NFEAT] as written by pr_token_features,
 *              16-byte aligned
 *   row_flags  device uint32 [n_rows] or NULL (then no row is flagged)
 *   n_rows     rows in feat; a request reaching past it gets PR_FLAG_BAD_OFFSETS
 *   offsets    device int64 [n_req + 1]; rows [offsets[r], offsets[r+1]) are read
 *   w          device float [PR_NAGG], b: bias; z = w . a + b, score = sigmoid(z)
 *   tau        threshold in (0, 1); ship = (z >= log(tau / (1 - tau)))
 *   agg        device float [n_req][PR_NAGG] or NULL      (output)
 *   score      device float [n_req]                       (output)
 *   ship       device uint8 [n_req], 1 = ship, 0 = escalate (output)
 *   req_flags  device uint32 [n_req]                      (output)
 * Sums run in a fixed order per request, so results do not depend on timing.
 */
pr_status pr_aggregate_score(pr_ctx* ctx, const float* feat, const uint32_t* row_flags,
                             int64_t n_rows, const int64_t* offsets, int32_t n_req,
                             const float* w, float b, float tau, float* agg, float* score,
                             uint8_t* ship, uint32_t* req_flags, void* stream);

/*
 * Fused verification: logit rows -> ship / escalate, in one launch.  Rows are
 * rows [row_base, row_base + n_rows) of a batch whose requests are described
 * by `offsets` (global row indices, n_req + 1 entries, offsets[n_req] <=
 * max_rows).  A batch may be fed in several chunks on one stream, each call
 * with its own row_base, in any order, each row exactly once; a request that
 * straddles chunks is finished by the call that delivers its last row.  Per
 * request, when all its rows are done, the kernel that finished the last row
 * pools, scores and writes score / ship / req_flags (and agg if not NULL).
 * Empty requests are written by every call whose row range touches their
 * offset.  K and the entropy mode come from the context options.
 */
pr_status pr_route(pr_ctx* ctx, const void* logits, pr_dtype dt, int64_t row_base,
                   int64_t n_rows, int64_t vocab, int64_t row_stride, const int32_t* chosen,
                   const int64_t* offsets, int32_t n_req, const float* w, float b, float tau,
                   float* score, uint8_t* ship, uint32_t* req_flags, float* agg, void* stream);

/*
 * The same verification from HOST memory, end to end: the logits, token ids,
 * offsets and weights are host buffers (pinned memory copies fastest); rows
 * are copied to the device in chunks of `chunk_rows` rows through a
 * double-buffered staging area owned by the context, overlapped with the
 * fused kernel, and score / ship / req_flags (and agg if not NULL) are copied
 * back to the host buffers.  Synchronous: returns when the host outputs are
 * written.  chunk_rows >= 1; a chunk larger than the batch is taken as the
 * batch.  The staging area (2 chunks of rows and token ids) is allocated on
 * the first call and again whenever a larger chunk or another row size is
 * asked for (that call synchronises the device).
 */
pr_status pr_route_host(pr_ctx* ctx, const void* logits, pr_dtype dt, int64_t n_rows,
                        int64_t vocab, int64_t row_stride, const int32_t* chosen,
                        const int64_t* offsets, int32_t n_req, const float* w, float b, float tau,
                        int64_t chunk_rows, float* score, uint8_t* ship, uint32_t* req_flags,
                        float* agg, void* stream);

/* ---- incremental decode-step mode --------------------------------------------- */

/*
 * One decode step over n_live live requests, each in its own slot of the
 * context (0 <= slot < max_requests, no slot twice in one step).  Row i of
 * `logits` is the distribution that produced token chosen[i] of the request in
 * slot[i].  Each row's features are folded in place into that slot's running
 * accumulators (count, compensated sums, minima) in step order.  When eos[i]
 * is non-zero the request ends with this row: its aggregates (mean rho =
 * (T+1)/(2T)) are scored and thresholded, score_out / ship_out / slot_flags
 * (and agg_out if not NULL) at index slot[i] are written, and the slot is
 * cleared for the next request.  Output arrays have max_requests entries;
 * entries of slots that did not end in this step are left untouched.
 */
pr_status pr_decode_step(pr_ctx* ctx, const void* logits, pr_dtype dt, int32_t n_live,
                         int64_t vocab, int64_t row_stride, const int32_t* slot,
                         const int32_t* chosen, const uint8_t* eos, const float* w, float b,
                         float tau, float* score_out, uint8_t* ship_out, uint32_t* slot_flags,
                         float* agg_out, void* stream);

/*
 * Checkpoint of the decode slots.  pr_state_export with host_buf == NULL
 * stores the needed size in *bytes; otherwise it copies the state into
 * host_buf (*bytes must be at least that size).  pr_state_import restores a
 * state exported from a context with the same max_requests.  Both synchronise
 * the device.
 */
pr_status pr_state_export(pr_ctx* ctx, void* host_buf, size_t* bytes);
pr_status pr_state_import(pr_ctx* ctx, const void* host_buf, size_t bytes);

/* ---- transformer scorer head ------------------------------------------------------ */

#define PR_HEAD_D 64          /* model width */
#define PR_HEAD_HEADS 4       /* attention heads (width 16 each) */
#define PR_HEAD_FF 128        /* feed-forward width */
#define PR_HEAD_MAX_LAYERS 8  /* largest number of encoder layers accepted */

/* Number of floats of the head's weights for n_layers encoder layers
 * (67,329 for 2 layers); -1 if n_layers is outside [1, PR_HEAD_MAX_LAYERS]. */
int64_t pr_head_param_count(int32_t n_layers);

/*
 * The paper's learned scorer (Section 3.1) over per-request feature
 * sequences: for request r the T = offsets[r+1] - offsets[r] rows give
 * x_t = (l_t, m_t, h_t, rho_t) (record slots LOGP, MAXP, TOPK, RHO of Eq. 3);
 * h_0 = W_in x_t + b_in + PE(t) with the sinusoidal encoding PE(t)[2i] =
 * sin(t / 10000^(2i/64)), PE(t)[2i+1] = cos(same), t = 0 .. T-1; n_layers
 * post-norm transformer encoder layers (4-head self-attention, residual,
 * LayerNorm; ReLU feed-forward of width 128, residual, LayerNorm; eps 1e-5);
 * z = w_out . mean_t(h_L) + b_out; score = sigmoid(z); ship = (z >= logit(tau)).
 *   feat       device float [n_rows][PR_NFEAT], 16-byte aligned, e.g. from
 *              pr_token_features with offsets (so that rho is filled in)
 *   row_flags  device uint32 [n_rows] or NULL; a request with a row flagged
 *              PR_FLAG_NONFINITE or PR_FLAG_BAD_CHOSEN escalates with score NaN
 *   offsets    device int64 [n_req + 1], non-decreasing for valid requests; a
 *              request with offsets[r] < 0, offsets[r+1] < offsets[r] or
 *              offsets[r+1] > n_rows gets score NaN and PR_FLAG_BAD_OFFSETS;
 *              an empty request gets score 0 and PR_FLAG_EMPTY_REQ
 *   w          device float [pr_head_param_count(n_layers)], 16-byte aligned,
 *              in this order (matrices row-major, y = W x + b):
 *                W_in[64][4] b_in[64]
 *                per layer: W_qkv[192][64] (rows q, k, v) b_qkv[192]
 *                  W_o[64][64] b_o[64] g1[64] be1[64] W_1[128][64] b_1[128]
 *                  W_2[64][128] b_2[64] g2[64] be2[64]
 *                w_out[64] b_out
 *   score, ship, req_flags   device [n_req]            (outputs)
 * The batch runs layer by layer in 2 n_layers + 3 launches on `stream`.  The
 * contractions (the attention's Q K^T and P V, the projections and the
 * feed-forward) run on the tensor cores (tcgen05) with each fp32 operand
 * split into two TF32 parts and three products per product (errors below
 * 2^-21 of a product); the softmax, LayerNorm and the rest are fp32 on the
 * CUDA cores; all sums run in a fixed order, so results are bit-reproducible.  A
 * bounded wait on the tensor cores that runs out raises PR_FLAG_TIMEOUT in
 * the context's flag word (that call's outputs are invalid).  The
 * context holds a device scratch of 1 KB per row, allocated (or grown) by the
 * first call with more rows than before -- that call synchronises the device;
 * calls on different streams must not overlap (they share that scratch).
 */
pr_status pr_head_score(pr_ctx* ctx, const float* feat, const uint32_t* row_flags,
                        int64_t n_rows, const int64_t* offsets, int32_t n_req, const float* w,
                        int32_t n_layers, float tau, float* score, uint8_t* ship,
                        uint32_t* req_flags, void* stream);

/* ---- LM head fused with the row reduction --------------------------------------------- */

#define PR_LMHEAD_MAX_VOCAB 2147483392LL /* 2^31 - 256: largest vocab of the LM-head calls */

/*
 * pr_token_features without logits in memory: the rows' logits x = W h are
 * computed on the tensor cores (tcgen05, bf16 inputs, fp32 accumulation) and
 * reduced to the Eq. 3 row record in the GEMM's epilogue, so the [n_rows][V]
 * logit matrix is never written (Section 3.1: the features need nothing the
 * small model's decoding does not already compute).
 *   hidden   device bf16 [n_rows][d], row-major, 16-byte aligned (the final
 *            hidden states of the small model)
 *   weight   device bf16 [vocab][d], row-major, 16-byte aligned (the LM head;
 *            x_v = sum_k weight[v][k] hidden[row][k])
 *   vocab    1 <= V <= PR_LMHEAD_MAX_VOCAB (the kernel's 32-bit column
 *            arithmetic runs up to the end of V's last 256-column tile)
 *   d        hidden size, a multiple of 8, at most 2^20
 *   chosen, topk, offsets, n_req, feat, top2, row_flags: as pr_token_features
 * The record has pr_token_features' slots and conventions, computed from the
 * fp32 logits; uses the context's PR_OPT_TOPK_RENORM.  Two launches on
 * `stream` (the first in thread-block clusters of two CTAs sharing each
 * tcgen05 MMA); the context holds a state buffer of 288 bytes per row and
 * vocabulary split (grown on demand; that call synchronises the device).  A
 * device-side wait that runs out (2 s) raises PR_FLAG_TIMEOUT in the context
 * flag word.
 */
pr_status pr_lmhead_features(pr_ctx* ctx, const void* hidden, const void* weight, int64_t n_rows,
                             int64_t d, int64_t vocab, const int32_t* chosen, int32_t topk,
                             const int64_t* offsets, int32_t n_req, float* feat, int32_t* top2,
                             uint32_t* row_flags, void* stream);

/*
 * pr_decode_step without logits in memory: row i's logits x = W h_i are
 * computed from the hidden state of the token in slot[i] on the tensor cores
 * (as pr_lmhead_features) and its Eq. 3 features are folded into that slot
 * (as pr_decode_step: running count, compensated sums and minima in step
 * order; at eos[i] the request's aggregates are scored and thresholded, the
 * outputs at index slot[i] written and the slot cleared).
 *   hidden   device bf16 [n_live][d], row-major, 16-byte aligned
 *   weight   device bf16 [vocab][d], row-major, 16-byte aligned
 *   vocab    as pr_lmhead_features
 *   d        a multiple of 8, at most 2^20
 *   slot, chosen, eos, w, b, tau, score_out, ship_out, slot_flags, agg_out:
 *            as pr_decode_step (n_live <= the context's max_requests)
 * Uses the context's PR_OPT_TOPK and PR_OPT_TOPK_RENORM.  Two launches on
 * `stream`; the state buffer as pr_lmhead_features; PR_FLAG_TIMEOUT as there.
 */
pr_status pr_lmhead_decode_step(pr_ctx* ctx, const void* hidden, const void* weight,
                                int32_t n_live, int64_t d, int64_t vocab, const int32_t* slot,
                                const int32_t* chosen, const uint8_t* eos, const float* w,
                                float b, float tau, float* score_out, uint8_t* ship_out,
                                uint32_t* slot_flags, float* agg_out, void* stream);

/*
 * Failure-detection self-test: runs the bounded device-side wait that
 * pr_lmhead_features' kernels use on an mbarrier that nothing completes, with
 * a limit of `limit_ns` nanoseconds (0 .. 2e9) instead of 2 s.  *completed (host)
 * receives 0 when the wait ran out, and the run-out raises PR_FLAG_TIMEOUT in
 * the context flag word, exactly as a stalled pr_lmhead_features would; the
 * context stays usable.  One launch on the default stream, synchronous.
 */
pr_status pr_selftest_wait(pr_ctx* ctx, int64_t limit_ns, int32_t* completed);

/* ---- quantile-summary + MLP aggregator ------------------------------------------------ */

#define PR_QMLP_SUMMARY 28   /* summary length: 4 features x 7 quantile levels */
#define PR_QMLP_PARAMS 6081  /* weights of the 28 -> 64 -> 64 -> 1 MLP */

/*
 * The verifier-architecture ablation's alternative scorer (Section 4.2,
 * Table 2): an MLP over quantiles pooled per request.  Per request, for each feature x in
 * (l, m, h, rho) (record slots LOGP, MAXP, TOPK, RHO of Eq. 3) over its T
 * rows, the quantiles at levels 0, 1/10, 1/4, 1/2, 3/4, 9/10, 1 by linear
 * interpolation between order statistics (x_(0) <= ... <= x_(T-1); level a/b:
 * i = floor(a (T-1) / b), f = (a (T-1) mod b) / b, q = x_(i) + f (x_(i+1) -
 * x_(i))), then z = w3 . ReLU(W2 ReLU(W1 s + b1) + b2) + b3, score =
 * sigmoid(z), ship = (z >= logit(tau)).
 *   feat, row_flags, offsets, n_rows: as pr_head_score (flags escalate with
 *              score NaN, empty requests score 0, bad offsets PR_FLAG_BAD_OFFSETS)
 *   w          device float [PR_QMLP_PARAMS]: W1[64][28] b1[64] W2[64][64] b2[64]
 *              w3[64] b3 (row-major, y = W x + b)
 *   summary    device float [n_req][PR_QMLP_SUMMARY] or NULL: the quantiles,
 *              feature-major (written for requests that are scored)
 *   score, ship, req_flags   device [n_req]                     (outputs)
 * One launch, one CTA per request; requests of up to 256 rows are sorted in
 * registers (one warp per feature), up to 2,048 rows in shared memory, longer
 * ones use radix selection over global memory (exact, slower).  fp32,
 * fixed-order sums.  n_rows < 2^31; feat must be 16-byte aligned
 * (PR_ERR_INVALID_ARG otherwise).
 */
pr_status pr_quantile_score(pr_ctx* ctx, const float* feat, const uint32_t* row_flags,
                            int64_t n_rows, const int64_t* offsets, int32_t n_req, const float* w,
                            float tau, float* summary, float* score, uint8_t* ship,
                            uint32_t* req_flags, void* stream);

/* ---- operating point and selective-prediction metrics ------------------------------ */

typedef struct {
  float tau;           /* threshold: the k-th largest finite score; +inf when k = 0 */
  int32_t reserved;
  int64_t n_finite;    /* requests with a finite score (the others never ship) */
  int64_t k;           /* requests the coverage rule ships: min(floor(q n + 1/2), n_finite) */
  int64_t n_ship;      /* finite scores >= tau: k plus the ties at tau */
  int64_t n_pos;       /* correct answers among the finite-scored requests (0 without labels) */
  double auroc;        /* P(correct scores above incorrect), ties 1/2; NaN without both classes */
  double auarc;        /* area under accuracy-among-shipped vs ship rate; NaN without labels */
  double acc_shipped;  /* accuracy among the n_ship requests with score >= tau */
} pr_selective;

/*
 * Calibrate the operating point on a validation pool and score the ranking
 * (Section 3.1: tau is fixed in advance on a validation pool; Section 4.1:
 * the coverage rule of selective prediction fixes a ship fraction q, and
 * AUROC and AUARC, the area under accuracy-of-what-ships against ship rate,
 * measure the ranking).
 *   scores  device float [n], e.g. the score output of pr_route or
 *           pr_head_score; non-finite entries (flagged requests) never ship
 *           and are left out of the metrics
 *   labels  device uint8 [n] (non-zero = correct) or NULL (calibration only;
 *           with the pairwise label the AUARC field is the paper's AUACC)
 *   n       0 <= n < 2^31;  q: ship fraction in [0, 1]
 *   out     host struct, written before the call returns
 * A tie group's order is undefined, so AUARC spreads its correct answers
 * evenly over its ranks (the expectation over orders) and AUROC counts ties
 * as 1/2.  Runs as one stable radix sort of the scores plus scans on
 * `stream` (17 kernels) and synchronises it; results are deterministic.  The
 * context holds a sort workspace of about 15 bytes per score, allocated (or
 * grown) by the first call with more scores than before -- that call
 * synchronises the device.
 */
pr_status pr_selective_metrics(pr_ctx* ctx, const float* scores, const uint8_t* labels, int64_t n,
                               double q, pr_selective* out, void* stream);

/* ---- verification without allocation ------------------------------------------------- */

#define PR_NOALLOC_MAX_ROWS 16384    /* largest n_rows pr_route_noalloc accepts */
#define PR_NOALLOC_MAX_REQUESTS 1024 /* largest n_req pr_route_noalloc accepts */

/*
 * pr_route without a context and without allocating anything.  The paper has
 * no counterpart: this call exists for hosts that cannot let a library call
 * cudaMalloc -- an inference engine that reserves the GPU's memory for its own
 * pool at start-up (so a later cudaMalloc fails or fragments that pool), or a
 * serving loop that must not take the device-wide synchronisation a cudaMalloc
 * or cudaFree can imply while other streams are running.
 *
 * It does what pr_route does for a whole batch in one call (row_base 0, no
 * chunking), with K = 20 and the raw top-K entropy, on the current CUDA
 * device.  The caller still passes every input and output buffer (device
 * memory, the same layouts as pr_route).  The per-row records and request
 * counters live in a fixed scratch array compiled into the library: each
 * device that loads it keeps that array (about 580 KB) until the process
 * exits.  Limits: 1 <= n_rows <= PR_NOALLOC_MAX_ROWS and
 * 1 <= n_req <= PR_NOALLOC_MAX_REQUESTS; larger batches are rejected with
 * PR_ERR_INVALID_ARG before anything is queued (use pr_route with a context
 * instead).  The offsets must cover the batch exactly, offsets[n_req] ==
 * n_rows: there is no flag word the caller could read afterwards, so a
 * request reaching past n_rows gets PR_FLAG_BAD_OFFSETS, and when
 * offsets[n_req] < n_rows the last request is reported with
 * PR_FLAG_BAD_OFFSETS and a NaN score while the rows after offsets[n_req],
 * which belong to no request, are not verified.
 *
 * The first call on a device looks up the scratch array's device address and
 * the launch shape, once, with that device current; make that first call
 * before any stream capture.  The address is kept for the life of the
 * process: after cudaDeviceReset (which unloads the library's device code)
 * this call must not be used on that device again.  Every call clears the counters it needs on
 * `stream` and then reuses the same array, which keeps the previous call's
 * contents: two calls whose work overlaps on the GPU (different streams, no
 * ordering between them) race on the scratch and give undefined results.
 * Calls issued on one stream, or otherwise ordered, are safe.
 */
pr_status pr_route_noalloc(const void* logits, pr_dtype dt, int64_t n_rows, int64_t vocab,
                           int64_t row_stride, const int32_t* chosen, const int64_t* offsets,
                           int32_t n_req, const float* w, float b, float tau, float* score,
                           uint8_t* ship, uint32_t* req_flags, float* agg, void* stream);

/* ---- the prompt pre-scorer (host CPU) ----------------------------------------------- */

/*
 * Pro-Router's first stage (Section 3.1, Eq. 2): before any token is
 * generated a logistic regression over cheap prompt features guides the
 * request, p_pre(x) = sigmoid(w . phi(x) + b), phi(x) = [TF-IDF vector of the
 * prompt text, image count, prompt length].  The paper keeps this step off
 * the accelerator; these calls run on the host CPU and touch no device.
 *
 * Readings of what the paper leaves open: a token is a maximal run of word
 * bytes ([0-9A-Za-z_] and every byte >= 0x80) at least two bytes long, ASCII
 * letters lowercased; the vocabulary is every term of the fitting corpus with
 * document frequency >= min_df, columns in byte order of the terms; tf is the
 * raw count, idf = ln((1 + n) / (1 + df)) + 1 (n documents), the row tf * idf
 * is scaled to unit Euclidean length (a prompt without vocabulary terms has a
 * zero row); the length is the prompt's token count (in or out of the
 * vocabulary).  Sums run in double precision in ascending column order.
 *
 * pr_prescorer_fit: vocabulary and idf of n_docs NUL-terminated texts (host
 *   pointers, read during the call only).  *out receives a new pre-scorer,
 *   owned by the caller (pr_prescorer_destroy).  PR_ERR_INVALID_ARG for a
 *   NULL text, n_docs < 0 or min_df < 1; PR_ERR_NO_MEMORY if an allocation fails.
 * pr_prescorer_vocab_size: V, the number of TF-IDF columns (-1 for NULL).
 * pr_prescorer_term: the term of a column (NUL-terminated, owned by the
 *   pre-scorer), NULL outside [0, V).
 * pr_prescorer_features: phi of one prompt: the nonzero TF-IDF entries in
 *   ascending column order into columns / values (host arrays of cap
 *   entries), their count into *nnz and the token count into *length;
 *   PR_ERR_INVALID_ARG (with *nnz set) when cap is too small.
 * pr_prescorer_score: for each of n prompts (host NUL-terminated texts) with
 *   n_images[i] >= 0 images, score[i] = p_pre and, if logit is not NULL,
 *   logit[i] = w . phi + b.  w: host float [V + 2] (V TF-IDF weights, then the
 *   image-count weight, then the length weight).  n_threads host threads (0:
 *   all hardware threads); the results do not depend on it.  Thread-safe for
 *   concurrent calls on one pre-scorer (it is only read).
 */
typedef struct pr_prescorer pr_prescorer;
pr_status pr_prescorer_fit(const char* const* docs, int32_t n_docs, int32_t min_df,
                           pr_prescorer** out);
void pr_prescorer_destroy(pr_prescorer* ps);
int64_t pr_prescorer_vocab_size(const pr_prescorer* ps);
const char* pr_prescorer_term(const pr_prescorer* ps, int64_t column);
pr_status pr_prescorer_features(const pr_prescorer* ps, const char* prompt, int32_t cap,
                                int32_t* columns, float* values, int32_t* nnz, int64_t* length);
pr_status pr_prescorer_score(const pr_prescorer* ps, const char* const* prompts,
                             const int32_t* n_images, int32_t n, const float* w, float b,
                             int32_t n_threads, float* score, float* logit);

/* ---- diagnostics ------------------------------------------------------------------ */

/* Static description of a status code. */
const char* pr_status_string(pr_status status);

/* The CUDA error string of the last PR_ERR_CUDA on this thread ("" if none). */
const char* pr_last_cuda_error(void);

/* Number of kernel launches this library has issued in this process. */
uint64_t pr_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* PRO_ROUTER_H */
