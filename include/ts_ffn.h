/*
 * ts_ffn.h -- C ABI of libtsffn: the decode-time activation-sparse dReLU FFN
 * of Turbo Sparse (arXiv 2406.05955) on one GB300 (sm_103a).
 *
 * The operation (Eq. 1 in Sec. 2 with the dReLU of Eq. 2 in Sec. 3.2):
 *     g = x W_gate,  u = x W_up,  c = max(0, g) * max(0, u),  y = c W_down
 * Only neurons with g_j > 0 cost W_up bytes and only neurons with g_j > 0 and
 * u_j > 0 ("active", the non-zero activations counted in Sec. 6.2) cost
 * W_down bytes; the result equals the dense formula.
 *
 * Layout. All three weight matrices are neuron-major, [m][d] row-major:
 * row j of w_gate / w_up is neuron j's input weights (column j of the paper's
 * d x m matrices), row j of w_down is neuron j's output row (row j of the
 * paper's m x d W_down). Activations x are [batch][d] in the weight dtype;
 * outputs y and the residual stream h are [batch][d] fp32. Rows of every
 * weight matrix must start on 16-byte boundaries (pointer 16-byte aligned
 * and d * sizeof(element) a multiple of 16).
 *
 * Ownership. Weights, x, y, h and index lists are caller-owned device
 * memory; a handle borrows the weight pointers (they must outlive it) and
 * owns only its scratch, allocated once by *_create.
 *
 * Execution. Every *_forward call is asynchronous on `stream`, performs no
 * host synchronisation and no allocation, and may be captured in a CUDA
 * graph. One forward may be in flight per handle at a time.
 *
 * Errors. Argument errors are returned synchronously and nothing is
 * launched. Errors the GPU detects (an out-of-range or unsorted index list)
 * never trap: the offending entries are skipped, a status word in the
 * handle's scratch records it, and ts_*_get_error reports it.
 */
#ifndef TS_FFN_H
#define TS_FFN_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    TS_OK = 0,
    TS_ERR_INVALID_ARG = 1,  /* bad pointer, size, alignment or batch       */
    TS_ERR_CUDA = 2,         /* a CUDA runtime call failed                   */
    TS_ERR_OOM = 3,          /* scratch allocation failed                    */
    TS_ERR_BAD_INDEX = 4,    /* the GPU saw an out-of-range/unsorted list    */
    TS_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up           */
    TS_ERR_UNSUPPORTED = 6,  /* valid request this build does not handle     */
    TS_ERR_SCRATCH = 7       /* a scratch guard zone was overwritten         */
} ts_status;

/*
 * Weight storage. TS_F32 and TS_BF16 rows hold d elements. TS_INT4 rows (the
 * weight-only 4-bit storage of the paper's INT4 models, Tables 7-9) hold d/2
 * bytes of 4-bit codes followed by d/32 little-endian IEEE binary16 scales,
 * one per group of 32 consecutive elements: weight i = scale[i/32] *
 * (code[i] - 8). Group G's codes are the 16 bytes at offset 16G, read as four
 * little-endian 32-bit words w0..w3; element 8s + 2t + h of the group
 * (s, t in 0..3, h in 0..1) is nibble s + 4h of word t, i.e. bits
 * [4(s + 4h), 4(s + 4h) + 4) of w_t (the order in which one tensor-core lane
 * consumes them). An INT4 row is 9d/16 bytes and needs d to be a multiple of
 * 256; its activations x are bf16.
 */
typedef enum { TS_F32 = 0, TS_BF16 = 1, TS_INT4 = 2 } ts_dtype;

typedef struct ts_ffn ts_ffn;     /* one dReLU FFN (one layer or one expert) */
typedef struct ts_moe ts_moe;     /* one top-k MoE layer over ts_ffn experts */
typedef struct ts_graph ts_graph; /* a captured multi-layer forward          */
typedef struct ts_predictor ts_predictor; /* one layer's activation predictor */

/* Human-readable name of a status code (static string, never NULL). */
const char* ts_status_str(ts_status s);

/* ABI version of this library (major * 100 + minor). */
int ts_version(void);

/*
 * Create a handle for one dReLU FFN (Eq. 1 + Eq. 2).
 *   d, m       model width and number of neurons (d >= 1, m >= 1)
 *   wdtype     storage type of the weights (and of x, except INT4: bf16 x)
 *   w_gate, w_up, w_down  device pointers, [m][d] each, or [m][9d/16] bytes
 *              for TS_INT4 (borrowed)
 *   max_batch  largest batch a forward may pass (1..64); INT4 handles run
 *              passes of up to 2 tokens
 * Allocates the handle's scratch on the current device.
 * Returns TS_ERR_INVALID_ARG for bad sizes/pointers/alignment, TS_ERR_OOM if
 * scratch cannot be allocated, TS_ERR_CUDA for other CUDA failures.
 */
ts_status ts_ffn_create(ts_ffn** out, int d, int m, ts_dtype wdtype, const void* w_gate,
                        const void* w_up, const void* w_down, int max_batch);
void ts_ffn_destroy(ts_ffn* h);

/*
 * y = dReLU-FFN(x) for `batch` tokens (Eq. 1 + Eq. 2), on `stream`.
 *   x          device [batch][d], wdtype
 *   y          device [batch][d] fp32, overwritten
 *   active_idx NULL: the active sets are detected from the signs of g and u.
 *              Otherwise a device list of n_active neuron ids (0 <= n_active
 *              <= m), strictly ascending, shared by every token of the
 *              batch: the predictor-driven mode of Sec. 7. Gate, up and
 *              down then touch only listed rows, and listed neurons that
 *              are not dReLU-active contribute 0; unlisted neurons are
 *              skipped even if they would be active.
 * batch == 0 is a no-op. Equivalent to ts_ffn_gate_up then ts_ffn_down.
 */
ts_status ts_ffn_forward(ts_ffn* h, const void* x, int batch, float* y, cudaStream_t stream,
                         const int32_t* active_idx, int n_active);

/*
 * y = (Combined(x) * Mask(x)) W_down with the top-k magnitude mask of Eq. 3
 * and Eq. 4 (Sec. 3.2): per token, Mask keeps the `keep` neurons with the
 * largest |Combined| = max(0, g) max(0, u) (Eq. 2), a lower neuron index
 * winning a tie; the others contribute 0.
 *   x, batch, y, stream   as ts_ffn_forward (no predictor list)
 *   keep                  0 <= keep <= m; keep >= the number of dReLU-active
 *                         neurons gives ts_ffn_forward's result up to the
 *                         fp32 summation order of the down projection (the
 *                         masked path gathers W_down by column slices)
 * The per-token both-active sets that ts_ffn_get_active reports afterwards
 * are the kept active neurons. The selection compares the fp32 c values.
 * Errors: TS_ERR_INVALID_ARG for a bad keep or batch, TS_ERR_UNSUPPORTED for
 * INT4 rows.
 */
ts_status ts_ffn_forward_topk(ts_ffn* h, const void* x, int batch, float* y, cudaStream_t stream, int keep);

/*
 * First step alone: gate GEMV + ReLU + compaction, then the gathered up
 * projection over gate-active rows + dReLU product + second compaction
 * (into the handle's scratch). Arguments as ts_ffn_forward. For batch > 8
 * the steps run in passes of 8 tokens and ts_ffn_forward must be used.
 */
ts_status ts_ffn_gate_up(ts_ffn* h, const void* x, int batch, cudaStream_t stream,
                         const int32_t* active_idx, int n_active);

/* Second step alone: gathered down projection of the rows the preceding
   ts_ffn_gate_up on this handle marked active; writes y [batch][d] fp32. */
ts_status ts_ffn_down(ts_ffn* h, int batch, float* y, cudaStream_t stream);

/*
 * Pre-norm residual stack of n_layers FFNs on the fp32 residual h [batch][d]
 * (updated in place): for each layer l,
 *     x = round_wdtype(h / sqrt(mean(h^2) + 1e-5)),  x[d-1] = 1,
 *     h = h + FFN_l(x).
 * (The normalisation and bias channel are synthetic glue: the paper studies
 * the FFN alone.) active_idx / n_active: NULL, or per-layer lists as in
 * ts_ffn_forward (an entry may be NULL). All layers need the same d, wdtype.
 */
ts_status ts_stack_forward(ts_ffn* const* layers, int n_layers, float* h, int batch,
                           cudaStream_t stream, const int32_t* const* active_idx,
                           const int* n_active);

/*
 * Active sets of the last forward on this handle, copied to host memory
 * (synchronises `stream`). token >= 0 selects one token, -1 the union over
 * the batch. gate_idx / both_idx are host arrays of at least m entries
 * (either may be NULL); the lists come back ascending (neuron ids).
 */
ts_status ts_ffn_get_active(ts_ffn* h, cudaStream_t stream, int token, int32_t* gate_idx,
                            int* n_gate, int32_t* both_idx, int* n_both);

/* Synchronise `stream`, return and clear the device status word:
   TS_OK, TS_ERR_BAD_INDEX, or TS_ERR_TIMEOUT (a bounded device-side wait ran
   out; the kernels wound down instead of hanging and the results of that
   forward are undefined). */
ts_status ts_ffn_get_error(ts_ffn* h, cudaStream_t stream);

/*
 * Scratch guard check (a debugging aid, not part of the method). Every block
 * of a handle's device scratch (partial sums, bitmaps, c values, status
 * word, ...) is followed by a guard zone filled with one byte value when the
 * handle is created. This call synchronises `stream` and compares every zone
 * with its fill: TS_OK if all are intact, TS_ERR_SCRATCH if a kernel wrote
 * past the end of a block, TS_ERR_INVALID_ARG for a NULL handle.
 * ts_ffn_poke_guard overwrites one byte of guard zone i (0 <= i < the number
 * of blocks; TS_ERR_INVALID_ARG otherwise) from the host, so that a test can
 * check that the check fires; the handle stays usable.
 */
ts_status ts_ffn_check_scratch(ts_ffn* h, cudaStream_t stream);
ts_status ts_ffn_poke_guard(ts_ffn* h, int i);

/*
 * Test hook for the failure-detection path (not part of the method): while
 * `on` is nonzero, forwards on this handle make one consumer warp of every
 * gate+up CTA wait on a barrier that nothing arrives at. The wait, like every
 * device-side wait of the library, gives up after about one second, records
 * TS_ERR_TIMEOUT in the status word and lets the kernels wind down, so the
 * CUDA context stays usable. Such a forward takes a few seconds and its
 * output is undefined. Returns TS_ERR_INVALID_ARG for a NULL handle.
 */
ts_status ts_ffn_set_test_stall(ts_ffn* h, int on);

/*
 * One FFN forward with no handle and no device allocation. The paper has no
 * counterpart: this is a calling convention, not part of the method. It
 * computes exactly what ts_ffn_forward computes, with the same kernels, for
 * callers that cannot allocate device memory when they run the FFN (a memory
 * pool that is full or must not grow, code that must not take the implicit
 * device synchronisation of cudaFree, a plain C caller with nowhere to keep
 * a handle).
 *   d, m, wdtype, w_gate, w_up, w_down   as ts_ffn_create (borrowed for the call)
 *   x, batch, y, stream, active_idx, n_active   as ts_ffn_forward
 * Scratch: a fixed array of the library's static device memory (~0.8 MB per
 * device), sized for m <= TS_NOALLOC_MAX_M and batch <= TS_NOALLOC_MAX_BATCH;
 * larger sizes return TS_ERR_UNSUPPORTED and launch nothing. Nothing is
 * allocated or freed by this call.
 * Set-up: the first call on a device (that device current) looks up the
 * scratch address and sets kernel attributes; make that first call before
 * any stream capture on the device. Each call compares the current context
 * with the one the set-up was made in and repeats the set-up when the
 * context was recreated (e.g. after cudaDeviceReset).
 * Concurrency: all calls on a device share the one scratch, so calls whose
 * executions overlap (other streams, unordered host threads) race; the
 * caller serialises them.
 * Errors: argument errors as ts_ffn_create / ts_ffn_forward. A device-side
 * list error (unsorted or out-of-range ids) skips the offending entries but
 * is not reported by this entry point.
 */
#define TS_NOALLOC_MAX_M 16384
#define TS_NOALLOC_MAX_BATCH 64
ts_status ts_ffn_forward_noalloc(int d, int m, ts_dtype wdtype, const void* w_gate,
                                 const void* w_up, const void* w_down, const void* x, int batch,
                                 float* y, cudaStream_t stream, const int32_t* active_idx,
                                 int n_active);

/*
 * Top-k MoE layer (Sec. 4; Mixtral: 2 of 8 experts, Sec. 6.2):
 *     r = x W_r^T, pick the top_k largest logits (lower expert index wins a
 *     tie), w = softmax over the picked logits,
 *     y_t = sum_k w_{t,k} * FFN_{e_{t,k}}(x_t),
 * each expert itself a neuron-sparse dReLU FFN.
 *   w_router   device [n_experts][d], wdtype (bf16 when the experts are
 *              TS_INT4; borrowed)
 *   experts    n_experts handles (same d and wdtype; borrowed)
 *   n_experts  1..16, top_k 1..min(4, n_experts), max_batch 1..8 (1..2 for
 *              INT4 experts)
 */
ts_status ts_moe_create(ts_moe** out, int d, int n_experts, int top_k, ts_dtype wdtype,
                        const void* w_router, ts_ffn* const* experts, int max_batch);
void ts_moe_destroy(ts_moe* h);

/* y [batch][d] fp32 = MoE(x [batch][d] wdtype), on `stream`. */
ts_status ts_moe_forward(ts_moe* h, const void* x, int batch, float* y, cudaStream_t stream);

/* Pre-norm residual stack of MoE layers on h [batch][d] fp32 (in place),
   with the same glue as ts_stack_forward. */
ts_status ts_moe_stack_forward(ts_moe* const* layers, int n_layers, float* h, int batch,
                               cudaStream_t stream);

/* Routing of the last forward, to host memory (synchronises `stream`):
   sel [batch][top_k] expert ids (largest logit first), w [batch][top_k]. */
ts_status ts_moe_get_routing(ts_moe* h, cudaStream_t stream, int32_t* sel, float* w);

/* Per-expert active sets of the last MoE forward (synchronises `stream`):
   as ts_ffn_get_active for expert `expert` and batch token `token` (-1: the
   union over the tokens routed to that expert). */
ts_status ts_moe_get_active(ts_moe* h, cudaStream_t stream, int expert, int token,
                            int32_t* gate_idx, int* n_gate, int32_t* both_idx, int* n_both);

/* As ts_ffn_get_error, for the MoE layer's router and grouped kernels. */
ts_status ts_moe_get_error(ts_moe* h, cudaStream_t stream);

/* As ts_ffn_check_scratch, for the MoE layer's scratch. */
ts_status ts_moe_check_scratch(ts_moe* h, cudaStream_t stream);

/*
 * Activation predictor of one FFN layer (Sec. 7: a predictor per FFN block,
 * per expert for MoE; the paper gives no architecture, so this is a reading):
 * a two-layer ReLU MLP over the layer's input x,
 *     hid = max(0, W1 x),   s = W2 hid      (s[j]: score of neuron j),
 * and a batch's list is the K neurons with the largest key
 * key[j] = max over the batch's tokens of s[t][j], a lower neuron id winning
 * a tie, emitted in ascending id order -- the input of the predictor-driven
 * mode of ts_ffn_forward / ts_stack_forward.
 *   d, r, m    input width, hidden width, neurons; d and r multiples of 256
 *              (bf16) or 128 (fp32), r / that multiple one of 1, 2, 4, 8
 *   dtype      TS_BF16 or TS_F32: the type of W1, W2 and x
 *   w1, w2     device [r][d] and [m][r], row-major (borrowed, 16-byte aligned)
 *   max_batch  largest batch of a prediction, 1..8
 * Scores accumulate in fp32. Returns TS_ERR_UNSUPPORTED for sizes without a
 * kernel, TS_ERR_OOM if scratch cannot be allocated. The handle owns its
 * scratch (hidden-layer partials, per-neuron keys and a histogram of the
 * keys), which serves one prediction at a time: predictions with the same
 * handle must not overlap on the GPU (use one stream, or one handle per
 * stream).
 */
ts_status ts_predictor_create(ts_predictor** out, int d, int r, int m, ts_dtype dtype, const void* w1,
                              const void* w2, int max_batch);
void ts_predictor_destroy(ts_predictor* p);

/* As ts_ffn_check_scratch, for the predictor's scratch. */
ts_status ts_predictor_check_scratch(ts_predictor* p, cudaStream_t stream);

/*
 * list[0..K) = the predicted neurons for the batch x [batch][d] (device,
 * predictor dtype), ascending; `list` is a caller-owned device buffer of at
 * least K int32. scores: NULL, or a device [batch][m] fp32 buffer that
 * receives s. batch == 0 or K == 0 is a no-op. 0 <= K <= m, else
 * TS_ERR_INVALID_ARG. Asynchronous on `stream`.
 */
ts_status ts_predict(ts_predictor* p, const void* x, int batch, int K, int32_t* list, float* scores,
                     cudaStream_t stream);

/*
 * ts_stack_forward with a predictor per layer: for each layer l,
 *     x = round_wdtype(h / sqrt(mean(h^2) + 1e-5)),  x[d-1] = 1,
 *     lists[l][0..K[l]) = ts_predict(preds[l], x, K[l]),
 *     h = h + FFN_l(x) over the listed neurons only (predictor-driven mode).
 * preds[l] must match layer l's d, m and activation dtype (bf16 for INT4
 * layers). lists[l]: caller-owned device buffers of K[l] int32 that keep the
 * lists for inspection. K[l] == 0 leaves h unchanged for that layer.
 */
ts_status ts_stack_forward_predicted(ts_ffn* const* layers, ts_predictor* const* preds, int n_layers,
                                     float* h, int batch, const int* K, int32_t* const* lists,
                                     cudaStream_t stream);

/*
 * Capture a whole multi-layer forward once as a CUDA graph and replay it.
 * The captured calls keep the pointers given here; replaying reads and
 * writes the same buffers. ts_graph_capture_stack captures
 * ts_stack_forward(layers, n_layers, h, batch, ., active_idx, n_active);
 * ts_graph_capture_moe_stack captures ts_moe_stack_forward.
 */
ts_status ts_graph_capture_stack(ts_graph** out, ts_ffn* const* layers, int n_layers, float* h,
                                 int batch, const int32_t* const* active_idx, const int* n_active);
ts_status ts_graph_capture_moe_stack(ts_graph** out, ts_moe* const* layers, int n_layers,
                                     float* h, int batch);
/* Captures ts_stack_forward_predicted(layers, preds, n_layers, h, batch, K, lists, .). */
ts_status ts_graph_capture_stack_predicted(ts_graph** out, ts_ffn* const* layers, ts_predictor* const* preds,
                                           int n_layers, float* h, int batch, const int* K,
                                           int32_t* const* lists);
/*
 * The same stack as ts_graph_capture_stack (Eq. 1 with the dReLU of Eq. 2 per
 * layer, the stack glue between layers), fused into one persistent launch:
 * every CTA (one per SM, all resident at once by a cooperative launch) runs
 * each layer's gate+up phases and its share of the down projection, then the
 * CTAs meet at a grid barrier, sum the partial down projections by column
 * slices into h, meet again and go on with the next layer. No launch gaps
 * between layers; one launch per replay, plus a memset that clears the
 * barrier words.
 *   layers, n_layers, h, batch, active_idx, n_active   as ts_graph_capture_stack
 * Supported: bf16 layers of one width d, batch 1 or 2, the same grid for
 * every layer; otherwise TS_ERR_UNSUPPORTED (capture the unfused stack then).
 * The graph owns a small device table of the layers' parameters (allocated
 * here, freed by ts_graph_destroy). Replays are bitwise identical to the
 * unfused graph's only up to the fp32 summation order of the reduction (the
 * partials are added in CTA order in both, in different groupings).
 * Device-side errors (bad list entries, a barrier that waited past its
 * bound: TS_ERR_TIMEOUT, after which the CTAs stop and h is undefined) are
 * reported by ts_ffn_get_error on layers[0] (barriers) and on each layer
 * (lists).
 */
ts_status ts_graph_capture_stack_fused(ts_graph** out, ts_ffn* const* layers, int n_layers, float* h,
                                       int batch, const int32_t* const* active_idx, const int* n_active);
ts_status ts_graph_launch(ts_graph* g, cudaStream_t stream);
void ts_graph_destroy(ts_graph* g);

#ifdef __cplusplus
}
#endif
#endif /* TS_FFN_H */
