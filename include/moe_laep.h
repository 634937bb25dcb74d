/*
 * moe_laep.h - C ABI of the GB300 (sm_103a) MoE expert-layer hot path that
 * Layer-Adaptive Expert Pruning (LAEP; Yuan3.0 Ultra report, arXiv 2601.14327)
 * accelerates during pre-training.
 *
 * One MoE layer step on one GPU:
 *   moe_route              router logits, top-k, gates, per-expert histogram
 *   moe_load_stats         per-expert histogram of an existing routing
 *   laep_prune_mask        LAEP pruning decision (host)
 *   moe_permute            contiguous per-expert groups of token rows
 *   moe_grouped_ffn_fwd    grouped SwiGLU expert FFN (tcgen05 / TMEM / TMA)
 *   moe_unpermute_combine  gate-weighted combine back to token order
 * and the backward companions moe_unpermute_combine_bwd, moe_grouped_ffn_bwd
 * (or its halves moe_grouped_ffn_bwd_dgrad / _wgrad), moe_route_bwd,
 * moe_permute_bwd. Fused variants, same results, slower on GB300 and so not
 * the default: moe_permute_map with the *_gather GEMM entry points (X_perm read
 * from x by TMA gathers) and moe_grouped_ffn_fwd_combine (the combine in the
 * down GEMM's epilogue). Host-side LAEP: laep_prune_mask, laep_prune_layers,
 * laep_layer_alpha, laep_rearrange.
 *
 * Conventions (all entry points):
 *  - Pointers are DEVICE pointers owned by the caller unless marked "host".
 *    The library allocates no memory; scratch comes from the caller's `ws`
 *    (size from moe_workspace_size) or from explicit scratch arguments.
 *  - bf16 tensors are passed as uint16_t (IEEE bfloat16 bit patterns).
 *  - Every device call is asynchronous on `stream` (NULL = legacy default
 *    stream) and returns a status: MOE_OK, or a negative MOE_ERR_* when the
 *    host-side argument check failed (nothing was launched) or a launch
 *    failed. moe_last_error_string() describes the last failure of the
 *    calling thread.
 *  - Problems the kernels detect on the device (an expert id out of range,
 *    fewer than k live experts, a histogram that disagrees with the routing,
 *    a bounded wait that expired) are recorded in a device error word, read
 *    with moe_device_error(). Kernels never trap.
 *  - Row-major layouts. Shapes use T tokens, d = d_model, E experts (pruned
 *    ones included), k experts per token, F = d_ff, A = T*k assignments and
 *    R = moe_perm_rows_max(T,k,E) rows in the grouped (permuted) layout.
 *  - Grouped layout: group e holds the assignments routed to expert e in
 *    (token, slot) order; it starts at group_offsets[e], a multiple of 128,
 *    and its rows past group_counts[e] up to group_offsets[e+1] are zero
 *    padding. group_offsets[E] is the number of rows in use (<= R).
 */
#ifndef MOE_LAEP_H
#define MOE_LAEP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st *moe_stream_t;

enum {
  MOE_OK = 0,
  MOE_ERR_ARG = -1,          /* invalid argument: null pointer, size or alignment */
  MOE_ERR_UNSUPPORTED = -2,  /* valid but outside the supported shapes */
  MOE_ERR_CUDA = -3,         /* a CUDA runtime/driver call failed */
  MOE_ERR_INVARIANT = -4,    /* a device-side consistency check failed */
  MOE_ERR_TIMEOUT = -5,      /* a bounded device-side wait expired */
  MOE_ERR_WORKSPACE = -6     /* workspace too small */
};

/* Codes stored in the device error word (first error wins). */
enum {
  MOE_DEV_OK = 0,
  MOE_DEV_BAD_EXPERT = 1,    /* topk_idx entry outside [0, E) */
  MOE_DEV_TOO_FEW_LIVE = 2,  /* a token saw fewer than k live experts */
  MOE_DEV_COUNT_MISMATCH = 3,/* counts disagree with the routing */
  MOE_DEV_WAIT_TIMEOUT = 4,  /* a pipeline wait in a GEMM kernel gave up */
  MOE_DEV_ROWS_OVERFLOW = 5  /* grouped layout would exceed R rows */
};

/* Library version (major*10000 + minor*100 + patch). */
int moe_version(void);

/* Text of the last error of the calling thread ("" if none). */
const char *moe_last_error_string(void);

/* Reads the device error word into *code (MOE_DEV_*), clearing it when
 * `clear` is nonzero. Synchronizes the current device first. Returns MOE_OK
 * or MOE_ERR_CUDA. */
int moe_device_error(int *code, int clear);

/* Kernel timing (instrumentation; not part of the paper's method). While
 * enabled, every kernel the library launches is bracketed by two CUDA events
 * recorded on its stream. moe_timing_read() waits for those events and
 * writes one line per kernel name, "name launches total_ms\n", in first-seen
 * order into buf (NUL-terminated); reset != 0 then forgets the records.
 * Host calls; they return MOE_OK, MOE_ERR_ARG or MOE_ERR_CUDA. */
int moe_timing_enable(int enable);
int moe_timing_read(char *buf, size_t buf_len, int reset);

/* Rows to allocate for every grouped-layout buffer: T*k + 128*E. */
int64_t moe_perm_rows_max(int T, int k, int E);

/* Bytes of scratch `ws` every device entry point below may use for a layer of
 * this shape (one buffer serves all calls of a step issued on one stream).
 * Its first 256 bytes hold the weight-gradient GEMMs' tile counter: the
 * moe_grouped_ffn_* entry points need a ws of at least 256 bytes (16-byte
 * aligned), and two weight-gradient calls whose kernels may overlap on the GPU
 * need separate workspaces. The other calls use disjoint regions after them, so the router
 * backward and the unpermute-sum may share one workspace with GEMM calls running
 * beside them on another stream. */
size_t moe_workspace_size(int T, int d, int E, int k, int F);

/*
 * moe_route - router of the MoE layer: which experts each token goes to.
 * Sec. 3.2 defines the routing indicator E[i,j,l] (token j of layer l sent to
 * expert i) and Sec. 4 / Table 5 require pruned experts to receive no token;
 * the router itself is an fp32 linear layer with a fixed bias.
 *   z[t,e] = sum_i x[t,i] * w_router[i,e] + bias[e]     (fp32 accumulation)
 *   z[t,e] = -inf where active_mask[e] == 0
 *   topk_idx[t,0..k-1] = the k largest z (descending, ties to lower index)
 *   topk_gate[t,j]     = softmax over the k selected z (fp32)
 *   counts[e]          = #{(t,j) : topk_idx[t,j] == e}   (overwritten)
 * x [T,d] bf16; w_router [d,E] fp32; bias [E] fp32 or NULL; active_mask [E]
 * uint8 or NULL (all live); logits_in [T,E] fp32 or NULL: when given it
 * replaces x*w_router+bias (x, w_router, bias are then not read; the mask is
 * still applied); logits_out [T,E] fp32 or NULL receives the masked z;
 * topk_idx [T,k] int32; topk_gate [T,k] fp32; counts [E] int32 or NULL;
 * ws, ws_bytes: workspace (moe_workspace_size; may be NULL with logits_in),
 * it holds w_router as three bf16 terms (hi + mid + lo, which together keep
 * every bit of an fp32 weight) for the tensor cores, whose bf16 products are
 * exact and accumulate in fp32, and the partial logits of the split reduction
 * over d. The partials are summed in a fixed order and every launch shape is a
 * function of (T, d, E), so the routing is deterministic.
 * Limits: 1 <= E <= 256, 1 <= k <= min(E, 8), d % 8 == 0, T >= 0.
 * A token with fewer than k live experts sets MOE_DEV_TOO_FEW_LIVE.
 */
int moe_route(const uint16_t *x, const float *w_router, const float *bias,
              const uint8_t *active_mask, int T, int d, int E, int k,
              const float *logits_in, float *logits_out, int32_t *topk_idx,
              float *topk_gate, int32_t *counts, void *ws, size_t ws_bytes,
              moe_stream_t stream);

/*
 * moe_load_stats - per-expert token number of one routing: the ETN statistic
 * of Algorithm 1 Step 1 (and the left-hand side of Eq. 1).
 *   counts[e] (+)= #{(t,j) : topk_idx[t,j] == e}
 * topk_idx [T,k] int32; counts [E] int32, overwritten when accumulate == 0,
 * added to otherwise (recording over iterations). Out-of-range ids are
 * skipped and set MOE_DEV_BAD_EXPERT.
 */
int moe_load_stats(const int32_t *topk_idx, int T, int k, int E, int32_t *counts,
                   int accumulate, moe_stream_t stream);

/*
 * laep_prune_mask - LAEP expert-pruning decision for one layer (HOST call).
 * Sec. 3.2 Eq. 1-2 and Algorithm 1 (one histogram): experts are visited in
 * ascending load order (ties: lower index first); with a running load sum,
 * an expert is pruned when the sum is < S*k*beta and its own load is
 * < S*k*alpha/E (E = experts before pruning). With prune_count >= 0 the rule
 * is instead "prune the prune_count least-loaded experts" (the largest=False
 * top-K of Eq. 2). At least k experts are always kept.
 * counts_host [E] int32 (host); S = tokens of the layer; active_mask_host [E]
 * uint8 (host, out: 1 keep, 0 pruned); n_pruned (host, out, may be NULL).
 */
int laep_prune_mask(const int32_t *counts_host, int E, int64_t S, int k, double alpha,
                    double beta, int prune_count, uint8_t *active_mask_host, int *n_pruned);

/*
 * laep_layer_alpha - layer-adaptive alpha (Sec. 3.4.3; Table 5 caption): the
 * first and the last floor(L/6) layers use alpha_edge (0.2 in the paper), the
 * other layers alpha_middle (0.4). HOST call; returns alpha for `layer`.
 */
double laep_layer_alpha(int L, int layer, double alpha_edge, double alpha_middle);

/*
 * laep_prune_layers - Algorithm 1 (Expert Pruning) over a recorded history.
 * Step 1's ETN[ITER, L, E] is etn_host (row-major, e.g. filled by
 * moe_load_stats into slot (iter*L + layer)*E). Step 2: for every iteration and
 * layer, experts are visited in ascending load order (ties: lower id) with a
 * running load sum that restarts per (iteration, layer); an expert is flagged
 * when the sum is < S*k*beta and its load is < S*k*alpha[layer]/E; Exp_dis
 * counts the flags of a layer and Marker those of each expert. Step 3: a layer
 * prunes N = the mean flagged count over the iterations (rounded half up) of
 * its experts, in descending Marker order (ties: lower total load, then lower
 * id), only experts flagged at least once, and keeps at least k.
 * HOST call. alpha_host [L]; mask_host [L, E] (out: 1 keep, 0 pruned);
 * n_pruned_host [L] (out, may be NULL). With ITER = 1 it equals
 * laep_prune_mask's alpha/beta rule layer by layer.
 */
int laep_prune_layers(const int32_t *etn_host, int iters, int L, int E, int64_t S, int k,
                      const double *alpha_host, double beta, uint8_t *mask_host,
                      int32_t *n_pruned_host);

/*
 * laep_rearrange - Algorithm 2 (Expert Rearranging): experts taken in
 * descending load order (ties: lower id) each go to the group with the
 * smallest load sum that still has room (ties: lower group; a full group
 * leaves the choice); capacity n/n_groups, rounded up when it does not divide.
 * HOST call. load_host [n]; order_host [n] (out: expert ids group after
 * group); group_of_host [n] and group_load_host [n_groups] (out, may be NULL).
 * In this library the same heaviest-first rule orders the weight-gradient
 * tiles of the grouped GEMM.
 */
int laep_rearrange(const int64_t *load_host, int n, int n_groups, int32_t *order_host,
                   int32_t *group_of_host, int64_t *group_load_host);

/*
 * moe_permute - dispatch: token rows into contiguous per-expert groups
 * (the data movement of expert-parallel dispatch, Sec. 3.3, on one GPU).
 * Stable counting sort of the A assignments by (expert, token, slot), then
 * x_perm[row_of_assignment[t*k+j], :] = x[t, :]; padding rows are zeroed.
 * x [T,d] bf16; topk_idx [T,k] int32; counts [E] int32 or NULL: when given it
 * is checked against the routing (MOE_DEV_COUNT_MISMATCH); rows_cap = rows
 * allocated in x_perm (>= moe_perm_rows_max); outputs group_offsets [E+1]
 * int32, group_counts [E] int32, row_of_assignment [T,k] int32,
 * x_perm [rows_cap, d] bf16. Limits: d % 8 == 0, E <= 256.
 */
int moe_permute(const uint16_t *x, const int32_t *topk_idx, const int32_t *counts, int T,
                int d, int E, int k, int64_t rows_cap, int32_t *group_offsets,
                int32_t *group_counts, int32_t *row_of_assignment, uint16_t *x_perm,
                void *ws, size_t ws_bytes, moe_stream_t stream);

/*
 * moe_permute_noalloc - moe_permute for callers that cannot allocate device
 * memory. The paper has no counterpart; this is a deployment variant.
 * Some callers may not call cudaMalloc or hand out a workspace: code that
 * runs inside an inference engine's plugin, for example, where the engine
 * planned and owns all device memory before execution and passes the plugin
 * only its input and output buffers. This entry point computes exactly what moe_permute computes
 * (same arguments minus ws/ws_bytes, same results) but keeps its per-block
 * histograms in a fixed 256 KiB array compiled into the library (65536
 * int32 entries) instead of a workspace; it allocates nothing.
 * Limit: E * ceil(T*k / 4096) <= 65536 (e.g. 256 experts with at most
 * 1,048,576 assignments); larger problems return MOE_ERR_UNSUPPORTED before
 * anything is launched.
 * The array's device address belongs to the CUDA context that loaded the
 * library: the first call in each context (the current one of the calling
 * thread: a device's primary context, another context of the same device, or
 * the new primary context after cudaDeviceReset) looks it up and caches it under
 * the context's unique id; make that first call in a context before any stream
 * capture on it. Every GPU that loads the library holds the array until the
 * process exits. All calls share the one array and it keeps the last call's
 * contents (nothing in it needs to start at zero): calls whose kernels may
 * overlap on the GPU (other streams, other host threads) race on it and must
 * be serialized by the caller.
 */
int moe_permute_noalloc(const uint16_t *x, const int32_t *topk_idx, const int32_t *counts, int T,
                        int d, int E, int k, int64_t rows_cap, int32_t *group_offsets,
                        int32_t *group_counts, int32_t *row_of_assignment, uint16_t *x_perm,
                        moe_stream_t stream);

/*
 * moe_grouped_ffn_fwd - the experts' SwiGLU FFN over the grouped layout.
 * Table A1 fixes three matrices per expert (gate, up, down); for each group
 * e with rows X_e:
 *   [A_e | B_e] = X_e * W_gate_up[e]^T;  H_e = silu(A_e) * B_e;
 *   O_e = H_e * W_down[e]^T
 * bf16 operands, fp32 accumulation in tensor memory, bf16 results.
 * x_perm [rows_cap,d]; group_offsets [E+1]; w_gate_up [E,2F,d] bf16 (rows
 * 0..F-1 gate, F..2F-1 up); w_down [E,d,F] bf16; outputs ab_saved (the
 * [rows, 2F] matrix [A|B], kept for the backward, rows_cap*2F bf16, stored in
 * 32-row blocks: element (r, c) at ((r/32)*(2F/8) + c/8)*256 + (r%32)*8 + c%8,
 * so that the 32 rows one warp handles are contiguous), h [rows_cap,F] bf16,
 * out_perm [rows_cap,d] bf16. Only rows below group_offsets[E] are written.
 * Groups of 0 rows cost nothing. ws: at least 256 bytes, 16-byte aligned (the
 * tile counter; see moe_workspace_size).
 * Schedule (all moe_grouped_ffn_* GEMMs): in the weight-gradient GEMMs, whose
 * tiles cost as much as their expert has rows, the tiles are listed heaviest
 * expert first (the longest-processing-time order of Algorithm 2's greedy) and
 * CTA pairs that run out of work take the next tile of the list from a counter in
 * ws, so the heaviest tile left always goes to the least-loaded pair (Algorithm 2
 * with the GPU's CTA pairs as its devices, applied online; a light expert's tiles
 * of 1-7 k-blocks of 128 rows are claimed 8, 4 or 2 at a time); the other GEMMs'
 * tiles all cost the same, are listed in expert order and each pair takes every
 * 76th one (with rows_cap >= 2^18, a group's odd last 128-row block is computed
 * by a second, one-SM launch on the same stream). A tile's arithmetic does not depend on which pair runs it: results
 * are bitwise reproducible.
 * Limits: d % 128 == 0, F % 128 == 0, all pointers 16-byte aligned.
 */
int moe_grouped_ffn_fwd(const uint16_t *x_perm, const int32_t *group_offsets, int E, int d,
                        int F, int64_t rows_cap, const uint16_t *w_gate_up,
                        const uint16_t *w_down, uint16_t *ab_saved, uint16_t *h,
                        uint16_t *out_perm, void *ws, size_t ws_bytes, moe_stream_t stream);

/*
 * moe_grouped_ffn_fwd_combine - moe_grouped_ffn_fwd with the combine of
 * moe_unpermute_combine done in the down GEMM's epilogue:
 *   y[t,:] = bf16( sum_j topk_gate[t,j] * O[row_of_assignment[t,j], :] )
 * The epilogue adds gate * O (its fp32 accumulator, before any bf16 rounding) into
 * y_acc with fp32 atomics, so the order of the k terms of a token, and the last
 * bits of y, can change from run to run (the unfused pair is bitwise
 * reproducible). out_perm may be NULL: O is then not stored (enough for a forward
 * without backward). y_acc [T,d] fp32 is caller-owned scratch (overwritten); y
 * [T,d] bf16 (out). row_of_assignment, topk_gate [T,k] as moe_permute/moe_route
 * wrote them; ws: moe_workspace_size(T, d, E, k, F) bytes (the token and gate of
 * each grouped row live there). Other arguments, outputs and limits as in
 * moe_grouped_ffn_fwd; 1 <= k <= min(8, E); rows_cap >= moe_perm_rows_max(T,k,E).
 * A row index outside [0, moe_perm_rows_max) sets MOE_DEV_ROWS_OVERFLOW.
 */
int moe_grouped_ffn_fwd_combine(const uint16_t *x_perm, const int32_t *group_offsets, int E, int d,
                                int F, int64_t rows_cap, const uint16_t *w_gate_up,
                                const uint16_t *w_down, const int32_t *row_of_assignment,
                                const float *topk_gate, int T, int k, uint16_t *ab_saved,
                                uint16_t *h, uint16_t *out_perm, float *y_acc, uint16_t *y,
                                void *ws, size_t ws_bytes, moe_stream_t stream);

/*
 * Gathered form of the dispatch (no X_perm in memory). The grouped operand X_perm
 * of the forward GEMM and of the dW_gate_up GEMM is taken from x itself through a
 * row -> token map: grouped
 * row r is x[token_of_row[r], :]. The GEMMs load those rows with 4-row TMA
 * gathers (one token row of d_model per gathered row, 128 bytes at a time), so
 * the (T*k + padding) x d copy that moe_permute writes is never materialized.
 * Results are the same as with moe_permute's X_perm, bit for bit, on every real
 * row and in every gradient: a padding row reads token 0 instead of zeros, and
 * every consumer multiplies padding rows by zero (d_out_perm's padding rows are
 * zero); on padding rows the
 * forward's ab_saved, h and out_perm hold finite values instead of zeros.
 * Cost on GB300: the two GEMMs that read X_perm run ~3.3x longer with 4-row
 * gathers than with tile loads of a materialized X_perm, far more than the
 * copy saves; moe_permute + the plain entry points are the fast path.
 */

/*
 * moe_permute_map - the grouped layout of moe_permute without the row copy:
 * group_offsets [E+1], group_counts [E], row_of_assignment [T,k] exactly as
 * moe_permute computes them, and token_of_row [rows_cap] int32 (out): the token
 * of each grouped row (real rows: the t of its assignment; padding rows: 0;
 * rows at or past group_offsets[E] are not written). ws: the workspace of
 * moe_permute (only its first region, the per-block histograms, is used).
 * Limits as in moe_permute; token_of_row 16-byte aligned.
 */
int moe_permute_map(const int32_t *topk_idx, const int32_t *counts, int T, int E, int k,
                    int64_t rows_cap, int32_t *group_offsets, int32_t *group_counts,
                    int32_t *row_of_assignment, int32_t *token_of_row, void *ws, size_t ws_bytes,
                    moe_stream_t stream);

/*
 * moe_grouped_ffn_fwd_gather - moe_grouped_ffn_fwd with X_perm read from
 * x [T,d] bf16 through token_of_row (from moe_permute_map). Other arguments,
 * outputs and limits as in moe_grouped_ffn_fwd; needs the CTA-pair GEMM kernel
 * (the default; MOE_ERR_UNSUPPORTED under MOE_GEMM_1SM=1).
 */
int moe_grouped_ffn_fwd_gather(const uint16_t *x, const int32_t *token_of_row, int T,
                               const int32_t *group_offsets, int E, int d, int F,
                               int64_t rows_cap, const uint16_t *w_gate_up,
                               const uint16_t *w_down, uint16_t *ab_saved, uint16_t *h,
                               uint16_t *out_perm, void *ws, size_t ws_bytes,
                               moe_stream_t stream);

/*
 * moe_unpermute_combine - gate-weighted combine back to token order: the
 * layer's output sums, for every token, the outputs of the experts its routing
 * indicator selects (E[i,j,l] = 1, Sec. 3.2), weighted by the gates; the dispatch
 * of Sec. 3.3 in reverse (the paper names the MoE layer but prints no combine
 * formula; the gates are the softmax over the selected experts of moe_route):
 *   y[t,:] = sum_j topk_gate[t,j] * out_perm[row_of_assignment[t,j], :]
 * summed in fp32, rounded once to bf16. out_perm [rows_cap,d] bf16;
 * row_of_assignment [T,k]; topk_gate [T,k] fp32; y [T,d] bf16. d % 8 == 0.
 */
int moe_unpermute_combine(const uint16_t *out_perm, const int32_t *row_of_assignment,
                          const float *topk_gate, int T, int d, int k, uint16_t *y,
                          moe_stream_t stream);

/*
 * moe_unpermute_combine_bwd - backward of the combine (the paper gives no
 * backward; this is the derivative of moe_unpermute_combine):
 *   d_out_perm[row(t,j), :] = topk_gate[t,j] * dy[t, :]   (bf16)
 *   d_gate[t,j] = <dy[t,:], out_perm[row(t,j),:]>         (fp32)
 * and zeroes the padding rows of d_out_perm (group_offsets/group_counts from
 * moe_permute). dy [T,d] bf16; d_out_perm [rows_cap,d] bf16; d_gate [T,k].
 * Either output may be NULL (not both, unless T == 0): that half is skipped. A
 * caller whose router is frozen needs d_out_perm only, which never reads out_perm;
 * out_perm is read for d_gate only, group_offsets / group_counts are used for
 * d_out_perm only. (Running the d_gate half on a second stream beside the dH GEMM
 * measured no faster on GB300 than the fused call: it slows the GEMM by as much.)
 */
int moe_unpermute_combine_bwd(const uint16_t *dy, const uint16_t *out_perm,
                              const int32_t *row_of_assignment, const float *topk_gate,
                              const int32_t *group_offsets, const int32_t *group_counts,
                              int T, int d, int E, int k, uint16_t *d_out_perm,
                              float *d_gate, moe_stream_t stream);

/*
 * moe_grouped_ffn_bwd - backward of moe_grouped_ffn_fwd (dgrad and wgrad) for
 * the three-matrix SwiGLU expert of Table A1 (the paper gives no backward; this
 * is the derivative of moe_grouped_ffn_fwd):
 *   dH_e = dO_e * W_down[e];  dA_e = dH_e * B_e * silu'(A_e);
 *   dB_e = dH_e * silu(A_e);  dX_e = [dA_e | dB_e] * W_gate_up[e]
 *   dW_down[e] = dO_e^T * H_e;  dW_gate_up[e] = [dA_e | dB_e]^T * X_e
 * active_mask [E] uint8 or NULL (all live): the LAEP mask the routing used. A
 * pruned expert (active_mask[e] == 0) is removed from the model (Sec. 4,
 * Table 5), so it has no weight gradient: its dw_gate_up[e] and dw_down[e] are
 * not written and keep what the caller left there. A live expert whose group is
 * empty gets exactly zero weight gradients.
 * d_out_perm [rows_cap,d] (padding rows zero); x_perm, ab_saved, h from the
 * forward; d_ab [rows_cap,2F] bf16 caller scratch (receives [dA|dB]);
 * outputs dx_perm [rows_cap,d] bf16, dw_gate_up [E,2F,d] bf16,
 * dw_down [E,d,F] bf16 (fp32 accumulation). ws as in moe_grouped_ffn_fwd.
 * Gate gradient (optional, d_gate_out [T,k] fp32 not NULL; needs topk_gate and
 * row_of_assignment unless T == 0): the dH GEMM's epilogue recomputes
 * H = silu(A) * B from ab_saved and sums dH * H over each grouped row; since
 * dH = g * dy W_down, that sum is g * <dy, O>, and d_gate_out[t,j] = sum / g[t,j]
 * (0 where the gate is 0, an fp32 softmax that underflowed: the routing backward
 * multiplies d_gate by its gate, so no gradient changes), the d_gate of
 * moe_unpermute_combine_bwd without its read of out_perm (call that one with
 * d_gate NULL). Sums in a fixed order: bitwise reproducible.
 * Router term (optional, on when w_router is not NULL; topk_gate and
 * row_of_assignment are then needed unless T == 0, and d_gate unless d_gate_out is
 * given, whose values it then uses; d_gate is NULL whenever w_router is): with
 * topk_gate [T,k] and row_of_assignment [T,k] (moe_route, moe_permute), d_gate [T,k]
 * (moe_unpermute_combine_bwd, or d_gate_out) and w_router [d,E] fp32, the dX GEMM's epilogue adds
 * the router's share of the input gradient to every grouped row before rounding:
 *   dx_perm[row(t,j), :] = dX(t,j) + dz[t,j] * w_router[:, e_j],
 *   dz[t,j] = g[t,j] * (d_gate[t,j] - sum_i g[t,i] * d_gate[t,i])
 * (the d_logits of moe_route_bwd, same arithmetic), so that moe_permute_bwd, called
 * without its router term, sums the rows into the full dx. The epilogue reads one
 * 256-wide slice of a w_router column per tile instead of k columns per token.
 * ws then needs moe_workspace_size(T, d, E, k, F) bytes (dz per grouped row);
 * 1 <= k <= min(8, E), rows_cap >= moe_perm_rows_max(T, k, E).
 * Limits as in the forward.
 */
int moe_grouped_ffn_bwd(const uint16_t *d_out_perm, const uint16_t *x_perm,
                        const uint16_t *ab_saved, const uint16_t *h,
                        const int32_t *group_offsets, const uint8_t *active_mask, int E, int d,
                        int F, int64_t rows_cap, const uint16_t *w_gate_up,
                        const uint16_t *w_down, const float *topk_gate, const float *d_gate,
                        const int32_t *row_of_assignment, const float *w_router, int T, int k,
                        float *d_gate_out, uint16_t *d_ab, uint16_t *dx_perm,
                        uint16_t *dw_gate_up, uint16_t *dw_down, void *ws, size_t ws_bytes,
                        moe_stream_t stream);

/*
 * moe_grouped_ffn_bwd_dgrad / moe_grouped_ffn_bwd_wgrad - the two halves of
 * moe_grouped_ffn_bwd (which calls them in this order on one stream), for
 * callers that overlap other work with the weight gradients (the derivative of
 * Table A1's three-matrix expert; the paper gives no backward):
 *   dgrad: dH = dO W_down, [dA|dB] (into d_ab), dX = [dA|dB] W_gate_up
 *          (+ the router term when its arguments are given)
 *   wgrad: dW_down = dO^T H, dW_gate_up = [dA|dB]^T X  (needs d_ab from dgrad;
 *          pruned experts of active_mask are not written)
 * Arguments as in moe_grouped_ffn_bwd.
 */
int moe_grouped_ffn_bwd_dgrad(const uint16_t *d_out_perm, const uint16_t *ab_saved,
                              const int32_t *group_offsets, int E, int d, int F, int64_t rows_cap,
                              const uint16_t *w_gate_up, const uint16_t *w_down,
                              const float *topk_gate, const float *d_gate,
                              const int32_t *row_of_assignment, const float *w_router, int T,
                              int k, float *d_gate_out, uint16_t *d_ab, uint16_t *dx_perm,
                              void *ws, size_t ws_bytes, moe_stream_t stream);
int moe_grouped_ffn_bwd_wgrad(const uint16_t *d_out_perm, const uint16_t *x_perm,
                              const uint16_t *h, const uint16_t *d_ab,
                              const int32_t *group_offsets, const uint8_t *active_mask, int E,
                              int d, int F, int64_t rows_cap, uint16_t *dw_gate_up,
                              uint16_t *dw_down, void *ws, size_t ws_bytes, moe_stream_t stream);

/*
 * moe_grouped_ffn_bwd_wgrad_gather - moe_grouped_ffn_bwd_wgrad with X_e read
 * from x [T,d] bf16 through token_of_row (moe_permute_map). Other arguments
 * and limits as in moe_grouped_ffn_bwd_wgrad (CTA-pair kernel only).
 */
int moe_grouped_ffn_bwd_wgrad_gather(const uint16_t *d_out_perm, const uint16_t *x,
                                     const int32_t *token_of_row, int T, const uint16_t *h,
                                     const uint16_t *d_ab, const int32_t *group_offsets,
                                     const uint8_t *active_mask, int E, int d, int F,
                                     int64_t rows_cap, uint16_t *dw_gate_up, uint16_t *dw_down,
                                     void *ws, size_t ws_bytes, moe_stream_t stream);

/*
 * moe_route_bwd - backward of the router's softmax over the selected experts
 * (the routing scores of Sec. 3.2 as a trainable linear router):
 *   d_logits[t,j] = g[t,j] * (d_gate[t,j] - sum_i g[t,i] * d_gate[t,i])
 *   dw_router[:, e] = sum over assignments (t,j) to e of d_logits[t,j] * x[t,:]
 * (the bias is fixed; unselected and pruned experts get zero). x [T,d] bf16 is the
 * layer input (16-byte aligned); topk_idx, topk_gate [T,k] as moe_route wrote them;
 * d_gate [T,k] fp32 (from moe_unpermute_combine_bwd). d_logits [T,k] fp32 (out);
 * dw_router [d,E] fp32 (out, overwritten; zero when T == 0).
 * dw_router is the product x^T dZ on the tensor cores, dZ [T,E] split into three
 * bf16 terms (bf16 x bf16 products are exact in fp32), accumulated in fp32 in a
 * fixed order: bitwise reproducible from run to run. ws/ws_bytes: workspace of
 * moe_workspace_size(T, d, E, k, F) bytes, 16-byte aligned.
 */
int moe_route_bwd(const uint16_t *x, const int32_t *topk_idx, const float *topk_gate,
                  const float *d_gate, int T, int d, int E, int k, float *d_logits,
                  float *dw_router, void *ws, size_t ws_bytes, moe_stream_t stream);

/*
 * moe_permute_bwd - gradient of the layer input (the paper gives no backward;
 * this is the derivative of moe_permute's gather x_perm[row(t,j)] = x[t], the
 * dispatch of Sec. 3.3 that sends each token to the experts its routing
 * indicator E[i,j,l] selects (Sec. 3.2), plus the router's term from
 * moe_route_bwd's d_logits):
 *   dx[t,:] = sum_j dx_perm[row(t,j), :] + sum_j d_logits[t,j] * w_router[:, e_j]
 * summed in fp32, one bf16 rounding. d_logits and w_router may both be NULL
 * (no router term): the form to use after moe_grouped_ffn_bwd_dgrad added the router
 * term to dx_perm (the layer's default; a pure gather-sum at the HBM rate), while
 * with them each token reads k fp32 rows of w_router. dx [T,d] bf16 (out).
 */
int moe_permute_bwd(const uint16_t *dx_perm, const int32_t *row_of_assignment,
                    const int32_t *topk_idx, const float *d_logits, const float *w_router,
                    int T, int d, int E, int k, uint16_t *dx, void *ws, size_t ws_bytes,
                    moe_stream_t stream);

/*
 * moe_selftest_wait_timeout - failure-detection self-test (no counterpart in the
 * paper). Launches one thread that waits, with the bounded pipeline wait the GEMM
 * and router kernels use on their mbarriers, on an mbarrier nothing arrives on.
 * After limit_ns nanoseconds (1e6 .. 2e9) the wait gives up, the kernel records
 * MOE_DEV_WAIT_TIMEOUT in the device error word (read with moe_device_error) and
 * returns; the context stays usable. Nothing else is touched.
 */
int moe_selftest_wait_timeout(int64_t limit_ns, moe_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* MOE_LAEP_H */
