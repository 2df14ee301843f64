/*
 * bacon.h -- C ABI of the GB300 (sm_103a) BACON KV-cache compression library.
 *
 * BACON (Boundary Attention CalibratiON) scores every cached prompt token of
 * every (layer, kv-head) at the end of prefill and keeps the best ones:
 *
 *   window score   B_i = mean over the window queries of their causal
 *                        attention to key i                       (Sec. 4.1, Eq. 1)
 *   last query     Q_i = attention of the last prompt query to i  (Sec. 4.2, Eq. 2)
 *   residual       E_i = max(Q_i - B_i, 0)                        (Sec. 4.2, Eq. 4)
 *   coherence      L   = radius-r box mean of E, truncated at the ends
 *                                                                 (Sec. 4.3, Eqs. 5-7)
 *   persistence    T   = mean of E over the preceding min(m, l) layers
 *                                                                 (Sec. 4.3, Eqs. 8-9)
 *   evidence       V   = E + L + T                                (Sec. 4.3, Eqs. 10-11)
 *   scale          lambda = gamma Std_M(B~) / (Std_M(V) + eps), M = the
 *                        top-min(rho K, |I|) candidates by B~     (Sec. 4.4, Eqs. 12-15)
 *   score          S_i = B~_i + lambda V_i                        (Sec. 4.4, Eq. 16)
 *   selection      the K best candidates by S                     (Sec. 4.4, Eq. 17)
 *   compaction     their K/V rows gathered into a dense cache     (Sec. 4.4, after Eq. 17)
 *
 * where B~ is B max-pooled (odd width `pool`, stride 1, out-of-range
 * positions ignored) over the candidates.  Readings where the paper is
 * silent: the G = q_heads / kv_heads query heads of a kv-head are averaged
 * into one B and one Q; the candidates are positions [0, N - W) and the W
 * window tokens are always kept, so K = budget - W; gamma = 1, eps = 1e-8;
 * Std is the population standard deviation; ties go to the lower position.
 *
 * Layouts (all row-major, contiguous, element type bf16 unless stated):
 *   q_win  [Hq][W][d]      the last W prompt queries of one layer, post-RoPE;
 *                          query w sits at position N - W + w
 *   k, v   [Hkv][N][d]     one layer's prefill cache
 *   idx    [Hkv][budget]   int32 kept positions, ascending per head
 *   k_out, v_out [Hkv][budget][d]
 * Only head_dim 64 and 128 are supported.  Every device pointer must be
 * 16-byte aligned.
 *
 * Ownership: the caller owns every tensor passed in or out.  The library
 * owns the context, its device scratch and the per-request state.  All calls
 * are asynchronous on the caller's CUDA stream (`bacon_stream` is a
 * cudaStream_t; NULL means the legacy default stream).  A call returns the
 * launch-time status; no exception crosses the ABI.  On error the message of
 * the failing call is available from bacon_last_error() on the same thread.
 *
 * Errors: BACON_EINVAL for a bad argument (null or misaligned pointer, a
 * size out of range, budget < W, q_heads not a multiple of kv_heads,
 * unsupported head_dim, seq_len above max_seq_len, requests above
 * max_requests); BACON_ENOMEM when device or host allocation fails;
 * BACON_ECUDA for a CUDA launch or copy failure; BACON_ESTATE when layers
 * of a request are scored out of order or select runs before any layer was
 * scored; BACON_EUNSUPPORTED for sizes beyond the allocation-free entry
 * point's static scratch.  Errors found on the device are latched in the
 * context and returned by the next bacon_sync (the first one wins):
 * BACON_ETIMEOUT when a kernel's bounded pipeline wait (about a second) ran
 * out, after which the kernel drained its own work and returned, so the
 * context stays usable; BACON_EINVAL when bacon_compact was given an index
 * outside [0, seq_len); BACON_ECUDA when an internal consistency check of a
 * selection kernel failed (it emitted a different number of positions than
 * its budget; never expected, its message says so).  A context must not be
 * used from two threads at once.
 */
#ifndef BACON_H
#define BACON_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    BACON_OK = 0,
    BACON_EINVAL = 1,
    BACON_ENOMEM = 2,
    BACON_ECUDA = 3,
    BACON_ESTATE = 4,
    BACON_ETIMEOUT = 5,
    BACON_EUNSUPPORTED = 6
} bacon_status;

typedef void* bacon_stream; /* a cudaStream_t */

typedef struct bacon_ctx bacon_ctx;
typedef struct bacon_state bacon_state;

/* Hyper-parameters (Secs. 4.3-4.4) and capacity limits. */
typedef struct {
    int r;            /* coherence radius, default 5 (Sec. 4.3)            */
    int m;            /* persistence depth, default 4 (Sec. 4.3)           */
    int rho;          /* scale-matching expansion, default 2 (Sec. 4.4)    */
    float gamma;      /* calibration strength, default 1 (Eq. 14)          */
    float eps;        /* stabiliser, default 1e-8 (Eq. 15)                 */
    int use_E;        /* terms of Eq. 10, default 1, 1, 1 (0 = ablated)    */
    int use_L;
    int use_T;
    int keep_window;  /* 1 (default): window kept, candidates [0, N - W)   */
    int max_seq_len;  /* largest N any call may pass (default 16384)       */
    int max_requests; /* largest request count of one call (default 4)     */
    int keep_scores;  /* 1: keep V, pooled B and S of the last whole-step
                         call for bacon_get_scores (default 0)            */
} bacon_params;

/* Fill *p with the defaults listed above. */
void bacon_default_params(bacon_params* p);

/* Create a context for one model shape.  `layers` transformer layers with
 * `q_heads` query heads sharing `kv_heads` kv heads of dimension head_dim;
 * window W; odd max-pool width `pool` (1 = no pooling); default budget.
 * p may be NULL for the defaults.  Allocates the device scratch for
 * max_requests x layers x kv_heads x max_seq_len scores on the current
 * device.  For tests of failure detection only: when the environment
 * variable BACON_FAULT is "missing_arrival" at this call, the context's
 * next two-pass window step withholds one K-tile load, its bounded pipeline
 * waits run out and bacon_sync reports BACON_ETIMEOUT (nothing faults). */
bacon_status bacon_init(bacon_ctx** out, int layers, int kv_heads, int q_heads,
                        int head_dim, int window, int pool, int budget,
                        const bacon_params* p);
void bacon_destroy(bacon_ctx* ctx);

/* Message of the last failing call on this thread ("" if none). */
const char* bacon_last_error(void);

/* Per-request state for layer-by-layer scoring: the residuals E of the
 * preceding m layers (persistence, Eqs. 8-9), the scores of the last scored
 * layer and the index of the next layer expected. */
bacon_status bacon_state_create(bacon_ctx* ctx, bacon_state** out);
bacon_status bacon_state_reset(bacon_state* st);
void bacon_state_destroy(bacon_state* st);

/* Score one layer of one request (Eqs. 1-16 for every kv-head).  Layers
 * must arrive as 0, 1, 2, ... per state, else BACON_ESTATE.  q_win and k
 * are device pointers in the layouts above.  scores_out, if not NULL,
 * receives S as fp32 [Hkv][seq_len] (0 at non-candidates). */
bacon_status bacon_score_layer(bacon_ctx* ctx, bacon_state* st, int layer,
                               const void* q_win, const void* k, int seq_len,
                               float* scores_out, bacon_stream stream);

/* Select (Eq. 17) on the last layer scored with `st`: idx_out receives
 * int32 [Hkv][min(budget, N)] kept positions, ascending per head. */
bacon_status bacon_select(bacon_ctx* ctx, bacon_state* st, int budget,
                          int32_t* idx_out, bacon_stream stream);

/* Gather the kept rows of one layer: k_out[h][j] = k[h][idx[h][j]] and the
 * same for v (bitwise copies).  `count` indices per head. */
bacon_status bacon_compact(bacon_ctx* ctx, const void* k, const void* v,
                           const int32_t* idx, int seq_len, int count,
                           void* k_out, void* v_out, bacon_stream stream);

/* The whole step for `requests` independent prompts of seq_len tokens:
 * every layer and kv-head is scored, selected and compacted.  The pointer
 * arrays are HOST arrays of DEVICE pointers, indexed [request * layers +
 * layer], each pointing at one layer's tensor in the layouts above.
 * idx_out is one device array int32 [requests][layers][Hkv][kept] with
 * kept = min(budget, seq_len).  The host pointer arrays may be reused as
 * soon as the call returns. */
bacon_status bacon_compress_all_layers(bacon_ctx* ctx, int requests,
                                       const void* const* q_win,
                                       const void* const* k,
                                       const void* const* v, int seq_len,
                                       int budget, void* const* k_out,
                                       void* const* v_out, int32_t* idx_out,
                                       bacon_stream stream);

/* The whole step with one budget per layer (window included), e.g. the
 * pyramid schedule of bacon_pyramid_budgets (PyramidKV-style allocation,
 * Sec. 5 / App. B: BACON replaces only the within-head score, the base
 * compressor's layer budgets are kept).  layer_budgets is a HOST array of
 * `layers` ints; K_{l,h} of Eq. 12 is the layer's own budget minus W.
 * idx_out is a HOST array of DEVICE pointers [request * layers + layer], each
 * int32 [Hkv][kept_l] with kept_l = min(layer_budgets[l], seq_len); k_out and
 * v_out point at [Hkv][kept_l][d] per pair.  Other arguments and errors as
 * bacon_compress_all_layers. */
bacon_status bacon_compress_layer_budgets(bacon_ctx* ctx, int requests,
                                          const void* const* q_win, const void* const* k,
                                          const void* const* v, int seq_len,
                                          const int* layer_budgets, void* const* k_out,
                                          void* const* v_out, int32_t* const* idx_out,
                                          bacon_stream stream);

/* The whole step when the caller's prefill attention already produced the
 * softmax normalisers of the window rows (a fused attention kernel keeps
 * the log-sum-exp of every query row; Eq. 1's rows need nothing else to be
 * normalised), so the first pass over K is skipped.  lse is a HOST array of
 * DEVICE pointers [request * layers + layer], each fp32 [Hq][W]: for window
 * query w of query head g, ln sum_{i <= N-W+w} exp(q . k_i / sqrt(d)).
 * Everything else, including outputs and errors, as bacon_compress_all_layers.
 * Results equal that call's up to the rounding of the supplied values. */
bacon_status bacon_compress_with_lse(bacon_ctx* ctx, int requests, const void* const* q_win,
                                     const void* const* k, const void* const* v,
                                     const float* const* lse, int seq_len, int budget,
                                     void* const* k_out, void* const* v_out, int32_t* idx_out,
                                     bacon_stream stream);

/* The whole step with AdaKV-style adaptive head budgets (Sec. 5 / App. B:
 * the base compressor spreads a layer's budget over its kv-heads; BACON
 * supplies the score, Eq. 16, with K of Eq. 12 the average per-head budget).
 * Per (request, layer), with K = min(budget, N) - W per head on average:
 * every head first keeps its own top floor(alpha K) candidates; the other
 * Hkv K - Hkv floor(alpha K) slots go to the best remaining candidates of
 * all heads together (larger score first, ties to the lower head, then the
 * lower position).  Outputs are flat per (request, layer) pair, heads in
 * order: idx_out[pair] -> int32 [Hkv * kept] (each head's kept positions
 * ascending, then its window), k_out/v_out[pair] -> [Hkv * kept][d], with
 * kept = min(budget, N); counts_out is a DEVICE int32 [requests][layers][Hkv]
 * array receiving each head's kept count (window included).  alpha in
 * [0, 1]; BACON_EUNSUPPORTED when kv_heads x candidates exceeds 204800.
 * Other arguments and errors as bacon_compress_all_layers. */
bacon_status bacon_compress_adaptive(bacon_ctx* ctx, int requests, const void* const* q_win,
                                     const void* const* k, const void* const* v, int seq_len,
                                     int budget, float alpha, void* const* k_out,
                                     void* const* v_out, int32_t* const* idx_out,
                                     int32_t* counts_out, bacon_stream stream);

/* Ablation / sensitivity sweep (Sec. 5's component ablation of E, L and T
 * and its sensitivity study over m and r): every unit is scored under
 * several hyper-parameter sets while the window passes (Eqs. 1-4, the
 * dominant cost) run once.  Each variant overrides these fields of the
 * context's parameters; eps, keep_window and the pool width stay the
 * context's. */
#define BACON_MAX_VARIANTS 32
typedef struct {
    int r;           /* coherence radius (Eqs. 5-7), >= 0              */
    int m;           /* persistence depth (Eqs. 8-9), >= 0; 0 = no T  */
    int rho;         /* scale-matching expansion (Eq. 12), >= 0        */
    float gamma;     /* calibration strength (Eq. 14), finite, >= 0    */
    int use_E;       /* terms of Eq. 10 (0 = ablated)                  */
    int use_L;
    int use_T;
} bacon_variant;

/* Selection (Eq. 17) of every (request, layer, kv-head) under each of
 * n_variants variants (1 <= n_variants <= BACON_MAX_VARIANTS, HOST array),
 * from one set of window passes.  q_win and k as in
 * bacon_compress_all_layers; no K/V is gathered.  idx_out is one device
 * array int32 [n_variants][requests][layers][Hkv][kept], kept =
 * min(budget, seq_len), each variant's block laid out as that call's;
 * lambda_out, if not NULL, a device array fp32
 * [n_variants][requests][layers][Hkv] receiving Eq. 15's lambda.  Variant j
 * gives the indices bacon_compress_all_layers gives with its fields in the
 * context's parameters.  Afterwards bacon_get_scores reports BACON_ESTATE
 * until the next whole-step call.  EINVAL for a variant field out of range;
 * other errors as bacon_compress_all_layers. */
bacon_status bacon_sweep(bacon_ctx* ctx, int requests, const void* const* q_win,
                         const void* const* k, int seq_len, int budget, int n_variants,
                         const bacon_variant* variants, int32_t* idx_out, float* lambda_out,
                         bacon_stream stream);

/* Pyramid budget schedule over `layers` layers averaging `budget` (window
 * included): with K = budget - window, K_min = floor(K / beta) and
 * K_max = 2 K - K_min, layer l keeps W + K_min +
 * floor((layers - 1 - l) (K_max - K_min) / (layers - 1)) tokens, so the first
 * layer keeps the most, the last the fewest, and the layers together keep
 * at most layers x budget.  Host-only; writes out[0 .. layers). */
void bacon_pyramid_budgets(int layers, int window, int budget, int beta, int* out);

/* The same step on HOST buffers: inputs are copied to library-owned device
 * buffers, compressed, and the outputs copied back, all on `stream`; the
 * call returns once the outputs are on the host.  Contiguous host layouts:
 *   q_win [requests][layers][Hq][W][d], k, v [requests][layers][Hkv][N][d],
 *   k_out, v_out [requests][layers][Hkv][kept][d],
 *   idx_out [requests][layers][Hkv][kept].
 * Page-locked host memory gives the full copy bandwidth.  When `v` is
 * page-locked memory the device can address (allocated or registered
 * through CUDA, 16-byte aligned), it is not uploaded: the gather reads only
 * the kept rows from it in place. */
bacon_status bacon_compress_host(bacon_ctx* ctx, int requests,
                                 const void* q_win, const void* k,
                                 const void* v, int seq_len, int budget,
                                 void* k_out, void* v_out, int32_t* idx_out,
                                 bacon_stream stream);

/* Intermediate per-token arrays of the last bacon_compress_all_layers /
 * bacon_compress_host call, for inspection: fp32 [requests][layers][Hkv][N]
 * (lambda: [requests][layers][Hkv]).  `out` is a device pointer of at least
 * `count` floats.  V, the pooled B and S are kept only when the context was
 * created with keep_scores = 1 (else BACON_ESTATE). */
typedef enum {
    BACON_SCORE_B = 0,      /* window score, Eq. 1               */
    BACON_SCORE_Q = 1,      /* last-query score, Eq. 2           */
    BACON_SCORE_E = 2,      /* residual, Eq. 4                   */
    BACON_SCORE_V = 3,      /* calibrated evidence, Eq. 10       */
    BACON_SCORE_BPOOL = 4,  /* pooled window score (0 off-candidates) */
    BACON_SCORE_S = 5,      /* final score, Eq. 16 (0 off-candidates) */
    BACON_SCORE_LAMBDA = 6  /* lambda, Eq. 15                    */
} bacon_score_kind;

bacon_status bacon_get_scores(bacon_ctx* ctx, bacon_score_kind kind,
                              float* out, size_t count, bacon_stream stream);

/* Per-kernel device timing of the whole-step path: when enabled, CUDA events
 * are recorded on the caller's stream around each launch of
 * bacon_compress_all_layers / bacon_compress_host. */
bacon_status bacon_profile_enable(bacon_ctx* ctx, int enable);

/* Kernel stages reported by bacon_profile_read, in this order. */
#define BACON_PROFILE_STAGES 5 /* window_stats, window_combine, window_scores,
                                  calibrate_select, gather */

/* Waits for the recorded work, then writes per stage the summed device time
 * in ms and the launch count since the previous read (arrays of at least
 * `n` entries; n <= BACON_PROFILE_STAGES), and clears the record.  A stage
 * that launched nothing in a call is not counted: when every unit's logits
 * fit in tensor memory (at most 32 window rows and 1024 tokens) the window
 * score is one kernel, reported as window_scores, with no window_stats or
 * window_combine launch. */
bacon_status bacon_profile_read(bacon_ctx* ctx, double* ms, int* launches, int n);

/* Window scores of one layer (B, Q and E of Eqs. 1, 2 and 4 for every
 * kv-head) WITHOUT ANY DEVICE ALLOCATION.  The paper has no counterpart:
 * this entry point exists for callers that cannot call cudaMalloc, such as
 * a serving engine that reserves all of HBM for its KV cache up front, or
 * code that must not pay the device-wide synchronisation of cudaMalloc /
 * cudaFree in the middle of prefill.  It needs no context: the kernels'
 * scratch (softmax statistics and two TMA descriptors) lives in one static
 * __device__ array of about 528 KiB, which every GPU that loads the library
 * holds until the process exits.
 *
 * Inputs as in the layouts above (q_win [Hq][W][d], k [Hkv][N][d] bf16);
 * outputs B_out, Q_out, E_out fp32 [Hkv][N], all caller-owned device
 * pointers, 16-byte aligned.  Limits: seq_len <= 16384,
 * q_heads * window <= 4096 and (q_heads / kv_heads) * window <= 512 (beyond
 * them: BACON_EUNSUPPORTED); malformed
 * arguments give BACON_EINVAL, a CUDA failure at launch BACON_ECUDA.  No
 * message is recorded for bacon_last_error.  The status is returned before
 * the kernels run, so an error found on the device (a bounded pipeline wait
 * of about a second that ran out) is reported in the outputs instead: B_out,
 * Q_out and E_out are then all NaN once the stream reaches the end of the
 * call.  A caller that must tell this case apart checks one output value
 * after synchronising.
 *
 * The first call on a device looks up the array's device address (with
 * that device current) and caches it.  Every call uses the same array:
 * calls whose work can overlap on the GPU (different streams, or several
 * host threads) race and must be serialised by the caller.  The array keeps
 * the last call's contents; its error word, the one entry that must start
 * at zero, is cleared by each call on its stream, and every other entry a
 * call reads it has written first. */
bacon_status bacon_window_scores_noalloc(int kv_heads, int q_heads, int head_dim, int window,
                                         const void* q_win, const void* k, int seq_len,
                                         float* B_out, float* Q_out, float* E_out,
                                         bacon_stream stream);

/* Wait for the stream and report any error latched by a kernel. */
bacon_status bacon_sync(bacon_ctx* ctx, bacon_stream stream);

#ifdef __cplusplus
}
#endif
#endif /* BACON_H */
