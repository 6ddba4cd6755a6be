/*
 * kvec.h -- C ABI of the GB300 (sm_103a) K-VEC eviction-selection library.
 *
 * K-VEC ("KV cache Eviction with Coverage") decides, at the end of prefill and
 * layer by layer, which B tokens each KV head keeps in its cache:
 *   - window scores: Eq. 1, the mean attention of the last O queries (O' for
 *     the cross-head heads), summed over the query heads of a GQA group;
 *   - cross-head coverage (Section 4.1): the delta KV heads whose scores have
 *     the lowest standard deviation use the extended window O';
 *   - cross-layer coverage (Section 4.2): P' = P + lambda * I * (1 - n_t/(l+1)),
 *     with I the head-max importance and n_t the number of earlier layers that
 *     kept token t; the top floor(beta*B) tokens by P are preserved;
 *   - per-KV-head top-B (Section 4.1, "each head selects the top-B tokens"),
 *     then the gather of the selected K/V rows into the budget-sized cache.
 * Algorithm 1 of the paper lists the same steps.
 *
 * Conventions shared by every entry point:
 *   - Pointers marked "device" are CUDA device memory owned by the caller
 *     (torch tensors, cudaMalloc, ...).  The library never frees them.
 *   - Work is asynchronous and stream ordered on the stream argument; results
 *     are valid once that stream reaches the call.  Host-side validation runs
 *     first and a rejected call launches nothing.
 *   - Errors are returned as kvec_status; kvec_last_error() gives a message
 *     for the calling thread.  No C++ exception crosses this boundary.
 *   - A handle is used from one host thread at a time.
 *   - bf16 tensors are raw IEEE bfloat16 (2 bytes per element).
 */
#ifndef KVEC_H
#define KVEC_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define KVEC_API __attribute__((visibility("default")))
#else
#define KVEC_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    KVEC_OK = 0,
    KVEC_ERR_INVALID_ARG = 1,     /* a pointer, size or parameter is out of range */
    KVEC_ERR_UNSUPPORTED = 2,     /* valid per the paper, not supported by these kernels */
    KVEC_ERR_CUDA = 3,            /* a CUDA runtime call failed (message has the CUDA error) */
    KVEC_ERR_DEVICE_TIMEOUT = 4,  /* a bounded device-side wait gave up; outputs are invalid */
    KVEC_ERR_OOM = 5              /* workspace allocation in kvec_create failed */
} kvec_status;

typedef struct kvec_handle kvec_handle;
/* Same object as cudaStream_t; declared here so the header needs no CUDA include. */
typedef struct CUstream_st* kvec_stream_t;

/* Hyper-parameters (names follow Algorithm 1) and workspace sizing. */
typedef struct {
    int   num_q_heads;    /* H_q query heads */
    int   num_kv_heads;   /* H_kv KV heads; query head hq uses KV head hq / (H_q/H_kv) */
    int   head_dim;       /* d; these kernels support 128 */
    int   window;         /* w: observation query rows given per sequence; the last w
                             tokens are always kept and count toward the budget unless
                             all_positions = 1 */
    int   obs_window;     /* O of Eq. 1 (paper: "e.g., 16"), 1 <= O <= min(w, 64) */
    int   ext_window;     /* O' of Section 4.1 (paper default 32), 1 <= O' <= w */
    int   pool_kernel;    /* odd width of the 1-D max-pool over candidate scores, 1..15 */
    int   num_ext_heads;  /* delta of Section 4.1 (paper default 3), 0..H_kv */
    float lambda;         /* lambda of Section 4.2 (paper default 1.0), finite */
    float beta;           /* beta of Section 4.2 (paper's best 0.25), 0..1 */
    float softmax_scale;  /* <= 0 selects 1/sqrt(head_dim) */
    int   max_batch;      /* largest batch a call may pass */
    int   max_seqlen;     /* largest prefix length L a call may pass (<= 131072) */
    int   max_layers;     /* layers one coverage state may see (<= 255; n_t is 8-bit) */
    int   pool_mode;      /* 0: max-pool (the paper's setting, default); 1: average of the
                             in-range neighbours (variant of the SnapKV lineage) */
    int   head_criterion; /* 0: the delta heads with the lowest standard deviation of pooled
                             P_O take O' (Section 4.1, default); 1: those with the highest
                             entropy of pooled P_O normalised over the candidates (the
                             Section 5.4 ablation "Head Selection Criteria") */
    int   all_positions;  /* 0: the last w tokens are always kept and count toward the
                             budget; the candidates are [0, L - w) (SnapKV's retained
                             observation window, default).  1: every position [0, L) is a
                             candidate, the window part scored by its causal attention, and
                             each head keeps the top B of them (Section 4.1's top-B over
                             the T input tokens); budget >= 1 instead of >= window */
    int   head_budget;    /* 0: every KV head keeps B tokens (default).  1: head-wise
                             adaptive fill (the AdaKV-style allocation Section 2 names
                             as a plug-and-play addition): each head keeps its window,
                             its preserved tokens and the floor(ada_floor * F) best of
                             its own other candidates by P' (F = B - w - K, K the
                             preserved count); the layer's other H_kv * (F - that)
                             fill slots go to the best P' over all its heads'
                             remaining candidates together (ties: lower head, then
                             lower position), so heads keep different numbers of
                             tokens, H_kv * B in total.  Not available through
                             kvec_select_layer_noalloc. */
    float ada_floor;      /* 0..1, with head_budget = 1: the share of its fill a head
                             ranks on its own (1 gives the uniform fill) */
} kvec_params;

/* Creates a handle and allocates its device workspace on the current device.
 * Returns INVALID_ARG / UNSUPPORTED for bad parameters (nothing allocated),
 * OOM or CUDA on allocation failure.  *out is NULL on failure. */
KVEC_API kvec_status kvec_create(const kvec_params* params, kvec_handle** out);

/* Frees the workspace; waits for the handle's pending work first. */
KVEC_API kvec_status kvec_destroy(kvec_handle* h);

/* Rows per KV head of every selection output (out_idx, out_k, out_v below):
 * budget, or with head_budget = 1 the most tokens one head can keep,
 * budget + (H_kv - 1) * (F - floor(ada_floor * F)).  -1 if params or budget are
 * invalid.  Host only; needs no device. */
KVEC_API int kvec_output_capacity(const kvec_params* params, int budget);

/* Bytes of coverage state per sequence (Section 4.2's counters n_t).  The
 * caller allocates batch * kvec_state_bytes(max_seqlen) bytes of device memory.
 * Layout of one sequence's state (little endian, 16-byte aligned):
 *   u32 layers_done   layers processed so far (l in coverage = n_t/(l+1))
 *   u32 seqlen        L of the last call
 *   u32 reserved[2]   zero
 *   u8  n[round_up(max_seqlen, 16)]      n_t: layers that kept token t
 *   u32 last_union[ceil(max_seqlen/32)]  bit t set if any head kept t in the last layer
 * padded to a multiple of 16 bytes.  Copying it is a checkpoint. */
KVEC_API size_t kvec_state_bytes(int max_seqlen);

/* Zeroes `batch` consecutive states (a new prompt starts at layer 0). */
KVEC_API kvec_status kvec_reset(kvec_handle* h, void* coverage_state, int batch, kvec_stream_t stream);

/* One layer of eviction selection for a varlen-packed batch (Algorithm 1 followed
 * by per-KV-head top-B and the K/V gather).
 *   cu_seqlens_host [batch+1] host, cu_seqlens_dev [batch+1] device: same values,
 *       cu[0] = 0, L_s = cu[s+1] - cu[s] with w <= L_s <= max_seqlen.
 *   q_obs  device bf16 [batch][w][H_q][d]: the last w query rows of every sequence
 *          (post-RoPE, as the attention saw them).
 *   k, v   device bf16 [cu[batch]][H_kv][d]: the layer's prefix keys and values.
 *   coverage_state  device, batch states (kvec_state_bytes each); read and updated.
 *   budget B: tokens kept per KV head, the w window tokens included; B >= w
 *          (with all_positions = 1 nothing is kept by rule and B >= 1).
 *   out_idx device int32 [batch][H_kv][C]: kept positions (0-based within the
 *          sequence), ascending; -1 after a head's last one.  C is
 *          kvec_output_capacity(params, B): B for the uniform fill.
 *   out_k, out_v device bf16 [batch][H_kv][C][d]: gathered rows, zero padded.
 * When L_s <= B every token is kept.  All device pointers must be 16-byte aligned. */
KVEC_API kvec_status kvec_select_layer(kvec_handle* h, int batch,
                              const int32_t* cu_seqlens_host, const int32_t* cu_seqlens_dev,
                              const void* q_obs, const void* k, const void* v,
                              void* coverage_state, int budget,
                              int32_t* out_idx, void* out_k, void* out_v,
                              kvec_stream_t stream);

/* num_layers consecutive layers of one prefill (same batch, lengths and state),
 * as if kvec_select_layer were called for layer 0, 1, ... in order.  Each array
 * holds num_layers device pointers with the per-layer meaning above.  The
 * library overlaps the score work of later layers with the coverage-dependent
 * selection of earlier ones; the results are identical to the layer-by-layer
 * calls.  num_layers must not exceed max_layers.  A sequence whose state would
 * pass 255 layers (layers_done + num_layers > 255) keeps its state unchanged and
 * gets no selection for any layer of the call; kvec_sync_status then returns
 * KVEC_ERR_INVALID_ARG. */
KVEC_API kvec_status kvec_select_layers(kvec_handle* h, int num_layers, int batch,
                               const int32_t* cu_seqlens_host, const int32_t* cu_seqlens_dev,
                               const void* const* q_obs, const void* const* k, const void* const* v,
                               void* coverage_state, int budget,
                               int32_t* const* out_idx, void* const* out_k, void* const* out_v,
                               kvec_stream_t stream);

/* kvec_select_layers with the window rows' softmax denominators supplied by the
 * caller, who has them from the prefill attention it just ran (the step right
 * before eviction, Section 5.1: selection happens in the prefill of each layer).
 * The library then skips its own statistics pass over K (score kernel) and
 * forms the attention A of Eq. 1 as exp(scale * <q, k> - lse) directly.
 *   lse  array of num_layers device pointers, each fp32 [batch][w][H_q]:
 *        lse[s][q][hq] = ln( sum over every key t the row sees (the prefix and
 *        the causal part of the window, t <= L_s - w + q) of
 *        exp(scale * <q_obs[s][q][hq], k_t>) ), with the same scale as
 *        params.softmax_scale (1/sqrt(d) when that is <= 0).  4-byte aligned.
 * Everything else as kvec_select_layers.  The library cannot check that lse
 * matches q_obs and K; a wrong lse gives a wrong selection. */
KVEC_API kvec_status kvec_select_layers_lse(kvec_handle* h, int num_layers, int batch,
                               const int32_t* cu_seqlens_host, const int32_t* cu_seqlens_dev,
                               const void* const* q_obs, const void* const* k, const void* const* v,
                               const float* const* lse, void* coverage_state, int budget,
                               int32_t* const* out_idx, void* const* out_k, void* const* out_v,
                               kvec_stream_t stream);

/* One layer of kvec_select_layers_lse. */
KVEC_API kvec_status kvec_select_layer_lse(kvec_handle* h, int batch,
                              const int32_t* cu_seqlens_host, const int32_t* cu_seqlens_dev,
                              const void* q_obs, const void* k, const void* v, const float* lse,
                              void* coverage_state, int budget,
                              int32_t* out_idx, void* out_k, void* out_v,
                              kvec_stream_t stream);

/* kvec_select_layer for callers that cannot allocate device memory: the
 * library then needs no handle and calls no cudaMalloc, cudaFree or other
 * allocating routine.  It serves hosts whose device memory belongs to someone
 * else (an inference server or framework plugin that hands out all memory
 * from its own pool and forbids extra allocations), which cannot create a
 * handle because kvec_create allocates its workspace.  The paper has no
 * counterpart; this is a deployment convenience.
 *   Arguments: as kvec_select_layer, with the hyper-parameters and the sizing
 *   limits (max_batch, max_seqlen; max_seqlen also fixes the state layout)
 *   given in *params instead of a handle.
 *   Scratch: one 32 MiB static device array inside the library, held by every
 *   GPU that loads the library until the process exits.  A call needs about
 *   (28 * H_kv + 9) * ML bytes per sequence (ML = max_seqlen + 4 rounded up to
 *   a multiple of 32) plus (8 * H_kv * g * w + 512 * O * ceil(H_kv / 8)) bytes
 *   per 128-token tile of its sequences; one 8192-token Llama-3.1-8B-shaped
 *   sequence needs about 3 MiB.  A call that needs more than the array is
 *   rejected with KVEC_ERR_INVALID_ARG and a message giving both sizes.
 *   Every call shares that array and it keeps the last call's contents; each
 *   part of it is written before it is read within a call.  Calls whose work
 *   overlaps on the GPU (different streams, or several host threads) race on
 *   it: serialise them.
 *   The first call on each device resolves the array's device address, sets
 *   kernel attributes and clears the array's error word, synchronously (no
 *   allocation); make that first call before any stream capture.
 *   Device-side errors (a bounded wait that gave up, or the refusal of a call
 *   that would take a state past 255 layers, which leaves that state unchanged)
 *   are recorded in the array's error word and reported by
 *   kvec_noalloc_sync_status. */
KVEC_API kvec_status kvec_select_layer_noalloc(const kvec_params* params, int batch,
                                      const int32_t* cu_seqlens_host, const int32_t* cu_seqlens_dev,
                                      const void* q_obs, const void* k, const void* v,
                                      void* coverage_state, int budget,
                                      int32_t* out_idx, void* out_k, void* out_v,
                                      kvec_stream_t stream);

/* Device-side status of kvec_select_layer_noalloc on the current device:
 * synchronises `stream`, then returns KVEC_ERR_DEVICE_TIMEOUT if a bounded
 * wait of any call since the last check gave up, KVEC_ERR_INVALID_ARG if a
 * call was refused because a state would have passed 255 layers (that state
 * is unchanged), else KVEC_OK; the recorded error is cleared.  The outputs of
 * a call that recorded an error are invalid.  Allocates nothing; KVEC_OK when
 * no call has run on this device yet. */
KVEC_API kvec_status kvec_noalloc_sync_status(kvec_stream_t stream);

/* One decoding step of attention over the compacted cache that the selection
 * produced.  Section 4.1: once each KV head has kept its B tokens, their keys
 * and values are the cache that the subsequent decoding steps read; Section
 * 5.3 (Computational Complexity) times decoding over that cache.  For every
 * sequence s and query head hq (KV head h = hq / (H_q/H_kv)):
 *   out[s][hq] = sum_{j < n_s} p_j * v_cache[s][h][j],
 *   p_j = softmax_j( scale * <q[s][hq], k_cache[s][h][j]> ),
 * with n_s = lens[s] clamped to [0, cap]; n_s = 0 gives a zero row.  scale is
 * params.softmax_scale (1/sqrt(d) when that is <= 0).
 *   q        device bf16 [batch][H_q][d]: the step's query rows.
 *   k_cache, v_cache  device bf16 [batch][H_kv][cap][d]: for instance out_k and
 *            out_v of kvec_select_layer (cap = B, lens[s] = min(L_s, B): the kept
 *            rows come first), or that cache with decoded tokens appended.
 *   lens     device int32 [batch].
 *   out      device fp32 [batch][H_q][d].
 * 1 <= batch <= max_batch, 1 <= cap <= 2^20, H_q/H_kv <= 8 (else UNSUPPORTED);
 * q, k_cache, v_cache 16-byte aligned, lens 4-byte and out 8-byte aligned.
 * Asynchronous on `stream`; the handle's decode workspace is reused by every
 * call, so calls on different streams must not overlap. */
KVEC_API kvec_status kvec_decode_attention(kvec_handle* h, int batch, const void* q,
                                           const void* k_cache, const void* v_cache,
                                           const int32_t* lens, int cap, float* out,
                                           kvec_stream_t stream);

/* Device views of the last processed layer's intermediates (valid until the
 * next call on the handle; read after synchronising the stream).  Row strides
 * use ML = max_seqlen + 4 rounded up to a multiple of 32 (reported in max_seqlen).
 * Only candidate positions hold scores: t < L_s - w by default, t < L_s with
 * all_positions = 1.  Pprime is written only for sequences with L_s > budget. */
typedef struct {
    const float*    P_O;        /* [max_batch][H_kv][ML]  Eq. 1 with O, max-pooled */
    const float*    P_Oext;     /* [max_batch][H_kv][ML]  Eq. 1 with O', max-pooled */
    const float*    I;          /* [max_batch][ML]        Section 4.2 importance, max-pooled */
    const float*    sigma;      /* [max_batch][H_kv]      the heads' ranking key (lowest first):
                                   std of pooled P_O over candidates, or minus its
                                   entropy when head_criterion = 1 */
    const int32_t*  htop;       /* [max_batch][H_kv]      1 if the head uses O' */
    const uint32_t* pres_bits;  /* [max_batch][H_kv][ceil(ML/32)] preserved top-K tokens */
    const float*    Pprime;     /* [max_batch][H_kv][ML]  P + lambda * focus */
    const float*    row_stats;  /* [max_batch][H_kv][g*w][2]  softmax row max (log2 units)
                                   and denominator; row r = q*g + j is query head
                                   h*g + j at window row q */
    int max_seqlen;             /* ML: the row stride of the arrays above */
    int words_per_row;          /* ceil(max_seqlen/32): words of pres_bits per row */
} kvec_debug_view;

KVEC_API kvec_status kvec_debug_scores(kvec_handle* h, kvec_debug_view* out);

/* Synchronises the handle's streams and reports a device-side error recorded
 * by a bounded wait (KVEC_ERR_DEVICE_TIMEOUT), then clears it. */
KVEC_API kvec_status kvec_sync_status(kvec_handle* h);

/* Per-kernel device time recorded since the last kvec_set_profiling(h, 1)
 * call, from CUDA events on the launching stream.  kernel: 0 score (QK^T and
 * softmax statistics), 1 window sums + pooling, 2 cross-head choice +
 * preserved tokens, 3 coverage-adjusted selection, 4 gather.  Synchronises. */
KVEC_API kvec_status kvec_set_profiling(kvec_handle* h, int enable);
KVEC_API kvec_status kvec_kernel_time(kvec_handle* h, int kernel, double* total_ms, int* launches);

/* For tests of the error path only; never set in production.  fault = 1 makes
 * every window kernel launched from then on withhold the signal of its first
 * accumulator, so that the epilogue's bounded wait for it gives up after about
 * 20 us: the kernel records KVEC_ERR_DEVICE_TIMEOUT in the error word (read by
 * kvec_sync_status or kvec_noalloc_sync_status), drains its copies and returns,
 * and that call's outputs are invalid.  fault = 0 (the default) switches it
 * off.  Process-wide; while it is set, multi-layer calls are neither captured
 * into nor replayed from the handle's graph cache. */
KVEC_API void kvec_set_test_fault(int fault);

KVEC_API const char* kvec_status_string(kvec_status s);
KVEC_API const char* kvec_last_error(void);

#ifdef __cplusplus
}
#endif
#endif
