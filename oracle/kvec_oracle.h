/*
 * kvec_oracle.h -- plain, slow fp64 CPU oracle of K-VEC's end-of-prefill
 * KV-cache eviction selection (cross-head and cross-layer coverage,
 * Section 4 and Algorithm 1 of the K-VEC paper).
 *
 * TEST INFRASTRUCTURE ONLY.  The oracle exists to check the CUDA path; only
 * the test suite, the smoke check and the benchmark's CPU-baseline leg call
 * it.  It shares no code, header, table or helper with the CUDA library.
 *
 * Every input is host memory.  bf16 values are passed as their raw 16-bit
 * patterns and widened exactly to double.
 */
#ifndef KVEC_ORACLE_H
#define KVEC_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
    int num_q_heads;     /* H_q */
    int num_kv_heads;    /* H_kv; query head hq reads KV head hq / (H_q / H_kv) */
    int head_dim;        /* d */
    int window;          /* w: query rows supplied per sequence, also the always-kept tail */
    int obs_window;      /* O  (Eq. 1) */
    int ext_window;      /* O' (Section 4.1, extended window) */
    int pool_kernel;     /* odd width of the 1-D max-pool over candidate scores; 1 = none */
    int num_ext_heads;   /* delta (Section 4.1) */
    double lambda;       /* lambda (Section 4.2) */
    double beta;         /* beta: preserved fraction of the budget (Section 4.2) */
    double softmax_scale;/* <= 0 selects 1/sqrt(d) */
    int pool_mode;       /* 0: max-pool (default); 1: average over the in-range neighbours */
    int head_criterion;  /* 0: standard deviation (Section 4.1, default); 1: entropy
                            (Section 5.4 ablation, "Head Selection Criteria") */
    int all_positions;   /* 0: the last w tokens are always kept and count toward B,
                            candidates are [0, L-w) (default); 1: every position
                            [0, L) is a candidate and each head keeps the top B of
                            them (Section 4.1's top-B over the T input tokens) */
    int head_budget;     /* 0: every KV head keeps B tokens (default); 1: head-wise
                            adaptive fill (the AdaKV-style allocation Section 2 calls
                            plug-and-play): each head keeps its window and preserved
                            tokens and the floor(ada_floor * F) best of its own other
                            candidates by P', F = B - w - K; the layer's remaining
                            H_kv * F - H_kv * floor(ada_floor * F) fill slots go to the
                            best P' over all heads' remaining candidates together
                            (ties: lower head, then lower position) */
    double ada_floor;    /* in [0, 1]; 1 gives the uniform fill */
} kvo_params;

/* Optional debug outputs.  Any pointer may be NULL.  Sizes use the caller's
 * max_seqlen (ML) as the per-row stride.  Entries outside their domain are 0. */
typedef struct {
    double* P_O_raw;     /* [batch][H_kv][ML] Eq. 1 with window O, every key t < L */
    double* P_Oext_raw;  /* [batch][H_kv][ML] same with window O' */
    double* I_raw;       /* [batch][ML] global importance (Section 4.2), every key t < L */
    double* P_O;         /* [batch][H_kv][ML] max-pooled over candidates t < L - w */
    double* P_Oext;      /* [batch][H_kv][ML] */
    double* I;           /* [batch][ML] */
    double* sigma;       /* [batch][H_kv] the heads' ranking key (lowest first): the std of
                            pooled P_O over candidates, or minus its entropy */
    int32_t* htop;       /* [batch][H_kv] 1 if the head gets the extended window */
    double* P;           /* [batch][H_kv][ML] priority after the cross-head step */
    uint8_t* pres;       /* [batch][H_kv][ML] 1 for the preserved top-K tokens */
    double* Pprime;      /* [batch][H_kv][ML] P + lambda * focus on candidates */
    double* row_sums;    /* [batch][H_q][w] sum of every softmax row (should be 1) */
    int64_t* coverage;   /* [batch] #tokens with n_t > 0 after this layer */
    int64_t literal_override_differs; /* heads where setting P'=1.0 literally would change S_h */
} kvo_debug;

/* Rows per KV head of the outputs: budget for the uniform fill; with the
 * adaptive fill a head may keep up to budget + (H_kv - 1) * (F - floor(ada_floor * F))
 * tokens.  -1 for invalid parameters. */
int kvo_head_capacity(const kvo_params* p, int budget);

/* Bytes of coverage state per sequence for a given max_seqlen.  Layout:
 *   u32 layers_done, u32 seqlen, u32 reserved[2],
 *   u8  n[round_up(max_seqlen, 16)],
 *   u32 last_union[ceil(max_seqlen / 32)],
 * padded to a multiple of 16 bytes. */
size_t kvo_state_bytes(int max_seqlen);

/* One layer of eviction selection for a packed (varlen) batch.
 *   cu_seqlens [batch+1]; q_obs [batch][w][H_q][d]; k, v [total][H_kv][d];
 *   state: batch consecutive per-sequence states (stride kvo_state_bytes);
 *   out_idx [batch][H_kv][cap] (ascending, -1 padded), cap = kvo_head_capacity;
 *   out_k, out_v [batch][H_kv][cap][d] (zero padded).
 * Returns 0 on success, a negative code on invalid arguments. */
int kvo_select_layer(const kvo_params* p, int batch, const int32_t* cu_seqlens, int max_seqlen,
                     const uint16_t* q_obs, const uint16_t* k, const uint16_t* v,
                     uint8_t* state, int budget,
                     int32_t* out_idx, uint16_t* out_k, uint16_t* out_v,
                     kvo_debug* dbg);

/* Number of threads the OpenMP runtime would use (1 when built without it). */
int kvo_num_threads(void);

#ifdef __cplusplus
}
#endif
#endif
