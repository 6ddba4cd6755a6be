/*
 * kvec_oracle.c -- plain fp64 CPU oracle of K-VEC eviction selection.
 *
 * TEST INFRASTRUCTURE ONLY: called by the tests, the smoke check and the
 * benchmark's CPU-baseline leg; never by the product path.  Written from the
 * K-VEC paper (Section 4.1 "Cross-Head Coverage", Section 4.2 "Cross-Layer
 * Coverage", Algorithm 1), following its steps in its order.  Deliberately
 * unoptimised: full softmax rows in fp64, full sorts for every top-k.
 *
 * Readings of points the paper leaves open (each listed in the design notes):
 *  - Attention A is the model's causal softmax: row q of the window (absolute
 *    position L-w+q) normalises over every key t <= L-w+q.
 *  - "Heads" are KV heads; A is summed over the query heads of a GQA group.
 *  - Candidates are t in [0, L-w); the last w tokens are always kept and
 *    count toward the budget B (observation-window retention of SnapKV).
 *    With all_positions = 1 every t in [0, L) is a candidate (the window part
 *    scored by its causal attention) and nothing is kept unconditionally:
 *    the top-B over the T input tokens of Section 4.1, read literally.
 *  - Scores are max-pooled (odd width, stride 1, neighbours outside the
 *    candidate range ignored) before sigma, preservation and focus.
 *  - sigma is the sample standard deviation (n-1); 0 when fewer than 2
 *    candidates.  Ties in sigma go to the lower head index.
 *  - The "P'=1.0" override of Section 4.2 is read as force-keep: the
 *    floor(beta*B) preserved tokens (clamped to B-w) always stay, the rest of
 *    the budget goes to the highest P' among the other candidates.
 *  - Every top-k orders by higher score, then lower position.
 *  - coverage_t = n_t / (l+1) with l the number of layers already processed.
 *  - Head-wise adaptive fill (head_budget = 1; Section 2 names AdaKV's head-wise
 *    budget allocation as a plug-and-play addition without defining it): each
 *    head keeps its window and preserved tokens and its own floor(a * F) best
 *    other candidates by P' (F = B - w - K, a = ada_floor); the rest of the
 *    layer's fill, H_kv * (F - floor(a * F)) slots, goes to the best P' among all
 *    heads' remaining candidates ranked together (higher P', then lower head,
 *    then lower position).  a = 1 is the uniform fill.
 */
#include "kvec_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

size_t kvo_state_bytes(int max_seqlen) {
    size_t ns = round_up((size_t)max_seqlen, 16);
    size_t words = ((size_t)max_seqlen + 31) / 32;
    return round_up(16 + ns + 4 * words, 16);
}

int kvo_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* bf16 -> double, exact: a bf16 is the top half of an IEEE binary32. */
static double widen_bf16(uint16_t bits) {
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

typedef struct {
    double key;
    int32_t t;
} ranked_t;

/* Higher key first; on equal keys the lower position first. */
static int by_key_desc(const void* a, const void* b) {
    const ranked_t* x = (const ranked_t*)a;
    const ranked_t* y = (const ranked_t*)b;
    if (x->key > y->key) return -1;
    if (x->key < y->key) return 1;
    return (x->t > y->t) - (x->t < y->t);
}

/* Marks in sel[] the k best entries among positions t in [0, n) with allowed[t] != 0. */
static void top_k(const double* key, const uint8_t* allowed, int n, int k, uint8_t* sel) {
    ranked_t* r = (ranked_t*)malloc(sizeof(ranked_t) * (size_t)(n > 0 ? n : 1));
    int m = 0;
    for (int t = 0; t < n; ++t)
        if (!allowed || allowed[t]) { r[m].key = key[t]; r[m].t = t; ++m; }
    qsort(r, (size_t)m, sizeof(ranked_t), by_key_desc);
    for (int i = 0; i < k && i < m; ++i) sel[r[i].t] = 1;
    free(r);
}

/* 1-D average pool, width `kernel`, stride 1, over x[0, n): the mean of the
 * neighbours inside [0, n) (the pooling variant of the SnapKV lineage the paper
 * builds on; the paper's own setting is the max-pool below). */
static void avg_pool(const double* x, int n, int kernel, double* y) {
    int r = kernel / 2;
    for (int t = 0; t < n; ++t) {
        int lo = t - r < 0 ? 0 : t - r;
        int hi = t + r > n - 1 ? n - 1 : t + r;
        double s = 0.0;
        for (int j = lo; j <= hi; ++j) s += x[j];
        y[t] = s / (hi - lo + 1);
    }
}

/* 1-D max-pool, width `kernel`, stride 1, over x[0, n); neighbours outside [0, n) are ignored. */
static void max_pool(const double* x, int n, int kernel, double* y) {
    int r = kernel / 2;
    for (int t = 0; t < n; ++t) {
        int lo = t - r < 0 ? 0 : t - r;
        int hi = t + r > n - 1 ? n - 1 : t + r;
        double m = x[lo];
        for (int j = lo + 1; j <= hi; ++j) if (x[j] > m) m = x[j];
        y[t] = m;
    }
}

/* Preserved tokens and fill per head: K = min(floor(beta * B), B - wk), F = B - wk - K. */
static void budget_split(const kvo_params* p, int budget, int* Kp, int* F, int* f0) {
    const int wk = p->all_positions ? 0 : p->window;
    int k = (int)floor(p->beta * (double)budget);
    if (k > budget - wk) k = budget - wk;
    *Kp = k;
    *F = budget - wk - k;
    *f0 = p->head_budget ? (int)floor(p->ada_floor * (double)*F) : *F;
}

int kvo_head_capacity(const kvo_params* p, int budget) {
    if (!p || budget < 1 || p->num_kv_heads < 1) return -1;
    if (p->head_budget != 0 && p->head_budget != 1) return -1;
    if (p->head_budget && !(p->ada_floor >= 0.0 && p->ada_floor <= 1.0)) return -1;
    const int wk = p->all_positions ? 0 : p->window;
    if (budget < wk) return -1;
    int Kp, F, f0;
    budget_split(p, budget, &Kp, &F, &f0);
    return budget + (p->num_kv_heads - 1) * (F - f0);
}

int kvo_select_layer(const kvo_params* p, int batch, const int32_t* cu_seqlens, int max_seqlen,
                     const uint16_t* q_obs, const uint16_t* k, const uint16_t* v,
                     uint8_t* state, int budget,
                     int32_t* out_idx, uint16_t* out_k, uint16_t* out_v,
                     kvo_debug* dbg) {
    if (!p || batch < 1 || !cu_seqlens || !q_obs || !k || !v || !state || !out_idx || !out_k || !out_v)
        return -1;
    const int Hq = p->num_q_heads, Hkv = p->num_kv_heads, d = p->head_dim, w = p->window;
    const int O = p->obs_window, Oe = p->ext_window;
    if (Hkv < 1 || Hq < Hkv || Hq % Hkv != 0 || d < 1 || w < 1) return -2;
    if (O < 1 || Oe < 1 || O > w || Oe > w) return -3;
    if (p->pool_kernel < 1 || p->pool_kernel % 2 == 0) return -4;
    if (p->pool_mode != 0 && p->pool_mode != 1) return -4;
    if (p->head_criterion != 0 && p->head_criterion != 1) return -5;
    if (p->num_ext_heads < 0 || p->num_ext_heads > Hkv) return -5;
    if (!(p->beta >= 0.0 && p->beta <= 1.0)) return -6;
    if (p->all_positions != 0 && p->all_positions != 1) return -4;
    /* wk: the tail kept unconditionally (the window, or nothing). */
    const int wk = p->all_positions ? 0 : w;
    if (budget < wk || budget < 1) return -7;
    if (p->head_budget != 0 && p->head_budget != 1) return -4;
    if (p->head_budget && !(p->ada_floor >= 0.0 && p->ada_floor <= 1.0)) return -6;
    const int cap = kvo_head_capacity(p, budget);
    for (int b = 0; b < batch; ++b) {
        int L = cu_seqlens[b + 1] - cu_seqlens[b];
        if (L < w || L > max_seqlen) return -8;
    }
    const int g = Hq / Hkv;
    const double scale = p->softmax_scale > 0.0 ? p->softmax_scale : 1.0 / sqrt((double)d);
    const size_t sbytes = kvo_state_bytes(max_seqlen);
    const size_t ns = round_up((size_t)max_seqlen, 16);
    const int ML = max_seqlen;
    if (dbg) dbg->literal_override_differs = 0;

    for (int b = 0; b < batch; ++b) {
        const int L = cu_seqlens[b + 1] - cu_seqlens[b];
        const int Lc = L - wk;                 /* candidates t in [0, Lc) */
        const uint16_t* kb = k + (size_t)cu_seqlens[b] * Hkv * d;
        const uint16_t* vb = v + (size_t)cu_seqlens[b] * Hkv * d;
        uint8_t* st = state + (size_t)b * sbytes;
        uint32_t layers_done;
        memcpy(&layers_done, st, 4);
        if (layers_done >= 255) return -9;
        uint8_t* n_t = st + 16;
        uint32_t* last_union = (uint32_t*)(st + 16 + ns);

        /* Step 1 (Eq. 1 input): attention rows of the w window queries.
         * A[hq][q][t] = exp(s_t - max) / sum, s_t = scale * <q, k_t>, t <= L-w+q. */
        double* A = (double*)calloc((size_t)Hq * w * L, sizeof(double));
        #pragma omp parallel for schedule(dynamic)
        for (int row = 0; row < Hq * w; ++row) {
            const int hq = row / w, q = row % w, h = hq / g;
            const int pos = L - w + q;
            double* qv = (double*)malloc(sizeof(double) * (size_t)d);
            const uint16_t* qs = q_obs + (((size_t)b * w + q) * Hq + hq) * d;
            for (int j = 0; j < d; ++j) qv[j] = widen_bf16(qs[j]);
            double* a = A + ((size_t)hq * w + q) * L;
            double mx = -INFINITY;
            for (int t = 0; t <= pos; ++t) {
                const uint16_t* kt = kb + ((size_t)t * Hkv + h) * d;
                double s = 0.0;
                for (int j = 0; j < d; ++j) s += qv[j] * widen_bf16(kt[j]);
                a[t] = scale * s;
                if (a[t] > mx) mx = a[t];
            }
            double Z = 0.0;
            for (int t = 0; t <= pos; ++t) { a[t] = exp(a[t] - mx); Z += a[t]; }
            for (int t = 0; t <= pos; ++t) a[t] /= Z;
            free(qv);
        }
        if (dbg && dbg->row_sums) {
            for (int hq = 0; hq < Hq; ++hq)
                for (int q = 0; q < w; ++q) {
                    const double* a = A + ((size_t)hq * w + q) * L;
                    double s = 0.0;
                    for (int t = 0; t < L; ++t) s += a[t];
                    dbg->row_sums[((size_t)b * Hq + hq) * w + q] = s;
                }
        }

        /* Steps 2-3: Eq. 1 with windows O and O' on the group-summed attention,
         * and the global importance I_t = (1/O) sum_q max_h A[h,q,t] (Section 4.2). */
        /* Akv[h][q][t]: attention of KV head h = sum over its g query heads. */
        double* Akv = (double*)calloc((size_t)Hkv * w * L, sizeof(double));
        for (int h = 0; h < Hkv; ++h)
            for (int j = 0; j < g; ++j)
                for (int q = 0; q < w; ++q) {
                    const double* a = A + ((size_t)(h * g + j) * w + q) * L;
                    double* dst = Akv + ((size_t)h * w + q) * L;
                    for (int t = 0; t < L; ++t) dst[t] += a[t];
                }
        free(A);
        double* PO = (double*)calloc((size_t)Hkv * L, sizeof(double));
        double* POe = (double*)calloc((size_t)Hkv * L, sizeof(double));
        double* Iraw = (double*)calloc((size_t)L, sizeof(double));
        for (int h = 0; h < Hkv; ++h) {
            for (int q = w - O; q < w; ++q)
                for (int t = 0; t < L; ++t) PO[(size_t)h * L + t] += Akv[((size_t)h * w + q) * L + t];
            for (int q = w - Oe; q < w; ++q)
                for (int t = 0; t < L; ++t) POe[(size_t)h * L + t] += Akv[((size_t)h * w + q) * L + t];
            for (int t = 0; t < L; ++t) {
                PO[(size_t)h * L + t] /= O;
                POe[(size_t)h * L + t] /= Oe;
            }
        }
        for (int q = w - O; q < w; ++q)
            for (int t = 0; t < L; ++t) {
                double m = Akv[(size_t)q * L + t];
                for (int h = 1; h < Hkv; ++h) {
                    double x = Akv[((size_t)h * w + q) * L + t];
                    if (x > m) m = x;
                }
                Iraw[t] += m;
            }
        for (int t = 0; t < L; ++t) Iraw[t] /= O;
        free(Akv);

        /* Step 4: pool every row over the candidates [0, Lc) (max, or the average variant). */
        void (*pool)(const double*, int, int, double*) = p->pool_mode == 1 ? avg_pool : max_pool;
        double* PpO = (double*)calloc((size_t)Hkv * (Lc > 0 ? Lc : 1), sizeof(double));
        double* PpOe = (double*)calloc((size_t)Hkv * (Lc > 0 ? Lc : 1), sizeof(double));
        double* Ip = (double*)calloc((size_t)(Lc > 0 ? Lc : 1), sizeof(double));
        for (int h = 0; h < Hkv && Lc > 0; ++h) {
            pool(PO + (size_t)h * L, Lc, p->pool_kernel, PpO + (size_t)h * Lc);
            pool(POe + (size_t)h * L, Lc, p->pool_kernel, PpOe + (size_t)h * Lc);
        }
        if (Lc > 0) pool(Iraw, Lc, p->pool_kernel, Ip);

        /* Step 5 (Section 4.1): sigma_h = std(P_h) over candidates; the delta heads
         * with the lowest sigma take the extended-window scores. */
        double* sigma = (double*)calloc((size_t)Hkv, sizeof(double));
        int* htop = (int*)calloc((size_t)Hkv, sizeof(int));
        for (int h = 0; h < Hkv && p->head_criterion == 1; ++h) {
            /* Entropy variant (Section 5.4, "Head Selection Criteria"): the least
             * focused heads have the highest entropy of their pooled scores
             * normalised over the candidates; the key is minus that entropy so the
             * same lowest-first ranking applies.  0 with no mass. */
            const double* x = PpO + (size_t)h * Lc;
            double S = 0.0;
            for (int t = 0; t < Lc; ++t) S += x[t];
            double H = 0.0;
            if (S > 0.0)
                for (int t = 0; t < Lc; ++t)
                    if (x[t] > 0.0) H -= (x[t] / S) * log(x[t] / S);
            sigma[h] = -H;
        }
        for (int h = 0; h < Hkv && p->head_criterion == 0; ++h) {
            if (Lc < 2) { sigma[h] = 0.0; continue; }
            const double* x = PpO + (size_t)h * Lc;
            double mean = 0.0;
            for (int t = 0; t < Lc; ++t) mean += x[t];
            mean /= Lc;
            double ss = 0.0;
            for (int t = 0; t < Lc; ++t) ss += (x[t] - mean) * (x[t] - mean);
            sigma[h] = sqrt(ss / (Lc - 1));
        }
        for (int h = 0; h < Hkv; ++h) {
            int rank = 0;
            for (int o = 0; o < Hkv; ++o)
                if (sigma[o] < sigma[h] || (sigma[o] == sigma[h] && o < h)) ++rank;
            htop[h] = rank < p->num_ext_heads;
        }
        double* P = (double*)calloc((size_t)Hkv * (Lc > 0 ? Lc : 1), sizeof(double));
        for (int h = 0; h < Hkv; ++h)
            for (int t = 0; t < Lc; ++t)
                P[(size_t)h * Lc + t] = htop[h] ? PpOe[(size_t)h * Lc + t] : PpO[(size_t)h * Lc + t];

        /* Steps 6-8 (Section 4.2): preserve top-K of P, add lambda*focus, fill the rest. */
        const int keep_all = L <= budget;
        int Kp, k2, f0;
        budget_split(p, budget, &Kp, &k2, &f0);
        uint8_t* pres = (uint8_t*)calloc((size_t)Hkv * (Lc > 0 ? Lc : 1), 1);
        double* Pp = (double*)calloc((size_t)Hkv * (Lc > 0 ? Lc : 1), sizeof(double));
        uint8_t* keep = (uint8_t*)calloc((size_t)Hkv * L, 1);   /* S_h as a mask over [0, L) */
        for (int h = 0; h < Hkv; ++h) {
            uint8_t* ph = pres + (size_t)h * (Lc > 0 ? Lc : 1);
            double* pph = Pp + (size_t)h * (Lc > 0 ? Lc : 1);
            const double* Ph = P + (size_t)h * Lc;
            for (int t = 0; t < Lc; ++t) {
                double coverage = (double)n_t[t] / ((double)layers_done + 1.0);
                double focus = Ip[t] * (1.0 - coverage);
                pph[t] = Ph[t] + p->lambda * focus;
            }
            uint8_t* kh = keep + (size_t)h * L;
            if (keep_all) {
                for (int t = 0; t < L; ++t) kh[t] = 1;
                continue;
            }
            top_k(Ph, NULL, Lc, Kp, ph);
            uint8_t* others = (uint8_t*)malloc((size_t)Lc);
            for (int t = 0; t < Lc; ++t) others[t] = !ph[t];
            top_k(pph, others, Lc, f0, kh);   /* the whole fill (uniform) or the head's floor */
            for (int t = 0; t < Lc; ++t) if (ph[t]) kh[t] = 1;
            for (int t = Lc; t < L; ++t) kh[t] = 1;
            /* Literal reading: P' = 1.0 on preserved tokens, then top-(B-w) of P'. */
            if (dbg && !p->head_budget) {
                double* lit = (double*)malloc(sizeof(double) * (size_t)Lc);
                uint8_t* lsel = (uint8_t*)calloc((size_t)Lc, 1);
                for (int t = 0; t < Lc; ++t) lit[t] = ph[t] ? 1.0 : pph[t];
                top_k(lit, NULL, Lc, budget - wk, lsel);
                int differs = 0;
                for (int t = 0; t < Lc; ++t) if (lsel[t] != kh[t]) differs = 1;
                dbg->literal_override_differs += differs;
                free(lit);
                free(lsel);
            }
            free(others);
        }

        /* Adaptive fill: the rest of the layer's fill to the best P' over all
         * heads' remaining candidates, ranked together (entry h * Lc + t, so ties
         * go to the lower head, then the lower position). */
        if (p->head_budget && !keep_all && Lc > 0) {
            const size_t n = (size_t)Hkv * Lc;
            double* jk = (double*)malloc(sizeof(double) * n);
            uint8_t* ja = (uint8_t*)calloc(n, 1);
            uint8_t* js = (uint8_t*)calloc(n, 1);
            for (int h = 0; h < Hkv; ++h)
                for (int t = 0; t < Lc; ++t) {
                    const size_t i = (size_t)h * Lc + t;
                    jk[i] = Pp[i];
                    ja[i] = !pres[i] && !keep[(size_t)h * L + t];
                }
            top_k(jk, ja, (int)n, Hkv * (k2 - f0), js);
            for (int h = 0; h < Hkv; ++h)
                for (int t = 0; t < Lc; ++t)
                    if (js[(size_t)h * Lc + t]) keep[(size_t)h * L + t] = 1;
            free(jk);
            free(ja);
            free(js);
        }

        /* Outputs: ascending positions per head, then gather of K and V rows. */
        for (int h = 0; h < Hkv; ++h) {
            int32_t* oi = out_idx + ((size_t)b * Hkv + h) * cap;
            uint16_t* ok = out_k + ((size_t)b * Hkv + h) * cap * d;
            uint16_t* ov = out_v + ((size_t)b * Hkv + h) * cap * d;
            int j = 0;
            for (int t = 0; t < L; ++t) {
                if (!keep[(size_t)h * L + t]) continue;
                oi[j] = t;
                memcpy(ok + (size_t)j * d, kb + ((size_t)t * Hkv + h) * d, sizeof(uint16_t) * d);
                memcpy(ov + (size_t)j * d, vb + ((size_t)t * Hkv + h) * d, sizeof(uint16_t) * d);
                ++j;
            }
            for (; j < cap; ++j) {
                oi[j] = -1;
                memset(ok + (size_t)j * d, 0, sizeof(uint16_t) * d);
                memset(ov + (size_t)j * d, 0, sizeof(uint16_t) * d);
            }
        }

        /* Step 9 (Section 4.2): n_t counts the layers in which t was kept by at least one head. */
        const size_t words = ((size_t)max_seqlen + 31) / 32;
        memset(last_union, 0, 4 * words);
        int64_t covered = 0;
        for (int t = 0; t < L; ++t) {
            int any = 0;
            for (int h = 0; h < Hkv; ++h) any |= keep[(size_t)h * L + t];
            if (any) {
                n_t[t] = (uint8_t)(n_t[t] + 1);
                last_union[t / 32] |= 1u << (t % 32);
            }
            covered += n_t[t] > 0;
        }
        layers_done += 1;
        memcpy(st, &layers_done, 4);
        uint32_t seqlen = (uint32_t)L;
        memcpy(st + 4, &seqlen, 4);

        if (dbg) {
            for (int h = 0; h < Hkv; ++h) {
                size_t row = ((size_t)b * Hkv + h) * ML;
                for (int t = 0; t < ML; ++t) {
                    int cand = t < Lc;
                    if (dbg->P_O_raw) dbg->P_O_raw[row + t] = t < L ? PO[(size_t)h * L + t] : 0.0;
                    if (dbg->P_Oext_raw) dbg->P_Oext_raw[row + t] = t < L ? POe[(size_t)h * L + t] : 0.0;
                    if (dbg->P_O) dbg->P_O[row + t] = cand ? PpO[(size_t)h * Lc + t] : 0.0;
                    if (dbg->P_Oext) dbg->P_Oext[row + t] = cand ? PpOe[(size_t)h * Lc + t] : 0.0;
                    if (dbg->P) dbg->P[row + t] = cand ? P[(size_t)h * Lc + t] : 0.0;
                    if (dbg->Pprime) dbg->Pprime[row + t] = cand ? Pp[(size_t)h * Lc + t] : 0.0;
                    if (dbg->pres) dbg->pres[row + t] = cand ? pres[(size_t)h * Lc + t] : 0;
                }
                if (dbg->sigma) dbg->sigma[(size_t)b * Hkv + h] = sigma[h];
                if (dbg->htop) dbg->htop[(size_t)b * Hkv + h] = htop[h];
            }
            for (int t = 0; t < ML; ++t) {
                if (dbg->I_raw) dbg->I_raw[(size_t)b * ML + t] = t < L ? Iraw[t] : 0.0;
                if (dbg->I) dbg->I[(size_t)b * ML + t] = t < Lc ? Ip[t] : 0.0;
            }
            if (dbg->coverage) dbg->coverage[b] = covered;
        }

        free(PO); free(POe); free(Iraw); free(PpO); free(PpOe); free(Ip);
        free(sigma); free(htop); free(P); free(pres); free(Pp); free(keep);
    }
    return 0;
}
