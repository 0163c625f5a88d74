/*
 * PHSA CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, deliberately unoptimised fp64 restatement of what the PHSA
 * (Punctuation-aware Hybrid Sparse Attention) layer computes, written from the
 * paper's Section 3 and Algorithm 1. It exists to check the CUDA library and
 * must never be called from the product path: only the tests, the smoke check
 * and the CPU-baseline leg of the benchmark load it. It shares no code, header
 * or constant with the CUDA sources.
 *
 * Conventions
 *   - bf16 tensors arrive as uint16 bit patterns; they are decoded exactly to
 *     double. All arithmetic is fp64 in the order the definitions state.
 *   - Layout [B, H, L, D] row-major; head h reads KV head h / (Hq / Hkv).
 *   - Block t covers tokens [t*m, (t+1)*m) (Eq. 3); T = floor(L/m) blocks have
 *     a representative key; NQB = ceil(L/m) query blocks exist.
 *   - Selection is made per (query block, KV head): all G*m query rows of the
 *     block and of the KV head's query heads share one block set.
 *
 * Readings of the paper taken here (each is also listed in the design notes):
 *   R1 (Eq. 7 with no punctuation): M_p := M_0, so M = M_0 (Eq. 7's text and
 *      Algorithm 1's else-branch agree).
 *   R2 (Eq. 8, Algorithm 1 step 3): the relevance of block t to a query row is
 *      the softmax probability of q.M_t * scale taken over the candidate
 *      blocks only (forced and future blocks masked before the softmax); the
 *      group's relevance A_t is the sum of those probabilities over its rows.
 *   R3 (forced blocks): F_b = {0..n_init-1} U {b-n_local+1..b}, clipped to
 *      [0, b]. Candidates are the strictly earlier full blocks not in F_b.
 *   R4 (Top-K budget): `topk` counts forced blocks; min(topk-|F_b|, |C_b|)
 *      candidates are chosen, by A descending then block index ascending.
 *      The ranking compares A rounded to binary32, the precision in which the
 *      kernel takes the same decision.
 *   R5 (Eq. 10 inside the diagonal block): only keys at positions <= the
 *      query's own position take part (token-level causal mask).
 *   R6 (backward): selection is a hard choice; gradients flow to Q, K, V only.
 *   R7 (Krepr precision): the representative keys are stored as bf16 (round
 *      to nearest even) and scoring reads the stored values.
 *   R8 (max-logit variant, agg_mode 1): the group's relevance A_t is the
 *      largest raw score S_{r,t} = q_r . M_t * scale over its rows; for a
 *      single row this ranks exactly as Eq. 8's softmax does.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static int g_threads = 0;

void phsa_oracle_set_threads(int n) { g_threads = n; }

int phsa_oracle_max_threads(void) {
#ifdef _OPENMP
    return g_threads > 0 ? g_threads : omp_get_max_threads();
#else
    return 1;
#endif
}

#ifdef _OPENMP
#define NTH phsa_oracle_max_threads()
#endif

/* ---- bf16 <-> double -------------------------------------------------- */

double phsa_oracle_bf16_to_f64(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round a double to the nearest bf16 value, ties to even, in one step (no
 * intermediate float rounding). bf16 keeps 8 significant bits, so a finite
 * value of binary exponent e (x = f * 2^e, f in [0.5, 1)) is rounded to a
 * multiple of 2^(e-8); below the normal range the grid is fixed at 2^-133. */
uint16_t phsa_oracle_f64_to_bf16(double x) {
    if (isnan(x)) return 0x7FC0;
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (a == 0.0) return sign;
    if (isinf(a)) return sign | 0x7F80;
    int e;
    (void)frexp(a, &e);
    int q = e - 8;
    if (q < -133) q = -133;
    double r = nearbyint(ldexp(a, -q)); /* default mode: nearest, ties to even */
    double v = ldexp(r, q);
    if (v > 3.3895313892515355e38) return sign | 0x7F80; /* beyond bf16 max */
    float f = (float)v; /* exact: v has at most 8 significant bits */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return sign | (uint16_t)(u >> 16);
}

void phsa_oracle_bf16_to_f64_array(const uint16_t* h, int64_t n, double* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = phsa_oracle_bf16_to_f64(h[i]);
}

void phsa_oracle_f64_to_bf16_array(const double* x, int64_t n, uint16_t* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = phsa_oracle_f64_to_bf16(x[i]);
}

/* ---- Eq. 4-5: punctuation indicator from token ids --------------------- */

/* mask[i] = 1 if ids[i] is in the punctuation id set P, else 0. */
void phsa_oracle_punct_mask(const int32_t* ids, int64_t n, const int32_t* punct_ids,
                            int n_punct, uint8_t* mask) {
    for (int64_t i = 0; i < n; ++i) {
        uint8_t in = 0;
        for (int p = 0; p < n_punct; ++p)
            if (ids[i] == punct_ids[p]) in = 1;
        mask[i] = in;
    }
}

/* ---- Eq. 3, 6, 7, 8 / Algorithm 1 step 2: representative keys ----------- */

/* K [B,Hkv,L,D] bf16, mask [B,L]; Krepr [B,Hkv,T,D] bf16 (rounded, R7) and,
 * when Krepr64 is not NULL, the unrounded fp64 values. */
void phsa_oracle_block_repr(const uint16_t* K, const uint8_t* mask, int B, int Hkv, int L,
                            int D, int m, double lambda, uint16_t* Krepr, double* Krepr64) {
    const int T = L / m; /* Eq. 3: floor(L/m) full blocks */
    double* M0 = (double*)malloc(sizeof(double) * D);
    double* Sp = (double*)malloc(sizeof(double) * D);
    for (int b = 0; b < B; ++b)
        for (int g = 0; g < Hkv; ++g)
            for (int t = 0; t < T; ++t) {
                const uint16_t* Kbg = K + ((int64_t)b * Hkv + g) * L * D;
                int c = 0; /* number of punctuation tokens in the block */
                for (int d = 0; d < D; ++d) { M0[d] = 0.0; Sp[d] = 0.0; }
                for (int i = t * m; i < (t + 1) * m; ++i) {
                    int is_p = mask[(int64_t)b * L + i] != 0;
                    c += is_p;
                    for (int d = 0; d < D; ++d) {
                        double k = phsa_oracle_bf16_to_f64(Kbg[(int64_t)i * D + d]);
                        M0[d] += k;            /* Eq. 6 numerator */
                        if (is_p) Sp[d] += k;  /* Eq. 7 numerator */
                    }
                }
                for (int d = 0; d < D; ++d) {
                    double m0 = M0[d] / m;                    /* Eq. 6 */
                    double M;
                    if (c > 0) {
                        double mp = Sp[d] / c;                /* Eq. 7 */
                        M = lambda * m0 + (1.0 - lambda) * mp; /* Eq. 8 */
                    } else {
                        M = m0;                               /* R1 */
                    }
                    int64_t o = (((int64_t)b * Hkv + g) * T + t) * D + d;
                    Krepr[o] = phsa_oracle_f64_to_bf16(M);
                    if (Krepr64) Krepr64[o] = M;
                }
            }
    free(M0);
    free(Sp);
}

/* ---- Algorithm 1 step 3: scoring and block selection ------------------- */

typedef struct {
    float a32; /* aggregate rounded to binary32 (R4) */
    int t;
} cand_t;

static int cand_cmp(const void* x, const void* y) {
    const cand_t* a = (const cand_t*)x;
    const cand_t* b = (const cand_t*)y;
    if (a->a32 > b->a32) return -1;
    if (a->a32 < b->a32) return 1;
    return (a->t < b->t) ? -1 : (a->t > b->t);
}

static int is_forced(int t, int qb, int n_init, int n_local) {
    if (t > qb || t < 0) return 0;
    return t < n_init || t >= qb - n_local + 1;
}

/* The selection rule (R2-R4) for one query block qb of one KV head, whose
 * query rows are rows[0..nrows) (D bf16 values each, in the order their
 * probabilities are summed). Kr holds the KV head's representative keys, one
 * per block; only the first T of them exist. Writes topk entries to out and
 * returns the count, or -1 if topk < |F_b|. If agg is not NULL it receives A_t
 * for t < T (NaN where t was not scored). */
static int select_core(const uint16_t* const* rows, int nrows, const uint16_t* Kr, int T, int qb,
                       int D, int topk, int n_init, int n_local, double scale, int agg_mode,
                       int32_t* out, double* agg) {
    double* A = (double*)calloc((size_t)(T > 0 ? T : 1), sizeof(double));
    int* cand = (int*)malloc(sizeof(int) * (size_t)(qb + 1));
    int* chosen = (int*)calloc((size_t)(qb + 1), sizeof(int));
    int nC = 0, nF = 0, n = -1;
    for (int t = 0; t <= qb; ++t) {
        if (is_forced(t, qb, n_init, n_local)) { chosen[t] = 1; ++nF; }
        else if (t <= qb - 1 && t < T) cand[nC++] = t; /* causal: strictly past */
    }
    if (agg)
        for (int t = 0; t < T; ++t) agg[t] = NAN;
    if (topk >= nF) {
        int ksel = topk - nF;
        if (ksel >= nC) {
            for (int c = 0; c < nC; ++c) chosen[cand[c]] = 1;
        } else if (ksel > 0) {
            double* s = (double*)malloc(sizeof(double) * (size_t)nC);
            if (agg_mode == 1)
                for (int c = 0; c < nC; ++c) A[cand[c]] = -INFINITY;
            for (int r = 0; r < nrows; ++r) {
                const uint16_t* q = rows[r];
                double mx = -INFINITY;
                for (int c = 0; c < nC; ++c) {
                    const uint16_t* M = Kr + (int64_t)cand[c] * D;
                    double dot = 0.0;
                    for (int d = 0; d < D; ++d)
                        dot += phsa_oracle_bf16_to_f64(q[d]) * phsa_oracle_bf16_to_f64(M[d]);
                    s[c] = dot * scale; /* S_{r,t} */
                    if (s[c] > mx) mx = s[c];
                }
                if (agg_mode == 1) { /* R8 */
                    for (int c = 0; c < nC; ++c)
                        if (s[c] > A[cand[c]]) A[cand[c]] = s[c];
                    continue;
                }
                double z = 0.0;
                for (int c = 0; c < nC; ++c) z += exp(s[c] - mx);
                for (int c = 0; c < nC; ++c) A[cand[c]] += exp(s[c] - mx) / z; /* R2 */
            }
            free(s);
            cand_t* order = (cand_t*)malloc(sizeof(cand_t) * (size_t)nC);
            for (int c = 0; c < nC; ++c) {
                order[c].a32 = (float)A[cand[c]];
                order[c].t = cand[c];
                if (agg) agg[cand[c]] = A[cand[c]];
            }
            qsort(order, (size_t)nC, sizeof(cand_t), cand_cmp);
            for (int c = 0; c < ksel; ++c) chosen[order[c].t] = 1;
            free(order);
        }
        n = 0;
        for (int t = 0; t <= qb; ++t)
            if (chosen[t]) out[n++] = t; /* Unique, ascending */
        for (int j = n; j < topk; ++j) out[j] = -1;
    }
    free(A);
    free(cand);
    free(chosen);
    return n;
}

/* Selection for one (b, g, qb) unit u = (b*Hkv + g)*NQB + qb: the rows are the
 * block's tokens of each query head of the group, head by head. */
static int select_unit(const uint16_t* Q, const uint16_t* Krepr, int Hq, int Hkv, int L, int D,
                       int m, int topk, int n_init, int n_local, double scale, int agg_mode,
                       int64_t u, int32_t* out, double* agg) {
    const int G = Hq / Hkv, T = L / m, NQB = (L + m - 1) / m;
    const int qb = (int)(u % NQB);
    const int g = (int)((u / NQB) % Hkv);
    const int b = (int)(u / ((int64_t)NQB * Hkv));
    const uint16_t** rows = (const uint16_t**)malloc(sizeof(uint16_t*) * (size_t)(G * m));
    int nrows = 0;
    for (int hh = 0; hh < G; ++hh) {
        const int h = g * G + hh;
        for (int i = qb * m; i < (qb + 1) * m && i < L; ++i)
            rows[nrows++] = Q + (((int64_t)b * Hq + h) * L + i) * D;
    }
    int n = select_core(rows, nrows, Krepr + ((int64_t)b * Hkv + g) * T * D, T, qb, D, topk,
                        n_init, n_local, scale, agg_mode, out, agg);
    free(rows);
    return n;
}

/* Q [B,Hq,L,D] bf16, Krepr [B,Hkv,T,D] bf16.
 * Outputs block_idx [B,Hkv,NQB,topk] (ascending, -1 padded), block_cnt
 * [B,Hkv,NQB]. If agg is not NULL it receives A_t [B,Hkv,NQB,T] for every
 * scored candidate and NaN elsewhere (including blocks that were selected
 * without scoring because the budget covered every candidate).
 * Returns 0, or -1 if topk < |F_b| for some query block. */
int phsa_oracle_select_blocks(const uint16_t* Q, const uint16_t* Krepr, int B, int Hq,
                              int Hkv, int L, int D, int m, int topk, int n_init, int n_local,
                              double scale, int agg_mode, int32_t* block_idx, int32_t* block_cnt,
                              double* agg) {
    const int T = L / m, NQB = (L + m - 1) / m;
    int bad = 0;
    const int64_t units = (int64_t)B * Hkv * NQB;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(NTH) reduction(| : bad)
#endif
    for (int64_t u = 0; u < units; ++u) {
        int n = select_unit(Q, Krepr, Hq, Hkv, L, D, m, topk, n_init, n_local, scale, agg_mode,
                            u, block_idx + u * topk, agg ? agg + u * T : NULL);
        block_cnt[u] = n;
        if (n < 0) bad = 1;
    }
    return bad ? -1 : 0;
}

/* The same selection for a list of units only (sampled checks of large
 * problems): idx [n_units, topk], cnt [n_units], agg [n_units, T] or NULL. */
int phsa_oracle_select_units(const uint16_t* Q, const uint16_t* Krepr, int B, int Hq, int Hkv,
                             int L, int D, int m, int topk, int n_init, int n_local,
                             double scale, int agg_mode, const int64_t* units, int64_t n_units,
                             int32_t* idx, int32_t* cnt, double* agg) {
    const int T = L / m;
    int bad = 0;
    (void)B;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(NTH) reduction(| : bad)
#endif
    for (int64_t k = 0; k < n_units; ++k) {
        int n = select_unit(Q, Krepr, Hq, Hkv, L, D, m, topk, n_init, n_local, scale, agg_mode,
                            units[k], idx + k * topk, agg ? agg + k * T : NULL);
        cnt[k] = n;
        if (n < 0) bad = 1;
    }
    return bad ? -1 : 0;
}

/* ---- Eq. 10-11 / Algorithm 1 step 4: sparse attention, one row ---------- */

/* Collects the key positions row i attends: every position of every listed
 * block, up to and including i (R5). Returns their number. */
static int row_keys(const int32_t* idx, int cnt, int i, int L, int m, int* keys) {
    int n = 0;
    for (int c = 0; c < cnt; ++c) {
        int t = idx[c];
        if (t < 0) continue;
        for (int j = t * m; j < (t + 1) * m && j < L; ++j)
            if (j <= i) keys[n++] = j;
    }
    return n;
}

/* Computes one output row o_i (D values) and its log-sum-exp. */
static void attn_row(const uint16_t* q, const uint16_t* Kg, const uint16_t* Vg, const int* keys,
                     int nk, int D, double scale, double* s, double* o, double* lse) {
    double mx = -INFINITY;
    for (int n = 0; n < nk; ++n) {
        const uint16_t* k = Kg + (int64_t)keys[n] * D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d)
            dot += phsa_oracle_bf16_to_f64(q[d]) * phsa_oracle_bf16_to_f64(k[d]);
        s[n] = dot * scale;
        if (s[n] > mx) mx = s[n];
    }
    double z = 0.0;
    for (int n = 0; n < nk; ++n) z += exp(s[n] - mx);
    for (int d = 0; d < D; ++d) o[d] = 0.0;
    for (int n = 0; n < nk; ++n) {
        double p = exp(s[n] - mx) / z; /* Eq. 11 */
        const uint16_t* v = Vg + (int64_t)keys[n] * D;
        for (int d = 0; d < D; ++d) o[d] += p * phsa_oracle_bf16_to_f64(v[d]); /* Eq. 10 */
    }
    *lse = mx + log(z);
}

/* Rows listed as (b, h, i) triples; O_rows [n_rows, D], lse_rows [n_rows]. */
void phsa_oracle_sparse_attn_rows(const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                                  const int32_t* block_idx, const int32_t* block_cnt, int B,
                                  int Hq, int Hkv, int L, int D, int m, int topk, double scale,
                                  const int32_t* rows, int64_t n_rows, double* O_rows,
                                  double* lse_rows) {
    const int G = Hq / Hkv, NQB = (L + m - 1) / m;
    (void)B;
#ifdef _OPENMP
#pragma omp parallel num_threads(NTH)
#endif
    {
        int* keys = (int*)malloc(sizeof(int) * (size_t)L);
        double* s = (double*)malloc(sizeof(double) * (size_t)L);
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 16)
#endif
        for (int64_t r = 0; r < n_rows; ++r) {
            const int b = rows[3 * r], h = rows[3 * r + 1], i = rows[3 * r + 2];
            const int g = h / G, qb = i / m;
            const int64_t u = ((int64_t)b * Hkv + g) * NQB + qb;
            int nk = row_keys(block_idx + u * topk, block_cnt[u], i, L, m, keys);
            attn_row(Q + (((int64_t)b * Hq + h) * L + i) * D, K + ((int64_t)b * Hkv + g) * L * D,
                     V + ((int64_t)b * Hkv + g) * L * D, keys, nk, D, scale, s, O_rows + r * D,
                     lse_rows + r);
        }
        free(keys);
        free(s);
    }
}

/* Full forward: O [B,Hq,L,D] fp64, lse [B,Hq,L] fp64 (natural log). */
void phsa_oracle_sparse_attn_fwd(const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                                 const int32_t* block_idx, const int32_t* block_cnt, int B,
                                 int Hq, int Hkv, int L, int D, int m, int topk, double scale,
                                 double* O, double* lse) {
    const int G = Hq / Hkv, NQB = (L + m - 1) / m;
    const int64_t n_rows = (int64_t)B * Hq * L;
#ifdef _OPENMP
#pragma omp parallel num_threads(NTH)
#endif
    {
        int* keys = (int*)malloc(sizeof(int) * (size_t)L);
        double* s = (double*)malloc(sizeof(double) * (size_t)L);
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 16)
#endif
        for (int64_t r = 0; r < n_rows; ++r) {
            const int i = (int)(r % L);
            const int h = (int)((r / L) % Hq);
            const int b = (int)(r / ((int64_t)L * Hq));
            const int g = h / G, qb = i / m;
            const int64_t u = ((int64_t)b * Hkv + g) * NQB + qb;
            int nk = row_keys(block_idx + u * topk, block_cnt[u], i, L, m, keys);
            attn_row(Q + r * D, K + ((int64_t)b * Hkv + g) * L * D,
                     V + ((int64_t)b * Hkv + g) * L * D, keys, nk, D, scale, s, O + r * D,
                     lse + r);
        }
        free(keys);
        free(s);
    }
}

/* ---- Backward of the sparse attention (R6) ------------------------------
 * For each row i with keys J_i: P_ij = exp(S_ij - lse_i), o_i = sum_j P_ij v_j,
 * Delta_i = dO_i . o_i, dP_ij = dO_i . v_j, dS_ij = P_ij (dP_ij - Delta_i);
 * dV_j += P_ij dO_i, dK_j += dS_ij q_i * scale, dQ_i += dS_ij k_j * scale.
 * All quantities, o_i and lse_i included, are recomputed here in fp64.
 * Parallel over (b, kv head); each thread owns its dK/dV slices. */
void phsa_oracle_sparse_attn_bwd(const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                                 const uint16_t* dO, const int32_t* block_idx,
                                 const int32_t* block_cnt, int B, int Hq, int Hkv, int L, int D,
                                 int m, int topk, double scale, double* dQ, double* dK,
                                 double* dV) {
    const int G = Hq / Hkv, NQB = (L + m - 1) / m;
    memset(dQ, 0, sizeof(double) * (size_t)B * Hq * L * D);
    memset(dK, 0, sizeof(double) * (size_t)B * Hkv * L * D);
    memset(dV, 0, sizeof(double) * (size_t)B * Hkv * L * D);
    const int64_t units = (int64_t)B * Hkv;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(NTH)
#endif
    for (int64_t u = 0; u < units; ++u) {
        const int g = (int)(u % Hkv), b = (int)(u / Hkv);
        int* keys = (int*)malloc(sizeof(int) * (size_t)L);
        double* s = (double*)malloc(sizeof(double) * (size_t)L);
        double* o = (double*)malloc(sizeof(double) * (size_t)D);
        const uint16_t* Kg = K + u * L * D;
        const uint16_t* Vg = V + u * L * D;
        double* dKg = dK + u * L * D;
        double* dVg = dV + u * L * D;
        for (int hh = 0; hh < G; ++hh) {
            const int h = g * G + hh;
            for (int i = 0; i < L; ++i) {
                const int64_t r = ((int64_t)b * Hq + h) * L + i;
                const int64_t su = ((int64_t)b * Hkv + g) * NQB + i / m;
                int nk = row_keys(block_idx + su * topk, block_cnt[su], i, L, m, keys);
                double lse;
                attn_row(Q + r * D, Kg, Vg, keys, nk, D, scale, s, o, &lse);
                const uint16_t* q = Q + r * D;
                const uint16_t* go = dO + r * D;
                double delta = 0.0;
                for (int d = 0; d < D; ++d) delta += phsa_oracle_bf16_to_f64(go[d]) * o[d];
                for (int n = 0; n < nk; ++n) {
                    const int j = keys[n];
                    const uint16_t* k = Kg + (int64_t)j * D;
                    const uint16_t* v = Vg + (int64_t)j * D;
                    double p = exp(s[n] - lse);
                    double dp = 0.0;
                    for (int d = 0; d < D; ++d)
                        dp += phsa_oracle_bf16_to_f64(go[d]) * phsa_oracle_bf16_to_f64(v[d]);
                    double ds = p * (dp - delta);
                    for (int d = 0; d < D; ++d) {
                        dVg[(int64_t)j * D + d] += p * phsa_oracle_bf16_to_f64(go[d]);
                        dKg[(int64_t)j * D + d] += ds * phsa_oracle_bf16_to_f64(q[d]) * scale;
                        dQ[r * D + d] += ds * phsa_oracle_bf16_to_f64(k[d]) * scale;
                    }
                }
            }
        }
        free(keys);
        free(s);
        free(o);
    }
}

/* Sampled gradients for large problems. Same definitions as above.
 * dQ for the listed rows (b, h, i): dQ_rows [n_rows, D]. */
void phsa_oracle_sparse_attn_bwd_dq_rows(const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                                         const uint16_t* dO, const int32_t* block_idx,
                                         const int32_t* block_cnt, int B, int Hq, int Hkv, int L,
                                         int D, int m, int topk, double scale, const int32_t* rows,
                                         int64_t n_rows, double* dQ_rows) {
    const int G = Hq / Hkv, NQB = (L + m - 1) / m;
    (void)B;
#ifdef _OPENMP
#pragma omp parallel num_threads(NTH)
#endif
    {
        int* keys = (int*)malloc(sizeof(int) * (size_t)L);
        double* s = (double*)malloc(sizeof(double) * (size_t)L);
        double* o = (double*)malloc(sizeof(double) * (size_t)D);
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 4)
#endif
        for (int64_t r = 0; r < n_rows; ++r) {
            const int b = rows[3 * r], h = rows[3 * r + 1], i = rows[3 * r + 2];
            const int g = h / G;
            const int64_t su = ((int64_t)b * Hkv + g) * NQB + i / m;
            const uint16_t* Kg = K + ((int64_t)b * Hkv + g) * L * D;
            const uint16_t* Vg = V + ((int64_t)b * Hkv + g) * L * D;
            const uint16_t* q = Q + (((int64_t)b * Hq + h) * L + i) * D;
            const uint16_t* go = dO + (((int64_t)b * Hq + h) * L + i) * D;
            int nk = row_keys(block_idx + su * topk, block_cnt[su], i, L, m, keys);
            double lse;
            attn_row(q, Kg, Vg, keys, nk, D, scale, s, o, &lse);
            double delta = 0.0;
            for (int d = 0; d < D; ++d) delta += phsa_oracle_bf16_to_f64(go[d]) * o[d];
            double* dq = dQ_rows + r * D;
            for (int d = 0; d < D; ++d) dq[d] = 0.0;
            for (int n = 0; n < nk; ++n) {
                const uint16_t* k = Kg + (int64_t)keys[n] * D;
                const uint16_t* v = Vg + (int64_t)keys[n] * D;
                double p = exp(s[n] - lse), dp = 0.0;
                for (int d = 0; d < D; ++d)
                    dp += phsa_oracle_bf16_to_f64(go[d]) * phsa_oracle_bf16_to_f64(v[d]);
                double ds = p * (dp - delta);
                for (int d = 0; d < D; ++d) dq[d] += ds * phsa_oracle_bf16_to_f64(k[d]) * scale;
            }
        }
        free(keys);
        free(s);
        free(o);
    }
}

/* dK and dV of every key of the listed KV blocks (b, g, t): dK_out, dV_out
 * [n_blocks, m, D] (rows past L are zero). Every query row that attends a
 * key of block t lies in a query block qb >= t whose list contains t. */
void phsa_oracle_sparse_attn_bwd_kv_blocks(const uint16_t* Q, const uint16_t* K,
                                           const uint16_t* V, const uint16_t* dO,
                                           const int32_t* block_idx, const int32_t* block_cnt,
                                           int B, int Hq, int Hkv, int L, int D, int m, int topk,
                                           double scale, const int32_t* blocks, int64_t n_blocks,
                                           double* dK_out, double* dV_out) {
    const int G = Hq / Hkv, NQB = (L + m - 1) / m;
    (void)B;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(NTH)
#endif
    for (int64_t k = 0; k < n_blocks; ++k) {
        const int b = blocks[3 * k], g = blocks[3 * k + 1], t = blocks[3 * k + 2];
        int* keys = (int*)malloc(sizeof(int) * (size_t)L);
        double* s = (double*)malloc(sizeof(double) * (size_t)L);
        double* o = (double*)malloc(sizeof(double) * (size_t)D);
        double* dKb = dK_out + k * (int64_t)m * D;
        double* dVb = dV_out + k * (int64_t)m * D;
        memset(dKb, 0, sizeof(double) * (size_t)m * D);
        memset(dVb, 0, sizeof(double) * (size_t)m * D);
        const uint16_t* Kg = K + ((int64_t)b * Hkv + g) * L * D;
        const uint16_t* Vg = V + ((int64_t)b * Hkv + g) * L * D;
        for (int qb = t; qb < NQB; ++qb) {
            const int64_t su = ((int64_t)b * Hkv + g) * NQB + qb;
            int listed = 0;
            for (int c = 0; c < block_cnt[su]; ++c) listed |= block_idx[su * topk + c] == t;
            if (!listed) continue;
            for (int hh = 0; hh < G; ++hh) {
                const int h = g * G + hh;
                for (int i = qb * m; i < (qb + 1) * m && i < L; ++i) {
                    const uint16_t* q = Q + (((int64_t)b * Hq + h) * L + i) * D;
                    const uint16_t* go = dO + (((int64_t)b * Hq + h) * L + i) * D;
                    int nk = row_keys(block_idx + su * topk, block_cnt[su], i, L, m, keys);
                    double lse;
                    attn_row(q, Kg, Vg, keys, nk, D, scale, s, o, &lse);
                    double delta = 0.0;
                    for (int d = 0; d < D; ++d) delta += phsa_oracle_bf16_to_f64(go[d]) * o[d];
                    for (int n = 0; n < nk; ++n) {
                        const int j = keys[n];
                        if (j / m != t) continue;
                        const uint16_t* v = Vg + (int64_t)j * D;
                        double p = exp(s[n] - lse), dp = 0.0;
                        for (int d = 0; d < D; ++d)
                            dp += phsa_oracle_bf16_to_f64(go[d]) * phsa_oracle_bf16_to_f64(v[d]);
                        double ds = p * (dp - delta);
                        for (int d = 0; d < D; ++d) {
                            dVb[(int64_t)(j - t * m) * D + d] += p * phsa_oracle_bf16_to_f64(go[d]);
                            dKb[(int64_t)(j - t * m) * D + d] +=
                                ds * phsa_oracle_bf16_to_f64(q[d]) * scale;
                        }
                    }
                }
            }
        }
        free(keys);
        free(s);
        free(o);
    }
}

/* ---- Decode: one new token per sequence ----------------------------------
 * Sequence b holds lens[b] tokens of a cache with capacity Lc: K, V
 * [B,Hkv,Lc,D], Krepr [B,Hkv,Lc/m,D] (the representative keys of its full
 * blocks), q [B,Hq,D] the token at position p = lens[b] - 1. This is the same
 * rule as for a query block that holds the single row p (Section 3.3,
 * Algorithm 1 for one token, with the group's G heads as its rows): forced
 * F = {0..n_init-1} U {qb-n_local+1..qb} with qb = floor(p/m); candidates are
 * the strictly earlier full blocks. A sequence with lens[b] <= 0 has no query:
 * count 0, indices -1, output 0 and lse -inf. */
int phsa_oracle_decode_select(const uint16_t* q, const uint16_t* Krepr, const int32_t* lens,
                              int B, int Hq, int Hkv, int Lc, int D, int m, int topk, int n_init,
                              int n_local, double scale, int agg_mode, int32_t* block_idx,
                              int32_t* block_cnt, double* agg) {
    const int G = Hq / Hkv, Tc = Lc / m;
    int bad = 0;
    const int64_t units = (int64_t)B * Hkv;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(NTH) reduction(| : bad)
#endif
    for (int64_t u = 0; u < units; ++u) {
        const int b = (int)(u / Hkv), g = (int)(u % Hkv);
        const int len = lens[b];
        int32_t* out = block_idx + u * topk;
        double* ag = agg ? agg + u * Tc : NULL;
        if (ag)
            for (int t = 0; t < Tc; ++t) ag[t] = NAN;
        if (len <= 0 || len > Lc) {
            for (int j = 0; j < topk; ++j) out[j] = -1;
            block_cnt[u] = 0;
            if (len > Lc) bad = 1;
            continue;
        }
        const int p = len - 1;
        const uint16_t* rows[64];
        for (int hh = 0; hh < G && hh < 64; ++hh) rows[hh] = q + ((int64_t)b * Hq + g * G + hh) * D;
        int n = select_core(rows, G, Krepr + ((int64_t)b * Hkv + g) * Tc * D, len / m, p / m, D,
                            topk, n_init, n_local, scale, agg_mode, out, ag);
        block_cnt[u] = n;
        if (n < 0) bad = 1;
    }
    return bad ? -1 : 0;
}

/* Decode attention (Eq. 10-11 for row p): O [B,Hq,D] fp64, lse [B,Hq]. */
void phsa_oracle_decode_attn(const uint16_t* q, const uint16_t* K, const uint16_t* V,
                             const int32_t* block_idx, const int32_t* block_cnt,
                             const int32_t* lens, int B, int Hq, int Hkv, int Lc, int D, int m,
                             int topk, double scale, double* O, double* lse) {
    const int G = Hq / Hkv;
    const int64_t n_rows = (int64_t)B * Hq;
#ifdef _OPENMP
#pragma omp parallel num_threads(NTH)
#endif
    {
        int* keys = (int*)malloc(sizeof(int) * (size_t)(Lc > 0 ? Lc : 1));
        double* s = (double*)malloc(sizeof(double) * (size_t)(Lc > 0 ? Lc : 1));
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 4)
#endif
        for (int64_t r = 0; r < n_rows; ++r) {
            const int b = (int)(r / Hq), h = (int)(r % Hq), g = h / G;
            const int len = lens[b];
            if (len <= 0 || len > Lc) {
                for (int d = 0; d < D; ++d) O[r * D + d] = 0.0;
                lse[r] = -INFINITY;
                continue;
            }
            const int64_t u = (int64_t)b * Hkv + g;
            int nk = row_keys(block_idx + u * topk, block_cnt[u], len - 1, len, m, keys);
            attn_row(q + r * D, K + u * Lc * D, V + u * Lc * D, keys, nk, D, scale, s, O + r * D,
                     lse + r);
        }
        free(keys);
        free(s);
    }
}

/* ---- Eq. 1-2: dense causal attention (for the full-budget special case) -- */
void phsa_oracle_dense_causal(const uint16_t* Q, const uint16_t* K, const uint16_t* V, int B,
                              int Hq, int Hkv, int L, int D, double scale, double* O,
                              double* lse) {
    const int G = Hq / Hkv;
    const int64_t n_rows = (int64_t)B * Hq * L;
#ifdef _OPENMP
#pragma omp parallel num_threads(NTH)
#endif
    {
        int* keys = (int*)malloc(sizeof(int) * (size_t)L);
        double* s = (double*)malloc(sizeof(double) * (size_t)L);
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 16)
#endif
        for (int64_t r = 0; r < n_rows; ++r) {
            const int i = (int)(r % L);
            const int h = (int)((r / L) % Hq);
            const int b = (int)(r / ((int64_t)L * Hq));
            const int g = h / G;
            for (int j = 0; j <= i; ++j) keys[j] = j; /* every preceding key, Eq. 1 */
            attn_row(Q + r * D, K + ((int64_t)b * Hkv + g) * L * D,
                     V + ((int64_t)b * Hkv + g) * L * D, keys, i + 1, D, scale, s, O + r * D,
                     lse + r);
        }
        free(keys);
        free(s);
    }
}
