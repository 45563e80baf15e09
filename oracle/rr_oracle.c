/*
 * rr_oracle.c -- plain, slow, fp64 CPU oracle for the extend-attention path.
 *
 * TEST INFRASTRUCTURE.  Only the tests, __graft_entry__.smoke() and the CPU
 * baseline leg of bench.py may load or call this file.  It shares no code,
 * header, table or helper with the CUDA library; it never reads anything the
 * CUDA path produced.
 *
 * What it computes (the paper never writes the attention formula; these are
 * the readings used throughout, each stated where it is used):
 *
 *  (A) KV append ("materializes their KV tensors", Sec. 2; into the shared
 *      pool, Sec. 2 / Sec. 3.1).  For agent b with cached prefix P_b and
 *      uncached suffix S_b, suffix token j (0 <= j < S_b) sits at absolute
 *      position pos = P_b + j, in page page_table[b][pos / ps], slot pos % ps.
 *      Its K row k_new[cu_b + j] (cu_b = sum of S over agents before b) is
 *      copied to k_pool[page][slot] and likewise for V.  Nothing else changes.
 *
 *  (B) Extend attention ("reuses the cached KV tensors for the shared prefix
 *      and computes the uncached suffix", Sec. 1 and Sec. 2).  For agent b,
 *      suffix row i, query head h, with G = Hq / Hkv, KV head g = floor(h / G)
 *      (contiguous GQA groups) and absolute position p = P_b + i:
 *          K_j, V_j = pool rows of position j of agent b, KV head g, j = 0..p
 *          s_j  = scale * <q, K_j>
 *          m    = max_j s_j
 *          w_j  = exp(s_j - m)
 *          o    = sum_j w_j V_j / sum_j w_j
 *          lse  = m + log(sum_j w_j)
 *      i.e. causal attention aligned bottom-right: the row sees the whole
 *      cached prefix and the suffix up to and including itself.  bf16 inputs
 *      are widened to double exactly; everything is computed in double.
 *      `wsum` returns sum_j (w_j / sum_j w_j), which is 1 up to rounding.
 *
 *  (C) Rotary position embedding of the suffix's q and k rows at positions
 *      P_b + j (not in the paper; the models its agents run use it -- see
 *      section (C) below for the reading), and the rounding of a rotated K row
 *      to the bf16 the pool stores.
 *
 * Parity of this oracle is pinned in tests/test_oracle_pins.py against a
 * dense brute force with an explicit mask matrix, closed forms and the
 * invariants (prefix-extend equals full causal attention; page permutation
 * leaves the result unchanged; softmax weights sum to 1).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_BAD_ARG 1
#define ORACLE_BAD_PAGE 2
#define ORACLE_NO_MEM 3

static double widen_bf16(uint16_t x) {
    uint32_t u = (uint32_t)x << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------------ (A) append */

int oracle_kv_append(const uint16_t* k_new, const uint16_t* v_new, uint16_t* k_pool, uint16_t* v_pool,
                     const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens,
                     int32_t B, int32_t Hkv, int32_t D, int32_t ps, int32_t max_pages, int64_t num_pages) {
    if (B < 0 || Hkv <= 0 || D <= 0 || ps <= 0 || max_pages < 0) return ORACLE_BAD_ARG;
    const int64_t row = (int64_t)Hkv * D; /* elements of one token's K (all KV heads) */
    int64_t cu = 0;
    for (int32_t b = 0; b < B; ++b) {
        int64_t P = prefix_lens[b], S = suffix_lens[b];
        if (P < 0 || S < 0 || P + S > (int64_t)max_pages * ps) return ORACLE_BAD_ARG;
        for (int64_t j = 0; j < S; ++j) {
            int64_t pos = P + j;
            int64_t page = page_table[(int64_t)b * max_pages + pos / ps];
            int64_t slot = pos % ps;
            if (page < 0 || page >= num_pages) return ORACLE_BAD_PAGE;
            int64_t dst = (page * ps + slot) * row;
            int64_t src = (cu + j) * row;
            for (int64_t e = 0; e < row; ++e) {
                k_pool[dst + e] = k_new[src + e];
                v_pool[dst + e] = v_new[src + e];
            }
        }
        cu += S;
    }
    return ORACLE_OK;
}

/* --------------------------------------------------------- (B) one attention row */

/*
 * Row at absolute position p over the logical key/value rows K[0..p], V[0..p]
 * (each D doubles, row stride D), query qv (D doubles).
 */
static void attention_row(const double* qv, const double* K, const double* V, int64_t p, int32_t D, double scale,
                          double* s /* scratch, p+1 */, double* o, double* lse, double* wsum) {
    double m = -INFINITY;
    for (int64_t j = 0; j <= p; ++j) {
        double dot = 0.0;
        for (int32_t d = 0; d < D; ++d) dot += qv[d] * K[j * D + d];
        s[j] = scale * dot;
        if (s[j] > m) m = s[j];
    }
    double l = 0.0;
    for (int64_t j = 0; j <= p; ++j) {
        s[j] = exp(s[j] - m);
        l += s[j];
    }
    for (int32_t d = 0; d < D; ++d) o[d] = 0.0;
    for (int64_t j = 0; j <= p; ++j)
        for (int32_t d = 0; d < D; ++d) o[d] += s[j] * V[j * D + d];
    for (int32_t d = 0; d < D; ++d) o[d] /= l;
    if (lse) *lse = m + log(l);
    if (wsum) {
        double t = 0.0;
        for (int64_t j = 0; j <= p; ++j) t += s[j] / l;
        *wsum = t;
    }
}

/* -------------------------------------------- (B) over the paged pool, all rows */

typedef struct {
    const uint16_t *q, *k_pool, *v_pool;
    const double* q64;       /* if set: q as doubles (already rotated by (C)), used instead of q */
    const int32_t *page_table, *prefix_lens, *suffix_lens;
    const int64_t* cu;
    int32_t B, Hq, Hkv, D, ps, max_pages;
    int64_t num_pages;
    double scale;
    double *out, *lse, *wsum;
    int64_t next;            /* next (b, g) work item, shared */
    pthread_mutex_t mu;
    int status;
} paged_job;

static void paged_item(paged_job* J, int32_t b, int32_t g, double* K, double* V, double* s, double* qv) {
    const int32_t G = J->Hq / J->Hkv, D = J->D;
    const int64_t P = J->prefix_lens[b], S = J->suffix_lens[b], L = P + S;
    /* gather agent b's keys and values of KV head g, position by position */
    for (int64_t j = 0; j < L; ++j) {
        int64_t page = J->page_table[(int64_t)b * J->max_pages + j / J->ps];
        if (page < 0 || page >= J->num_pages) {
            J->status = ORACLE_BAD_PAGE;
            return;
        }
        int64_t base = ((page * J->ps + j % J->ps) * J->Hkv + g) * (int64_t)D;
        for (int32_t d = 0; d < D; ++d) {
            K[j * D + d] = widen_bf16(J->k_pool[base + d]);
            V[j * D + d] = widen_bf16(J->v_pool[base + d]);
        }
    }
    for (int64_t i = 0; i < S; ++i) {
        int64_t t = J->cu[b] + i; /* row of q/out */
        for (int32_t hh = 0; hh < G; ++hh) {
            int32_t h = g * G + hh;
            if (J->q64) {
                const double* qsrc = J->q64 + (t * J->Hq + h) * (int64_t)D;
                for (int32_t d = 0; d < D; ++d) qv[d] = qsrc[d];
            } else {
                const uint16_t* qsrc = J->q + (t * J->Hq + h) * (int64_t)D;
                for (int32_t d = 0; d < D; ++d) qv[d] = widen_bf16(qsrc[d]);
            }
            int64_t r = t * J->Hq + h;
            attention_row(qv, K, V, P + i, D, J->scale, s, J->out + r * D, J->lse ? J->lse + r : NULL,
                          J->wsum ? J->wsum + r : NULL);
        }
    }
}

static void* paged_worker(void* arg) {
    paged_job* J = (paged_job*)arg;
    int64_t Lmax = 1;
    for (int32_t b = 0; b < J->B; ++b) {
        int64_t L = (int64_t)J->prefix_lens[b] + J->suffix_lens[b];
        if (L > Lmax) Lmax = L;
    }
    double* K = (double*)malloc(sizeof(double) * (size_t)Lmax * J->D);
    double* V = (double*)malloc(sizeof(double) * (size_t)Lmax * J->D);
    double* s = (double*)malloc(sizeof(double) * (size_t)Lmax);
    double* qv = (double*)malloc(sizeof(double) * (size_t)J->D);
    if (!K || !V || !s || !qv) {
        J->status = ORACLE_NO_MEM;
    } else {
        for (;;) {
            pthread_mutex_lock(&J->mu);
            int64_t item = J->next++;
            pthread_mutex_unlock(&J->mu);
            if (item >= (int64_t)J->B * J->Hkv || J->status) break;
            paged_item(J, (int32_t)(item / J->Hkv), (int32_t)(item % J->Hkv), K, V, s, qv);
        }
    }
    free(K); free(V); free(s); free(qv);
    return NULL;
}

static int run_threads(void* (*fn)(void*), void* job, int nthreads) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 512) nthreads = 512;
    pthread_t th[512];
    int started = 0;
    for (int t = 0; t < nthreads; ++t)
        if (pthread_create(&th[started], NULL, fn, job) == 0) ++started;
    if (started == 0) fn(job);
    for (int t = 0; t < started; ++t) pthread_join(th[t], NULL);
    return 0;
}

/*
 * out: [T, Hq, D] doubles; lse, wsum: [T, Hq] doubles or NULL.
 * scale <= 0 is NOT replaced here: the caller passes the scale it wants
 * (1/sqrt(D) for the workloads), and scale == 0 is a legal input (uniform weights).
 */
static int extend_attention_any(const uint16_t* q, const double* q64, const uint16_t* k_pool,
                                const uint16_t* v_pool, const int32_t* page_table, const int32_t* prefix_lens,
                                const int32_t* suffix_lens, int32_t B, int32_t Hq, int32_t Hkv, int32_t D, int32_t ps,
                                int32_t max_pages, int64_t num_pages, double scale, double* out, double* lse,
                                double* wsum, int32_t nthreads) {
    if (B < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || D <= 0 || ps <= 0 || max_pages < 0) return ORACLE_BAD_ARG;
    int64_t* cu = (int64_t*)malloc(sizeof(int64_t) * (size_t)(B + 1));
    if (!cu) return ORACLE_NO_MEM;
    cu[0] = 0;
    for (int32_t b = 0; b < B; ++b) {
        if (prefix_lens[b] < 0 || suffix_lens[b] < 0 ||
            (int64_t)prefix_lens[b] + suffix_lens[b] > (int64_t)max_pages * ps) {
            free(cu);
            return ORACLE_BAD_ARG;
        }
        cu[b + 1] = cu[b] + suffix_lens[b];
    }
    paged_job J;
    memset(&J, 0, sizeof J);
    J.q = q; J.q64 = q64; J.k_pool = k_pool; J.v_pool = v_pool;
    J.page_table = page_table; J.prefix_lens = prefix_lens; J.suffix_lens = suffix_lens; J.cu = cu;
    J.B = B; J.Hq = Hq; J.Hkv = Hkv; J.D = D; J.ps = ps; J.max_pages = max_pages; J.num_pages = num_pages;
    J.scale = scale; J.out = out; J.lse = lse; J.wsum = wsum;
    pthread_mutex_init(&J.mu, NULL);
    run_threads(paged_worker, &J, nthreads);
    pthread_mutex_destroy(&J.mu);
    free(cu);
    return J.status;
}

int oracle_extend_attention(const uint16_t* q, const uint16_t* k_pool, const uint16_t* v_pool,
                            const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens,
                            int32_t B, int32_t Hq, int32_t Hkv, int32_t D, int32_t ps, int32_t max_pages,
                            int64_t num_pages, double scale, double* out, double* lse, double* wsum,
                            int32_t nthreads) {
    return extend_attention_any(q, NULL, k_pool, v_pool, page_table, prefix_lens, suffix_lens, B, Hq, Hkv, D, ps,
                                max_pages, num_pages, scale, out, lse, wsum, nthreads);
}

/* The same with q given as doubles [T, Hq, D] (a q rotated by (C) in double precision, not rounded). */
int oracle_extend_attention_q64(const double* q, const uint16_t* k_pool, const uint16_t* v_pool,
                                const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens,
                                int32_t B, int32_t Hq, int32_t Hkv, int32_t D, int32_t ps, int32_t max_pages,
                                int64_t num_pages, double scale, double* out, double* lse, double* wsum,
                                int32_t nthreads) {
    return extend_attention_any(NULL, q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, B, Hq, Hkv, D, ps,
                                max_pages, num_pages, scale, out, lse, wsum, nthreads);
}

/* ------------------------------- (B) selected rows over one agent's logical K/V */

typedef struct {
    const uint16_t *q, *K, *V;
    const double* q64;       /* if set: q as doubles, used instead of q */
    const int64_t* positions;
    int64_t n_rows, n_keys;
    int32_t G, D;
    double scale;
    double *Kd, *Vd;
    double *out, *lse, *wsum;
    int64_t next;
    pthread_mutex_t mu;
    int status;
} rows_job;

static void* rows_worker(void* arg) {
    rows_job* J = (rows_job*)arg;
    double* s = (double*)malloc(sizeof(double) * (size_t)(J->n_keys > 0 ? J->n_keys : 1));
    double* qv = (double*)malloc(sizeof(double) * (size_t)J->D);
    if (!s || !qv) {
        J->status = ORACLE_NO_MEM;
    } else {
        for (;;) {
            pthread_mutex_lock(&J->mu);
            int64_t item = J->next++;
            pthread_mutex_unlock(&J->mu);
            if (item >= J->n_rows * J->G) break;
            int64_t r = item / J->G;
            int32_t hh = (int32_t)(item % J->G);
            if (J->q64) {
                const double* qsrc = J->q64 + (r * J->G + hh) * (int64_t)J->D;
                for (int32_t d = 0; d < J->D; ++d) qv[d] = qsrc[d];
            } else {
                const uint16_t* qsrc = J->q + (r * J->G + hh) * (int64_t)J->D;
                for (int32_t d = 0; d < J->D; ++d) qv[d] = widen_bf16(qsrc[d]);
            }
            attention_row(qv, J->Kd, J->Vd, J->positions[r], J->D, J->scale, s, J->out + item * J->D,
                          J->lse ? J->lse + item : NULL, J->wsum ? J->wsum + item : NULL);
        }
    }
    free(s); free(qv);
    return NULL;
}

/*
 * Rows of one agent and one KV head, given that agent's LOGICAL keys/values
 * K, V: [n_keys, D] bf16 (position j at row j).  q: [n_rows, G, D] bf16 holds
 * the G query heads of the group for each selected row; positions[r] is the
 * row's absolute position (it sees keys 0..positions[r]).
 * out: [n_rows, G, D]; lse, wsum: [n_rows, G] or NULL.
 */
static int attention_rows_any(const uint16_t* q, const double* q64, const int64_t* positions, int64_t n_rows,
                              const uint16_t* K, const uint16_t* V, int64_t n_keys, int32_t G, int32_t D,
                              double scale, double* out, double* lse, double* wsum, int32_t nthreads) {
    if (n_rows < 0 || n_keys < 0 || G <= 0 || D <= 0) return ORACLE_BAD_ARG;
    for (int64_t r = 0; r < n_rows; ++r)
        if (positions[r] < 0 || positions[r] >= n_keys) return ORACLE_BAD_ARG;
    rows_job J;
    memset(&J, 0, sizeof J);
    J.Kd = (double*)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1) * D);
    J.Vd = (double*)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1) * D);
    if (!J.Kd || !J.Vd) {
        free(J.Kd); free(J.Vd);
        return ORACLE_NO_MEM;
    }
    for (int64_t e = 0; e < n_keys * D; ++e) {
        J.Kd[e] = widen_bf16(K[e]);
        J.Vd[e] = widen_bf16(V[e]);
    }
    J.q = q; J.q64 = q64; J.K = K; J.V = V; J.positions = positions; J.n_rows = n_rows; J.n_keys = n_keys;
    J.G = G; J.D = D; J.scale = scale; J.out = out; J.lse = lse; J.wsum = wsum;
    pthread_mutex_init(&J.mu, NULL);
    run_threads(rows_worker, &J, nthreads);
    pthread_mutex_destroy(&J.mu);
    free(J.Kd); free(J.Vd);
    return J.status;
}

int oracle_attention_rows(const uint16_t* q, const int64_t* positions, int64_t n_rows, const uint16_t* K,
                          const uint16_t* V, int64_t n_keys, int32_t G, int32_t D, double scale, double* out,
                          double* lse, double* wsum, int32_t nthreads) {
    return attention_rows_any(q, NULL, positions, n_rows, K, V, n_keys, G, D, scale, out, lse, wsum, nthreads);
}

/* The same with q_rows given as doubles [n_rows, G, D]. */
int oracle_attention_rows_q64(const double* q, const int64_t* positions, int64_t n_rows, const uint16_t* K,
                              const uint16_t* V, int64_t n_keys, int32_t G, int32_t D, double scale, double* out,
                              double* lse, double* wsum, int32_t nthreads) {
    return attention_rows_any(NULL, q, positions, n_rows, K, V, n_keys, G, D, scale, out, lse, wsum, nthreads);
}

/* ------------------------------------------------- (C) rotary position embedding
 *
 * The paper never mentions positional encodings.  The models its agents run
 * (Llama-3, Qwen3) rotate every query and key row by its absolute position
 * before attention (RoPE: Su et al., "RoFormer: Enhanced Transformer with
 * Rotary Position Embedding", 2021), so an extend step that receives
 * un-rotated rows rotates the suffix's q and k at positions P_b + j -- the
 * positions that continue the cached prefix, which is why the cached keys stay
 * valid.  Reading used: the "rotate-half" pairing of GPT-NeoX and Llama (dim i
 * < D/2 pairs with dim i + D/2) and angle p * base^(-2i/D) for pair i:
 *     y[i]       = x[i]       cos(a) - x[i + D/2] sin(a)
 *     y[i + D/2] = x[i + D/2] cos(a) + x[i]       sin(a),   a = p * base^(-2i/D)
 * x: [rows, heads, D] doubles, pos: [rows]; out: [rows, heads, D] doubles.
 */
int oracle_rope(const double* x, const int64_t* pos, int64_t rows, int32_t heads, int32_t D, double base,
                double* out) {
    if (rows < 0 || heads <= 0 || D <= 0 || D % 2 || !(base > 0.0)) return ORACLE_BAD_ARG;
    const int32_t half = D / 2;
    for (int64_t r = 0; r < rows; ++r) {
        for (int32_t i = 0; i < half; ++i) {
            const double a = (double)pos[r] * pow(base, -2.0 * i / D);
            const double c = cos(a), s = sin(a);
            for (int32_t h = 0; h < heads; ++h) {
                const double* xr = x + (r * heads + h) * (int64_t)D;
                double* yr = out + (r * heads + h) * (int64_t)D;
                yr[i] = xr[i] * c - xr[i + half] * s;
                yr[i + half] = xr[i + half] * c + xr[i] * s;
            }
        }
    }
    return ORACLE_OK;
}

/*
 * Nearest bfloat16 of each double (8 significant bits, the binary32 exponent
 * range, subnormals down to 2^-133), ties to even, in ONE rounding from the
 * double value: the value is scaled so that the bf16 grid around it becomes
 * the integers, rounded by rint (ties to even in the default rounding mode) and
 * scaled back.  This is how a bf16 pool stores a K row rotated by (C).
 */
int oracle_round_bf16(const double* x, int64_t n, uint16_t* out) {
    for (int64_t e = 0; e < n; ++e) {
        double v = x[e];
        float f;
        if (isnan(v)) {
            f = NAN;
        } else if (v == 0.0 || isinf(v)) {
            f = (float)v;
        } else {
            int ex;
            frexp(v, &ex);                  /* |v| = m * 2^ex, m in [0.5, 1) */
            int q = ex - 8;                 /* bf16 spacing in [2^(ex-1), 2^ex) */
            if (q < -133) q = -133;         /* subnormal spacing */
            double r = ldexp(rint(ldexp(v, -q)), q);
            if (fabs(r) >= 0x1.0p128) r = v > 0 ? INFINITY : -INFINITY;
            f = (float)r;                   /* exact: r is on the bf16 grid */
        }
        uint32_t u;
        memcpy(&u, &f, sizeof u);
        out[e] = (uint16_t)(u >> 16);
    }
    return ORACLE_OK;
}
