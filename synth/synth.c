/*
 * Seeded synthetic inputs for the extend-attention path (CPU side).
 *
 * This module holds no arithmetic of the attention or append method: it only
 * produces input values.  Both the oracle harness (tests) and the GPU inputs
 * (bench, parity tests) draw from the same definition, so a value never has to
 * travel from one side to the other.
 *
 * Generator.  Every bf16 element is a pure function of its LOGICAL coordinates
 * (seed, tensor, owner, position, head, dim), never of the physical page it
 * lands in.  The hash is SplitMix64's output function (Steele, Lea, Flood,
 * "Fast Splittable Pseudorandom Number Generators", OOPSLA 2014, with the
 * "Mix13" finaliser constants published by D. Stafford): for a state z,
 *   z += 0x9e3779b97f4a7c15;
 *   z  = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9;
 *   z  = (z ^ (z >> 27)) * 0x94d049bb133111eb;
 *   return z ^ (z >> 31);
 * The element key is a chain of mixes over the coordinates; three more mixes
 * give twelve 16-bit uniform fields u_k, and the value is the Irwin-Hall sum
 *   x = (sum_k u_k - 393210) / 65536          (12 uniforms: mean 0, variance 1)
 * which is exact in fp32 (|numerator| < 2^20) and is rounded to bf16 with
 * round-to-nearest-even.  The result is bit-identical on any machine and on
 * the GPU (synth_fill.cu implements the same definition), with no libm.
 *
 * Owner.  Positions below `shared_len` belong to a prefix that all agents
 * share (one set of physical pages), so their owner is RRS_SHARED instead of
 * the agent index.
 */
#include <stdint.h>
#include <stddef.h>
#include <string.h>
#include <pthread.h>

#define RRS_SHARED 0xFFFFFFFFu
#define RRS_TENSOR_Q 1u
#define RRS_TENSOR_K 2u
#define RRS_TENSOR_V 3u

static inline uint64_t rrs_mix(uint64_t z) {
    z += 0x9e3779b97f4a7c15ull;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

/* Key of one token row: (seed, tensor, owner, pos). */
static inline uint64_t rrs_row_key(uint64_t seed, uint32_t tensor, uint32_t owner, uint64_t pos) {
    uint64_t h = rrs_mix(seed);
    h = rrs_mix(h ^ (uint64_t)tensor);
    h = rrs_mix(h ^ (uint64_t)owner);
    h = rrs_mix(h ^ pos);
    return h;
}

static inline uint16_t rrs_f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static inline uint16_t rrs_elem(uint64_t row_key, uint32_t head, uint32_t dim) {
    uint64_t h = rrs_mix(row_key ^ (((uint64_t)head << 20) | (uint64_t)dim));
    int32_t s = 0;
    for (uint64_t k = 1; k <= 3; ++k) {
        uint64_t r = rrs_mix(h + k);
        s += (int32_t)(r & 0xFFFF) + (int32_t)((r >> 16) & 0xFFFF) +
             (int32_t)((r >> 32) & 0xFFFF) + (int32_t)((r >> 48) & 0xFFFF);
    }
    float x = (float)(s - 393210) * (1.0f / 65536.0f);
    return rrs_f32_to_bf16_rne(x);
}

static inline uint32_t rrs_owner(int32_t agent, int64_t pos, int64_t shared_len) {
    return pos < shared_len ? RRS_SHARED : (uint32_t)agent;
}

/* ---- public scalar API ------------------------------------------------- */

uint64_t rrs_mix64(uint64_t z) { return rrs_mix(z); }

uint16_t rrs_value(uint64_t seed, uint32_t tensor, uint32_t owner, uint64_t pos, uint32_t head, uint32_t dim) {
    return rrs_elem(rrs_row_key(seed, tensor, owner, pos), head, dim);
}

/* ---- threaded fills ------------------------------------------------------ */

typedef struct {
    uint16_t* dst;            /* [n_rows, n_heads, D] */
    const int32_t* row_agent; /* [n_rows] */
    const int64_t* row_pos;   /* [n_rows] */
    int64_t n_rows;
    int32_t n_heads, D, head0, head_count;
    uint32_t tensor;
    uint64_t seed;
    int64_t shared_len;
    int64_t r0, r1;
} rrs_rows_job;

static void* rrs_rows_worker(void* arg) {
    rrs_rows_job* j = (rrs_rows_job*)arg;
    for (int64_t r = j->r0; r < j->r1; ++r) {
        uint32_t owner = rrs_owner(j->row_agent[r], j->row_pos[r], j->shared_len);
        uint64_t key = rrs_row_key(j->seed, j->tensor, owner, (uint64_t)j->row_pos[r]);
        uint16_t* out = j->dst + (size_t)r * (size_t)j->head_count * (size_t)j->D;
        for (int32_t h = 0; h < j->head_count; ++h)
            for (int32_t d = 0; d < j->D; ++d)
                out[(size_t)h * j->D + d] = rrs_elem(key, (uint32_t)(j->head0 + h), (uint32_t)d);
    }
    return NULL;
}

/*
 * dst[r, h, d] = value(seed, tensor, owner(row_agent[r], row_pos[r]), row_pos[r], head0 + h, d)
 * for h < head_count.  `n_heads` is informational (total heads of the tensor).
 */
void rrs_fill_rows(uint16_t* dst, const int32_t* row_agent, const int64_t* row_pos, int64_t n_rows,
                   int32_t head0, int32_t head_count, int32_t D, uint32_t tensor, uint64_t seed,
                   int64_t shared_len, int32_t nthreads) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    if (n_rows < 4096) nthreads = 1;
    pthread_t th[256];
    rrs_rows_job jobs[256];
    int64_t per = (n_rows + nthreads - 1) / nthreads;
    int started = 0;
    for (int t = 0; t < nthreads; ++t) {
        rrs_rows_job* j = &jobs[t];
        j->dst = dst; j->row_agent = row_agent; j->row_pos = row_pos; j->n_rows = n_rows;
        j->n_heads = head0 + head_count; j->D = D; j->head0 = head0; j->head_count = head_count;
        j->tensor = tensor; j->seed = seed; j->shared_len = shared_len;
        j->r0 = (int64_t)t * per;
        j->r1 = j->r0 + per < n_rows ? j->r0 + per : n_rows;
        if (j->r0 >= j->r1) continue;
        if (nthreads == 1) { rrs_rows_worker(j); continue; }
        if (pthread_create(&th[t], NULL, rrs_rows_worker, j) == 0) { ++started; } else { rrs_rows_worker(j); j->r0 = j->r1; }
    }
    if (nthreads > 1)
        for (int t = 0; t < nthreads; ++t)
            if (jobs[t].r0 < jobs[t].r1) pthread_join(th[t], NULL);
    (void)started;
}

/*
 * Write every cached-prefix position (pos < prefix_lens[b]) of every agent into
 * the paged pool [num_pages, ps, Hkv, D] through the page table.  Shared
 * positions are written by agent 0 only (all agents map them to the same
 * physical pages and the values are identical by construction).
 */
typedef struct {
    uint16_t* k_pool; uint16_t* v_pool;
    const int32_t* page_table; const int32_t* prefix_lens;
    int32_t B, max_pages, ps, Hkv, D;
    uint64_t seed; int64_t shared_len;
    int32_t b0, b1;
} rrs_pool_job;

static void* rrs_pool_worker(void* arg) {
    rrs_pool_job* j = (rrs_pool_job*)arg;
    size_t row_elems = (size_t)j->Hkv * (size_t)j->D;
    for (int32_t b = j->b0; b < j->b1; ++b) {
        int64_t P = j->prefix_lens[b];
        for (int64_t pos = (b == 0 ? 0 : (j->shared_len < P ? j->shared_len : P)); pos < P; ++pos) {
            int32_t page = j->page_table[(size_t)b * j->max_pages + (size_t)(pos / j->ps)];
            size_t base = ((size_t)page * j->ps + (size_t)(pos % j->ps)) * row_elems;
            uint32_t owner = rrs_owner(b, pos, j->shared_len);
            uint64_t kk = rrs_row_key(j->seed, RRS_TENSOR_K, owner, (uint64_t)pos);
            uint64_t kv = rrs_row_key(j->seed, RRS_TENSOR_V, owner, (uint64_t)pos);
            for (int32_t h = 0; h < j->Hkv; ++h)
                for (int32_t d = 0; d < j->D; ++d) {
                    j->k_pool[base + (size_t)h * j->D + d] = rrs_elem(kk, (uint32_t)h, (uint32_t)d);
                    j->v_pool[base + (size_t)h * j->D + d] = rrs_elem(kv, (uint32_t)h, (uint32_t)d);
                }
        }
    }
    return NULL;
}

void rrs_fill_pool_prefix(uint16_t* k_pool, uint16_t* v_pool, const int32_t* page_table,
                          const int32_t* prefix_lens, int32_t B, int32_t max_pages, int32_t ps,
                          int32_t Hkv, int32_t D, uint64_t seed, int64_t shared_len, int32_t nthreads) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > B) nthreads = B > 0 ? B : 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    rrs_pool_job jobs[256];
    int32_t per = (B + nthreads - 1) / nthreads;
    for (int t = 0; t < nthreads; ++t) {
        rrs_pool_job* j = &jobs[t];
        j->k_pool = k_pool; j->v_pool = v_pool; j->page_table = page_table; j->prefix_lens = prefix_lens;
        j->B = B; j->max_pages = max_pages; j->ps = ps; j->Hkv = Hkv; j->D = D;
        j->seed = seed; j->shared_len = shared_len;
        j->b0 = t * per; j->b1 = j->b0 + per < B ? j->b0 + per : B;
        if (j->b0 >= j->b1) continue;
        if (nthreads == 1 || pthread_create(&th[t], NULL, rrs_pool_worker, j) != 0) {
            rrs_pool_worker(j);
            j->b0 = j->b1;
        }
    }
    if (nthreads > 1)
        for (int t = 0; t < nthreads; ++t)
            if (jobs[t].b0 < jobs[t].b1) pthread_join(th[t], NULL);
}

/*
 * Seeded Fisher-Yates permutation of 0..n-1 (Durstenfeld's form), driven by a
 * SplitMix64 stream.  The bounded draw uses Lemire's multiply-shift
 * ("Fast Random Integer Generation in an Interval", 2019) without the rejection
 * step; its bias (< n / 2^64) does not matter for page placement.
 */
void rrs_permutation(int32_t* out, int64_t n, uint64_t seed) {
    for (int64_t i = 0; i < n; ++i) out[i] = (int32_t)i;
    uint64_t state = seed;
    for (int64_t i = n - 1; i > 0; --i) {
        uint64_t r = rrs_mix(state);
        state += 0x9e3779b97f4a7c15ull;
        uint64_t j = (uint64_t)(((unsigned __int128)r * (unsigned __int128)(uint64_t)(i + 1)) >> 64);
        int32_t t = out[i]; out[i] = out[j]; out[j] = t;
    }
}

/* A stream of n uniform 64-bit words from SplitMix64 (used for seeded length draws). */
void rrs_stream(uint64_t* out, int64_t n, uint64_t seed) {
    uint64_t state = seed;
    for (int64_t i = 0; i < n; ++i) {
        out[i] = rrs_mix(state);
        state += 0x9e3779b97f4a7c15ull;
    }
}
