/*
 * rr.h -- C ABI of librr.so, the GB300 (sm_103a) extend-attention library.
 *
 * The path it implements is the "extend" prefill of agents that return to a
 * prefix-cached serving engine (RR-Evict, Sec. 1 and Sec. 2: the engine reuses
 * the cached KV tensors of an agent's surviving prefix and computes only the
 * uncached suffix; the suffix's new KV tensors are materialised into the
 * shared, paged KV pool, Sec. 2).  Which prefix survives is decided by the
 * eviction policy (round-robin tail-chunk eviction, Algorithm 1, versus LRU,
 * Sec. 3.1-3.2); the kernels take the resulting per-agent lengths as input.
 *
 * Conventions shared by every call
 * --------------------------------
 *  * B agents; Hq query heads; Hkv KV heads, G = Hq / Hkv query heads per KV
 *    head (query head h reads KV head h / G); D head dim; ps tokens per page.
 *  * Agent b has a cached prefix of P_b = prefix_lens[b] tokens and an
 *    uncached suffix of S_b = suffix_lens[b] tokens.  Suffix token j of agent
 *    b has absolute position P_b + j.  Agents' suffix rows are packed in agent
 *    order: agent b owns rows cu_b .. cu_b + S_b - 1 of q / out / k_new /
 *    v_new, cu_b = S_0 + ... + S_{b-1};  T = sum of S_b = dims->total_tokens.
 *  * Layouts (row-major, contiguous, bf16 = IEEE bfloat16):
 *        q, out        [T, Hq, D]                 bf16
 *        k_new, v_new  [T, Hkv, D]                bf16
 *        k_pool,v_pool [num_pages, ps, Hkv, D]    bf16
 *        page_table    [B, max_pages]             int32, physical page of
 *                      logical page i of agent b (position i*ps .. i*ps+ps-1);
 *                      entries past ceil((P_b+S_b)/ps) are never read.
 *        prefix_lens, suffix_lens  [B]            int32
 *  * Memory: every pointer is a DEVICE pointer on the current device, owned
 *    by the caller; q/out/k_new/v_new/pools must be 16-byte aligned.  The
 *    library keeps one growable per-device workspace (schedule, error word),
 *    allocated on first use and freed by rr_shutdown().
 *  * Streams: calls enqueue work on `stream` and return without waiting; the
 *    lens stay on the device (the schedule is built on the device).
 *  * Errors: a call returns RR_OK or an RR_ERR_* code and never aborts; the
 *    message of the last failure on the calling thread is rr_last_error().
 *    Problems only the device can see (lens inconsistent with total_tokens,
 *    a page id outside the pool, a wait that timed out) are recorded in a
 *    device error word instead of faulting: read it with rr_get_device_error.
 */
#ifndef RR_H_
#define RR_H_

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RR_OK 0
#define RR_ERR_INVALID_ARG 1   /* null pointer, negative size, misaligned pointer */
#define RR_ERR_UNSUPPORTED 2   /* D not 64/128, G not in {1,2,4,8,16}, ps not in {16,32,64,128} */
#define RR_ERR_CUDA 3          /* a CUDA runtime/driver call failed */
#define RR_ERR_TIMEOUT 4       /* device: a bounded pipeline wait gave up (the kernel returned early) */
#define RR_ERR_OOB 5           /* device or host: a page id outside [0, num_pages) */
#define RR_ERR_LENS 6          /* device: negative length, P_b+S_b > max_pages*ps, or sum S_b != T */
#define RR_ERR_OVERLAP 7       /* host validation: a suffix page is shared with another agent or a prefix */
#define RR_ERR_SHARED 8        /* device: an agent's page table differs from agent 0's inside the declared shared prefix */

/* Sizes of one call.  All counts are in elements or tokens, not bytes. */
typedef struct rr_dims {
    int32_t batch;         /* B, number of agents (>= 0) */
    int32_t num_q_heads;   /* Hq */
    int32_t num_kv_heads;  /* Hkv; Hq % Hkv == 0 */
    int32_t head_dim;      /* D: 64 or 128 */
    int32_t page_size;     /* ps: tokens per page */
    int32_t max_pages;     /* columns of page_table */
    int64_t num_pages;     /* pages in EACH of k_pool and v_pool */
    int64_t total_tokens;  /* T = sum of suffix_lens (rows of q/out/k_new/v_new) */
} rr_dims;

/*
 * rr_kv_append -- write the uncached suffix's K/V into the pool (Sec. 2: the
 * prefill "materializes" the KV tensors of the tokens it processes; they go
 * into the shared pool so later turns can reuse them, Sec. 2 / Sec. 3.1).
 *
 * For every agent b and j < S_b, with pos = P_b + j:
 *     k_pool[page_table[b][pos / ps], pos % ps, :, :] = k_new[cu_b + j, :, :]
 *     v_pool[ ... same slot ... ]                      = v_new[cu_b + j, :, :]
 * Bytes are copied unchanged; no other pool byte is written.  The pages that
 * hold suffix positions must be distinct across agents (rr_validate_page_table
 * checks this on the host); pages shared between agents (a common system
 * prompt) are only ever read.  A page id outside the pool is skipped and
 * recorded as RR_ERR_OOB in the device error word.
 *
 * For a batch of at most 2047 agents the call is a single kernel that checks
 * the lengths and takes their prefix sums itself (it uses no workspace); a
 * larger batch runs the device-side schedule first, in the workspace.  Either
 * way, lengths inconsistent with total_tokens (or a negative length, or one
 * past the page table) write nothing and record RR_ERR_LENS.
 */
int rr_kv_append(const void* k_new, const void* v_new, void* k_pool, void* v_pool, const int32_t* page_table,
                 const int32_t* prefix_lens, const int32_t* suffix_lens, const rr_dims* dims,
                 cudaStream_t stream);

/*
 * rr_extend_attention -- attention of every uncached suffix row over the
 * agent's cached prefix and its own suffix (Sec. 1 and Sec. 2: the returning
 * agent reuses its surviving prefix and prefills the missing suffix).
 *
 * For agent b, suffix row i, query head h, g = h / G, p = P_b + i:
 *     s_j = scale * <q[cu_b+i, h, :], K_j>      for keys j = 0 .. p
 *     out[cu_b+i, h, :] = sum_j softmax(s)_j V_j
 * where K_j, V_j are position j of agent b, KV head g, read from
 * k_pool/v_pool through page_table.  The row sees the whole prefix and the
 * suffix up to and including itself (causal mask aligned bottom-right).
 * softmax_scale <= 0 selects 1/sqrt(D).  bf16 inputs, fp32 accumulation and
 * softmax, bf16 output rounded to nearest even.
 *
 * The suffix's K/V must already be in the pool: call rr_kv_append first on
 * the same stream.  Pool slots past an agent's last position are never read
 * into the result, whatever they contain.  The output is a deterministic
 * function of the logical inputs: it does not depend on the physical page
 * placement or on the order in which agents are listed.
 */
int rr_extend_attention(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                        const int32_t* prefix_lens, const int32_t* suffix_lens, void* out, const rr_dims* dims,
                        float softmax_scale, cudaStream_t stream);

/*
 * rr_extend_step -- the whole extend step of Sec. 2 in one attention launch:
 * the same results as rr_kv_append followed by rr_extend_attention on the
 * same stream (the pools receive the suffix K/V bit for bit, and `out` is
 * bit-identical), with two kernels launched instead of three.
 *
 * The kernel first writes every suffix row of k_new / v_new [T][Hkv][D] into
 * the pool slots page_table assigns to it, with all its threads; then every
 * CTA waits at a grid-wide barrier (the kernel is launched cooperatively, one
 * CTA per SM, so all of them are resident); then it runs the attention over
 * the pool.  The barrier's wait is bounded like the pipeline's waits
 * (rr_set_wait_limit): if it runs out, RR_ERR_TIMEOUT is recorded and the
 * output is undefined.  Arguments, layouts, preconditions and errors are those
 * of the two calls it replaces; k_pool / v_pool are written, so they are
 * non-const here.
 *
 * Performance (GB300): 1.01-1.03x the two calls on the long-context batches,
 * and up to ~1.09x on a single small extend (one agent, a few thousand keys),
 * where the saved launches matter most.
 */
int rr_extend_step(const void* q, const void* k_new, const void* v_new, void* k_pool, void* v_pool,
                   const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens, void* out,
                   const rr_dims* dims, float softmax_scale, cudaStream_t stream);

/*
 * rr_decode_attention -- decode attention over the same paged pool: the
 * extend attention above for a suffix of exactly one token per agent, the
 * step that follows an extend in an agent's turn (Sec. 2: an agent's request
 * reuses the cached KV and computes only what is new).
 *
 * q [B][Hq][D] bf16: the one new query token of each agent (row b is agent b).
 * kv_lens [B] int32 (device): L_b >= 1 keys of agent b in the pool, the new
 * token's own K/V included (append it first with rr_kv_append, prefix_lens =
 * L_b - 1, suffix_lens = 1).  out [B][Hq][D] bf16.  dims: total_tokens must
 * equal batch; the other fields as for rr_extend_attention.
 *     out[b, h, :] = sum_j softmax_j(scale * <q[b, h, :], K_j>) V_j,  j < L_b
 * with K_j, V_j position j of agent b, KV head h / G, through page_table.
 *
 * Same accuracy, determinism and page-placement independence as
 * rr_extend_attention; a kernel built for one query row per KV head (the
 * tensor cores take the keys as rows), bound by HBM bandwidth.  Batches with
 * few (agent, KV head) pairs split each agent's keys over several CTAs and
 * merge the pieces, as rr_extend_attention does.  Errors: RR_ERR_INVALID_ARG
 * (nulls, misalignment, total_tokens != batch), RR_ERR_UNSUPPORTED as for
 * rr_extend_attention; on the device a length L_b < 1 or L_b > max_pages *
 * page_size records RR_ERR_LENS and a page id outside the pool RR_ERR_OOB.
 * Allocates only the library's cached per-device workspace.
 */
int rr_decode_attention(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                        const int32_t* kv_lens, void* out, const rr_dims* dims, float softmax_scale,
                        cudaStream_t stream);

/*
 * Rotary position embedding (RoPE) of the suffix's rows
 * -----------------------------------------------------
 * The paper applies no positional encoding of its own, but the models its
 * agents run (Llama-3, Qwen3) rotate each q and k row by its absolute
 * position before attention (RoPE: Su et al., "RoFormer", 2021).  The calls
 * below take the suffix's q and k un-rotated and rotate them at positions
 * P_b + j -- the positions that continue the cached prefix, which is why the
 * cached (already rotated) keys stay valid across turns.  Convention: the
 * "rotate-half" pairing of GPT-NeoX / Llama, dim i < D/2 paired with i + D/2,
 * pair i at position p turned by a = p * base^(-2i/D):
 *     y[i] = x[i] cos a - x[i+D/2] sin a,   y[i+D/2] = x[i+D/2] cos a + x[i] sin a
 * The rotation runs in fp32 from a (cos a, sin a) table and is rounded to
 * nearest-even bf16: a rotated K row in the pool may differ from the exactly
 * rounded rotation by one bf16 unit in the last place in rare elements.
 * Rotating costs no extra pass over HBM: K is rotated by the append as it
 * writes the pool, q by the attention kernel as each Q tile lands in shared
 * memory (extend and decode alike).  Cached prefix keys are read as stored
 * (rotated when they were appended).
 */

/*
 * rr_rope_table -- fill table [max_pos][head_dim/2][2] float (device, 16-byte
 * aligned, caller-owned) with (cos a, sin a), a = p * base^(-2i/head_dim),
 * for positions 0 <= p < max_pos and pairs 0 <= i < head_dim/2.  Angles,
 * cosines and sines are computed in double precision and rounded once to
 * float.  Build it once per model (base 500000 for Llama-3, 10000 for older
 * models) with max_pos above the longest context.  head_dim 64 or 128,
 * base > 1.  Asynchronous on `stream`.
 */
int rr_rope_table(float* table, int32_t max_pos, int32_t head_dim, double base, cudaStream_t stream);

/*
 * rr_kv_append_rope -- rr_kv_append with each K row rotated at its position
 * P_b + j on its way into the pool (V is copied unchanged).  rope_table /
 * rope_max_pos: a table built by rr_rope_table for the same head_dim.  A
 * suffix position >= rope_max_pos is not written and records RR_ERR_LENS in
 * the device error word.  Other arguments, preconditions and errors as for
 * rr_kv_append.
 */
int rr_kv_append_rope(const void* k_new, const void* v_new, void* k_pool, void* v_pool, const int32_t* page_table,
                      const int32_t* prefix_lens, const int32_t* suffix_lens, const rr_dims* dims,
                      const float* rope_table, int32_t rope_max_pos, cudaStream_t stream);

/*
 * rr_extend_attention_rope -- rr_extend_attention with each suffix query row
 * rotated at its position P_b + i before its scores are taken (the rotated q
 * is rounded to bf16 for the tensor cores; q itself is not modified).  The
 * pool must hold rotated keys (rr_kv_append_rope for the suffix, and the same
 * for every earlier turn's keys).  A row whose position is >= rope_max_pos is
 * left un-rotated and records RR_ERR_LENS.  Other arguments as for
 * rr_extend_attention.
 */
int rr_extend_attention_rope(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                             const int32_t* prefix_lens, const int32_t* suffix_lens, void* out, const rr_dims* dims,
                             float softmax_scale, const float* rope_table, int32_t rope_max_pos,
                             cudaStream_t stream);

/*
 * rr_extend_step_rope -- the extend step with rotary embedding in one
 * launch: the same results as rr_kv_append_rope followed by
 * rr_extend_attention_rope on `stream` (pools and `out` bit-identical).  The
 * kernel's first phase rotates each K row at its position P_b + j as it
 * writes the pool (the same arithmetic as rr_kv_append_rope); after the grid
 * barrier the attention rotates q as each Q tile lands.  Other arguments,
 * preconditions and errors as for rr_extend_step and rr_kv_append_rope.
 */
int rr_extend_step_rope(const void* q, const void* k_new, const void* v_new, void* k_pool, void* v_pool,
                        const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens, void* out,
                        const rr_dims* dims, float softmax_scale, const float* rope_table, int32_t rope_max_pos,
                        cudaStream_t stream);

/*
 * rr_extend_attention_shared -- rr_extend_attention for a batch whose agents
 * all share their first shared_len positions (a common system prompt, the
 * same physical pages at the start of every page table: Sec. 2's shared
 * prefix cache), computed as a cascade.  A first pass attends every suffix
 * row of the batch to the shared keys only, in dense Q tiles of consecutive
 * rows whatever their agent (no causal mask is needed there: every suffix
 * position lies past the shared keys), and keeps each (token, query head)'s
 * unnormalised output and (max, sum) in fp32; a second pass attends each
 * agent's rows to its keys from shared_len on, as rr_extend_attention does,
 * and merges the two by their log-sum-exp weights.  Same result as
 * rr_extend_attention within the parity tolerance (the summation order
 * differs).  Measured slower than rr_extend_attention on GB300 (the shared
 * keys cost the tensor-bound kernel nothing it could save, and the partials
 * add a write and a read per row); provided for the comparison and for
 * batches where that changes.
 *
 * shared_len: a positive multiple of 128 with shared_len <= prefix_lens[b]
 * for every agent.  The device records RR_ERR_LENS if an agent's prefix is
 * shorter, and RR_ERR_SHARED if an agent's first shared_len / page_size
 * page-table entries differ from agent 0's; in either case no output is
 * written.  The workspace grows by total_tokens x Hq x (D + 2) x 4 bytes for
 * the partials.  Other arguments, layouts and errors as for
 * rr_extend_attention.
 */
int rr_extend_attention_shared(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                               const int32_t* prefix_lens, const int32_t* suffix_lens, int32_t shared_len, void* out,
                               const rr_dims* dims, float softmax_scale, cudaStream_t stream);

/*
 * rr_decode_attention_shared -- rr_decode_attention for a batch whose agents
 * all share their first shared_len positions (a common system prompt, the
 * same physical pages at the start of every page table: Sec. 2's shared
 * prefix cache).  Same result as rr_decode_attention (within the parity
 * tolerance: the merge order differs), fewer bytes: the shared pages are read
 * once per group of 16 / G agents of a KV head -- their queries fill the 16
 * columns the tensor-core MMA has, which G query heads alone leave mostly
 * padding -- instead of once per agent; each agent's keys from shared_len on
 * are read as by rr_decode_attention, and the two partial results of every
 * (agent, query head) are merged by their log-sum-exp weights.
 *
 * shared_len: a positive multiple of 128 with shared_len < kv_lens[b] for
 * every agent (each agent's own new token lies past the shared prefix).  The
 * device records RR_ERR_LENS if an agent's kv_lens is not larger, and
 * RR_ERR_SHARED if an agent's first shared_len / page_size page-table entries
 * differ from agent 0's.  Batches of more than 1024 (agent, KV head) pairs are
 * computed by rr_decode_attention.  Other arguments, layouts and errors as for
 * rr_decode_attention.
 */
int rr_decode_attention_shared(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                               const int32_t* kv_lens, int32_t shared_len, void* out, const rr_dims* dims,
                               float softmax_scale, cudaStream_t stream);

/*
 * rr_decode_attention_rope -- rr_decode_attention with each agent's query
 * rotated at its position L_b - 1 (the new token's) before its scores are
 * taken; the pool holds rotated keys (the new token's K appended with
 * rr_kv_append_rope, prefix_lens = L_b - 1, suffix_lens = 1).  A position >=
 * rope_max_pos leaves that agent's query un-rotated and records RR_ERR_LENS.
 * Other arguments as for rr_decode_attention.
 */
int rr_decode_attention_rope(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                             const int32_t* kv_lens, void* out, const rr_dims* dims, float softmax_scale,
                             const float* rope_table, int32_t rope_max_pos, cudaStream_t stream);

/*
 * rr_extend_attention_noalloc -- rr_extend_attention for callers that cannot
 * allocate device memory.  The paper has no counterpart; this is a deployment
 * convenience of this library.
 *
 * Some callers must not allocate during a call: a serving engine whose device
 * memory is entirely owned by its own pool allocator (the KV pool takes nearly
 * all of HBM), or a latency-critical loop that cannot afford the implicit
 * device-wide synchronisation of cudaMalloc/cudaFree.  This entry point
 * computes exactly what rr_extend_attention computes (same kernels, same
 * arguments and layouts), but keeps its schedule scratch in one fixed array
 * of static device memory (1,344,256 bytes, ~1.28 MiB) that every GPU
 * loading the library holds until the process exits.  It calls no
 * cudaMalloc, cudaFree or other allocating routine.
 *
 * Limits: at most 4096 agents, and at most 65536 schedule work units, where
 * the units needed are bounded by Hkv * (T / (256 / G) + B + 1).  Larger
 * batches return RR_ERR_UNSUPPORTED without launching anything.  It never
 * splits a unit's key range across CTAs (that needs partial-result buffers),
 * so small batches of long contexts run slower than through
 * rr_extend_attention; results agree within the parity tolerance.
 *
 * device_error: optional device int32 (4-byte aligned) that receives a
 * device-side error code (RR_ERR_LENS, RR_ERR_OOB, RR_ERR_TIMEOUT) if one
 * occurs; the kernels only ever write a nonzero code into it when it is still
 * zero, so the caller clears it.  With NULL, such errors are not reported.
 *
 * The first call on a device looks up the device address of the static array
 * (cudaGetSymbolAddress) and the device's SM count; make that first call
 * before any stream capture.  All calls on a device share the one array and
 * it keeps the last call's contents (every field is rewritten by each call
 * before it is read), so calls that overlap on the GPU -- on different
 * streams, or from different threads without ordering -- race on it and must
 * not be issued.
 */
int rr_extend_attention_noalloc(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                                const int32_t* prefix_lens, const int32_t* suffix_lens, void* out,
                                const rr_dims* dims, float softmax_scale, int32_t* device_error,
                                cudaStream_t stream);

/*
 * rr_validate_page_table -- HOST-side check of a page table before use
 * (host arrays, not device).  Returns RR_OK, RR_ERR_LENS (bad lengths),
 * RR_ERR_OOB (a page an agent uses is outside [0, num_pages)) or
 * RR_ERR_OVERLAP (a page holding suffix positions of one agent is used by
 * any other agent, or by the same agent twice).  Reads only; allocates a
 * bitmap of num_pages bits on the host.
 */
int rr_validate_page_table(const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens,
                           const rr_dims* dims);

/*
 * rr_get_device_error -- synchronise `stream`, return the device error word
 * of the current device (RR_OK or an RR_ERR_* code recorded by a kernel since
 * the last read) and reset it to RR_OK.
 */
int rr_get_device_error(cudaStream_t stream);

/* Message of the last failing call on this thread ("" if none). */
const char* rr_last_error(void);

/* Library version string. */
const char* rr_version(void);

/*
 * rr_set_wait_limit -- the budget, in GPU clock cycles, of the pipeline waits
 * of the attention kernels launched from now on by this process: every wait of
 * the decode kernel, and in the extend kernel the waits of its stage watcher
 * (the one thread that every K/V tile passes; the other roles keep the default
 * budget).  cycles <= 0 restores the default (2^33, about 4 s at 2 GHz).  A
 * wait that runs out does not trap: the kernel records RR_ERR_TIMEOUT in the
 * device error word, every role of every CTA leaves at its next unfinished
 * wait, in-flight copies and tensor-core operations are drained, tensor memory
 * is freed and the kernel returns, so the context stays usable.  A budget far
 * below a tile's load time makes that path run (the tests do this); results of
 * such a call are undefined.  One try of a wait suspends the thread for at
 * most a quarter of the budget (0.2 ms by default).
 */
void rr_set_wait_limit(long long cycles);

/* Free the per-device workspaces (synchronises each device that has one). */
void rr_shutdown(void);

/*
 * Self-describing tensors: the two calls of the extend step (rr_kv_append and
 * rr_extend_attention, Sec. 2) with every argument carrying its shape,
 * strides and element type, so that the library itself checks layouts a
 * caller might get wrong (a strided view, a transposed pool, an int64 length
 * array) instead of trusting the documented ones.  The plain-pointer calls
 * above stay the primary form: their sizes travel in one rr_dims and their
 * layouts are fixed by this header, which costs no per-call checks.
 *
 *   data    device pointer (same alignment rules as the plain calls)
 *   ndim    number of dimensions (1 to 4)
 *   shape   extent of each dimension, outermost first
 *   stride  distance in ELEMENTS between consecutive indices of each
 *           dimension; a dimension of extent 1 may have any stride
 *   dtype   RR_DTYPE_BF16 or RR_DTYPE_I32
 *
 * Accepted layouts are the plain calls' ones, row-major and contiguous:
 *   q, out [T, Hq, D] bf16; k_new, v_new [T, Hkv, D] bf16;
 *   k_pool, v_pool [num_pages, ps, Hkv, D] bf16 (same shape);
 *   page_table [B, max_pages] int32; prefix_lens, suffix_lens [B] int32.
 * Errors, returned before anything is launched: a null tensor or data
 * pointer, a wrong ndim, a negative extent or shapes that disagree with each
 * other -> RR_ERR_INVALID_ARG; a wrong dtype or any stride other than
 * row-major contiguous -> RR_ERR_UNSUPPORTED.  rr_last_error() names the
 * argument and the dimension.  Everything else (ownership, streams, device
 * errors, preconditions, results) is that of the plain call, which these
 * forward to with the rr_dims derived from the shapes.
 */
#define RR_DTYPE_BF16 1
#define RR_DTYPE_I32 2

typedef struct rr_tensor {
    void* data;
    int32_t ndim;
    int64_t shape[4];
    int64_t stride[4];
    int32_t dtype;
} rr_tensor;

int rr_kv_append_tensors(const rr_tensor* k_new, const rr_tensor* v_new, const rr_tensor* k_pool,
                         const rr_tensor* v_pool, const rr_tensor* page_table, const rr_tensor* prefix_lens,
                         const rr_tensor* suffix_lens, cudaStream_t stream);

int rr_extend_attention_tensors(const rr_tensor* q, const rr_tensor* k_pool, const rr_tensor* v_pool,
                                const rr_tensor* page_table, const rr_tensor* prefix_lens,
                                const rr_tensor* suffix_lens, const rr_tensor* out, float softmax_scale,
                                cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RR_H_ */
