// decode_attn.cu -- paged-KV decode attention for sm_103a (tcgen05 + TMEM + TMA).
//
// What it computes: the extend attention of Sec. 2 for a suffix of one token --
// the next token of every agent attends to all L_b keys the agent has in the
// pool (its cached history plus the token itself, appended beforehand):
//
//   out[b, h, :] = softmax_j( scale * q[b, h, :] . K_j ) V_j,   j = 0 .. L_b - 1
//
// Decode reads every K/V byte of the batch once per KV head and does 4 G D flops
// per key -- about 4 flop per byte at G = 4: the work is bound by HBM, and the
// kernel's job is to keep enough page-gather loads in flight.
//
// Transposed formulation: the G query heads of one KV head are too few rows for
// an M = 128 MMA, so the keys take the M dimension and the heads the N dimension
// (padded to 16):
//   S^T (128 keys x 16)  = K_tile (128 x D, K-major)      . Q^T (D x 16, K-major)
//   O^T (D x 16)        += V_tile^T (D x 128, MN-major)   . P^T (128 keys x 16, K-major)
// S^T and O^T live in TMEM (lane = key, resp. lane = head dimension; column =
// head); P^T is written by the softmax threads to shared memory.
//
// Roles (one persistent CTA per SM, 7 warps):
//   * warps 0-3, softmax and epilogue: thread t owns key t of the tile (TMEM
//     lane t of S^T).  Per head: mask keys past the agent's end, the tile max
//     (warp shuffles, then the four warps' maxima through shared memory), a
//     running max in log2 units updated lazily (O^T is rescaled only when the
//     max grows by more than 2^8), p = 2^(s scale log2e - m) written to P^T as
//     bf16, and a per-thread partial weight sum.  At the end of a work item
//     thread t owns output dimension t: O^T row t / l, stored as bf16 (or the
//     fp32 partial of a split item, merged by the combine kernel).
//   * warps 4 and 6, TMA producers, taking the 128-key tiles in turn: per tile
//     one 2-D box per page and chunk for K and for V (the page gather), into a
//     ring of NS stages; slots of the agent's last page past its end are
//     cleared in shared memory before the MMA may read V.  Warp 4 also loads
//     Q^T (one 3-D box of G rows per 64-column chunk).
//   * warp 5, MMA issuer (one thread): S^T(t) into one of two TMEM buffers,
//     then O^T += V(t-1)^T P^T(t-1), so the scores of tile t are computed while
//     the softmax works on tile t-1.
//
// The work items and their split-K pieces come from the same on-device
// schedule as extend attention (one unit per agent and KV head; the schedule
// also writes the lengths as prefix = L - 1, suffix = 1), and a split
// item's partial uses the same layout (rows 0..G-1 of the unit), so the same
// combine kernel merges them.
//
// Every wait is bounded (clock64 budget); a wait that runs out sets the device
// error word to RR_ERR_TIMEOUT and a shared abort flag, every role leaves its
// loop, in-flight copies and MMAs are drained, TMEM is freed and the kernel
// returns.  No trap, no unbounded spin.
#include <cuda_bf16.h>

#include "ptx.cuh"
#include "rope.cuh"
#include "rr_internal.h"

namespace rr {

namespace {

// TMA producer warps: warp 4, then 6, 7, ...  One warp issuing every page box of K and V (32 boxes per tile at
// 16-token pages; a warp issues its lanes' boxes one after another) streamed c2_decode at 5.69 TB/s; two warps
// taking the tiles in turn, 6.25 TB/s; three, 6.26 TB/s.
constexpr int kDecProducers = 2;
constexpr int kDecThreads = 32 * (6 + kDecProducers - 1);  // warps 0-3 softmax / epilogue, 5 MMA, the rest producers
constexpr int kDecWarpProducer = 4;     // Q, and the K / V tiles the first producer takes
constexpr int kDecWarpMMA = 5;
constexpr int kHeadCols = 16;          // N of both MMAs: the G heads of a KV head, padded
constexpr uint32_t kDecTmemCols = 64;  // S^T buffers at columns 0 and 16, O^T at 32
constexpr long long kDecWaitLimit = 1ll << 33;  // ~4 s at 2 GHz: the TMEM release wait (pipeline waits: a.wait_limit)

template <int D, int NS>
struct DecCfg {
    static constexpr int kChunks = D / 64;
    static constexpr int kTileChunkBytes = kBN * 128;      // 16 KiB: one 64-column chunk of a 128-key tile
    static constexpr int kTileBytes = kBN * D * 2;         // K (or V) of one tile
    static constexpr int kStageBytes = 2 * kTileBytes;     // K, then V
    static constexpr int kNarrowChunkBytes = kHeadCols * 128;  // 2 KiB: 16 rows of one 64-element chunk
    static constexpr int kOffStage = 0;
    static constexpr int kOffQ = NS * kStageBytes;          // Q^T: 16 head rows x D
    static constexpr int kOffP = kOffQ + kChunks * kNarrowChunkBytes;  // P^T x 2: 16 head rows x 128 keys
    static constexpr int kPBytes = 2 * kNarrowChunkBytes;
    static constexpr int kOffRed = kOffP + 2 * kPBytes;     // float [2][4 warps][16 heads]
    static constexpr int kOffBar = kOffRed + 2 * 4 * kHeadCols * 4;
    // barrier indices
    static constexpr int kQFull = 0, kQEmpty = 1;
    static constexpr int kKFull = 2, kVFull = kKFull + NS, kKVEmpty = kVFull + NS, kVTmp = kKVEmpty + NS;
    static constexpr int kSFull = kVTmp + 1, kSEmpty = kSFull + 2, kPFull = kSEmpty + 2, kPEmpty = kPFull + 2;
    static constexpr int kOFinal = kPEmpty + 2, kOEmpty = kOFinal + 1, kXch = kOEmpty + 1, kDrain = kXch + 1;
    static constexpr int kDone = kDrain + 1;
    static constexpr int kQRot = kDone + 1;  // rotary q: the item's Q^T rows rotated in shared memory
    static constexpr int kVTmp2 = kQRot + 1;  // the other producers' side barriers for a partly owned last page
    static constexpr int kNumBars = kVTmp2 + kDecProducers - 1;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // u32 TMEM base, i32 abort flag
    static constexpr int kSmemBytes = kOffMisc + 16 + 1024;  // + slack to align the base to 1 KiB
    static_assert(kStageBytes % 1024 == 0 && kOffQ % 1024 == 0 && kOffP % 1024 == 0,
                  "swizzled tiles must start on 1 KiB boundaries");
    static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

struct DecCtl {
    volatile int32_t* abort_flag;
    int32_t* err;
    long long limit;  // cycles a pipeline wait may take before it gives up
    uint32_t hint;    // ns a try may suspend the thread (less than the budget)
};

__device__ __forceinline__ bool dec_wait(uint32_t bar, uint32_t parity, const DecCtl& c) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (ptx::mbar_try_wait_sleep(bar, parity, c.hint)) return true;
        if (*c.abort_flag) return false;
        if (clock64() - t0 > c.limit) {
            *c.abort_flag = 1;
            atomicCAS(c.err, 0, RR_ERR_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ void dec_drain(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!ptx::mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > (1ll << 31)) break;
    }
}

// 16 consecutive 32-bit TMEM columns of this thread's lane, and the matching store / register-carrying wait.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}
__device__ __forceinline__ void tmem_wait_ld16(uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.wait::ld.sync.aligned;"
        : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
          "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
        :
        : "memory");
}

__device__ __forceinline__ int dec_unit_of(int wave, int cta, int grid) {
    return wave * grid + ((wave & 1) ? (grid - 1 - cta) : cta);
}

// Rotary embedding of the item's Q^T rows (rope.cuh): the G head rows of the agent's new token, all at
// position pos = L_b - 1, in the 128-byte swizzled layout TMA wrote (16 rows per 64-column chunk).
// Softmax thread t takes head row t / (D/16) and rotation pair unit t % (D/16): G * D/16 <= 128 units.
// Not inlined, to keep the per-tile loop's code as it is without rotation.
template <int D, int G>
__device__ __noinline__ void dec_rope_q(uint8_t* qs, int t, const float2* __restrict__ rope, int rope_max_pos, int pos,
                                        int32_t* err) {
    constexpr int kUnits = D / 16;
    const int row = t / kUnits, u = t - row * kUnits;
    if (row >= G) return;
    if (pos >= rope_max_pos) {
        atomicCAS(err, 0, RR_ERR_LENS);
        return;
    }
    auto at = [&](int d) -> uint4* {
        return reinterpret_cast<uint4*>(qs + (d >> 6) * (kHeadCols * 128) + row * 128 + ((((d & 63) >> 3) ^ (row & 7)) << 4));
    };
    uint4* p0 = at(8 * u);
    uint4* p1 = at(8 * u + D / 2);
    uint4 x0 = *p0, x1 = *p1;
    float4 t4[4];
    rope_load8(t4, rope + (long long)pos * (D / 2) + 8 * u);
    rope_rotate8(x0, x1, t4);
    *p0 = x0;
    *p1 = x1;
}

// One work item: agent b (the first of the group for a shared-prefix item), KV head g, piece sp, its KV
// tiles [kb, ke) counted from the first tile the item's range starts at, and the number of keys L of that
// range (its last key is L - 1).
struct DecItem {
    int b, g, sp, kb, ke, L;
};

template <bool kGroup>
__device__ __forceinline__ DecItem dec_item(const AttnArgs& a, int ui) {
    DecItem it;
    if constexpr (kGroup) {
        // shared-prefix item ui = ((g * groups_per_head) + group) * group_ns + piece
        const int ns = a.group_ns;
        it.sp = ui % ns;
        const int t = ui / ns;
        it.g = t / a.groups_per_head;
        it.b = (t % a.groups_per_head) * a.group_agents;
        it.kb = it.sp * a.shared_tiles / ns;
        it.ke = (it.sp + 1) * a.shared_tiles / ns;
        it.L = a.shared_tiles * kBN;
    } else {
        const int4 U = a.units[ui];
        it.b = U.x;
        it.g = U.y & 0xFF;
        it.sp = (U.y >> 8) & 0xFF;
        const int ns = (U.y >> 16) & 0xFF;
        it.kb = it.sp * U.w / ns;
        it.ke = (it.sp + 1) * U.w / ns;
        it.L = a.prefix[it.b] + 1;  // keys of the agent (its private keys over a shared prefix), the new token's included
    }
    return it;
}

// G (query heads per KV head) is a template parameter: every per-head loop below is then unrolled
// without branches, so the heads' shuffle reductions, shared-memory reads and exponentials
// interleave instead of running one head after another.  kRope: q arrives un-rotated and the softmax
// warps rotate the item's Q^T rows once they land (dec_rope_q); the MMA thread waits for that.
//
// kGroup: the shared-prefix items of rr_decode_attention_shared.  G is then 16, the MMA's columns: the
// a.G query heads of a.group_agents consecutive agents (Q^T loaded through tm_qg), all over the same
// shared pages; each column's partial result goes to its agent's unit slot.
template <int D, int NS, int G, bool kRope, bool kGroup = false>
__global__ void __launch_bounds__(kDecThreads, 1) decode_attn_kernel(const __grid_constant__ AttnArgs a) {
    using C = DecCfg<D, NS>;
    static_assert(!(kRope && kGroup), "shared-prefix items take rotated queries only");
    static_assert(G >= 1 && G <= kHeadCols, "one KV head's query heads must fit the 16 MMA columns");
    // A producer waits for a stage's previous phase by parity, which is exact only while the barrier can be at
    // most one phase behind: a producer's own previous tile (kDecProducers tiles back) bounds its lead to that
    // only if kDecProducers <= NS.
    static_assert(kDecProducers >= 1 && kDecProducers <= NS, "more producers than stages");
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sb = ptx::smem_u32(smem);
    auto bar = [&](int i) -> uint32_t { return sb + C::kOffBar + 8u * (uint32_t)i; };
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(smem + C::kOffMisc + 4);
    const DecCtl ctl{abort_flag, a.err, a.wait_limit, a.wait_hint_ns};
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // Q^T rows G..15 and both P^T buffers start at zero: the padded head columns of S^T and O^T then
    // hold zeros, not whatever the shared memory held
    for (int i = threadIdx.x; i < (C::kOffRed - C::kOffQ) / 16; i += kDecThreads)
        reinterpret_cast<uint4*>(smem + C::kOffQ)[i] = make_uint4(0u, 0u, 0u, 0u);
    ptx::fence_proxy_async_smem();
    if (threadIdx.x == 0) {
        ptx::mbar_init(bar(C::kQFull), 1);
        ptx::mbar_init(bar(C::kQEmpty), 1);
        ptx::mbar_init(bar(C::kQRot), 128);  // the softmax warps
        for (int s = 0; s < NS; ++s) {
            ptx::mbar_init(bar(C::kKFull + s), 1);
            ptx::mbar_init(bar(C::kVFull + s), 1);
            ptx::mbar_init(bar(C::kKVEmpty + s), 1);
        }
        ptx::mbar_init(bar(C::kVTmp), 1);
        for (int i = 0; i < kDecProducers - 1; ++i) ptx::mbar_init(bar(C::kVTmp2 + i), 1);
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(bar(C::kSFull + i), 1);
            ptx::mbar_init(bar(C::kSEmpty + i), 4);   // one arrival per softmax warp
            ptx::mbar_init(bar(C::kPFull + i), kBM);  // every softmax thread
            ptx::mbar_init(bar(C::kPEmpty + i), 1);
        }
        ptx::mbar_init(bar(C::kOFinal), 1);
        ptx::mbar_init(bar(C::kOEmpty), kBM);
        ptx::mbar_init(bar(C::kXch), 4);
        ptx::mbar_init(bar(C::kDrain), 1);
        ptx::mbar_init(bar(C::kDone), kBM);
        *abort_flag = 0;
        ptx::fence_mbar_init();
    }
    if (warp == kDecWarpMMA) {
        ptx::tmem_alloc(sb + C::kOffMisc, kDecTmemCols);
        ptx::tmem_relinquish();
    }
    if (warp == kDecWarpProducer && lane == 0) {
        ptx::prefetch_tmap(&a.tm_q);
        ptx::prefetch_tmap(&a.tm_k);
        ptx::prefetch_tmap(&a.tm_v);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + C::kOffMisc);
    ptx::griddep_wait();  // the schedule kernel's output (launched as its dependent)
    // shared-prefix items: as many as the host set up, but none if the schedule rejected the batch (it then
    // lists no private items and has written no unit slots)
    const int n_units = kGroup ? (*a.n_units > 0 ? a.group_items : 0) : *a.n_units;
    const int grid = gridDim.x, cta = blockIdx.x;
    const int page0 = kGroup ? 0 : a.page0;  // page-table column of the item range's first key

    if (warp == kDecWarpProducer || warp > kDecWarpMMA) {
        // ------------------------------------------------------------ TMA producers
        // A tile of small pages is many TMA boxes (K and V: 32 at 16-token pages), and a warp issues its lanes'
        // boxes one after another; one warp alone kept too few bytes in flight for HBM.  The producers take the
        // tiles in turn (by the running tile count), each waiting for its own tiles' stages.
        const bool first_warp = warp == kDecWarpProducer;
        const uint32_t pi = first_warp ? 0u : (uint32_t)(warp - kDecWarpMMA);  // producer index
        const uint32_t vtmp_bar = bar(first_warp ? C::kVTmp : C::kVTmp2 + (int)pi - 1);
        const int ppt = kBN / a.ps;  // pages per tile (<= 16)
        uint32_t gt = 0, item_i = 0, vtmp_phase = 0;
        int armed_q = -1, armed_vtmp = -1;  // copies in flight, for the abort drain
        uint32_t armed_k = 0, armed_v = 0, par_k = 0, par_v = 0;
        bool ok = true;
        for (int w = 0; ok; ++w) {
            const int ui = dec_unit_of(w, cta, grid);
            if (ui >= n_units) break;
            const DecItem it = dec_item<kGroup>(a, ui);
            const int b = it.b, g = it.g, kb = it.kb, ke = it.ke, L = it.L;
            const int last_page_end = ((L + a.ps - 1) / a.ps) * a.ps;
            if (first_warp && lane == 0) {
                if (item_i > 0) ok = dec_wait(bar(C::kQEmpty), (item_i - 1) & 1, ctl);
                if (ok) {
                    // one box of 16 Q^T rows (group: group_agents agents x a.G heads; rows past the batch are
                    // zero-filled) or G rows, per 64-column chunk
                    ptx::mbar_arrive_expect_tx(bar(C::kQFull), C::kChunks * G * 128);
                    for (int c = 0; c < C::kChunks; ++c) {
                        if constexpr (kGroup)
                            ptx::tma_load_3d(sb + C::kOffQ + c * C::kNarrowChunkBytes, &a.tm_qg, c * 64, g * a.G, b,
                                             bar(C::kQFull));
                        else
                            ptx::tma_load_3d(sb + C::kOffQ + c * C::kNarrowChunkBytes, &a.tm_q, c * 64, g * G, a.cu[b],
                                             bar(C::kQFull));
                    }
                    armed_q = (int)(item_i & 1);
                }
            }
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            for (int j = kb; j < ke; ++j, ++gt) {
                if (gt % (uint32_t)kDecProducers != pi) continue;  // another producer's tile
                const int s = (int)(gt % NS);
                const uint32_t use = gt / NS;
                int row = a.oob_row;  // page past the agent's keys: zero fill
                if (lane < ppt) {
                    const int lp = j * ppt + lane;
                    if (lp * a.ps < L) {
                        const int pid = a.page_table[(long long)b * a.max_pages + page0 + lp];
                        if (pid >= 0 && (long long)pid < a.num_pages) row = pid * a.ps;
                        else atomicCAS(a.err, 0, RR_ERR_OOB);
                    }
                }
                if (lane == 0) {
                    if (use > 0) ok = dec_wait(bar(C::kKVEmpty + s), (use - 1) & 1, ctl);
                    if (ok) ptx::mbar_arrive_expect_tx(bar(C::kKFull + s), C::kTileBytes);
                }
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                armed_k |= 1u << s;
                par_k = (par_k & ~(1u << s)) | ((use & 1u) << s);
                uint8_t* st = smem + C::kOffStage + s * C::kStageBytes;
                const uint32_t sk = sb + C::kOffStage + s * C::kStageBytes, sv = sk + C::kTileBytes;
                if (lane < ppt)
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_2d(sk + c * C::kTileChunkBytes + lane * a.ps * 128, &a.tm_k, g * D + c * 64, row,
                                         bar(C::kKFull + s));
                // V; if the agent's last page is only partly its own, land it on the side barrier, clear the
                // slots past the agent's end, then release it
                const bool clear_tail = (j == (L - 1) / kBN) && (last_page_end > L);
                const uint32_t vbar = clear_tail ? vtmp_bar : bar(C::kVFull + s);
                if (lane == 0) ptx::mbar_arrive_expect_tx(vbar, C::kTileBytes);
                __syncwarp();
                if (lane < ppt)
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_2d(sv + c * C::kTileChunkBytes + lane * a.ps * 128, &a.tm_v, g * D + c * 64, row,
                                         vbar);
                if (clear_tail) {
                    armed_vtmp = (int)vtmp_phase;
                    if (lane == 0) ok = dec_wait(vtmp_bar, vtmp_phase, ctl);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) break;
                    armed_vtmp = -1;
                    vtmp_phase ^= 1;
                    const int r0 = L - j * kBN;  // 0 < r0 < kBN: first row past the agent
                    for (int c = 0; c < C::kChunks; ++c) {
                        uint4* base = reinterpret_cast<uint4*>(st + C::kTileBytes + c * C::kTileChunkBytes);
                        for (int e = r0 * 8 + lane; e < kBN * 8; e += 32) base[e] = make_uint4(0u, 0u, 0u, 0u);
                    }
                    ptx::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(bar(C::kVFull + s));
                } else {
                    armed_v |= 1u << s;
                    par_v = (par_v & ~(1u << s)) | ((use & 1u) << s);
                }
            }
            ++item_i;
        }
        if (!ok && lane == 0) {  // abort: let every copy this warp started land before exit
            if (armed_q >= 0) dec_drain(bar(C::kQFull), (uint32_t)armed_q);
            if (armed_vtmp >= 0) dec_drain(vtmp_bar, (uint32_t)armed_vtmp);
            for (int s = 0; s < NS; ++s) {
                if (armed_k >> s & 1u) dec_drain(bar(C::kKFull + s), par_k >> s & 1u);
                if (armed_v >> s & 1u) dec_drain(bar(C::kVFull + s), par_v >> s & 1u);
            }
        }
        __syncwarp();
        return;
    }
    if (warp == kDecWarpMMA) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_s = ptx::idesc_bf16_f32(kBM, kHeadCols, false, false);  // K . Q^T
            constexpr uint32_t idesc_o = ptx::idesc_bf16_f32(kBM, kHeadCols, true, false);  // V^T . P^T (M = 128 rows of V^T)
            const uint64_t desc_q = ptx::sdesc_sw128(sb + C::kOffQ, 16, 1024);
            const uint64_t desc_k0 = ptx::sdesc_sw128(sb + C::kOffStage, 16, 1024);
            // V^T as an MN-major operand: 64-column chunks C::kTileChunkBytes apart; with D = 64 the MMA's
            // second group of 64 rows (M = 128) reads the same chunk again and fills O^T lanes 64-127 with a
            // copy that is never read
            const uint64_t desc_v0 =
                ptx::sdesc_sw128(sb + C::kOffStage + C::kTileBytes, D == 128 ? C::kTileChunkBytes : 0, 1024);
            const uint64_t desc_p0 = ptx::sdesc_sw128(sb + C::kOffP, 16, 1024);
            uint32_t gt = 0, item_i = 0;
            bool ok = true;
            auto issue_s = [&](uint32_t t) {  // S^T(t) = K(t) . Q^T
                const int s = (int)(t % NS), buf = (int)(t & 1);
                const uint64_t dk = desc_k0 + (uint64_t)((s * C::kStageBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint64_t ok_ = (uint64_t)(((kk >> 2) * C::kTileChunkBytes + (kk & 3) * 32) >> 4);
                    const uint64_t oq = (uint64_t)(((kk >> 2) * C::kNarrowChunkBytes + (kk & 3) * 32) >> 4);
                    ptx::mma_ss(tmem + (uint32_t)(buf * kHeadCols), dk + ok_, desc_q + oq, idesc_s, kk > 0 ? 1u : 0u);
                }
            };
            auto issue_o = [&](uint32_t t, bool first) {  // O^T (+)= V(t)^T . P^T(t)
                const int s = (int)(t % NS), buf = (int)(t & 1);
                const uint64_t dv = desc_v0 + (uint64_t)((s * C::kStageBytes) >> 4);
                const uint64_t dp = desc_p0 + (uint64_t)((buf * C::kPBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk) {
                    const uint64_t ov = (uint64_t)((kk * 16 * 128) >> 4);
                    const uint64_t op = (uint64_t)(((kk >> 2) * C::kNarrowChunkBytes + (kk & 3) * 32) >> 4);
                    ptx::mma_ss(tmem + 2u * kHeadCols, dv + ov, dp + op, idesc_o, (!first || kk > 0) ? 1u : 0u);
                }
            };
            // O^T(t): wait for P^T(t) (and, at an item's first tile, for the previous epilogue), issue, release
            auto step_o = [&](uint32_t t, bool first) -> bool {
                const int buf = (int)(t & 1);
                if (!dec_wait(bar(C::kPFull + buf), (t >> 1) & 1, ctl)) return false;
                if (!dec_wait(bar(C::kVFull + (int)(t % NS)), (t / NS) & 1, ctl)) return false;
                if (first && item_i > 0 && !dec_wait(bar(C::kOEmpty), (item_i - 1) & 1, ctl)) return false;
                ptx::tc_fence_after();
                issue_o(t, first);
                ptx::mma_commit(bar(C::kPEmpty + buf));
                ptx::mma_commit(bar(C::kKVEmpty + (int)(t % NS)));
                return true;
            };
            for (int w = 0; ok; ++w) {
                const int ui = dec_unit_of(w, cta, grid);
                if (ui >= n_units) break;
                const DecItem it = dec_item<kGroup>(a, ui);
                const int n_kv = it.ke - it.kb;
                if (!(ok = dec_wait(bar(C::kQFull), item_i & 1, ctl))) break;
                if (kRope && !(ok = dec_wait(bar(C::kQRot), item_i & 1, ctl))) break;
                for (int j = 0; j < n_kv && ok; ++j) {
                    const uint32_t t = gt + (uint32_t)j;
                    const int buf = (int)(t & 1);
                    if (!(ok = dec_wait(bar(C::kKFull + (int)(t % NS)), (t / NS) & 1, ctl))) break;
                    if (t >= 2 && !(ok = dec_wait(bar(C::kSEmpty + buf), ((t - 2) >> 1) & 1, ctl))) break;
                    ptx::tc_fence_after();
                    issue_s(t);
                    ptx::mma_commit(bar(C::kSFull + buf));
                    if (j == n_kv - 1) ptx::mma_commit(bar(C::kQEmpty));  // Q^T is read by S^T only
                    if (j > 0 && !(ok = step_o(t - 1, j == 1))) break;
                }
                if (!ok) break;
                if (!(ok = step_o(gt + (uint32_t)n_kv - 1, n_kv == 1))) break;
                ptx::mma_commit(bar(C::kOFinal));
                gt += (uint32_t)n_kv;
                ++item_i;
            }
            if (!ok) {  // abort: wait for every MMA this thread issued
                ptx::mma_commit(bar(C::kDrain));
                dec_drain(bar(C::kDrain), 0);
            }
            const long long t0 = clock64();
            while (!ptx::mbar_try_wait_sleep(bar(C::kDone), 0, 200000u))
                if (clock64() - t0 > kDecWaitLimit) { atomicCAS(a.err, 0, RR_ERR_TIMEOUT); break; }
        }
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kDecTmemCols);
        return;
    }

    // ================================================================ softmax / epilogue (warps 0-3)
    // Pipeline waits are warp-uniform (__all_sync): after an abort a lane that saw its phase complete must not go
    // on to a warp-collective tcgen05 instruction or shuffle while a lane of the same warp has left the loop.
    {
        const int t_in = threadIdx.x;  // key of the tile, and output dimension in the epilogue
        const uint32_t lane_bits = (uint32_t)(warp * 32) << 16;
        const float sl2 = a.scale_log2;
        float* red = reinterpret_cast<float*>(smem + C::kOffRed);  // [x parity][warp][head]
        uint32_t gt = 0, item_i = 0, x_par = 0;
        bool ok = true;
        // the P^T address of key t_in (even lanes store a pair of keys), row h added per head
        const int kc = t_in >> 6, col = t_in & 63;
        const uint32_t p_key_off = (uint32_t)(kc * C::kNarrowChunkBytes + ((col & 7) << 1));
        const int p_unit = col >> 3;
        for (int w = 0; ok; ++w) {
            const int ui = dec_unit_of(w, cta, grid);
            if (ui >= n_units) break;
            const DecItem it = dec_item<kGroup>(a, ui);
            const int b = it.b, g = it.g, kb = it.kb, ke = it.ke, L = it.L;
            if constexpr (kRope) {  // rotate the item's Q^T rows once they have landed
                if (!(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kQFull), item_i & 1, ctl)))) break;
                dec_rope_q<D, G>(smem + C::kOffQ, threadIdx.x, a.rope, a.rope_max_pos, L - 1, a.err);
                ptx::fence_proxy_async_smem();  // generic-proxy writes -> the tensor core's reads
                ptx::mbar_arrive(bar(C::kQRot));
            }
            float m[G], lp[G];
#pragma unroll
            for (int h = 0; h < G; ++h) { m[h] = -INFINITY; lp[h] = 0.f; }
            for (int j = kb; j < ke; ++j, ++gt) {
                const int buf = (int)(gt & 1);
                if (!(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kSFull + buf), (gt >> 1) & 1, ctl)))) break;
                ptx::tc_fence_after();
                uint32_t sr[16];
                tmem_ld16(tmem + lane_bits + (uint32_t)(buf * kHeadCols), sr);
                tmem_wait_ld16(sr);
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(bar(C::kSEmpty + buf));
                const bool valid = j * kBN + t_in < L;
                float x[G];
#pragma unroll
                for (int h = 0; h < G; ++h) x[h] = valid ? __uint_as_float(sr[h]) : -INFINITY;
                // tile max per head: within the warp (the heads' shuffle trees interleave), then across the
                // four warps
                float* rx = red + x_par * 4 * kHeadCols;
                {
                    float v[G];
#pragma unroll
                    for (int h = 0; h < G; ++h) v[h] = x[h];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
                        for (int h = 0; h < G; ++h) v[h] = fmaxf(v[h], __shfl_xor_sync(0xffffffffu, v[h], o));
                    }
                    if (lane == 0) {
#pragma unroll
                        for (int h = 0; h < G; ++h) rx[warp * kHeadCols + h] = v[h];
                    }
                }
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(bar(C::kXch));
                if (!(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kXch), x_par, ctl)))) break;
                x_par ^= 1u;
                bool grow = false;
                float f[G], p[G];
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    f[h] = 1.f;
                    const float tm =
                        fmaxf(fmaxf(rx[h], rx[kHeadCols + h]), fmaxf(rx[2 * kHeadCols + h], rx[3 * kHeadCols + h])) * sl2;
                    if (j == kb) {
                        m[h] = tm;  // a piece always holds at least one key of the agent: finite
                    } else if (tm > m[h] + 8.0f) {
                        f[h] = ptx::ex2_approx(m[h] - tm);
                        lp[h] *= f[h];
                        m[h] = tm;
                        grow = true;
                    }
                }
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    // x = -inf: p = 0.  p is rounded to bf16 here, so the weight sum and the P^T operand of
                    // the O^T GEMM hold the same weights and the output is a convex combination of V.
                    p[h] = __bfloat162float(__float2bfloat16_rn(ptx::ex2_approx(fmaf(x[h], sl2, -m[h]))));
                    lp[h] += p[h];
                }
                // P^T(gt) goes to buffer buf once O^T(gt-2) has read it
                if (gt >= 2 && !(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kPEmpty + buf), ((gt - 2) >> 1) & 1, ctl)))) break;
                const uint32_t pb = sb + C::kOffP + (uint32_t)(buf * C::kPBytes) + p_key_off;
                {
                    float nb[G];
#pragma unroll
                    for (int h = 0; h < G; ++h) nb[h] = __shfl_xor_sync(0xffffffffu, p[h], 1);
                    if ((lane & 1) == 0) {
#pragma unroll
                        for (int h = 0; h < G; ++h) {
                            const uint32_t v = ptx::pack_bf16x2(p[h], nb[h]);
                            const uint32_t addr = pb + (uint32_t)(h * 128 + ((p_unit ^ (h & 7)) << 4));
                            asm volatile("st.shared.b32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
                        }
                    }
                }
                // O^T holds V^T P^T of tiles < j once O^T(gt-1) has completed; bring it to the new max
                // before O^T(gt) may start.  The max is the same in every thread, so is the branch.
                if (grow) {
                    if (!(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kPEmpty + (int)((gt - 1) & 1)), ((gt - 1) >> 1) & 1, ctl)))) break;
                    ptx::tc_fence_after();
                    uint32_t o[16];
                    tmem_ld16(tmem + lane_bits + 2u * kHeadCols, o);
                    tmem_wait_ld16(o);
#pragma unroll
                    for (int h = 0; h < G; ++h) o[h] = __float_as_uint(__uint_as_float(o[h]) * f[h]);
                    tmem_st16(tmem + lane_bits + 2u * kHeadCols, o);
                    ptx::tmem_wait_st();
                }
                ptx::fence_proxy_async_smem();  // P^T: generic-proxy writes -> the MMA's async proxy
                ptx::tc_fence_before();
                ptx::mbar_arrive(bar(C::kPFull + buf));
            }
            if (!ok) break;
            // weight sums: per warp, then across the warps
            float* rx = red + x_par * 4 * kHeadCols;
            {
                float v[G];
#pragma unroll
                for (int h = 0; h < G; ++h) v[h] = lp[h];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
                    for (int h = 0; h < G; ++h) v[h] += __shfl_xor_sync(0xffffffffu, v[h], o);
                }
                if (lane == 0) {
#pragma unroll
                    for (int h = 0; h < G; ++h) rx[warp * kHeadCols + h] = v[h];
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(bar(C::kXch));
            if (!(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kXch), x_par, ctl)))) break;
            x_par ^= 1u;
            if (!(ok = __all_sync(0xffffffffu, dec_wait(bar(C::kOFinal), item_i & 1, ctl)))) break;
            ptx::tc_fence_after();
            uint32_t o[16];
            tmem_ld16(tmem + lane_bits + 2u * kHeadCols, o);
            tmem_wait_ld16(o);
            ptx::tc_fence_before();
            ptx::mbar_arrive(bar(C::kOEmpty));
            const int slot = kGroup ? 0 : a.item_slot[ui];
            if (t_in < D) {
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    const float lsum = (rx[h] + rx[kHeadCols + h]) + (rx[2 * kHeadCols + h] + rx[3 * kHeadCols + h]);
                    if constexpr (kGroup) {
                        // column h: query head h % a.G of agent b + h / a.G; its piece sp of the shared prefix goes to
                        // slot sp of the agent's unit (the unit's private pieces follow)
                        const int ag = b + h / a.G;
                        if (h / a.G < a.group_agents && ag < a.batch) {
                            const int us = a.unit_slot[(long long)ag * (a.Hq / a.G) + g] + it.sp;
                            const long long prow = (long long)us * a.rows_per_slot + h % a.G;
                            a.part_o[prow * D + t_in] = __uint_as_float(o[h]);
                            if (t_in == 0) a.part_ml[prow] = make_float2(m[h], lsum);
                        }
                    } else if (slot >= 0) {
                        // split item: fp32 unnormalised O row h of the unit plus (max, sum)
                        const long long prow = (long long)slot * a.rows_per_slot + h;
                        a.part_o[prow * D + t_in] = __uint_as_float(o[h]);
                        if (t_in == 0) a.part_ml[prow] = make_float2(m[h], lsum);
                    } else {
                        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(a.out) +
                                             ((long long)a.cu[b] * a.Hq + g * G + h) * D + t_in;
                        *dst = __float2bfloat16_rn(__uint_as_float(o[h]) / lsum);
                    }
                }
            }
            ++item_i;
        }
    }
    ptx::tc_fence_before();
    ptx::mbar_arrive(bar(C::kDone));
}

template <int D, int NS, int G, bool kRope, bool kGroup = false>
cudaError_t launch_dec(const AttnArgs& a, int grid, cudaStream_t st) {
    using C = DecCfg<D, NS>;
    static bool attr_done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!attr_done[dev]) {
        e = cudaFuncSetAttribute(decode_attn_kernel<D, NS, G, kRope, kGroup>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 C::kSmemBytes);
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    return launch_after_sched(decode_attn_kernel<D, NS, G, kRope, kGroup>, dim3(grid), dim3(kDecThreads), C::kSmemBytes,
                              st, a);
}

template <int D, int NS, bool kRope>
cudaError_t launch_dec_g(const AttnArgs& a, int grid, cudaStream_t st) {
    switch (a.G) {
        case 1: return launch_dec<D, NS, 1, kRope>(a, grid, st);
        case 2: return launch_dec<D, NS, 2, kRope>(a, grid, st);
        case 4: return launch_dec<D, NS, 4, kRope>(a, grid, st);
        case 8: return launch_dec<D, NS, 8, kRope>(a, grid, st);
        case 16: return launch_dec<D, NS, 16, kRope>(a, grid, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_decode_attention(const AttnArgs& a, int head_dim, int grid, cudaStream_t st) {
    if (head_dim == 128) return a.rope ? launch_dec_g<128, 3, true>(a, grid, st) : launch_dec_g<128, 3, false>(a, grid, st);
    if (head_dim == 64) return a.rope ? launch_dec_g<64, 6, true>(a, grid, st) : launch_dec_g<64, 6, false>(a, grid, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_decode_shared_prefix(const AttnArgs& a, int head_dim, int grid, cudaStream_t st) {
    if (a.rope || a.group_agents * a.G != kHeadCols) return cudaErrorInvalidValue;
    if (head_dim == 128) return launch_dec<128, 3, kHeadCols, false, true>(a, grid, st);
    if (head_dim == 64) return launch_dec<64, 6, kHeadCols, false, true>(a, grid, st);
    return cudaErrorInvalidValue;
}

}  // namespace rr
