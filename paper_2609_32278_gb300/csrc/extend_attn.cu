// extend_attn.cu -- paged-KV extend attention for sm_103a (tcgen05 + TMEM + TMA).
//
// What it computes (Sec. 1, Sec. 2): every uncached suffix row of a returning
// agent attends causally to the agent's cached prefix and to the suffix up to
// itself; K/V come from the shared paged pool through the agent's page table.
//
//   out[cu_b+i, h, :] = softmax_j( scale * q[cu_b+i, h, :] . K_j ) V_j,  j = 0 .. P_b + i
//
// Design (one persistent CTA per SM, 12 warps; warp 11 only lends its registers, except in the
// fused extend step, where it writes the suffix K/V into the pool):
//   * work unit = (agent b, KV head g, kNQ = 2 consecutive Q tiles).  A Q tile
//     packs 128/G suffix tokens x the G query heads that share KV head g into
//     128 rows (GQA packing), so each K/V tile is loaded once for the whole
//     group and feeds M = 128 MMAs.  Units come from the on-device schedule,
//     most expensive first, dealt to CTAs in a snake order.
//   * warp 8, TMA producer: Q tiles (one 3-D box per 64-column chunk) and, per
//     128-key KV tile, one 2-D box per page and chunk -- the page gather.  Pages
//     past the agent's keys are requested at a row past the pool, which TMA
//     fills with zeros; slots of the agent's last page that lie past its last
//     position are cleared in shared memory before the MMA may read V.
//   * warp 9, MMA issuer (one thread): S_q = Q_q K^T  (SS, both operands
//     K-major, 128B swizzle) into TMEM, and O_q += P_q V (TS: P read from TMEM,
//     V from shared memory as an MN-major operand).  Issue order per KV tile j:
//     PV_0(j), S_0(j+1), PV_1(j), S_1(j+1): the tensor core works on one Q
//     tile while the softmax warpgroup of the other runs, and a tile's PV and
//     next S run back to back, which keeps that tile's softmax-to-softmax
//     chain short.  (Two issuers, one per tile, were measured slower: the
//     tensor core then interleaves both tiles' GEMMs and every chain doubles.)
//     P_1(j) is tested with a non-blocking mbarrier.test_wait issued in the
//     same asm block as the last two MMAs of S_0(j+1), so the test's latency
//     hides behind them; the blocking wait runs only if the phase was open.
//     A unit's Q buffers are released with its last S GEMM, so the next unit's
//     Q tiles load while the last PVs and softmax passes run.
//   * warp 10, stage watcher (one thread): waits until V(j) and K(j+1) have
//     landed and adds one arrival to P_0(j), so the MMA issuer's wait for
//     P_0(j) covers both.  A wait on an mbarrier, even one already complete,
//     costs the issuing thread ~250 cycles while the tensor core is busy, and
//     with an MMA queue about one instruction deep every such wait idles the
//     tensor core; the issuer is left with one wait per Q tile and KV tile.
//   * warps 0-3 / 4-7, softmax warpgroups for Q tile 0 / 1: thread r owns row
//     r (= TMEM lane r).  It loads its S row from TMEM, applies the causal mask
//     on the tiles that need it, keeps a running max in log2 units and rescales
//     O only when the max grew by more than 2^8 (the stale max keeps every
//     probability <= 256, far inside bf16/fp32 range), writes P as bf16 back
//     over its S columns, and at the end of the unit normalises O and stores it.
//   TMEM: S_0 cols 0-127, S_1 128-255, O_0 256.., O_1 256+D.. (512 allocated).
//   Shared memory (D=128): Q 2 x 32 KiB, K 2 and V 3 stages of 32 KiB (the
//   producer loads K(i), V(i) in order; a third V stage keeps it from stalling
//   on V's stage while K(i+1)'s is already free).
//
// Rotary embedding (kRope; rope.cuh): q arrives un-rotated; as a unit's Q tiles land, each softmax
// thread rotates its own row at position P_b + i in shared memory and arrives on QRot[q], which the
// MMA issuer waits for before the unit's first S_q.  The keys were rotated by the append.
//
// Ordering facts the pipeline relies on: tcgen05.mma operations issued by one
// thread execute in order, and tcgen05.commit arrives only after every earlier
// MMA of that thread finished; so when S_q(j) is complete, PV_q(j-1) is too,
// and the softmax may rescale O_q without another wait.
//
// Every wait is bounded (clock64 budget); a wait that runs out sets the
// device error word to RR_ERR_TIMEOUT and a shared abort flag, every role
// leaves its loop, in-flight copies and MMAs are drained, TMEM is freed and
// the kernel returns.  No trap, no unbounded spin.
#include <cuda_bf16.h>

#include "ptx.cuh"
#include "rope.cuh"
#include "rr_internal.h"

namespace rr {

namespace {

constexpr int kThreads = 384;  // warpgroups: softmax Q tile 0, softmax Q tile 1, producer + MMA + stage (+1 idle)
// Register split (launch: 384 threads x 168 = 64512; 3 warps per SMSP): the producer/MMA warpgroup
// drops to kRegsControl and each softmax warpgroup rises to kRegsSoftmax.
constexpr uint32_t kRegsSoftmax = 192;
constexpr uint32_t kRegsControl = 112;
static_assert(2 * 128 * kRegsSoftmax + 128 * kRegsControl <= kThreads * 168, "register split exceeds the launch");
static_assert((2 * kRegsSoftmax + kRegsControl) * 32 <= 16384, "register split exceeds one SMSP's file");
constexpr int kWarpProducer = 8;
constexpr int kWarpMMA = 9;
constexpr int kWarpStage = 10;
constexpr long long kWaitLimitCycles = 1ll << 33;  // ~4 s at 2 GHz

template <int D, int NK, int NV>
struct Cfg {
    static constexpr int kChunks = D / 64;                 // 128-byte (64 x bf16) column chunks
    static constexpr int kChunkBytes = kBM * 128;          // one chunk of a 128-row tile: 16 KiB
    static constexpr int kQTileBytes = kBM * D * 2;
    static constexpr int kKVTileBytes = kBN * D * 2;
    static constexpr int kOffQ = 0;
    static constexpr int kOffK = kOffQ + kNQ * kQTileBytes;
    static constexpr int kOffV = kOffK + NK * kKVTileBytes;
    static constexpr int kOffBar = kOffV + NV * kKVTileBytes;
    // barrier indices
    static constexpr int kQFull = 0, kQEmpty = 1;
    static constexpr int kKFull = 2, kKEmpty = 2 + NK, kVFull = 2 + 2 * NK, kVEmpty = 2 + 2 * NK + NV;
    static constexpr int kSFull = 2 + 2 * NK + 2 * NV, kPFull = kSFull + kNQ, kOFinal = kPFull + kNQ;
    static constexpr int kVTmp = kOFinal + kNQ, kDrain = kVTmp + 1, kDone = kDrain + 1;
    static constexpr int kQRot = kDone + 1;  // rotary q: Q tile q rotated in shared memory (kNQ barriers)
    static constexpr int kNumBars = kQRot + kNQ;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // u32 TMEM base, i32 abort flag
    static constexpr int kSmemBytes = kOffMisc + 16 + 1024;  // + slack to align the base to 1 KiB
    static_assert(kChunkBytes % 1024 == 0, "swizzle atoms must stay 1 KiB aligned");
    static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
    static_assert(kSmemBytes > 114 * 1024, "one CTA per SM: each CTA owns all 512 TMEM columns");
};

struct Ctl {
    volatile int32_t* abort_flag;
    int32_t* err;
};

// Bounded wait on an mbarrier phase.  False: timed out (flag raised) or another role aborted.
// Each try may suspend the thread (up to `hint` ns, 0.2 ms by default) until the phase completes,
// so waiting warps leave the issue slots to the warps that are computing.  The stage watcher passes
// the launch's budget (rr_set_wait_limit); the other roles keep the fixed one, which leaves their
// code as it is, and leave at their next unfinished wait once any wait has run out.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, const Ctl& c,
                                         long long limit = kWaitLimitCycles, uint32_t hint = 200000u) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (ptx::mbar_try_wait_sleep(bar, parity, hint)) return true;
        if (*c.abort_flag) return false;
        if (clock64() - t0 > limit) {
            *c.abort_flag = 1;
            atomicCAS(c.err, 0, RR_ERR_TIMEOUT);
            return false;
        }
    }
}

// Bounded wait used only while draining after an abort (ignores the abort flag).
__device__ __forceinline__ void drain_bar(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!ptx::mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > (1ll << 31)) break;
    }
}

// 2^x for a pair of floats on the FMA pipe, taking part of the exponential load off the MUFU unit.
// Range reduction: x is clamped to [-126, +inf) (the lazy-rescale bound keeps x <= 8) and rounded to
// the nearest integer n by adding 1.5 * 2^23 (the sum's low mantissa bits then hold n, a standard
// round-to-nearest technique); r = x - n lies in [-1/2, 1/2].  2^r is a cubic whose coefficients
// were fitted to 2^r on [-1/2, 1/2] by iteratively reweighted least squares on Chebyshev nodes
// (Lawson's algorithm towards the minimax relative error): max relative error 7.5e-5 (2^-13.7),
// far inside the bf16 rounding (2^-9) that P gets next.  The exponent n is added to the result's
// exponent field by integer addition of n << 23 (the bits of the rounded sum shifted left by 23).
constexpr float kExp2C0 = 0.99992807f, kExp2C1 = 0.69326099f, kExp2C2 = 0.24261112f, kExp2C3 = 0.05517166f;
constexpr float kRoundMagic = 12582912.0f;  // 1.5 * 2^23

__device__ __forceinline__ void exp2_poly2(float& p0, float& p1, float x0, float x1) {
    x0 = fmaxf(x0, -126.f);
    x1 = fmaxf(x1, -126.f);
    float y0, y1, t0, t1, r0, r1, q0, q1;
    ptx::add2(y0, y1, x0, x1, kRoundMagic, kRoundMagic);
    ptx::add2(t0, t1, y0, y1, -kRoundMagic, -kRoundMagic);
    ptx::fma2(r0, r1, t0, t1, -1.f, -1.f, x0, x1);  // r = x - round(x)
    ptx::fma2(q0, q1, r0, r1, kExp2C3, kExp2C3, kExp2C2, kExp2C2);
    ptx::fma2(q0, q1, q0, q1, r0, r1, kExp2C1, kExp2C1);
    ptx::fma2(q0, q1, q0, q1, r0, r1, kExp2C0, kExp2C0);
    p0 = __int_as_float(__float_as_int(q0) + (__float_as_int(y0) << 23));
    p1 = __int_as_float(__float_as_int(q1) + (__float_as_int(y1) << 23));
}

// Every kEmuPairStride-th pair of scores goes through exp2_poly2, the others through MUFU ex2
// (0: MUFU only, the default: on GB300 the softmax is bound by instruction issue, not by the MUFU
// unit -- measured 1314 TFLOP/s with no offload against 1260 / 1219 / 1204 for 1/8 / 1/4 / 1/3).

#ifndef RR_EMU_PAIR_STRIDE
#define RR_EMU_PAIR_STRIDE 0
#endif
constexpr int kEmuPairStride = RR_EMU_PAIR_STRIDE;


// The cascade over a prefix every agent shares (rr_extend_attention_shared) runs the kernel twice.
// kCasShared: every suffix row of the batch against the shared keys, in dense Q tiles of consecutive rows
// whatever their agent (no causal mask: every suffix position lies past the shared keys), each row's
// unnormalised O and (max, sum) written at (token, head).  kCasPrivate: the schedule's work units over each
// agent's keys from the shared ones on, the epilogue merging the shared pass's partial into the output.
constexpr int kCasNone = 0, kCasShared = 1, kCasPrivate = 2;

// Work unit ui of the shared pass: KV head ui % Hkv, the Q tiles of rows (ui / Hkv) * unit_tokens.. of the
// whole batch, agent 0's page table (the schedule checks that every agent's shared pages are agent 0's),
// KV tiles [0, cas_tiles).  P = S + P = the shared keys, so every row's last visible key is the last shared one.
__device__ __forceinline__ void cas_shared_unit(const AttnArgs& a, int ui, int& b, int& g, int& u, int& n_kv,
                                                int& kb, int& ke, int& P, int& S, int& cu_b) {
    const int hkv = a.Hq / a.G;
    b = 0;
    g = ui % hkv;
    u = ui / hkv;
    n_kv = a.cas_tiles;
    kb = 0;
    ke = a.cas_tiles;
    P = a.cas_tiles * kBN;
    S = 0;
    cu_b = 0;
}

// KV tiles of item ui (the private pass never splits a unit; its first cas_tiles tiles are the shared pass's).
template <int kCas>
__device__ __forceinline__ int item_tiles(const AttnArgs& a, int ui) {
    if constexpr (kCas == kCasShared) {
        return a.cas_tiles;
    } else {
        const int4 U = a.units[ui];
        if constexpr (kCas == kCasPrivate) return U.w - a.cas_tiles;
        const int sp = (U.y >> 8) & 0xFF, ns = (U.y >> 16) & 0xFF;
        return (sp + 1) * U.w / ns - sp * U.w / ns;
    }
}

// Snake order: even waves left to right, odd waves right to left.
__device__ __forceinline__ int unit_of(int wave, int cta, int grid) {
    return wave * grid + ((wave & 1) ? (grid - 1 - cta) : cta);
}

// Rotary embedding of one Q row in shared memory (rope.cuh): row r of a Q tile in the 128-byte swizzled
// layout TMA wrote (16-byte unit u of row r of a 64-column chunk sits at unit u ^ (r & 7)); cs = the
// (cos, sin) table row of the row's position.  The table and shared-memory loads of four pair units are
// issued before any of their stores, so a row costs two table round trips, not eight.
// Not inlined: compiled into the softmax warps' function, this once-per-unit code changed the code of
// their per-tile loop, and the kernel ran 1.7 % slower with the rotation present but never executed; as
// a call, the rotating kernel runs at 1.024x the plain one's time on c2 instead of 1.033x.  The rest is
// the unit boundary: S_q of a unit waits until its Q tile has landed and been rotated.
template <int D>
__device__ __noinline__ void rope_q_row(uint8_t* tile, int r, const float2* __restrict__ cs) {
    auto at = [&](int d) -> uint4* {
        return reinterpret_cast<uint4*>(tile + (d >> 6) * (kBM * 128) + r * 128 + ((((d & 63) >> 3) ^ (r & 7)) << 4));
    };
    constexpr int kUnits = D / 16, kGroup = kUnits < 4 ? kUnits : 4;
#pragma unroll
    for (int u0 = 0; u0 < kUnits; u0 += kGroup) {
        float4 t[kGroup][4];
        uint4 x0[kGroup], x1[kGroup];
#pragma unroll
        for (int k = 0; k < kGroup; ++k) {
            rope_load8(t[k], cs + 8 * (u0 + k));
            x0[k] = *at(8 * (u0 + k));
            x1[k] = *at(8 * (u0 + k) + D / 2);
        }
#pragma unroll
        for (int k = 0; k < kGroup; ++k) {
            rope_rotate8(x0[k], x1[k], t[k]);
            *at(8 * (u0 + k)) = x0[k];
            *at(8 * (u0 + k) + D / 2) = x1[k];
        }
    }
}

// Phase 1 of the one-launch extend step: every suffix row of every KV head goes to its pool slot, K
// rotated at the row's position P_b + i when a rotary table is given, the same bytes rr_kv_append /
// rr_kv_append_rope write; then the grid waits until all of it is written, so that phase 2, the plain
// attention pipeline over the pool, finds each suffix key where a separate append would have put it.
// The work is handed out in tasks of 8 tokens of one unit's KV head over every warp of the grid (only
// units with split index 0: each (token, KV head) belongs to exactly one), with all of a lane's loads
// in flight before its stores.  Streaming (evict-first) loads and stores: this launch reads no k_new /
// v_new line again, and default-policy pool stores would push prefix K/V out of L2.
// The barrier needs every CTA resident at once (a cooperative launch, one CTA per SM); its spin is
// bounded by a.wait_limit, after which it reports RR_ERR_TIMEOUT and returns 0: the CTA then runs no
// unit of phase 2 (it still sets up and tears down its pipeline, so that every role ends as usual).
// Code generation note: the pipeline after this phase is sensitive to how the kernel gets past it.
// Leaving the kernel here on a failed barrier (before the mbarrier initialisation and the tensor-memory
// allocation), or ignoring the outcome, each made the whole step 7-8 % slower on the c2, c4 and c5
// batches than this form, in which the outcome only zeroes the unit count.
template <int D, bool kRope>
__device__ __forceinline__ int fused_append(const AttnArgs& a, int n_units, int unit_tokens) {
    constexpr int kPerTok = D / 8;  // 16-byte vectors of one head's row
    constexpr int kTask = 8;        // tokens per warp task (unit_tokens = 256 / G is a multiple of 16)
    const int lane = threadIdx.x & 31;
    const long long n_warps = (long long)gridDim.x * (kThreads / 32);
    const int tasks_per_unit = unit_tokens / kTask;
    const int ps_shift = __ffs(a.ps) - 1;  // page sizes are powers of two
    for (long long c = (long long)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); c < (long long)n_units * tasks_per_unit;
         c += n_warps) {
        const int ui = (int)(c / tasks_per_unit);
        const int4 U = a.units[ui];
        if (((U.y >> 8) & 0xFF) != 0) continue;  // a later piece of a split unit
        const int b = U.x, g = U.y & 0xFF;
        const int P = a.prefix[b], S = a.suffix[b];
        const int t0 = U.z * unit_tokens + (int)(c - (long long)ui * tasks_per_unit) * kTask;
        const int n = min(kTask, S - t0);
        if (n <= 0) continue;
        const int32_t* pt = a.page_table + (long long)b * a.max_pages;
        const long long src0 = (long long)(a.cu[b] + t0) * a.row16 + g * kPerTok;
        // the pool row of token t of the task (-1: not written, the error reported)
        auto dst_row = [&](int t) -> long long {
            if (t >= n) return -1;
            const int pos = P + t0 + t;
            if (kRope && pos >= a.rope_max_pos) {
                atomicCAS(a.err, 0, RR_ERR_LENS);
                return -1;
            }
            const int pid = pt[pos >> ps_shift];
            if (pid < 0 || (long long)pid >= a.num_pages) {
                atomicCAS(a.err, 0, RR_ERR_OOB);
                return -1;
            }
            return (((long long)pid << ps_shift) + (pos & (a.ps - 1))) * a.row16 + g * kPerTok;
        };
        {  // V, and K without a rotary table: one vector per lane and pass
            constexpr int kTokPerPass = 32 / kPerTok, kPasses = kTask / kTokPerPass;
            const int sub = lane / kPerTok, v = lane % kPerTok;
            long long dst[kPasses];
            uint4 kx[kPasses], vx[kPasses];
#pragma unroll
            for (int p = 0; p < kPasses; ++p) {
                const int t = p * kTokPerPass + sub;
                dst[p] = dst_row(t);
                if (dst[p] >= 0) {
                    const long long src = src0 + (long long)t * a.row16 + v;
                    if (!kRope) kx[p] = __ldcs(a.knew + src);
                    vx[p] = __ldcs(a.vnew + src);
                }
            }
#pragma unroll
            for (int p = 0; p < kPasses; ++p) {
                if (dst[p] < 0) continue;
                if (!kRope) __stcs(a.kpool + dst[p] + v, kx[p]);
                __stcs(a.vpool + dst[p] + v, vx[p]);
            }
        }
        if constexpr (kRope) {  // K: the two vectors of one rotation pair (elements 8u.. and 8u + D/2..) per lane
            constexpr int kHalf = kPerTok / 2, kTokPerPass = 32 / kHalf, kPasses = kTask / kTokPerPass;
            const int sub = lane / kHalf, u = lane % kHalf;
#pragma unroll
            for (int p = 0; p < kPasses; ++p) {
                const int t = p * kTokPerPass + sub;
                const long long dst = dst_row(t);
                if (dst < 0) continue;
                const long long src = src0 + (long long)t * a.row16;
                uint4 k0 = __ldcs(a.knew + src + u), k1 = __ldcs(a.knew + src + u + kHalf);
                float4 cs[4];
                rope_load8(cs, a.rope + (long long)(P + t0 + t) * (D / 2) + 8 * u);
                rope_rotate8(k0, k1, cs);
                __stcs(a.kpool + dst + u, k0);
                __stcs(a.kpool + dst + u + kHalf, k1);
            }
        }
    }
    // grid barrier: every CTA's pool stores, then its arrival; the attention reads the rows through TMA
    asm volatile("fence.proxy.async.global;" ::: "memory");
    __syncthreads();
    int ok = 1;
    if (threadIdx.x == 0) {
        __threadfence();
        atomicAdd(a.grid_sync, 1);
        const long long t_start = clock64();
        for (;;) {
            int arrived;
            asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(arrived) : "l"(a.grid_sync) : "memory");
            if (arrived >= (int)gridDim.x) break;
            if (clock64() - t_start > a.wait_limit) {
                atomicCAS(a.err, 0, RR_ERR_TIMEOUT);
                ok = 0;
                break;
            }
            __nanosleep(100);
        }
    }
    ok = __syncthreads_and(ok);
    asm volatile("fence.proxy.async.global;" ::: "memory");
    return ok;
}

// kFused: the one-launch extend step, fused_append above and then the attention over the pool; the
// result is bit-identical to rr_kv_append followed by rr_extend_attention (with kRope, to the _rope pair).
// kRope: q arrives un-rotated; as a unit's Q tiles land, each softmax thread rotates its own row at its
// position P_b + i in shared memory, and the MMA issuer starts S_q only once tile q is rotated (the
// keys were rotated on their way into the pool).
template <int D, int NK, int NV, bool kFused, bool kRope, int kCas = kCasNone>
__global__ void __launch_bounds__(kThreads, 1) extend_attn_kernel(const __grid_constant__ AttnArgs a) {
    using C = Cfg<D, NK, NV>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sb = ptx::smem_u32(smem);
    auto bar = [&](int i) -> uint32_t { return sb + C::kOffBar + 8u * (uint32_t)i; };
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(smem + C::kOffMisc + 4);
    const Ctl ctl{abort_flag, a.err};

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    bool phase2 = true;
    if constexpr (kFused) phase2 = fused_append<D, kRope>(a, *a.n_units, kNQ * a.tq);  // after the schedule kernel

    if (threadIdx.x == 0) {
        ptx::mbar_init(bar(C::kQFull), 1);
        ptx::mbar_init(bar(C::kQEmpty), 1);
        for (int s = 0; s < NK; ++s) {
            ptx::mbar_init(bar(C::kKFull + s), 1);
            ptx::mbar_init(bar(C::kKEmpty + s), 1);
        }
        for (int s = 0; s < NV; ++s) {
            ptx::mbar_init(bar(C::kVFull + s), 1);
            ptx::mbar_init(bar(C::kVEmpty + s), 1);
        }
        for (int q = 0; q < kNQ; ++q) {
            ptx::mbar_init(bar(C::kSFull + q), 1);
            ptx::mbar_init(bar(C::kPFull + q), q == 0 ? kBM + 1 : kBM);  // + the stage warp on P_0
            ptx::mbar_init(bar(C::kOFinal + q), 1);
        }
        ptx::mbar_init(bar(C::kVTmp), 1);
        for (int q = 0; q < kNQ; ++q) ptx::mbar_init(bar(C::kQRot + q), kBM);
        ptx::mbar_init(bar(C::kDrain), 1);
        ptx::mbar_init(bar(C::kDone), 2 * kBM);  // every softmax thread, once, at its end
        *abort_flag = 0;
        ptx::fence_mbar_init();
    }
    if (warp == kWarpMMA) {
        ptx::tmem_alloc(sb + C::kOffMisc, 512);
        ptx::tmem_relinquish();
    }
    if (warp == kWarpProducer && lane == 0) {
        ptx::prefetch_tmap(&a.tm_q);
        ptx::prefetch_tmap(&a.tm_k);
        ptx::prefetch_tmap(&a.tm_v);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + C::kOffMisc);
    ptx::griddep_wait();  // the schedule kernel's output (launched as its dependent)
    const int n_units = !phase2 ? 0 : kCas == kCasShared ? a.cas_units : *a.n_units;
    const int grid = gridDim.x, cta = blockIdx.x;
    const int unit_tokens = kNQ * a.tq;

    if (warp >= 8) {
    // ================================================================ control warpgroup (warps 8-11)
    ptx::setmaxnreg_dec<kRegsControl>();  // whole warpgroup, unconditionally: the softmax warpgroups wait for it
    if (warp == kWarpProducer) {
        // ------------------------------------------------------------ TMA producer
        const int ppt = kBN / a.ps;  // pages per KV tile (<= 16)
        uint32_t kv_count = 0, unit_i = 0, vtmp_phase = 0;
        // copies in flight, for the abort drain: bit s of armed_* = stage s armed, bit s of par_* = its parity
        int armed_q = -1, armed_vtmp = -1;
        uint32_t armed_k = 0, armed_v = 0, par_k = 0, par_v = 0;
        bool ok = true;
        for (int w = 0; ok; ++w) {
            const int ui = unit_of(w, cta, grid);
            if (ui >= n_units) break;
            // agent, KV head, unit, the unit's KV tiles, this item's [kb, ke), lengths, first row
            int b, g, u, n_kv, kb, ke, P, S, cu_b;
            if constexpr (kCas == kCasShared) {
                cas_shared_unit(a, ui, b, g, u, n_kv, kb, ke, P, S, cu_b);
            } else {
                const int4 U = a.units[ui];
                const int sp = (U.y >> 8) & 0xFF, ns = (U.y >> 16) & 0xFF;
                b = U.x, g = U.y & 0xFF, u = U.z;
                n_kv = U.w, kb = sp * n_kv / ns, ke = (sp + 1) * n_kv / ns;
                if constexpr (kCas == kCasPrivate) kb = a.cas_tiles;  // the shared keys are the shared pass's
                P = a.prefix[b], S = a.suffix[b], cu_b = a.cu[b];
            }
            const int t0 = u * unit_tokens;
            const int n_keys = P + min(S, t0 + unit_tokens);
            const int agent_len = P + S;
            // Q tiles of this unit, once the previous unit's last S GEMM has read its own (QEmpty)
            if (lane == 0) {
                if (unit_i > 0) ok = wait_bar(bar(C::kQEmpty), (unit_i - 1) & 1, ctl);
                if (ok) {
                    ptx::mbar_arrive_expect_tx(bar(C::kQFull), kNQ * C::kQTileBytes);
                    for (int q = 0; q < kNQ; ++q)
                        for (int c = 0; c < C::kChunks; ++c)
                            ptx::tma_load_3d(sb + C::kOffQ + q * C::kQTileBytes + c * C::kChunkBytes, &a.tm_q,
                                             c * 64, g * a.G, cu_b + t0 + q * a.tq, bar(C::kQFull));
                    armed_q = (int)(unit_i & 1);
                }
            }
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            const int last_page_end = ((n_keys + a.ps - 1) / a.ps) * a.ps;
            for (int j = kb; j < ke; ++j, ++kv_count) {
                const int sk = (int)(kv_count % NK), sv = (int)(kv_count % NV);
                const uint32_t usek = kv_count / NK, usev = kv_count / NV;
                // the page of this lane: from the pool, or past the agent's keys (a row past the pool: zero fill)
                int row = a.oob_row;
                if (lane < ppt) {
                    const int lp = j * ppt + lane;
                    if (lp * a.ps < n_keys) {
                        const int pid = a.page_table[(long long)b * a.max_pages + lp];
                        if (pid >= 0 && (long long)pid < a.num_pages) row = pid * a.ps;
                        else atomicCAS(a.err, 0, RR_ERR_OOB);
                    }
                }
                // K tile
                const uint32_t kbar = bar(C::kKFull + sk);
                if (lane == 0) {
                    if (usek > 0) ok = wait_bar(bar(C::kKEmpty + sk), (usek - 1) & 1, ctl);
                    if (ok) ptx::mbar_arrive_expect_tx(kbar, C::kKVTileBytes);
                }
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                armed_k |= 1u << sk;
                par_k = (par_k & ~(1u << sk)) | ((usek & 1u) << sk);
                if (lane < ppt)
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_2d(sb + C::kOffK + sk * C::kKVTileBytes + c * C::kChunkBytes + lane * a.ps * 128,
                                         &a.tm_k, g * D + c * 64, row, kbar);
                // V tile; if the agent's last page is only partly its own, land it on the side barrier, clear
                // the foreign slots, then release it to the MMA warp
                const bool clear_tail = (j == n_kv - 1) && (last_page_end > agent_len);
                const uint32_t vbar = clear_tail ? bar(C::kVTmp) : bar(C::kVFull + sv);
                if (lane == 0) {
                    if (usev > 0) ok = wait_bar(bar(C::kVEmpty + sv), (usev - 1) & 1, ctl);
                    if (ok) ptx::mbar_arrive_expect_tx(vbar, C::kKVTileBytes);
                }
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                if (lane < ppt)
                    for (int c = 0; c < C::kChunks; ++c)
                        ptx::tma_load_2d(sb + C::kOffV + sv * C::kKVTileBytes + c * C::kChunkBytes + lane * a.ps * 128,
                                         &a.tm_v, g * D + c * 64, row, vbar);
                if (clear_tail) {
                    armed_vtmp = (int)vtmp_phase;
                    if (lane == 0) ok = wait_bar(bar(C::kVTmp), vtmp_phase, ctl);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) break;
                    armed_vtmp = -1;
                    vtmp_phase ^= 1;
                    const int r0 = agent_len - j * kBN;  // 0 < r0 < kBN: first row past the agent
                    uint8_t* vt = smem + C::kOffV + sv * C::kKVTileBytes;
                    for (int c = 0; c < C::kChunks; ++c) {
                        uint4* base = reinterpret_cast<uint4*>(vt + c * C::kChunkBytes);
                        for (int e = r0 * 8 + lane; e < kBN * 8; e += 32) base[e] = make_uint4(0u, 0u, 0u, 0u);
                    }
                    ptx::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(bar(C::kVFull + sv));
                } else {
                    armed_v |= 1u << sv;
                    par_v = (par_v & ~(1u << sv)) | ((usev & 1u) << sv);
                }
            }
            ++unit_i;
        }
        if (!ok && lane == 0) {  // abort: let every copy this warp started land before exit
            if (armed_q >= 0) drain_bar(bar(C::kQFull), (uint32_t)armed_q);
            if (armed_vtmp >= 0) drain_bar(bar(C::kVTmp), (uint32_t)armed_vtmp);
            for (int s = 0; s < NK; ++s)
                if (armed_k >> s & 1u) drain_bar(bar(C::kKFull + s), par_k >> s & 1u);
            for (int s = 0; s < NV; ++s)
                if (armed_v >> s & 1u) drain_bar(bar(C::kVFull + s), par_v >> s & 1u);
        }
        __syncwarp();
    } else if (warp == kWarpStage) {
        // ------------------------------------------------------------ stage watcher
        if (lane == 0) {
            uint32_t kv_count = 0, p_phase = 0;
            const long long lim = a.wait_limit;
            const uint32_t hint = a.wait_hint_ns;
            bool ok = true;
            for (int w = 0; ok; ++w) {
                const int ui = unit_of(w, cta, grid);
                if (ui >= n_units) break;
                const int n_kv = item_tiles<kCas>(a, ui);
                for (int j = 0; j < n_kv; ++j, ++kv_count) {
                    const uint32_t nxt = kv_count + 1;
                    if (!(ok = wait_bar(bar(C::kVFull + (int)(kv_count % NV)), (kv_count / NV) & 1, ctl, lim, hint)))
                        break;
                    if (j + 1 < n_kv &&
                        !(ok = wait_bar(bar(C::kKFull + (int)(nxt % NK)), (nxt / NK) & 1, ctl, lim, hint)))
                        break;
                    ptx::mbar_arrive(bar(C::kPFull + 0));
                    // one arrival per phase: the next one only once this phase has completed
                    if (!(ok = wait_bar(bar(C::kPFull + 0), p_phase, ctl, lim, hint))) break;
                    p_phase ^= 1u;
                }
            }
        }
        __syncwarp();
    } else if (warp == kWarpMMA) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_qk = ptx::idesc_bf16_f32(kBM, kBN, false, false);
            constexpr uint32_t idesc_pv = ptx::idesc_bf16_f32(kBM, D, false, true);
            uint32_t kv_count = 0, unit_i = 0;
            uint32_t p_phase = 0;  // bit q: parity of the next P_q phase
            bool ok = true;
            // Shared-memory descriptors are built once; a K-step inside a 128-byte swizzle atom, a chunk or
            // a stage only moves the start address, i.e. adds (bytes >> 4) to the descriptor's low field
            // (no carry: shared addresses are below 256 KiB).
            const uint64_t desc_q0 = ptx::sdesc_sw128(sb + C::kOffQ, 16, 1024);
            const uint64_t desc_k0 = ptx::sdesc_sw128(sb + C::kOffK, 16, 1024);
            const uint64_t desc_v0 = ptx::sdesc_sw128(sb + C::kOffV, C::kChunkBytes, 1024);
            auto issue_qk = [&](int q, int s) {
                const uint32_t d_tmem = tmem + (uint32_t)(q * 128);
                const uint64_t da = desc_q0 + (uint64_t)((q * C::kQTileBytes) >> 4);
                const uint64_t db = desc_k0 + (uint64_t)((s * C::kKVTileBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint64_t off = (uint64_t)((((kk >> 2) * C::kChunkBytes) + (kk & 3) * 32) >> 4);
                    ptx::mma_ss(d_tmem, da + off, db + off, idesc_qk, kk > 0 ? 1u : 0u);
                }
            };
            // the same, with a non-blocking test of (bar, parity) issued ahead of the last two MMAs
            auto issue_qk_test = [&](int q, int s, uint32_t tbar, uint32_t parity) -> bool {
                const uint32_t d_tmem = tmem + (uint32_t)(q * 128);
                const uint64_t da = desc_q0 + (uint64_t)((q * C::kQTileBytes) >> 4);
                const uint64_t db = desc_k0 + (uint64_t)((s * C::kKVTileBytes) >> 4);
                constexpr int kSteps = D / 16;
#pragma unroll
                for (int kk = 0; kk < kSteps - 2; ++kk) {
                    const uint64_t off = (uint64_t)((((kk >> 2) * C::kChunkBytes) + (kk & 3) * 32) >> 4);
                    ptx::mma_ss(d_tmem, da + off, db + off, idesc_qk, kk > 0 ? 1u : 0u);
                }
                constexpr int k0 = kSteps - 2, k1 = kSteps - 1;
                const uint64_t off0 = (uint64_t)((((k0 >> 2) * C::kChunkBytes) + (k0 & 3) * 32) >> 4);
                const uint64_t off1 = (uint64_t)((((k1 >> 2) * C::kChunkBytes) + (k1 & 3) * 32) >> 4);
                return ptx::mma_ss2_test(d_tmem, da + off0, db + off0, da + off1, db + off1, idesc_qk, 1u, tbar,
                                         parity) != 0;
            };
            auto issue_pv = [&](int q, int s, bool accumulate) {
                const uint32_t d_tmem = tmem + 256u + (uint32_t)(q * D);
                const uint64_t db = desc_v0 + (uint64_t)((s * C::kKVTileBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk) {
                    const uint32_t a_tmem = tmem + (uint32_t)(q * 128 + kk * 8);  // P: bf16 pairs over S_q
                    ptx::mma_ts(d_tmem, a_tmem, db + (uint64_t)((kk * 16 * 128) >> 4), idesc_pv,
                                (accumulate || kk > 0) ? 1u : 0u);
                }
            };
            for (int w = 0; ok; ++w) {
                const int ui = unit_of(w, cta, grid);
                if (ui >= n_units) break;
                const int n_kv = item_tiles<kCas>(a, ui);  // KV tiles of this item
                if (!(ok = wait_bar(bar(C::kQFull), unit_i & 1, ctl))) break;
                {
                    const int sk = (int)(kv_count % NK);
                    if (!(ok = wait_bar(bar(C::kKFull + sk), (kv_count / NK) & 1, ctl))) break;
                    if (kRope && !(ok = wait_bar(bar(C::kQRot + 0), unit_i & 1, ctl))) break;
                    ptx::tc_fence_after();
                    issue_qk(0, sk);
                    ptx::mma_commit(bar(C::kSFull + 0));
                    if constexpr (kRope) {
                        if (!(ok = wait_bar(bar(C::kQRot + 1), unit_i & 1, ctl))) break;
                        ptx::tc_fence_after();
                    }
                    issue_qk(1, sk);
                    ptx::mma_commit(bar(C::kSFull + 1));
                    ptx::mma_commit(bar(C::kKEmpty + sk));
                    if (n_kv == 1) ptx::mma_commit(bar(C::kQEmpty));  // Q is read by the S GEMMs only
                }
                // P_q waits: a test for the next P rides on the last MMAs of the S GEMM before it; the
                // blocking wait runs only when that test found the phase still open.
                bool p_ready[kNQ] = {false, false};
                for (int j = 0; j < n_kv && ok; ++j) {
                    const uint32_t cur = kv_count + j, nxt = cur + 1;
                    const int sv = (int)(cur % NV), sk1 = (int)(nxt % NK);
                    const bool more = j + 1 < n_kv;
                    // PV_0(j), S_0(j+1), PV_1(j), S_1(j+1).  V(j) and K(j+1) are not waited for here: P_0(j)
                    // completes only after the stage warp has seen both land.
#pragma unroll
                    for (int q = 0; q < kNQ; ++q) {
                        if (!p_ready[q] && !(ok = wait_bar(bar(C::kPFull + q), (p_phase >> q) & 1u, ctl))) break;
                        p_ready[q] = false;  // consumed
                        p_phase ^= 1u << q;
                        ptx::tc_fence_after();
                        issue_pv(q, sv, j > 0);
                        if (q == kNQ - 1) ptx::mma_commit(bar(C::kVEmpty + sv));  // V(j) read by both PVs
                        if (!more) {
                            ptx::mma_commit(bar(C::kOFinal + q));
                            continue;
                        }
                        // test the P the next PV needs: P_1(j) after S_0(j+1), P_0(j+1) after S_1(j+1)
                        const int qn = (q + 1) % kNQ;
                        p_ready[qn] = issue_qk_test(q, sk1, bar(C::kPFull + qn), (p_phase >> qn) & 1u);
                        ptx::mma_commit(bar(C::kSFull + q));
                        if (q == kNQ - 1) {
                            ptx::mma_commit(bar(C::kKEmpty + sk1));
                            // the unit's last S GEMM: the next unit's Q may land while the last PVs run
                            if (j + 2 == n_kv) ptx::mma_commit(bar(C::kQEmpty));
                        }
                    }
                    if (!ok) break;
                }
                if (!ok) break;
                kv_count += n_kv;
                ++unit_i;
            }
            if (!ok) {  // abort: wait for every MMA this thread issued
                ptx::mma_commit(bar(C::kDrain));
                drain_bar(bar(C::kDrain), 0);
            }
            // TMEM is freed once every softmax thread has finished its last TMEM access (bounded like every
            // other wait; the columns must be released in any case, or the next kernel on this SM could not
            // allocate them)
            {
                const long long t0 = clock64();
                while (!ptx::mbar_try_wait_sleep(bar(C::kDone), 0, 200000u))
                    if (clock64() - t0 > kWaitLimitCycles) { atomicCAS(a.err, 0, RR_ERR_TIMEOUT); break; }
            }
        }
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 512);
    }
    return;
    }
    // ================================================================ softmax warpgroups (warps 0-7)
    // Their pipeline waits are warp-uniform (__all_sync): after an abort a lane that saw its phase complete must
    // not go on to a warp-collective tcgen05 instruction while a lane of the same warp has left the loop.
    ptx::setmaxnreg_inc<kRegsSoftmax>();
    {
        const int q = warp >> 2;                // Q tile of this warpgroup
        const int r = threadIdx.x & (kBM - 1);  // row == TMEM lane
        const uint32_t lane_bits = (uint32_t)((warp & 3) * 32) << 16;
        const uint32_t t_s = tmem + lane_bits + (uint32_t)(q * 128);
        const uint32_t t_o = tmem + lane_bits + 256u + (uint32_t)(q * D);
        const float sl2 = a.scale_log2;
        uint32_t s_phase = 0, o_phase = 0, q_phase = 0;
        bool ok = true;
        for (int w = 0; ok; ++w) {
            const int ui = unit_of(w, cta, grid);
            if (ui >= n_units) break;
            int b, g, u, kb, ke, P, agent_len;  // agent, KV head, unit, this item's KV tiles, keys
            if constexpr (kCas == kCasShared) {
                int n_kv, S, cu_b;
                cas_shared_unit(a, ui, b, g, u, n_kv, kb, ke, P, S, cu_b);
                agent_len = P;  // every row sees exactly the shared keys: P - 1 is each row's last key
            } else {
                const int4 U = a.units[ui];
                const int sp = (U.y >> 8) & 0xFF, ns = (U.y >> 16) & 0xFF;
                b = U.x, g = U.y & 0xFF, u = U.z;
                kb = sp * U.w / ns, ke = (sp + 1) * U.w / ns;
                if constexpr (kCas == kCasPrivate) kb = a.cas_tiles;
                P = a.prefix[b], agent_len = P + a.suffix[b];
            }
            const int tq0 = u * unit_tokens + q * a.tq;  // first suffix token of this Q tile
            const int row_limit = min(P + tq0 + r / a.G, agent_len - 1);     // last key this row may see
            const int mask_from = (min(P + tq0, agent_len - 1) + 1) / kBN;  // earlier tiles: no masking
            if constexpr (kRope) {  // rotate this thread's row of Q tile q once the tile has landed
                if (!(ok = __all_sync(0xffffffffu, wait_bar(bar(C::kQFull), q_phase, ctl)))) break;
                q_phase ^= 1u;
                const int tok = tq0 + r / a.G;
                if (tok < a.suffix[b]) {  // rows past the agent's suffix are never stored
                    const int pos = P + tok;
                    if (pos < a.rope_max_pos)
                        rope_q_row<D>(smem + C::kOffQ + q * C::kQTileBytes, r, a.rope + (long long)pos * (D / 2));
                    else
                        atomicCAS(a.err, 0, RR_ERR_LENS);
                }
                ptx::fence_proxy_async_smem();  // generic-proxy writes -> the tensor core's reads
                ptx::mbar_arrive(bar(C::kQRot + q));
            }
            float m_run = -INFINITY, l_run = 0.f;
            for (int j = kb; j < ke; ++j) {
                if (!(ok = __all_sync(0xffffffffu, wait_bar(bar(C::kSFull + q), s_phase, ctl)))) break;
                s_phase ^= 1;
                ptx::tc_fence_after();
                // S row in two halves: the second half's TMEM load overlaps the first half's max.
                uint32_t sr[kBN];
                auto chunk = [&](int c) -> uint32_t(&)[32] { return *reinterpret_cast<uint32_t(*)[32]>(&sr[c]); };
                ptx::tmem_ld32(t_s + 0, chunk(0));
                ptx::tmem_ld32(t_s + 32, chunk(32));
                ptx::tmem_wait_ld_regs(chunk(0));
                ptx::tmem_wait_ld_regs(chunk(32));
                ptx::tmem_ld32(t_s + 64, chunk(64));
                ptx::tmem_ld32(t_s + 96, chunk(96));
                float sv[kBN];
                const bool masked = j >= mask_from;
                const int lim = row_limit - j * kBN;  // columns past lim are invisible to this row
                float mx[8];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (h == 1) {
                        ptx::tmem_wait_ld_regs(chunk(64));
                        ptx::tmem_wait_ld_regs(chunk(96));
                    }
#pragma unroll
                    for (int c = h * 64; c < h * 64 + 64; ++c) sv[c] = __uint_as_float(sr[c]);
                    if (masked) {  // only the last tile or two of a unit
#pragma unroll
                        for (int c = h * 64; c < h * 64 + 64; ++c)
                            if (c > lim) sv[c] = -INFINITY;
                    }
                    // eight independent chains of 3-input max over this half
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        const int c = h * 64 + k * 8;
                        float m = ptx::max3(sv[c], sv[c + 1], sv[c + 2]);
                        m = ptx::max3(m, sv[c + 3], sv[c + 4]);
                        m = ptx::max3(m, sv[c + 5], sv[c + 6]);
                        m = h == 0 ? fmaxf(m, sv[c + 7]) : ptx::max3(m, sv[c + 7], mx[k]);
                        mx[k] = m;
                    }
                }
                const float mxs = ptx::max3(ptx::max3(mx[0], mx[1], mx[2]), ptx::max3(mx[3], mx[4], mx[5]),
                                            fmaxf(mx[6], mx[7])) * sl2;
                bool grow = false;
                float f = 1.0f;
                if (j == kb) {
                    m_run = mxs;  // -inf only for a row that sees no key of a later split's first tile
                } else if (mxs > m_run + 8.0f) {
                    grow = true;
                    f = ptx::ex2_approx(m_run - mxs);
                    l_run *= f;
                    m_run = mxs;
                }
                const float neg = m_run == -INFINITY ? 0.f : -m_run;  // a fully masked row keeps p = 0
                // p = 2^(s * scale * log2e - m): packed FMA, ex2, bf16 pairs; the first half of P goes to TMEM
                // while the second is computed
                uint32_t pk[kBN / 2];
#pragma unroll
                for (int c = 0; c < kBN; c += 2) {
                    float x0, x1, p0, p1;
                    ptx::fma2(x0, x1, sv[c], sv[c + 1], sl2, sl2, neg, neg);
                    if (kEmuPairStride > 0 && (c >> 1) % (kEmuPairStride > 0 ? kEmuPairStride : 1) ==
                                                  (kEmuPairStride > 0 ? kEmuPairStride - 1 : 0)) {
                        exp2_poly2(p0, p1, x0, x1);
                    } else {
                        p0 = ptx::ex2_approx(x0);
                        p1 = ptx::ex2_approx(x1);
                    }
                    pk[c >> 1] = ptx::pack_bf16x2(p0, p1);
                    if (c == kBN / 2 - 2) ptx::tmem_st32(t_s, *reinterpret_cast<uint32_t(*)[32]>(&pk[0]));
                }
                ptx::tmem_st32(t_s + 32, *reinterpret_cast<uint32_t(*)[32]>(&pk[32]));
                // O_q holds PV of tiles < j (complete: S_q(j) was issued after PV_q(j-1)); bring it to the
                // new max before PV_q(j) may start, i.e. before this thread signals P_q(j).
                if (__any_sync(0xffffffffu, grow)) {  // warp-uniform: tcgen05.ld/st are .sync.aligned
#pragma unroll
                    for (int c = 0; c < D; c += 32) {
                        uint32_t o[32];
                        ptx::tmem_ld32(t_o + c, o);
                        ptx::tmem_wait_ld_regs(o);
#pragma unroll
                        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
                        ptx::tmem_st32(t_o + c, o);
                    }
                }
                ptx::tmem_wait_st();
                ptx::tc_fence_before();
                ptx::mbar_arrive(bar(C::kPFull + q));
                // The weight sum, from the same bf16 weights the PV product multiplies (each half of a packed
                // pair widened exactly to f32), so that O / l is a convex combination of V rows.  It runs after
                // P is signalled, off the softmax-to-MMA chain that bounds the kernel.  Against a sum of the
                // unrounded f32 weights inside the chain this costs ~2 % of the attention time (c2 +1.9 %, c4
                // +2.3 %); widening by mixed-precision adds instead cost +3.3 % / +4.0 %, and either inside the
                // chain +5-10 %.
                {
                    float la[4] = {0.f, 0.f, 0.f, 0.f}, lb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int c = 0; c < kBN / 2; ++c)
                        ptx::add2(la[c & 3], lb[c & 3], la[c & 3], lb[c & 3], __uint_as_float(pk[c] << 16),
                                  __uint_as_float(pk[c] & 0xFFFF0000u));
                    float s0, s1, s2, s3;
                    ptx::add2(s0, s1, la[0], lb[0], la[1], lb[1]);
                    ptx::add2(s2, s3, la[2], lb[2], la[3], lb[3]);
                    l_run += (s0 + s2) + (s1 + s3);
                }
            }
            if (!ok) break;
            if constexpr (kCas == kCasShared) {
                if (!(ok = __all_sync(0xffffffffu, wait_bar(bar(C::kOFinal + q), o_phase, ctl)))) break;
                o_phase ^= 1;
                ptx::tc_fence_after();
                // this row's unnormalised O and (max, sum) at (token, head), for the private pass to merge
                const long long tok = (long long)tq0 + r / a.G;  // a row of the whole batch
                const bool valid = tok < a.cas_T;
                const long long prow = tok * a.Hq + g * a.G + r % a.G;
                float4* po = reinterpret_cast<float4*>(a.cas_o + prow * D);
#pragma unroll
                for (int c = 0; c < D; c += 32) {
                    uint32_t o[32];
                    ptx::tmem_ld32(t_o + c, o);
                    ptx::tmem_wait_ld_regs(o);
                    if (valid) {
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            po[c / 4 + i] = make_float4(__uint_as_float(o[4 * i]), __uint_as_float(o[4 * i + 1]),
                                                        __uint_as_float(o[4 * i + 2]), __uint_as_float(o[4 * i + 3]));
                    }
                }
                if (valid) a.cas_ml[prow] = make_float2(m_run, l_run);
                continue;
            }
            if constexpr (kCas == kCasPrivate) {
                // merge with the shared pass's partial of this (token, head): both are in log2 units of the same
                // scale, so o = (2^(m_s - M) O_s + 2^(m - M) O) / (2^(m_s - M) l_s + 2^(m - M) l), M = max(m_s, m)
                const int tok = tq0 + r / a.G;
                const bool valid = tok < a.suffix[b];
                const long long prow = (long long)(a.cu[b] + tok) * a.Hq + g * a.G + r % a.G;
                const float4* so = reinterpret_cast<const float4*>(a.cas_o + prow * D);
                const float2 ml = valid ? a.cas_ml[prow] : make_float2(-INFINITY, 0.f);  // in flight during the wait
                if (!(ok = __all_sync(0xffffffffu, wait_bar(bar(C::kOFinal + q), o_phase, ctl)))) break;
                o_phase ^= 1;
                ptx::tc_fence_after();
                const float M = fmaxf(ml.x, m_run);  // m_run is finite: a row sees at least its own key here
                const float ws = ml.x == -INFINITY ? 0.f : ptx::ex2_approx(ml.x - M);
                const float wp = ptx::ex2_approx(m_run - M);
                const float inv = 1.0f / (ws * ml.y + wp * l_run);
                __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(a.out) + prow * D;
                // 16 columns at a time (few registers: this is the epilogue of a kernel tuned to its limit), the
                // shared partial's next 16 columns in flight while these are merged and stored
                float4 nx[4];
                if (valid) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) nx[i] = so[i];
                }
#pragma unroll
                for (int c = 0; c < D; c += 16) {
                    uint32_t o[16];
                    ptx::tmem_ld16(t_o + c, o);
                    float4 sx[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) sx[i] = nx[i];
                    if (valid && c + 16 < D) {
#pragma unroll
                        for (int i = 0; i < 4; ++i) nx[i] = so[(c + 16) / 4 + i];
                    }
                    ptx::tmem_wait_ld_regs16(o);
                    uint32_t pk[8];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        pk[2 * i] = ptx::pack_bf16x2((wp * __uint_as_float(o[4 * i]) + ws * sx[i].x) * inv,
                                                     (wp * __uint_as_float(o[4 * i + 1]) + ws * sx[i].y) * inv);
                        pk[2 * i + 1] = ptx::pack_bf16x2((wp * __uint_as_float(o[4 * i + 2]) + ws * sx[i].z) * inv,
                                                         (wp * __uint_as_float(o[4 * i + 3]) + ws * sx[i].w) * inv);
                    }
                    if (valid) {
                        uint4* d4 = reinterpret_cast<uint4*>(dst + c);
                        d4[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                        d4[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                    }
                }
                continue;
            }
            if (!(ok = __all_sync(0xffffffffu, wait_bar(bar(C::kOFinal + q), o_phase, ctl)))) break;
            o_phase ^= 1;
            ptx::tc_fence_after();
            const int slot = a.item_slot[ui];
            if (slot >= 0) {
                // split item: unnormalised fp32 O row plus (max, sum); the combine kernel merges the splits
                const long long prow = (long long)slot * (kNQ * kBM) + q * kBM + r;
                float4* po = reinterpret_cast<float4*>(a.part_o + prow * D);
#pragma unroll
                for (int c = 0; c < D; c += 32) {
                    uint32_t o[32];
                    ptx::tmem_ld32(t_o + c, o);
                    ptx::tmem_wait_ld_regs(o);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        po[c / 4 + i] = make_float4(__uint_as_float(o[4 * i]), __uint_as_float(o[4 * i + 1]),
                                                    __uint_as_float(o[4 * i + 2]), __uint_as_float(o[4 * i + 3]));
                }
                a.part_ml[prow] = make_float2(m_run, l_run);
                continue;
            }
            const float inv_l = 1.0f / l_run;
            const int tok = tq0 + r / a.G;
            const bool valid = tok < a.suffix[b];
            __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(a.out) +
                                 ((long long)(a.cu[b] + tok) * a.Hq + g * a.G + r % a.G) * D;
#pragma unroll
            for (int c = 0; c < D; c += 32) {
                uint32_t o[32];
                ptx::tmem_ld32(t_o + c, o);
                ptx::tmem_wait_ld_regs(o);
                uint32_t pk[16];
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    pk[i] = ptx::pack_bf16x2(__uint_as_float(o[2 * i]) * inv_l, __uint_as_float(o[2 * i + 1]) * inv_l);
                if (valid) {
                    uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
                    for (int i = 0; i < 4; ++i) d4[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                }
            }
        }
    }
    ptx::tc_fence_before();
    ptx::mbar_arrive(bar(C::kDone));
}

template <int D, int NK, int NV, bool kFused, bool kRope, int kCas = kCasNone>
cudaError_t launch_cfg(const AttnArgs& a, int grid, cudaStream_t st) {
    using C = Cfg<D, NK, NV>;
    static bool attr_done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!attr_done[dev]) {
        e = cudaFuncSetAttribute(extend_attn_kernel<D, NK, NV, kFused, kRope, kCas>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    if constexpr (kCas == kCasShared) {  // needs no schedule: an ordinary launch
        extend_attn_kernel<D, NK, NV, kFused, kRope, kCas><<<grid, kThreads, C::kSmemBytes, st>>>(a);
        return cudaGetLastError();
    } else if constexpr (kFused) {
        // the grid barrier between the two phases needs every CTA resident: a cooperative launch (the
        // runtime refuses a grid larger than the device holds), started once the schedule has finished
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(grid);
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = C::kSmemBytes;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeCooperative;
        attr[0].val.cooperative = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, extend_attn_kernel<D, NK, NV, kFused, kRope, kCas>, a);
    } else {
        return launch_after_sched(extend_attn_kernel<D, NK, NV, kFused, kRope, kCas>, dim3(grid), dim3(kThreads),
                                  C::kSmemBytes, st, a);
    }
}

}  // namespace

size_t extend_attention_smem_bytes(int head_dim) {
    if (head_dim == 128) return Cfg<128, 2, 3>::kSmemBytes;
    if (head_dim == 64) return Cfg<64, 4, 4>::kSmemBytes;
    return 0;
}

cudaError_t launch_extend_cascade(const AttnArgs& a, int head_dim, int grid, cudaStream_t st, bool shared_pass) {
    if (head_dim == 128)
        return shared_pass ? launch_cfg<128, 2, 3, false, false, kCasShared>(a, grid, st)
                           : launch_cfg<128, 2, 3, false, false, kCasPrivate>(a, grid, st);
    if (head_dim == 64)
        return shared_pass ? launch_cfg<64, 4, 4, false, false, kCasShared>(a, grid, st)
                           : launch_cfg<64, 4, 4, false, false, kCasPrivate>(a, grid, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_extend_attention(const AttnArgs& a, int head_dim, int grid, cudaStream_t st, bool fused) {
    if (fused && !a.grid_sync) return cudaErrorInvalidValue;
    if (head_dim == 128) {
        if (fused) return a.rope ? launch_cfg<128, 2, 3, true, true>(a, grid, st) : launch_cfg<128, 2, 3, true, false>(a, grid, st);
        return a.rope ? launch_cfg<128, 2, 3, false, true>(a, grid, st) : launch_cfg<128, 2, 3, false, false>(a, grid, st);
    }
    if (head_dim == 64) {
        if (fused) return a.rope ? launch_cfg<64, 4, 4, true, true>(a, grid, st) : launch_cfg<64, 4, 4, true, false>(a, grid, st);
        return a.rope ? launch_cfg<64, 4, 4, false, true>(a, grid, st) : launch_cfg<64, 4, 4, false, false>(a, grid, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace rr
