// kv_append.cu -- write the uncached suffix's K/V rows into the paged pool.
//
// Sec. 2: the prefill materialises the KV tensors of the tokens it processes;
// the serving engine keeps them in a shared pool so the agent's next turn can
// reuse them.  Suffix token j of agent b (row cu_b + j of k_new / v_new) goes
// to position P_b + j: page page_table[b][pos / ps], slot pos % ps.
//
// One warp moves one token: the token's K row (all KV heads, Hkv*D bf16 =
// 2 KiB at Hkv=8, D=128) is contiguous in k_new and contiguous in the pool
// slot, so each lane issues 16-byte loads and stores that coalesce into whole
// 512-byte warp transactions on both sides.  Pure HBM copy: 4*T*Hkv*D*2 bytes
// of traffic, bound by HBM bandwidth.  The suffix rows are read once
// (streaming loads); the pool writes keep the default policy because the
// attention kernel reads those pages right after.
//
// Batches of up to kAppendSelfLensMaxB agents run as this one kernel: every block checks the lengths and takes
// the suffix prefix sums itself (self_lens), which takes the schedule kernel and its launch off the call.
//
// With a rotary table (kRope), each K row is rotated at its position P_b + j
// on the way into the pool (rope.cuh): a lane takes the two 16-byte vectors of
// one head that hold a rotation pair's halves (dims i0.. and i0 + D/2..), so
// the copy stays one pass over the same bytes plus a table read that the
// heads of one token share; V is copied unchanged.
#include "ptx.cuh"
#include "rope.cuh"
#include "rr_internal.h"

namespace rr {

namespace {

__device__ __forceinline__ int last_le(const int32_t* off, int n, long long x) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if ((long long)off[mid] <= x) lo = mid; else hi = mid - 1;
    }
    return lo;
}

constexpr int kAppendThreads = 256;
constexpr int kAppendBlocksPerSM = 4;  // resident blocks per SM: at most 64 registers a thread
constexpr int kCuSmem = 2048;  // agents whose suffix prefix sums a block stages in shared memory
static_assert(kAppendSelfLensMaxB < kCuSmem, "the self-checking path keeps B + 1 prefix sums in shared memory");

// The schedule kernel's length check and prefix sums, done by one block for itself (batches of fewer than
// kCuSmem agents): each thread takes a contiguous run of agents, checks 0 <= P, 0 <= S, P + S <= the page
// table's capacity, and the block scans the suffix lengths into s_cu[0..B]; the sum must equal T.  Every block
// reaches the same answer from the same lengths; block 0 reports a bad batch (RR_ERR_LENS) and no block writes.
__device__ bool self_lens(const AppendArgs& a, int32_t* s_cu, int32_t* s_pfx) {
    __shared__ long long s_w[kAppendThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int B = a.B;
    const int per = (B + kAppendThreads - 1) / kAppendThreads;
    const int b0 = min(B, (int)threadIdx.x * per), b1 = min(B, b0 + per);
    const long long cap = (long long)a.max_pages * a.ps;
    long long sum = 0;
    bool bad = false;
    for (int b = b0; b < b1; ++b) {
        const int P = a.prefix[b], S = a.suffix[b];
        if (P < 0 || S < 0 || (long long)P + S > cap) bad = true;
        sum += S;
    }
    long long inc = sum;  // inclusive scan over the block, in thread order
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31) s_w[warp] = inc;
    __syncthreads();
    long long before = 0, total = 0;
#pragma unroll
    for (int w = 0; w < kAppendThreads / 32; ++w) {
        if (w < warp) before += s_w[w];
        total += s_w[w];
    }
    long long off = before + inc - sum;
    const bool ok = !__syncthreads_or(bad) && total == a.T && total < (1ll << 31);
    if (!ok) {
        if (blockIdx.x == 0 && threadIdx.x == 0) atomicCAS(a.err, 0, RR_ERR_LENS);
        return false;
    }
    for (int b = b0; b < b1; ++b) {
        s_cu[b] = (int32_t)off;
        s_pfx[b] = a.prefix[b];
        off += a.suffix[b];
    }
    if (threadIdx.x == 0) s_cu[B] = (int32_t)total;
    __syncthreads();
    return true;
}


// kSelf: the lengths are checked and summed by the kernel itself (self_lens) instead of by the schedule kernel.
template <bool kRope, bool kSelf>
__global__ void __launch_bounds__(kAppendThreads, kAppendBlocksPerSM) kv_append_kernel(const AppendArgs a) {
    __shared__ int32_t s_cu[kCuSmem];
    __shared__ int32_t s_pfx[kCuSmem];
    // each token's agent is a binary search over the suffix prefix sums, and its position needs the agent's
    // prefix length: both from shared memory when they fit, so a token's copy does not wait behind dependent
    // global loads
    bool cu_in_smem = true;
    if constexpr (kSelf) {
        if (!self_lens(a, s_cu, s_pfx)) return;
    } else {
        ptx::griddep_wait();  // the schedule kernel's output (launched as its dependent)
        if (*a.lens_ok == 0) return;
        cu_in_smem = a.B < kCuSmem;
        if (cu_in_smem) {
            for (int i = threadIdx.x; i <= a.B; i += kAppendThreads) {
                s_cu[i] = a.cu[i];
                if (i < a.B) s_pfx[i] = a.prefix[i];
            }
            __syncthreads();
        }
    }
    const int32_t* __restrict__ cu = cu_in_smem ? s_cu : a.cu;
    const int32_t* __restrict__ pfx = cu_in_smem ? s_pfx : a.prefix;
    const int lane = threadIdx.x & 31;
    const long long warps = (long long)gridDim.x * (kAppendThreads / 32);
    const uint4* __restrict__ kn = a.k_new;
    const uint4* __restrict__ vn = a.v_new;
    uint4* __restrict__ kp = a.k_pool;
    uint4* __restrict__ vp = a.v_pool;
    for (long long t = (long long)blockIdx.x * (kAppendThreads / 32) + (threadIdx.x >> 5); t < a.T; t += warps) {
        const int b = last_le(cu, a.B, t);
        const long long pos = (long long)pfx[b] + (t - cu[b]);
        const long long src = t * a.row16;
        if constexpr (!kRope) {
            // 128 vectors of K and 128 of V at a time (the whole row up to Hkv * D = 1024), four of each per
            // lane; the first ones are read before the page-table entry comes back, so the two loads' latencies
            // overlap
            long long dst = -1;
            for (int c0 = 0; c0 < a.row16; c0 += 128) {
                uint4 kx[4], vx[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = c0 + lane + 32 * i;
                    if (e < a.row16) {
                        kx[i] = __ldcs(kn + src + e);
                        vx[i] = __ldcs(vn + src + e);
                    }
                }
                if (c0 == 0) {
                    const int page = a.page_table[(long long)b * a.max_pages + pos / a.ps];
                    if (page < 0 || (long long)page >= a.num_pages) {
                        if (lane == 0) atomicCAS(a.err, 0, RR_ERR_OOB);
                        break;
                    }
                    dst = ((long long)page * a.ps + pos % a.ps) * a.row16;
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = c0 + lane + 32 * i;
                    if (e < a.row16) {
                        kp[dst + e] = kx[i];
                        vp[dst + e] = vx[i];
                    }
                }
            }
        } else {
            const int page = a.page_table[(long long)b * a.max_pages + pos / a.ps];
            if (page < 0 || (long long)page >= a.num_pages) {
                if (lane == 0) atomicCAS(a.err, 0, RR_ERR_OOB);
                continue;
            }
            const long long dst = ((long long)page * a.ps + pos % a.ps) * a.row16;
            if (pos >= a.rope_max_pos) {  // no table row for this position: nothing written, reported
                if (lane == 0) atomicCAS(a.err, 0, RR_ERR_LENS);
                continue;
            }
            const float2* cs = a.rope + pos * (long long)(a.d16 * 8);  // this position's D/2 (cos, sin)
            int e = lane;
            for (; e + 96 < a.row16; e += 128) {  // V: four vectors in flight per lane, as below
                uint4 v0 = __ldcs(vn + src + e), v1 = __ldcs(vn + src + e + 32);
                uint4 v2 = __ldcs(vn + src + e + 64), v3 = __ldcs(vn + src + e + 96);
                vp[dst + e] = v0; vp[dst + e + 32] = v1; vp[dst + e + 64] = v2; vp[dst + e + 96] = v3;
            }
            for (; e < a.row16; e += 32) vp[dst + e] = __ldcs(vn + src + e);
#pragma unroll 2
            for (int x = lane; x < a.hkv * a.d16; x += 32) {  // K: the two vectors of one rotation pair unit
                const int h = x / a.d16, u = x - h * a.d16;
                const long long lo = (long long)h * 2 * a.d16 + u, hi = lo + a.d16;  // head h: 2 * d16 vectors
                uint4 k0 = __ldcs(kn + src + lo), k1 = __ldcs(kn + src + hi);
                float4 t[4];
                rope_load8(t, cs + u * 8);
                rope_rotate8(k0, k1, t);
                kp[dst + lo] = k0;
                kp[dst + hi] = k1;
            }
        }
    }
}

}  // namespace

cudaError_t launch_kv_append(const AppendArgs& a, int sm_count, cudaStream_t st) {
    const long long warps_needed = a.T;
    long long blocks = (warps_needed + (kAppendThreads / 32) - 1) / (kAppendThreads / 32);
    // two waves of resident blocks (a second-wave block starts as a first-wave one finishes): 2-7 % faster than
    // a grid of one wave on the c2 / c5 / c3_rr appends
    const long long cap = (long long)sm_count * kAppendBlocksPerSM * 2;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (a.self_lens) {  // an ordinary launch: it runs once the kernels before it on the stream have finished
        if (a.rope) kv_append_kernel<true, true><<<(unsigned)blocks, kAppendThreads, 0, st>>>(a);
        else kv_append_kernel<false, true><<<(unsigned)blocks, kAppendThreads, 0, st>>>(a);
        return cudaGetLastError();
    }
    cudaError_t e = a.rope ? launch_after_sched(kv_append_kernel<true, false>, dim3((unsigned)blocks), dim3(kAppendThreads), 0, st, a)
                           : launch_after_sched(kv_append_kernel<false, false>, dim3((unsigned)blocks), dim3(kAppendThreads), 0, st, a);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace rr
