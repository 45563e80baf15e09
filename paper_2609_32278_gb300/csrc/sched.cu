// sched.cu -- on-device schedule of one extend batch.
//
// The per-agent lengths live on the device, so the work list is built there
// too (one 1024-thread block, no host synchronisation):
//   1. validate the lengths and take exclusive prefix sums of the suffix
//      lengths (row offsets cu_b) and of the work units per agent;
//   2. (attention only) give every work unit -- one KV head of one agent,
//      kNQ consecutive Q tiles of its suffix -- its cost in KV tiles, the
//      number of 128-key tiles its last row must read (prefix + covered suffix);
//   3. counting-sort the units by cost, most expensive first, so a persistent
//      grid that takes them in order approximates longest-processing-time
//      scheduling.  This is what balances a batch whose agents have very
//      different cached prefixes and uncached suffixes (the skew an eviction
//      policy creates, Sec. 3.1-3.3).
// Within a cost bucket the order is not fixed (atomics), which is harmless: a
// unit's result does not depend on which CTA computes it or when.
#include "rr_internal.h"

namespace rr {

namespace {

// Last index b in [0, n) with off[b] <= x (off nondecreasing, off[0] == 0 <= x).
__device__ __forceinline__ int last_le(const int32_t* off, int n, long long x) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if ((long long)off[mid] <= x) lo = mid; else hi = mid - 1;
    }
    return lo;
}

__global__ void __launch_bounds__(1024) sched_kernel(SchedArgs a) {
    __shared__ long long s_ws[32], s_wu[32];
    __shared__ int s_hist[kCostBuckets];
    __shared__ int s_bad;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) s_bad = 0;
    __syncthreads();

    // ---- 1. validate, per-thread sums over a contiguous chunk of agents
    const int B = a.B;
    const int chunk = (B + 1023) / 1024;
    const int b0 = min(B, tid * chunk), b1 = min(B, b0 + chunk);
    const long long cap = (long long)a.max_pages * a.ps;
    long long sum_s = 0, sum_u = 0;
    bool bad = false;
    for (int b = b0; b < b1; ++b) {
        const long long P = a.prefix[b], S = a.suffix[b];
        if (P < 0 || S < 0 || P + S > cap) { bad = true; continue; }
        sum_s += S;
        sum_u += (long long)a.Hkv * ((S + a.unit_tokens - 1) / a.unit_tokens);
    }
    if (bad) s_bad = 1;
    long long inc_s = sum_s, inc_u = sum_u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        long long ys = __shfl_up_sync(0xffffffffu, inc_s, o);
        long long yu = __shfl_up_sync(0xffffffffu, inc_u, o);
        if (lane >= o) { inc_s += ys; inc_u += yu; }
    }
    if (lane == 31) { s_ws[warp] = inc_s; s_wu[warp] = inc_u; }
    __syncthreads();
    if (warp == 0) {
        long long xs = s_ws[lane], xu = s_wu[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            long long ys = __shfl_up_sync(0xffffffffu, xs, o);
            long long yu = __shfl_up_sync(0xffffffffu, xu, o);
            if (lane >= o) { xs += ys; xu += yu; }
        }
        s_ws[lane] = xs;
        s_wu[lane] = xu;
    }
    __syncthreads();
    const long long tot_s = s_ws[31], tot_u = s_wu[31];
    long long off_s = (warp ? s_ws[warp - 1] : 0) + inc_s - sum_s;
    long long off_u = (warp ? s_wu[warp - 1] : 0) + inc_u - sum_u;
    const bool ok = !s_bad && tot_s == a.T && tot_s < (1ll << 31) && (!a.build_units || tot_u <= a.max_units);
    if (ok) {
        for (int b = b0; b < b1; ++b) {
            const long long S = a.suffix[b];
            a.cu[b] = (int32_t)off_s;
            a.unit_off[b] = (int32_t)off_u;
            off_s += S;
            off_u += (long long)a.Hkv * ((S + a.unit_tokens - 1) / a.unit_tokens);
        }
        if (tid == 0) { a.cu[B] = (int32_t)tot_s; a.unit_off[B] = (int32_t)tot_u; }
    }
    if (!ok) {
        if (tid == 0) {
            atomicCAS(a.err, 0, RR_ERR_LENS);
            *a.lens_ok = 0;
            *a.n_units = 0;
        }
        return;  // uniform: every thread sees the same `ok`
    }
    if (tid == 0) *a.lens_ok = 1;
    if (!a.build_units) return;

    // ---- 2. histogram of unit costs
    for (int i = tid; i < kCostBuckets; i += 1024) s_hist[i] = 0;
    __syncthreads();  // also publishes cu / unit_off written above to the whole block
    for (long long idx = tid; idx < tot_u; idx += 1024) {
        const int b = last_le(a.unit_off, B, idx);
        const int S = a.suffix[b], P = a.prefix[b];
        const int nu = (S + a.unit_tokens - 1) / a.unit_tokens;
        const int local = (int)(idx - a.unit_off[b]);
        const int u = local % nu;
        const long long n_keys = (long long)P + min((long long)S, (long long)(u + 1) * a.unit_tokens);
        const long long cost = (n_keys + kBN - 1) / kBN;
        atomicAdd(&s_hist[(int)min(cost, (long long)kCostBuckets - 1)], 1);
    }
    __syncthreads();

    // ---- 3. exclusive scan in descending cost order: start[k] = sum of hist[k'] for k' > k
    {
        constexpr int kPer = kCostBuckets / 1024;
        int v[kPer];
        int local = 0;
#pragma unroll
        for (int i = 0; i < kPer; ++i) {  // descending position tid*kPer+i <-> bucket kCostBuckets-1-(tid*kPer+i)
            v[i] = s_hist[kCostBuckets - 1 - (tid * kPer + i)];
            local += v[i];
        }
        int inc = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += y;
        }
        __syncthreads();
        if (lane == 31) s_ws[warp] = inc;
        __syncthreads();
        if (warp == 0) {
            long long x = s_ws[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                long long y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            s_ws[lane] = x;
        }
        __syncthreads();
        int run = (int)((warp ? s_ws[warp - 1] : 0) + inc - local);
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            s_hist[kCostBuckets - 1 - (tid * kPer + i)] = run;  // becomes the bucket's cursor
            run += v[i];
        }
    }
    __syncthreads();

    // ---- 4. scatter
    for (long long idx = tid; idx < tot_u; idx += 1024) {
        const int b = last_le(a.unit_off, B, idx);
        const int S = a.suffix[b], P = a.prefix[b];
        const int nu = (S + a.unit_tokens - 1) / a.unit_tokens;
        const int local = (int)(idx - a.unit_off[b]);
        const int h = local / nu, u = local % nu;
        const long long n_keys = (long long)P + min((long long)S, (long long)(u + 1) * a.unit_tokens);
        const long long cost = (n_keys + kBN - 1) / kBN;
        const int pos = atomicAdd(&s_hist[(int)min(cost, (long long)kCostBuckets - 1)], 1);
        a.units[pos] = make_int4(b, h, u, (int)cost);
    }
    if (tid == 0) *a.n_units = (int32_t)tot_u;
}

}  // namespace

cudaError_t launch_sched(const SchedArgs& a, cudaStream_t st) {
    sched_kernel<<<1, 1024, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace rr
