// sched.cu -- on-device schedule of one extend batch.
//
// The per-agent lengths live on the device, so the work list is built there
// too (one 1024-thread block, no host synchronisation):
//   1. validate the lengths and take exclusive prefix sums of the suffix
//      lengths (row offsets cu_b) and of the work units per agent;
//   2. (attention only) give every work unit -- one KV head of one agent,
//      kNQ consecutive Q tiles of its suffix -- its cost in KV tiles, the
//      number of 128-key tiles its last row must read (prefix + covered suffix);
//   3. if the batch has fewer than two waves of units, split each unit's KV
//      range into items (split-K) so the grid stays full; the partial results
//      are merged by the combine kernel;
//   4. order the items most expensive first, so a persistent grid that takes
//      them in order approximates longest-processing-time scheduling: runs of
//      up to 128 consecutive units of one (agent, KV head) kept together and
//      ordered by their most expensive unit (unsplit batches of up to 1024
//      groups: a run's units share their K/V pages through L2), else a
//      counting sort of the items by cost.  This is what balances a batch whose agents have very
//      different cached prefixes and uncached suffixes (the skew an eviction
//      policy creates, Sec. 3.1-3.3).
// Within a cost bucket the order is not fixed (atomics), which is harmless: a
// unit's result does not depend on which CTA computes it or when.
#include "ptx.cuh"
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

// KV tiles of piece sp of a unit of `cost` tiles split into ns pieces: floor((sp+1) cost / ns) -
// floor(sp cost / ns), in 32-bit arithmetic (cost < 2^24, ns <= 64: the products stay below 2^31;
// 64-bit division is a long software sequence, and this runs once per item in two passes).
__device__ __forceinline__ int piece_tiles(int cost, int ns, int sp) {
    return (sp + 1) * cost / ns - sp * cost / ns;
}

// Sum over the 1024 threads of the block (every thread gets the total).
__device__ long long block_sum(long long v, long long* s_ws) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) s_ws[warp] = v;
    __syncthreads();
    long long t = 0;
#pragma unroll 4
    for (int w = 0; w < 32; ++w) t += s_ws[w];
    __syncthreads();
    return t;
}

// Block-wide exclusive prefix sums of two values at once, in thread order; also returns the totals.
__device__ void block_exclusive_scan2(long long x, long long y, long long& ex, long long& ey, long long& tx,
                                      long long& ty, long long* s_wx, long long* s_wy) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    long long ix = x, iy = y;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long px = __shfl_up_sync(0xffffffffu, ix, o);
        const long long py = __shfl_up_sync(0xffffffffu, iy, o);
        if (lane >= o) { ix += px; iy += py; }
    }
    __syncthreads();
    if (lane == 31) { s_wx[warp] = ix; s_wy[warp] = iy; }
    __syncthreads();
    if (warp == 0) {
        long long wx = s_wx[lane], wy = s_wy[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long px = __shfl_up_sync(0xffffffffu, wx, o);
            const long long py = __shfl_up_sync(0xffffffffu, wy, o);
            if (lane >= o) { wx += px; wy += py; }
        }
        s_wx[lane] = wx;
        s_wy[lane] = wy;
    }
    __syncthreads();
    ex = (warp ? s_wx[warp - 1] : 0) + ix - x;
    ey = (warp ? s_wy[warp - 1] : 0) + iy - y;
    tx = s_wx[31];
    ty = s_wy[31];
    __syncthreads();
}

__global__ void __launch_bounds__(1024) sched_kernel(SchedArgs a) {
    __shared__ long long s_ws[32], s_wu[32];
    __shared__ int s_hist[kCostBuckets];
    __shared__ long long s_key[2048];  // run order: chunk keys; before that, the agents' unit offsets
    __shared__ int s_bad;
    int32_t* s_uoff = reinterpret_cast<int32_t*>(s_key);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // the consumer kernel may start its prologue now; it waits for this kernel before reading its output
    ptx::griddep_launch_dependents();
    if (tid == 0) {
        s_bad = 0;
        if (a.grid_sync) *a.grid_sync = 0;
    }
    __syncthreads();

    // ---- 1. validate, per-thread sums over a contiguous chunk of agents
    const int B = a.B;
    const int chunk = (B + 1023) / 1024;
    const int b0 = min(B, tid * chunk), b1 = min(B, b0 + chunk);
    if (a.kv_lens) {  // decode: the lengths in prefix / suffix form (read back below by the same threads,
                      // and by every thread after the next barrier); over a shared prefix, the private keys
        for (int b = b0; b < b1; ++b) {
            const int L = a.kv_lens[b] - a.lens_offset;
            a.prefix_out[b] = L - 1;  // L < 1 fails the check below
            a.suffix_out[b] = 1;
        }
    }
    if (a.shared_pages > 0) {  // a batch over a shared prefix: every agent's shared-prefix pages are agent 0's
        for (long long i = tid; i < (long long)B * a.shared_pages; i += 1024) {
            const long long b = i / a.shared_pages, p = i % a.shared_pages;
            if (a.page_table[b * a.max_pages + p] != a.page_table[p]) {
                atomicCAS(a.err, 0, RR_ERR_SHARED);
                s_bad = 1;
            }
        }
    }
    const long long cap = (long long)a.max_pages * a.ps;
    long long sum_s = 0, sum_u = 0;
    bool bad = false;
    for (int b = b0; b < b1; ++b) {
        const int P = a.prefix[b], S = a.suffix[b];
        if (P < a.min_prefix || S < 0 || (long long)P + S > cap) { bad = true; continue; }
        sum_s += S;
        sum_u += (long long)a.Hkv * ((S + a.unit_tokens - 1) / a.unit_tokens);  // 32-bit division
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
    // the binary searches below read the unit offsets from shared memory when they fit (B + 1 <= 4096)
    const bool uoff_smem = B < 2 * 2048;
    if (ok) {
        for (int b = b0; b < b1; ++b) {
            const int S = a.suffix[b];
            a.cu[b] = (int32_t)off_s;
            a.unit_off[b] = (int32_t)off_u;
            if (uoff_smem) s_uoff[b] = (int32_t)off_u;
            off_s += S;
            off_u += (long long)a.Hkv * ((S + a.unit_tokens - 1) / a.unit_tokens);
        }
        if (tid == 0) {
            a.cu[B] = (int32_t)tot_s;
            a.unit_off[B] = (int32_t)tot_u;
            if (uoff_smem) s_uoff[B] = (int32_t)tot_u;
        }
    }
    if (!ok) {
        if (tid == 0) {
            atomicCAS(a.err, 0, RR_ERR_LENS);
            *a.lens_ok = 0;
            *a.n_units = 0;
            if (a.n_split) *a.n_split = 0;  // the combine must not replay a previous call's split list
        }
        return;  // uniform: every thread sees the same `ok`
    }
    if (tid == 0) *a.lens_ok = 1;
    if (!a.build_units) return;
    __syncthreads();  // every thread's cu / unit_off entries are written
    const int32_t* prefix = a.prefix;
    const int32_t* suffix = a.suffix;
    const int32_t* unit_off = uoff_smem ? s_uoff : a.unit_off;

    // ---- 2. split decision: a unit's cost is the number of 128-key tiles its last row reads.
    // Split the KV range of every unit when the batch has fewer than two waves of units: a unit of
    // `cost` KV tiles becomes ceil(cost / target) items (at most 64), target = total / (W waves), at
    // least 8 tiles.  Then items <= total/target + units <= (W + 2) waves, which bounds the partial buffers.
    const long long W = a.split_waves > 0 ? a.split_waves : 2;
    // extra_slots > 0 (decode over a shared prefix): every unit writes partials, split or not
    const bool split = tot_u > 0 && tot_u <= 1024 &&
                       (a.extra_slots > 0 || (a.split_grid > 0 && tot_u < 2ll * a.split_grid));
    const bool cut = split && a.split_grid > 0 && tot_u < 2ll * a.split_grid;  // pieces per unit > 1 allowed
    int my_b = 0, my_g = 0, my_u = 0, my_ns = 1;
    long long my_unit_cost = 0;
    int my_cost32 = 0;  // the same, in 32 bits (a unit reads fewer than 2^24 tiles: 2^31 keys)
    if (split && tid < tot_u) {  // a split batch has at most 1024 units: one per thread
        my_b = last_le(unit_off, B, tid);
        const int S = suffix[my_b], P = prefix[my_b];
        const int nu = (S + a.unit_tokens - 1) / a.unit_tokens;
        const int local = tid - unit_off[my_b];
        my_g = local / nu;
        my_u = local % nu;
        const long long n_keys = (long long)P + min((long long)S, (long long)(my_u + 1) * a.unit_tokens);
        my_unit_cost = (n_keys + kBN - 1) / kBN;
        my_cost32 = (int)my_unit_cost;
    }
    const long long tot_cost = cut ? block_sum(my_unit_cost, s_ws) : 0;  // `cut` is uniform over the block
    const long long target = cut ? max(8ll, (tot_cost + W * a.split_grid - 1) / (W * a.split_grid)) : (1ll << 40);
    if (split && tid < tot_u) {
        my_ns = (int)min(min(64ll, my_unit_cost), (my_unit_cost + target - 1) / target);
        if (my_ns < 1) my_ns = 1;
    }
    // partial-result slots and the rank of each split unit (exclusive scans over units)
    const bool my_partial = split && tid < tot_u && (my_ns > 1 || a.extra_slots > 0);
    const int my_slots = my_partial ? my_ns + a.extra_slots : 0;
    long long my_slot_base = 0, my_rank = 0, n_slots = 0, n_split_units = 0;
    block_exclusive_scan2(my_slots, my_partial ? 1 : 0, my_slot_base, my_rank, n_slots, n_split_units, s_ws, s_wu);
    if (my_partial && a.unit_slot) a.unit_slot[(long long)my_b * a.Hkv + my_g] = (int32_t)my_slot_base;

    // ---- 3'. unsplit batches of at most 1024 (agent, KV head) groups: list the units of a group in runs of
    // up to 128 consecutive units (a chunk), most expensive unit first, and order the chunks by their most
    // expensive unit.  A wave's CTAs then work on a few chunks at once, whose units stream the same K/V pages
    // at about the same time and share them through L2, instead of a group's units landing in different
    // waves and reading its pages from DRAM again; and since chunks are ordered by unit cost, the list stays
    // close to longest-first, which keeps the persistent grid's CTAs evenly loaded.  Deterministic.
    const long long n_groups = (long long)B * a.Hkv;
    // (decode: a group is one unit, so the counting sort below gives the same order, faster)
    if (!split && n_groups <= 1024 && !a.kv_lens) {
        int nu = 0, P = 0, S = 0;  // group tid = (agent tid / Hkv, KV head tid % Hkv)
        if (tid < n_groups) {
            S = suffix[tid / a.Hkv];
            P = prefix[tid / a.Hkv];
            nu = (S + a.unit_tokens - 1) / a.unit_tokens;
        }
        // the shortest chunk (128, 256 or 512 units) that keeps the batch within the sort's 2048 slots: a
        // group longer than that (a long suffix, whose units' costs spread widely) is cut for balance, the
        // others stay whole so that their units run in one wave
        int run = 0;
        for (int r = 128; r <= 512 && !run; r <<= 1)
            if (block_sum((nu + r - 1) / r, s_ws) <= 2048) run = r;
        if (run) {
            const int nch = (nu + run - 1) / run;
            long long cbase = 0, dummy = 0, t0 = 0, t1 = 0;
            block_exclusive_scan2(nch, 0, cbase, dummy, t0, t1, s_ws, s_wu);
            int n2 = 2;  // sort length: the chunks rounded up to a power of two (<= 2048)
            while (n2 < t0) n2 <<= 1;
            for (int i2 = tid; i2 < n2; i2 += 1024) s_key[i2] = -1;  // empty slots sort below every chunk
            __syncthreads();
            for (int c = 0; c < nch; ++c) {  // chunk c: units nu-1-c*run down to max(0, nu-(c+1)*run)
                const int u = nu - 1 - c * run;
                const long long top = ((long long)P + min((long long)S, (long long)(u + 1) * a.unit_tokens) + kBN - 1) / kBN;
                const long long id = ((long long)tid << 11) | c;  // group, chunk within it (< 2048)
                s_key[cbase + c] = (top << 21) | ((1ll << 21) - 1 - id);  // by cost, then group and chunk order
            }
            __syncthreads();
            for (int k = 2; k <= n2; k <<= 1) {  // bitonic sort of n2 keys, ascending
                for (int jj = k >> 1; jj > 0; jj >>= 1) {
                    for (int i2 = tid; i2 < n2; i2 += 1024) {
                        const int ixj = i2 ^ jj;
                        if (ixj > i2) {
                            const long long x = s_key[i2], y = s_key[ixj];
                            if (((i2 & k) == 0) ? (x > y) : (x < y)) {
                                s_key[i2] = y;
                                s_key[ixj] = x;
                            }
                        }
                    }
                    __syncthreads();
                }
            }
            // thread t takes ranks 2t and 2t + 1 (rank 0 = the chunk with the most expensive unit)
            int cg[2], cc[2], cn[2];
            for (int q = 0; q < 2; ++q) {
                const int rank = 2 * tid + q;
                const long long key = rank < n2 ? s_key[n2 - 1 - rank] : -1;
                cg[q] = -1; cc[q] = 0; cn[q] = 0;
                if (key >= 0) {
                    const long long id = (1ll << 21) - 1 - (key & ((1ll << 21) - 1));
                    cg[q] = (int)(id >> 11);
                    cc[q] = (int)(id & 2047);
                    const int gnu = (suffix[cg[q] / a.Hkv] + a.unit_tokens - 1) / a.unit_tokens;
                    cn[q] = min(run, gnu - cc[q] * run);
                }
            }
            long long start = 0, d2 = 0, t2 = 0, t3 = 0;
            block_exclusive_scan2(cn[0] + cn[1], 0, start, d2, t2, t3, s_ws, s_wu);
            for (int q = 0; q < 2; ++q) {
                if (cg[q] >= 0) {
                    const int gb = cg[q] / a.Hkv, gh = cg[q] % a.Hkv;
                    const int gS = suffix[gb], gP = prefix[gb];
                    const int gnu = (gS + a.unit_tokens - 1) / a.unit_tokens;
                    for (int i2 = 0; i2 < cn[q]; ++i2) {
                        const int u = gnu - 1 - cc[q] * run - i2;
                        const long long n_keys = (long long)gP + min((long long)gS, (long long)(u + 1) * a.unit_tokens);
                        a.units[start + i2] = make_int4(gb, gh | (1 << 16), u, (int)((n_keys + kBN - 1) / kBN));
                        a.item_slot[start + i2] = -1;
                    }
                }
                start += cn[q];
            }
            if (tid == 0) {
                *a.n_units = (int32_t)tot_u;
                *a.n_split = 0;
            }
            return;
        }
    }

    // ---- 3. histogram of item costs
    for (int i = tid; i < kCostBuckets; i += 1024) s_hist[i] = 0;
    __syncthreads();
    if (!split) {
        for (long long idx = tid; idx < tot_u; idx += 1024) {
            const int b = last_le(unit_off, B, idx);
            const int S = suffix[b], P = prefix[b];
            const int nu = (S + a.unit_tokens - 1) / a.unit_tokens;
            const int u = (int)(idx - unit_off[b]) % nu;
            const long long n_keys = (long long)P + min((long long)S, (long long)(u + 1) * a.unit_tokens);
            const long long cost = (n_keys + kBN - 1) / kBN;
            atomicAdd(&s_hist[(int)min(cost, (long long)kCostBuckets - 1)], 1);
        }
    } else if (tid < tot_u) {
        for (int sp = 0; sp < my_ns; ++sp) {
            const int c = piece_tiles(my_cost32, my_ns, sp);
            atomicAdd(&s_hist[min(c, kCostBuckets - 1)], 1);
        }
    }
    __syncthreads();

    // ---- 4. exclusive scan in descending cost order: start[k] = sum of hist[k'] for k' > k
    {
        constexpr int kPer = kCostBuckets / 1024;
        int v[kPer];
        int local = 0;
#pragma unroll
        for (int i = 0; i < kPer; ++i) {  // descending position tid*kPer+i <-> bucket kCostBuckets-1-(tid*kPer+i)
            v[i] = s_hist[kCostBuckets - 1 - (tid * kPer + i)];
            local += v[i];
        }
        long long ex = 0, dummy = 0, t0 = 0, t1 = 0;
        block_exclusive_scan2(local, 0, ex, dummy, t0, t1, s_ws, s_wu);
        int run = (int)ex;
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            s_hist[kCostBuckets - 1 - (tid * kPer + i)] = run;  // becomes the bucket's cursor
            run += v[i];
        }
    }
    __syncthreads();

    // ---- 5. scatter: item = (agent, kv head | split << 8 | nsplit << 16, unit, KV tiles of the whole unit)
    if (!split) {
        for (long long idx = tid; idx < tot_u; idx += 1024) {
            const int b = last_le(unit_off, B, idx);
            const int S = suffix[b], P = prefix[b];
            const int nu = (S + a.unit_tokens - 1) / a.unit_tokens;
            const int local = (int)(idx - unit_off[b]);
            const int h = local / nu, u = local % nu;
            const long long n_keys = (long long)P + min((long long)S, (long long)(u + 1) * a.unit_tokens);
            const long long cost = (n_keys + kBN - 1) / kBN;
            const int pos = atomicAdd(&s_hist[(int)min(cost, (long long)kCostBuckets - 1)], 1);
            a.units[pos] = make_int4(b, h | (1 << 16), u, (int)cost);
            a.item_slot[pos] = -1;
        }
    } else if (tid < tot_u) {
        for (int sp = 0; sp < my_ns; ++sp) {
            const int c = piece_tiles(my_cost32, my_ns, sp);
            const int pos = atomicAdd(&s_hist[min(c, kCostBuckets - 1)], 1);
            a.units[pos] = make_int4(my_b, my_g | (sp << 8) | (my_ns << 16), my_u, (int)my_unit_cost);
            a.item_slot[pos] = my_partial ? (int)(my_slot_base + a.extra_slots + sp) : -1;
        }
        if (my_partial) a.split_units[my_rank] = make_int4(my_b, my_g | (my_slots << 16), my_u, (int)my_slot_base);
    }
    if (tid == 0) {
        // items: the pieces of every unit (slots minus the reserved ones of units that write partials)
        *a.n_units = split ? (int32_t)(n_slots - (long long)a.extra_slots * n_split_units + (tot_u - n_split_units))
                           : (int32_t)tot_u;
        *a.n_split = split ? (int32_t)n_split_units : 0;
    }
}

}  // namespace

cudaError_t launch_sched(const SchedArgs& a, cudaStream_t st) {
    sched_kernel<<<1, 1024, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace rr
