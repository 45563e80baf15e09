// combine.cu -- merge the split-K partial results of extend attention.
//
// When a batch has too few work units to fill the GPU, the schedule splits each
// unit's key range into pieces; piece s of a row leaves an unnormalised output
// O_s, its running max m_s (log2 units, scale folded in) and its weight sum
// l_s = sum_j 2^(x_j - m_s).  The row's result is the log-sum-exp merge
//     M = max_s m_s,   w_s = 2^(m_s - M),   out = (sum_s w_s O_s) / (sum_s w_s l_s)
// which equals the unsplit softmax(x) V exactly in real arithmetic.  A piece in
// which a row sees no key has m_s = -inf, l_s = 0, O_s = 0 and weight 0; the
// first piece always holds key 0, so M is finite.  The pieces are merged in a
// fixed order, so the result is deterministic.
//
// One block per split unit (a.rows partial rows per piece: two Q tiles of 128
// packed rows for extend, one row per query head for decode); a warp takes a
// row at a time, each lane 4 of the D columns.  Memory bound: reads
// nsplit * (D + 2) floats per row, writes D bf16.
#include <cuda_bf16.h>

#include "ptx.cuh"
#include "rr_internal.h"

namespace rr {

namespace {

constexpr int kCombineThreads = 256;

template <int D>
__global__ void __launch_bounds__(kCombineThreads) combine_kernel(const CombineArgs a) {
    static_assert(D == 64 || D == 128, "lane mapping: 2 or 4 columns per lane");
    constexpr int kPer = D / 32;  // columns per lane
    ptx::griddep_wait();  // launched as the attention kernel's dependent: its partials must be complete
    const int n = *a.n_split;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int unit_tokens = kNQ * a.tq;
    for (int k = blockIdx.x; k < n; k += gridDim.x) {
        const int4 su = a.split_units[k];
        const int b = su.x, g = su.y & 0xFF, ns = (su.y >> 16) & 0xFF, u = su.z, base = su.w;
        const int S = a.suffix[b], cu_b = a.cu[b];
        for (int row = warp; row < a.rows; row += kCombineThreads / 32) {
            const int q = row / kBM, rr = row % kBM;
            const int tok = u * unit_tokens + q * a.tq + rr / a.G;
            if (tok >= S) continue;
            const int head = g * a.G + rr % a.G;
            // Both passes are unrolled so the loads of several pieces are in flight together (the merge
            // is a chain of dependent global loads otherwise: ~2 x nsplit memory latencies per row).
            float M = -INFINITY;
#pragma unroll 8
            for (int s = 0; s < ns; ++s) M = fmaxf(M, a.part_ml[(long long)(base + s) * a.rows + row].x);
            float L = 0.f, acc[kPer];
#pragma unroll
            for (int i = 0; i < kPer; ++i) acc[i] = 0.f;
#pragma unroll 4
            for (int s = 0; s < ns; ++s) {
                const long long prow = (long long)(base + s) * a.rows + row;
                const float2 ml = a.part_ml[prow];
                const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
                L += w * ml.y;
                const float* po = a.part_o + prow * D + lane * kPer;
                if constexpr (kPer % 4 == 0) {
#pragma unroll
                    for (int i = 0; i < kPer; i += 4) {
                        const float4 v = *reinterpret_cast<const float4*>(po + i);
                        acc[i] += w * v.x;
                        acc[i + 1] += w * v.y;
                        acc[i + 2] += w * v.z;
                        acc[i + 3] += w * v.w;
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < kPer; i += 2) {
                        const float2 v = *reinterpret_cast<const float2*>(po + i);
                        acc[i] += w * v.x;
                        acc[i + 1] += w * v.y;
                    }
                }
            }
            const float inv = 1.f / L;
            __nv_bfloat16* dst =
                reinterpret_cast<__nv_bfloat16*>(a.out) + ((long long)(cu_b + tok) * a.Hq + head) * D + lane * kPer;
#pragma unroll
            for (int i = 0; i < kPer; i += 2)
                *reinterpret_cast<__nv_bfloat162*>(dst + i) = __floats2bfloat162_rn(acc[i] * inv, acc[i + 1] * inv);
        }
    }
}

}  // namespace

cudaError_t launch_combine(const CombineArgs& a, int grid, cudaStream_t st) {
    if (grid < 1) grid = 1;
    cudaError_t e;
    if (a.D == 128) e = launch_after_sched(combine_kernel<128>, dim3(grid), dim3(kCombineThreads), 0, st, a);
    else if (a.D == 64) e = launch_after_sched(combine_kernel<64>, dim3(grid), dim3(kCombineThreads), 0, st, a);
    else return cudaErrorInvalidValue;
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace rr
