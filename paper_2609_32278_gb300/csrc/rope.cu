// rope.cu -- the (cos, sin) table of the rotary position embedding (see rope.cuh for the rotation).
//
// table[p][i] = (cos a, sin a), a = p * base^(-2i/D), for 0 <= p < max_pos, 0 <= i < D/2.  The angle
// and its cosine and sine are computed in double precision (the angle reaches ~10^5 radians at the
// longest contexts, where a float angle would be off by ~10^-2) and rounded once to float.  Built once
// per model; the append and attention kernels read it.
#include "rr_internal.h"

namespace rr {

namespace {

__global__ void __launch_bounds__(256) rope_table_kernel(float2* __restrict__ out, long long n, int half, double base) {
    const double two_over_d = 1.0 / half;  // 2 / D
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long p = idx / half;
        const int i = (int)(idx - p * half);
        const double a = (double)p * pow(base, -two_over_d * i);
        double s, c;
        sincos(a, &s, &c);
        out[idx] = make_float2((float)c, (float)s);
    }
}

}  // namespace

cudaError_t launch_rope_table(float2* out, int max_pos, int head_dim, double base, int sm_count, cudaStream_t st) {
    const int half = head_dim / 2;
    const long long n = (long long)max_pos * half;
    if (n == 0) return cudaSuccess;
    long long blocks = (n + 255) / 256;
    const long long cap = (long long)sm_count * 8;
    if (blocks > cap) blocks = cap;
    rope_table_kernel<<<(unsigned)blocks, 256, 0, st>>>(out, n, half, base);
    return cudaGetLastError();
}

}  // namespace rr
