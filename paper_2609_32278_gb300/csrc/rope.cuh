// rope.cuh -- rotary position embedding on the device, shared by the append and attention kernels.
//
// The paper uses no positional encoding of its own; the models its agents run (Llama-3, Qwen3) rotate
// every q and k row by its absolute position before attention (RoPE, Su et al., "RoFormer", 2021), so
// an extend step fed un-rotated rows rotates the suffix's rows at positions P_b + j -- the positions
// that continue the cached prefix, which is what keeps the cached keys valid.  Pairing: dim i < D/2
// with dim i + D/2 (the GPT-NeoX / Llama "rotate-half" layout); pair i at position p turns by
// a = p * base^(-2i/D):
//     y[i]       = x[i] cos a - x[i + D/2] sin a
//     y[i + D/2] = x[i + D/2] cos a + x[i] sin a
// cos a and sin a come from a table [max_pos][D/2] of float2 (cos, sin) built once in double
// precision (rope_table_kernel); the rotation runs in fp32 and is rounded to nearest-even bf16.
#pragma once
#include <cstdint>

#include "ptx.cuh"

namespace rr {

// Rotate the eight pairs (lo[e], hi[e]), e = 0..7: lo holds dims i0 .. i0+7 and hi dims i0+D/2 .. i0+D/2+7
// of one row as bf16; t holds the table's eight (cos, sin) entries of pairs i0 .. i0+7 as four float4
// (c, s, c, s).
__device__ __forceinline__ void rope_rotate8(uint4& lo, uint4& hi, const float4 (&t)[4]) {
    uint32_t* l = reinterpret_cast<uint32_t*>(&lo);
    uint32_t* h = reinterpret_cast<uint32_t*>(&hi);
#pragma unroll
    for (int w = 0; w < 4; ++w) {  // word w: pairs 2w (low half) and 2w + 1 (high half)
        const float a0 = __uint_as_float(l[w] << 16), a1 = __uint_as_float(l[w] & 0xffff0000u);
        const float b0 = __uint_as_float(h[w] << 16), b1 = __uint_as_float(h[w] & 0xffff0000u);
        const float c0 = t[w].x, s0 = t[w].y, c1 = t[w].z, s1 = t[w].w;
        const float y0 = fmaf(a0, c0, -(b0 * s0)), z0 = fmaf(b0, c0, a0 * s0);
        const float y1 = fmaf(a1, c1, -(b1 * s1)), z1 = fmaf(b1, c1, a1 * s1);
        l[w] = ptx::pack_bf16x2(y0, y1);
        h[w] = ptx::pack_bf16x2(z0, z1);
    }
}

// The table's eight (cos, sin) entries starting at cs (16-byte aligned).
__device__ __forceinline__ void rope_load8(float4 (&t)[4], const float2* __restrict__ cs) {
    const float4* c4 = reinterpret_cast<const float4*>(cs);
#pragma unroll
    for (int k = 0; k < 4; ++k) t[k] = __ldg(c4 + k);
}

}  // namespace rr
