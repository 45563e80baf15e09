/*
 * Seeded synthetic inputs for the extend-attention path (GPU side).
 *
 * Implements the same counter-based generator as synth.c (SplitMix64 output
 * function chained over logical coordinates, Irwin-Hall sum of twelve 16-bit
 * uniforms, round-to-nearest-even to bf16) so that full-size inputs can be
 * written straight into device memory.  Integer-only arithmetic: the values
 * are bit-identical to the CPU ones.  Holds no arithmetic of the attention or
 * append method.  Built as its own shared library, separate from the product
 * library, and used only by tests and the benchmark to create inputs.
 */
#include <cstdint>
#include <cuda_runtime.h>

#define RRS_SHARED 0xFFFFFFFFu

__device__ __forceinline__ uint64_t rrs_mix(uint64_t z) {
    z += 0x9e3779b97f4a7c15ull;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t rrs_row_key(uint64_t seed, uint32_t tensor, uint32_t owner, uint64_t pos) {
    uint64_t h = rrs_mix(seed);
    h = rrs_mix(h ^ (uint64_t)tensor);
    h = rrs_mix(h ^ (uint64_t)owner);
    h = rrs_mix(h ^ pos);
    return h;
}

__device__ __forceinline__ uint16_t rrs_elem(uint64_t row_key, uint32_t head, uint32_t dim) {
    uint64_t h = rrs_mix(row_key ^ (((uint64_t)head << 20) | (uint64_t)dim));
    int32_t s = 0;
#pragma unroll
    for (uint64_t k = 1; k <= 3; ++k) {
        uint64_t r = rrs_mix(h + k);
        s += (int32_t)(r & 0xFFFF) + (int32_t)((r >> 16) & 0xFFFF) +
             (int32_t)((r >> 32) & 0xFFFF) + (int32_t)((r >> 48) & 0xFFFF);
    }
    float x = (float)(s - 393210) * (1.0f / 65536.0f);
    uint32_t u = __float_as_uint(x);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

// dst[r, h, d] for h in [head0, head0 + head_count): one block per row.
__global__ void rrs_fill_rows_kernel(uint16_t* __restrict__ dst, const int32_t* __restrict__ row_agent,
                                     const int64_t* __restrict__ row_pos, int64_t n_rows, int32_t head0,
                                     int32_t head_count, int32_t D, uint32_t tensor, uint64_t seed,
                                     int64_t shared_len) {
    for (int64_t r = blockIdx.x; r < n_rows; r += gridDim.x) {
        int64_t pos = row_pos[r];
        uint32_t owner = pos < shared_len ? RRS_SHARED : (uint32_t)row_agent[r];
        uint64_t key = rrs_row_key(seed, tensor, owner, (uint64_t)pos);
        int32_t n = head_count * D;
        uint16_t* out = dst + r * (int64_t)n;
        for (int32_t e = threadIdx.x; e < n; e += blockDim.x)
            out[e] = rrs_elem(key, (uint32_t)(head0 + e / D), (uint32_t)(e % D));
    }
}

// One block per listed page: tokens pos0 .. min(pos0 + ps, pos_end) of page page_ids[i].
__global__ void rrs_fill_pool_kernel(uint16_t* __restrict__ pool, const int32_t* __restrict__ page_ids,
                                     const int32_t* __restrict__ page_agent, const int64_t* __restrict__ page_pos0,
                                     const int64_t* __restrict__ page_pos_end, int64_t n_list, int32_t ps,
                                     int32_t Hkv, int32_t D, uint32_t tensor, uint64_t seed, int64_t shared_len) {
    int32_t row = Hkv * D;
    for (int64_t i = blockIdx.x; i < n_list; i += gridDim.x) {
        int64_t page = page_ids[i];
        int64_t p0 = page_pos0[i], pe = page_pos_end[i];
        for (int32_t slot = 0; slot < ps; ++slot) {
            int64_t pos = p0 + slot;
            if (pos >= pe) break;
            uint32_t owner = pos < shared_len ? RRS_SHARED : (uint32_t)page_agent[i];
            uint64_t key = rrs_row_key(seed, tensor, owner, (uint64_t)pos);
            uint16_t* out = pool + (page * ps + slot) * (int64_t)row;
            for (int32_t e = threadIdx.x; e < row; e += blockDim.x)
                out[e] = rrs_elem(key, (uint32_t)(e / D), (uint32_t)(e % D));
        }
    }
}

static int grid_for(int64_t n) {
    int64_t g = n < 65535 * 8 ? n : 65535 * 8;
    return (int)(g > 0 ? g : 1);
}

extern "C" int rrs_cuda_fill_rows(void* dst, const int32_t* row_agent, const int64_t* row_pos, int64_t n_rows,
                                  int32_t head0, int32_t head_count, int32_t D, uint32_t tensor, uint64_t seed,
                                  int64_t shared_len, void* stream) {
    if (n_rows <= 0) return 0;
    rrs_fill_rows_kernel<<<grid_for(n_rows), 256, 0, (cudaStream_t)stream>>>(
        (uint16_t*)dst, row_agent, row_pos, n_rows, head0, head_count, D, tensor, seed, shared_len);
    return (int)cudaGetLastError();
}

extern "C" int rrs_cuda_fill_pool(void* pool, const int32_t* page_ids, const int32_t* page_agent,
                                  const int64_t* page_pos0, const int64_t* page_pos_end, int64_t n_list, int32_t ps,
                                  int32_t Hkv, int32_t D, uint32_t tensor, uint64_t seed, int64_t shared_len,
                                  void* stream) {
    if (n_list <= 0) return 0;
    rrs_fill_pool_kernel<<<grid_for(n_list), 256, 0, (cudaStream_t)stream>>>(
        (uint16_t*)pool, page_ids, page_agent, page_pos0, page_pos_end, n_list, ps, Hkv, D, tensor, seed,
        shared_len);
    return (int)cudaGetLastError();
}
