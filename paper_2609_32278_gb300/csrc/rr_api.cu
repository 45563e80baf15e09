// rr_api.cu -- the C ABI of librr.so (include/rr.h): argument validation,
// the per-device workspace, TMA tensor-map encoding and kernel launches.
#include <cstdarg>
#include <cstdio>
#include <algorithm>
#include <climits>
#include <cstring>
#include <atomic>
#include <mutex>
#include <vector>

#include <cudaTypedefs.h>

#include "rr_internal.h"

namespace {

thread_local char g_msg[512] = "";
std::atomic<long long> g_wait_limit{0};  // 0: the default budget

int fail(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(RR_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

constexpr int kMaxDevices = 64;

struct Device {
    std::mutex mu;
    bool init = false;
    int sm_count = 0;
    int32_t* err = nullptr;  // device error word (never moves once allocated)
    void* ws = nullptr;      // schedule workspace, grown on demand
    size_t ws_bytes = 0;
};

Device g_dev[kMaxDevices];
std::mutex g_encode_mu;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Workspace layout: [n_units, lens_ok, n_split][cu: B+1][unit_off: B+1][items: max_items x int4]
// [item_slot: max_items][split units: max_split x int4][part_ml: slots x 256 float2][part_o: slots x 256 x D]
// [decode only: prefix B][suffix B]
struct Layout {
    size_t off_cu, off_unit_off, off_units, off_slot, off_split, off_ml, off_o, off_lens, off_uslot, total;
};

// rows: partial rows per slot (two Q tiles for extend, 16 for decode); unit_slots: entries of the decode
// shared-prefix call's first-slot-per-unit array.
Layout layout_for(int64_t B, int64_t max_items, int64_t max_split = 0, int64_t slots = 0, int64_t D = 0,
                  bool lens = false, int64_t rows = rr::kNQ * rr::kBM, int64_t unit_slots = 0) {
    Layout L;
    L.off_cu = 256;
    L.off_unit_off = L.off_cu + align256((size_t)(B + 1) * 4);
    L.off_units = L.off_unit_off + align256((size_t)(B + 1) * 4);
    L.off_slot = L.off_units + align256((size_t)max_items * 16);
    L.off_split = L.off_slot + align256((size_t)max_items * 4);
    L.off_ml = L.off_split + align256((size_t)max_split * 16);
    L.off_o = L.off_ml + align256((size_t)slots * rows * 8);
    L.off_lens = L.off_o + align256((size_t)slots * rows * (size_t)D * 4);
    L.off_uslot = L.off_lens + (lens ? 2 * align256((size_t)B * 4) : 0);  // decode: prefix, suffix arrays
    L.total = L.off_uslot + align256((size_t)unit_slots * 4);
    return L;
}

int current_device(Device** out, int* dev_out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(RR_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
    Device& d = g_dev[dev];
    std::lock_guard<std::mutex> lk(d.mu);
    if (!d.init) {
        e = cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        e = cudaMalloc(&d.err, 256);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(error word)");
        e = cudaMemset(d.err, 0, 256);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemset(error word)");
        d.init = true;
    }
    *out = &d;
    if (dev_out) *dev_out = dev;
    return RR_OK;
}

// Make sure the workspace holds `bytes`.  Growing frees the old buffer, which
// synchronises the device (so no kernel can still be using it).
int ensure_ws(Device& d, size_t bytes) {
    std::lock_guard<std::mutex> lk(d.mu);
    if (d.ws_bytes >= bytes) return RR_OK;
    if (d.ws) {
        cudaError_t e = cudaFree(d.ws);
        d.ws = nullptr;
        d.ws_bytes = 0;
        if (e != cudaSuccess) return cuda_fail(e, "cudaFree(workspace)");
    }
    size_t want = bytes + bytes / 4;
    cudaError_t e = cudaMalloc(&d.ws, want);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(workspace)");
    d.ws_bytes = want;
    return RR_OK;
}

int get_encoder() {
    std::lock_guard<std::mutex> lk(g_encode_mu);
    if (g_encode) return RR_OK;
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
        return fail(RR_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return RR_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3) == 0; }

int check_dims(const rr_dims* d, bool attention) {
    if (!d) return fail(RR_ERR_INVALID_ARG, "dims is null");
    if (d->batch < 0 || d->total_tokens < 0 || d->num_pages < 0 || d->max_pages < 0)
        return fail(RR_ERR_INVALID_ARG, "negative size in dims");
    if (d->num_kv_heads <= 0 || d->num_q_heads <= 0 || d->num_q_heads % d->num_kv_heads)
        return fail(RR_ERR_INVALID_ARG, "num_q_heads (%d) must be a positive multiple of num_kv_heads (%d)",
                    d->num_q_heads, d->num_kv_heads);
    if (d->head_dim != 64 && d->head_dim != 128)
        return fail(RR_ERR_UNSUPPORTED, "head_dim %d unsupported (64 or 128)", d->head_dim);
    const int ps = d->page_size;
    if (ps != 8 && ps != 16 && ps != 32 && ps != 64 && ps != 128)
        return fail(RR_ERR_UNSUPPORTED, "page_size %d unsupported (8, 16, 32, 64 or 128)", ps);
    if (attention) {
        const int G = d->num_q_heads / d->num_kv_heads;
        if (G != 1 && G != 2 && G != 4 && G != 8 && G != 16)
            return fail(RR_ERR_UNSUPPORTED, "GQA group %d unsupported (1, 2, 4, 8 or 16)", G);
    }
    if (d->total_tokens >= (1ll << 31)) return fail(RR_ERR_UNSUPPORTED, "total_tokens must be < 2^31");
    if (d->num_pages * (int64_t)ps >= (1ll << 31) - ps)
        return fail(RR_ERR_UNSUPPORTED, "num_pages * page_size must be < 2^31");
    if (d->batch > 0 && d->max_pages == 0) return fail(RR_ERR_INVALID_ARG, "max_pages is 0");
    return RR_OK;
}

int encode_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
              uint32_t box_inner, uint32_t box_rows) {
    cuuint64_t dims[2] = {inner, rows};
    cuuint64_t strides[1] = {row_stride_bytes};
    cuuint32_t box[2] = {box_inner, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(RR_ERR_CUDA, "cuTensorMapEncodeTiled (2-D) failed: %d", (int)r);
    return RR_OK;
}

int encode_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1, uint64_t s2,
              uint32_t b0, uint32_t b1, uint32_t b2) {
    cuuint64_t dims[3] = {d0, d1, d2};
    cuuint64_t strides[2] = {s1, s2};
    cuuint32_t box[3] = {b0, b1, b2};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(RR_ERR_CUDA, "cuTensorMapEncodeTiled (3-D) failed: %d", (int)r);
    return RR_OK;
}

}  // namespace

namespace rr {
long long wait_limit_cycles() {
    const long long v = g_wait_limit.load(std::memory_order_relaxed);
    return v > 0 ? v : (1ll << 33);
}
}  // namespace rr

namespace {

// Extend attention; decode attention (decode = true: kv_lens in place of the prefix / suffix lengths,
// one query token per agent, the decode kernel in place of the extend kernel); or the fused extend
// step (k_new / v_new non-null: the extend kernel first writes them into the pools, rotating K when a
// rope table is given, then attends over the pools).
int attention_impl(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                   const int32_t* prefix_lens, const int32_t* suffix_lens, const int32_t* kv_lens, void* out,
                   const rr_dims* dims, float softmax_scale, cudaStream_t stream, bool decode,
                   const void* k_new = nullptr, const void* v_new = nullptr, const float* rope = nullptr,
                   int32_t rope_max_pos = 0) {
    g_msg[0] = 0;
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (dims->total_tokens == 0 && dims->batch == 0) return RR_OK;
    const bool fused = k_new != nullptr || v_new != nullptr;
    if (rope && dims->total_tokens > 0) {
        if (!aligned16(rope)) return fail(RR_ERR_INVALID_ARG, "rope table must be 16-byte aligned");
        if (rope_max_pos <= 0) return fail(RR_ERR_INVALID_ARG, "rope_max_pos must be positive");
    }
    if (fused) {
        if (!k_new || !v_new) return fail(RR_ERR_INVALID_ARG, "the fused step needs both k_new and v_new");
        if (!aligned16(k_new) || !aligned16(v_new)) return fail(RR_ERR_INVALID_ARG, "k_new / v_new must be 16-byte aligned");
    }
    if (decode) {
        if (!page_table || !kv_lens) return fail(RR_ERR_INVALID_ARG, "null kv_lens or page table");
        if (dims->total_tokens != dims->batch)
            return fail(RR_ERR_INVALID_ARG, "decode takes one query token per agent: total_tokens (%lld) != batch (%d)",
                        (long long)dims->total_tokens, dims->batch);
        if (!aligned4(kv_lens)) return fail(RR_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
    } else if (!page_table || !prefix_lens || !suffix_lens) {
        return fail(RR_ERR_INVALID_ARG, "null lens or page table");
    }
    if (dims->total_tokens > 0 && (!q || !k_pool || !v_pool || !out))
        return fail(RR_ERR_INVALID_ARG, "null q/pool/out pointer");
    if (!aligned16(q) || !aligned16(k_pool) || !aligned16(v_pool) || !aligned16(out))
        return fail(RR_ERR_INVALID_ARG, "q, pools and out must be 16-byte aligned");
    if (!aligned4(page_table) || (!decode && (!aligned4(prefix_lens) || !aligned4(suffix_lens))))
        return fail(RR_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
    if (dims->total_tokens > 0 && dims->num_pages == 0) return fail(RR_ERR_INVALID_ARG, "empty pool");
    const int Hq = dims->num_q_heads, Hkv = dims->num_kv_heads, D = dims->head_dim, ps = dims->page_size;
    const int G = Hq / Hkv;
    const int tq = rr::kBM / G;
    const int unit_tokens = rr::kNQ * tq;
    const int64_t T = dims->total_tokens, B = dims->batch;
    const int64_t max_units = (int64_t)Hkv * (T / unit_tokens + B + 1);
    if (max_units >= (1ll << 31)) return fail(RR_ERR_UNSUPPORTED, "too many work units");

    Device* d = nullptr;
    if ((rc = current_device(&d, nullptr))) return rc;
    if ((rc = get_encoder())) return rc;
    // Split-K is possible only when the batch may have fewer than two waves of units; the batch has at
    // least Hkv * T / unit_tokens units, so larger batches never split and need no partial buffers.
    const int grid_sm = d->sm_count;
    const bool may_split = (int64_t)Hkv * (T / unit_tokens) < 2ll * grid_sm;
    // Decode is bound by HBM and an item costs little beyond its bytes, so its splits aim at 6 waves
    // (a short last wave); extend splits aim at 2 (fewer partial rows to write and merge).
    const int split_waves = decode ? 6 : 2;
    const int64_t max_split = may_split ? 2ll * grid_sm : 0;
    const int64_t slots = may_split ? (int64_t)(split_waves + 2) * grid_sm : 0;
    const int64_t max_items = std::max<int64_t>(max_units, slots);
    const int64_t rows_per_slot = decode ? 16 : rr::kNQ * rr::kBM;
    const Layout L = layout_for(B, max_items, max_split, slots, D, decode, rows_per_slot);
    if ((rc = ensure_ws(*d, L.total))) return rc;
    uint8_t* ws = static_cast<uint8_t*>(d->ws);
    cudaError_t e = cudaSuccess;
    if (decode) {  // the schedule writes the lengths in prefix / suffix form itself
        prefix_lens = reinterpret_cast<int32_t*>(ws + L.off_lens);
        suffix_lens = reinterpret_cast<int32_t*>(ws + L.off_lens + align256((size_t)B * 4));
    }

    rr::SchedArgs s{};
    s.prefix = prefix_lens;
    s.suffix = suffix_lens;
    if (decode) {
        s.kv_lens = kv_lens;
        s.prefix_out = const_cast<int32_t*>(prefix_lens);
        s.suffix_out = const_cast<int32_t*>(suffix_lens);
    }
    s.B = (int32_t)B;
    s.Hkv = Hkv;
    s.unit_tokens = unit_tokens;
    s.T = T;
    s.max_pages = dims->max_pages;
    s.ps = ps;
    s.max_units = max_units;
    s.build_units = 1;
    s.cu = reinterpret_cast<int32_t*>(ws + L.off_cu);
    s.unit_off = reinterpret_cast<int32_t*>(ws + L.off_unit_off);
    s.units = reinterpret_cast<int4*>(ws + L.off_units);
    s.item_slot = reinterpret_cast<int32_t*>(ws + L.off_slot);
    s.split_units = reinterpret_cast<int4*>(ws + L.off_split);
    s.n_split = reinterpret_cast<int32_t*>(ws) + 2;
    s.split_grid = may_split ? grid_sm : 0;
    s.split_waves = split_waves;
    s.n_units = reinterpret_cast<int32_t*>(ws);
    s.lens_ok = reinterpret_cast<int32_t*>(ws) + 1;
    if (fused) s.grid_sync = reinterpret_cast<int32_t*>(ws) + 3;
    s.err = d->err;
    e = rr::launch_sched(s, stream);
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");
    if (T == 0) return RR_OK;

    rr::AttnArgs a;
    memset(&a, 0, sizeof a);
    // q [T][Hq][D]: a box is one 64-column chunk of G heads x (128/G tokens, or the one token of decode)
    if ((rc = encode_3d(&a.tm_q, q, (uint64_t)D, (uint64_t)Hq, (uint64_t)T, (uint64_t)D * 2, (uint64_t)Hq * D * 2, 64,
                        (uint32_t)G, decode ? 1u : (uint32_t)tq)))
        return rc;
    const uint64_t rows = (uint64_t)dims->num_pages * (uint64_t)ps;
    if ((rc = encode_2d(&a.tm_k, k_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
    if ((rc = encode_2d(&a.tm_v, v_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
    a.page_table = page_table;
    a.prefix = prefix_lens;
    a.suffix = suffix_lens;
    a.cu = s.cu;
    a.units = s.units;
    a.n_units = s.n_units;
    a.item_slot = s.item_slot;
    a.part_o = reinterpret_cast<float*>(ws + L.off_o);
    a.rows_per_slot = (int32_t)rows_per_slot;
    a.part_ml = reinterpret_cast<float2*>(ws + L.off_ml);
    a.err = d->err;
    a.out = out;
    a.num_pages = dims->num_pages;
    a.Hq = Hq;
    a.G = G;
    a.ps = ps;
    a.max_pages = dims->max_pages;
    a.tq = tq;
    a.oob_row = (int32_t)rows;
    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / sqrtf((float)D);
    a.scale_log2 = scale * 1.4426950408889634f;
    a.wait_limit = rr::wait_limit_cycles();
    a.wait_hint_ns = (uint32_t)std::min<long long>(200000, std::max<long long>(1, a.wait_limit / 4));
    const int64_t grid = std::min<int64_t>((int64_t)d->sm_count, max_items);
    if (fused) {
        // k_new / v_new [T][Hkv][D]: one row of Hkv * D per suffix token
        const uint64_t row_elems = (uint64_t)Hkv * D;
        a.grid_sync = s.grid_sync;
        a.knew = static_cast<const uint4*>(k_new);
        a.vnew = static_cast<const uint4*>(v_new);
        a.kpool = static_cast<uint4*>(const_cast<void*>(k_pool));
        a.vpool = static_cast<uint4*>(const_cast<void*>(v_pool));
        a.row16 = (int32_t)(row_elems * 2 / 16);
    }
    if (rope) {
        a.rope = reinterpret_cast<const float2*>(rope);
        a.rope_max_pos = rope_max_pos;
    }
    e = decode ? rr::launch_decode_attention(a, D, (int)std::max<int64_t>(grid, 1), stream)
               : rr::launch_extend_attention(a, D, (int)std::max<int64_t>(grid, 1), stream, fused);
    if (e != cudaSuccess) return cuda_fail(e, decode ? "decode attention kernel launch" : "extend attention kernel launch");
    if (may_split) {
        rr::CombineArgs c;
        c.split_units = s.split_units;
        c.n_split = s.n_split;
        c.part_o = a.part_o;
        c.part_ml = a.part_ml;
        c.suffix = suffix_lens;
        c.cu = s.cu;
        c.out = out;
        c.Hq = Hq;
        c.G = G;
        c.D = D;
        c.tq = tq;
        c.rows = (int32_t)rows_per_slot;
        e = rr::launch_combine(c, (int)max_split, stream);
        if (e != cudaSuccess) return cuda_fail(e, "split-K combine kernel launch");
    }
    return RR_OK;
}

// Extend attention over a prefix every agent of the batch shares (rr_extend_attention_shared), as a cascade:
// the shared pass runs every suffix row of the batch against the shared keys in dense Q tiles that cross
// agents, writing fp32 partials per (token, head); the private pass runs the schedule's units over each agent's
// remaining keys and merges the partial into the output in its epilogue.
int extend_shared_impl(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                       const int32_t* prefix_lens, const int32_t* suffix_lens, int32_t shared_len, void* out,
                       const rr_dims* dims, float softmax_scale, cudaStream_t stream) {
    g_msg[0] = 0;
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (dims->total_tokens == 0 && dims->batch == 0) return RR_OK;
    if (!page_table || !prefix_lens || !suffix_lens) return fail(RR_ERR_INVALID_ARG, "null lens or page table");
    if (dims->total_tokens > 0 && (!q || !k_pool || !v_pool || !out))
        return fail(RR_ERR_INVALID_ARG, "null q/pool/out pointer");
    if (!aligned16(q) || !aligned16(k_pool) || !aligned16(v_pool) || !aligned16(out))
        return fail(RR_ERR_INVALID_ARG, "q, pools and out must be 16-byte aligned");
    if (!aligned4(page_table) || !aligned4(prefix_lens) || !aligned4(suffix_lens))
        return fail(RR_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
    if (dims->total_tokens > 0 && dims->num_pages == 0) return fail(RR_ERR_INVALID_ARG, "empty pool");
    const int Hq = dims->num_q_heads, Hkv = dims->num_kv_heads, D = dims->head_dim, ps = dims->page_size;
    if (shared_len <= 0 || shared_len % rr::kBN != 0)
        return fail(RR_ERR_UNSUPPORTED, "shared_len (%d) must be a positive multiple of %d", shared_len, rr::kBN);
    if ((int64_t)shared_len > (int64_t)dims->max_pages * ps) return fail(RR_ERR_INVALID_ARG, "shared_len exceeds max_pages");
    const int G = Hq / Hkv;
    const int tq = rr::kBM / G;
    const int unit_tokens = rr::kNQ * tq;
    const int64_t T = dims->total_tokens, B = dims->batch;
    const int64_t max_units = (int64_t)Hkv * (T / unit_tokens + B + 1);
    const int64_t shared_units = (int64_t)Hkv * ((T + unit_tokens - 1) / unit_tokens);
    if (max_units >= (1ll << 31)) return fail(RR_ERR_UNSUPPORTED, "too many work units");

    Device* d = nullptr;
    if ((rc = current_device(&d, nullptr))) return rc;
    if ((rc = get_encoder())) return rc;
    const Layout L = layout_for(B, max_units);
    const size_t off_ml = align256(L.total);
    const size_t off_o = off_ml + align256((size_t)T * Hq * 8);
    if ((rc = ensure_ws(*d, off_o + (size_t)T * Hq * (size_t)D * 4))) return rc;
    uint8_t* ws = static_cast<uint8_t*>(d->ws);

    rr::AttnArgs a;
    memset(&a, 0, sizeof a);
    if (T > 0) {
        if ((rc = encode_3d(&a.tm_q, q, (uint64_t)D, (uint64_t)Hq, (uint64_t)T, (uint64_t)D * 2, (uint64_t)Hq * D * 2,
                            64, (uint32_t)G, (uint32_t)tq)))
            return rc;
        const uint64_t rows = (uint64_t)dims->num_pages * (uint64_t)ps;
        if ((rc = encode_2d(&a.tm_k, k_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
        if ((rc = encode_2d(&a.tm_v, v_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
        a.oob_row = (int32_t)rows;
    }
    a.page_table = page_table;
    a.prefix = prefix_lens;
    a.suffix = suffix_lens;
    a.err = d->err;
    a.out = out;
    a.num_pages = dims->num_pages;
    a.Hq = Hq;
    a.G = G;
    a.ps = ps;
    a.max_pages = dims->max_pages;
    a.tq = tq;
    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / sqrtf((float)D);
    a.scale_log2 = scale * 1.4426950408889634f;
    a.wait_limit = rr::wait_limit_cycles();
    a.wait_hint_ns = (uint32_t)std::min<long long>(200000, std::max<long long>(1, a.wait_limit / 4));
    a.cas_tiles = shared_len / rr::kBN;
    a.cas_units = (int32_t)shared_units;
    a.cas_T = T;
    a.cas_ml = reinterpret_cast<float2*>(ws + off_ml);
    a.cas_o = reinterpret_cast<float*>(ws + off_o);
    cudaError_t e = cudaSuccess;
    if (T > 0) {  // the shared pass needs nothing from the schedule
        const int64_t grid = std::min<int64_t>((int64_t)d->sm_count, shared_units);
        e = rr::launch_extend_cascade(a, D, (int)std::max<int64_t>(grid, 1), stream, true);
        if (e != cudaSuccess) return cuda_fail(e, "shared-prefix pass launch");
    }

    rr::SchedArgs s{};
    s.prefix = prefix_lens;
    s.suffix = suffix_lens;
    s.B = (int32_t)B;
    s.Hkv = Hkv;
    s.unit_tokens = unit_tokens;
    s.T = T;
    s.max_pages = dims->max_pages;
    s.ps = ps;
    s.max_units = max_units;
    s.build_units = 1;
    s.cu = reinterpret_cast<int32_t*>(ws + L.off_cu);
    s.unit_off = reinterpret_cast<int32_t*>(ws + L.off_unit_off);
    s.units = reinterpret_cast<int4*>(ws + L.off_units);
    s.item_slot = reinterpret_cast<int32_t*>(ws + L.off_slot);
    s.split_units = nullptr;  // the private pass never splits a unit
    s.n_split = reinterpret_cast<int32_t*>(ws) + 2;
    s.split_grid = 0;
    s.page_table = page_table;
    s.shared_pages = shared_len / ps;  // every agent's shared pages are agent 0's (RR_ERR_SHARED)
    s.min_prefix = shared_len;         // and every agent's prefix covers them (RR_ERR_LENS)
    s.n_units = reinterpret_cast<int32_t*>(ws);
    s.lens_ok = reinterpret_cast<int32_t*>(ws) + 1;
    s.err = d->err;
    e = rr::launch_sched(s, stream);
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");
    if (T == 0) return RR_OK;
    a.cu = s.cu;
    a.units = s.units;
    a.n_units = s.n_units;
    a.item_slot = s.item_slot;
    const int64_t grid = std::min<int64_t>((int64_t)d->sm_count, max_units);
    e = rr::launch_extend_cascade(a, D, (int)std::max<int64_t>(grid, 1), stream, false);
    if (e != cudaSuccess) return cuda_fail(e, "private-key pass launch");
    return RR_OK;
}

// Decode over a prefix every agent of the batch shares (rr_decode_attention_shared): the shared prefix's
// pages are read once per group of 16 / G agents (their queries fill the MMA's 16 columns) instead of once
// per agent, each agent's private keys by the plain decode kernel, and both partial results are merged.
int decode_shared_impl(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                       const int32_t* kv_lens, int32_t shared_len, void* out, const rr_dims* dims,
                       float softmax_scale, cudaStream_t stream) {
    g_msg[0] = 0;
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (dims->batch == 0) return RR_OK;
    if (!page_table || !kv_lens) return fail(RR_ERR_INVALID_ARG, "null kv_lens or page table");
    if (dims->total_tokens != dims->batch)
        return fail(RR_ERR_INVALID_ARG, "decode takes one query token per agent: total_tokens (%lld) != batch (%d)",
                    (long long)dims->total_tokens, dims->batch);
    if (!q || !k_pool || !v_pool || !out) return fail(RR_ERR_INVALID_ARG, "null q/pool/out pointer");
    if (!aligned16(q) || !aligned16(k_pool) || !aligned16(v_pool) || !aligned16(out))
        return fail(RR_ERR_INVALID_ARG, "q, pools and out must be 16-byte aligned");
    if (!aligned4(page_table) || !aligned4(kv_lens)) return fail(RR_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
    if (dims->num_pages == 0) return fail(RR_ERR_INVALID_ARG, "empty pool");
    const int Hq = dims->num_q_heads, Hkv = dims->num_kv_heads, D = dims->head_dim, ps = dims->page_size;
    const int G = Hq / Hkv;
    const int64_t B = dims->batch;
    if (shared_len <= 0 || shared_len % rr::kBN != 0)
        return fail(RR_ERR_UNSUPPORTED, "shared_len (%d) must be a positive multiple of %d", shared_len, rr::kBN);
    if ((int64_t)shared_len > (int64_t)dims->max_pages * ps) return fail(RR_ERR_INVALID_ARG, "shared_len exceeds max_pages");
    // the schedule gives each thread of one block one (agent, KV head) unit: larger batches take the plain call
    if (B * Hkv > 1024)
        return attention_impl(q, k_pool, v_pool, page_table, nullptr, nullptr, kv_lens, out, dims, softmax_scale, stream,
                              true);

    Device* d = nullptr;
    if ((rc = current_device(&d, nullptr))) return rc;
    if ((rc = get_encoder())) return rc;
    const int grid_sm = d->sm_count;
    const int tq = rr::kBM / G;
    const int unit_tokens = rr::kNQ * tq;
    const int64_t units = B * Hkv;
    // shared-prefix items: one KV head x group_agents agents x one of group_ns pieces of the shared tiles;
    // enough pieces for two waves, but none shorter than 8 tiles (a piece's fixed cost would dominate)
    const int group_agents = 16 / G;
    const int64_t groups_per_head = (B + group_agents - 1) / group_agents;
    const int shared_tiles = shared_len / rr::kBN;
    const int64_t groups = groups_per_head * Hkv;
    const int group_ns = (int)std::max<int64_t>(
        1, std::min<int64_t>(std::min(64, std::max(1, shared_tiles / 8)), (2ll * grid_sm + groups - 1) / groups));
    const int split_waves = 6;
    // slots: every unit's group_ns shared pieces plus its private pieces (1 each, or a split into at most
    // (waves + 2) x grid pieces over all units)
    const int64_t slots = units * group_ns + std::max<int64_t>(units, (int64_t)(split_waves + 2) * grid_sm);
    const int64_t max_items = std::max<int64_t>(units, (int64_t)(split_waves + 2) * grid_sm);
    const Layout L = layout_for(B, max_items, units, slots, D, true, 16, units);
    if ((rc = ensure_ws(*d, L.total))) return rc;
    uint8_t* ws = static_cast<uint8_t*>(d->ws);
    int32_t* prefix_lens = reinterpret_cast<int32_t*>(ws + L.off_lens);
    int32_t* suffix_lens = reinterpret_cast<int32_t*>(ws + L.off_lens + align256((size_t)B * 4));
    int32_t* unit_slot = reinterpret_cast<int32_t*>(ws + L.off_uslot);

    rr::SchedArgs s{};
    s.kv_lens = kv_lens;
    s.prefix_out = prefix_lens;
    s.suffix_out = suffix_lens;
    s.prefix = prefix_lens;
    s.suffix = suffix_lens;
    s.lens_offset = shared_len;
    s.extra_slots = group_ns;
    s.unit_slot = unit_slot;
    s.page_table = page_table;
    s.shared_pages = shared_len / ps;
    s.B = (int32_t)B;
    s.Hkv = Hkv;
    s.unit_tokens = unit_tokens;
    s.T = B;
    s.max_pages = dims->max_pages;
    s.ps = ps;
    s.max_units = units;
    s.build_units = 1;
    s.cu = reinterpret_cast<int32_t*>(ws + L.off_cu);
    s.unit_off = reinterpret_cast<int32_t*>(ws + L.off_unit_off);
    s.units = reinterpret_cast<int4*>(ws + L.off_units);
    s.item_slot = reinterpret_cast<int32_t*>(ws + L.off_slot);
    s.split_units = reinterpret_cast<int4*>(ws + L.off_split);
    s.n_split = reinterpret_cast<int32_t*>(ws) + 2;
    s.split_grid = grid_sm;
    s.split_waves = split_waves;
    s.n_units = reinterpret_cast<int32_t*>(ws);
    s.lens_ok = reinterpret_cast<int32_t*>(ws) + 1;
    s.err = d->err;
    cudaError_t e = rr::launch_sched(s, stream);
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");

    rr::AttnArgs a;
    memset(&a, 0, sizeof a);
    if ((rc = encode_3d(&a.tm_q, q, (uint64_t)D, (uint64_t)Hq, (uint64_t)B, (uint64_t)D * 2, (uint64_t)Hq * D * 2, 64,
                        (uint32_t)G, 1u)))
        return rc;
    if ((rc = encode_3d(&a.tm_qg, q, (uint64_t)D, (uint64_t)Hq, (uint64_t)B, (uint64_t)D * 2, (uint64_t)Hq * D * 2, 64,
                        (uint32_t)G, (uint32_t)group_agents)))
        return rc;
    const uint64_t rows = (uint64_t)dims->num_pages * (uint64_t)ps;
    if ((rc = encode_2d(&a.tm_k, k_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
    if ((rc = encode_2d(&a.tm_v, v_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
    a.page_table = page_table;
    a.prefix = prefix_lens;
    a.suffix = suffix_lens;
    a.cu = s.cu;
    a.units = s.units;
    a.n_units = s.n_units;
    a.item_slot = s.item_slot;
    a.part_o = reinterpret_cast<float*>(ws + L.off_o);
    a.part_ml = reinterpret_cast<float2*>(ws + L.off_ml);
    a.rows_per_slot = 16;
    a.err = d->err;
    a.out = out;
    a.num_pages = dims->num_pages;
    a.Hq = Hq;
    a.G = G;
    a.ps = ps;
    a.max_pages = dims->max_pages;
    a.tq = tq;
    a.oob_row = (int32_t)rows;
    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / sqrtf((float)D);
    a.scale_log2 = scale * 1.4426950408889634f;
    a.wait_limit = rr::wait_limit_cycles();
    a.wait_hint_ns = (uint32_t)std::min<long long>(200000, std::max<long long>(1, a.wait_limit / 4));
    a.unit_slot = unit_slot;
    a.batch = (int32_t)B;
    // 1. the shared prefix, once per group of agents
    a.group_items = (int32_t)(groups * group_ns);
    a.group_ns = group_ns;
    a.group_agents = group_agents;
    a.groups_per_head = (int32_t)groups_per_head;
    a.shared_tiles = shared_tiles;
    e = rr::launch_decode_shared_prefix(a, D, (int)std::min<int64_t>(grid_sm, groups * group_ns), stream);
    if (e != cudaSuccess) return cuda_fail(e, "shared-prefix decode kernel launch");
    // 2. every agent's private keys, from page-table column shared_len / ps on
    a.page0 = shared_len / ps;
    e = rr::launch_decode_attention(a, D, (int)std::min<int64_t>(grid_sm, max_items), stream);
    if (e != cudaSuccess) return cuda_fail(e, "decode attention kernel launch");
    // 3. merge each (agent, query head)'s shared and private pieces
    rr::CombineArgs c;
    c.split_units = s.split_units;
    c.n_split = s.n_split;
    c.part_o = a.part_o;
    c.part_ml = a.part_ml;
    c.suffix = suffix_lens;
    c.cu = s.cu;
    c.out = out;
    c.Hq = Hq;
    c.G = G;
    c.D = D;
    c.tq = tq;
    c.rows = 16;
    e = rr::launch_combine(c, (int)std::min<int64_t>(units, 2ll * grid_sm), stream);
    if (e != cudaSuccess) return cuda_fail(e, "split-K combine kernel launch");
    return RR_OK;
}

}  // namespace

extern "C" {

const char* rr_version(void) { return "rr-extend 0.1 (sm_103a)"; }

const char* rr_last_error(void) { return g_msg; }

void rr_set_wait_limit(long long cycles) { g_wait_limit.store(cycles > 0 ? cycles : 0, std::memory_order_relaxed); }

}  // extern "C"

namespace {

int append_impl(const void* k_new, const void* v_new, void* k_pool, void* v_pool, const int32_t* page_table,
                const int32_t* prefix_lens, const int32_t* suffix_lens, const rr_dims* dims, cudaStream_t stream,
                const float* rope, int32_t rope_max_pos) {
    g_msg[0] = 0;
    int rc = check_dims(dims, false);
    if (rc) return rc;
    if (dims->total_tokens == 0 && dims->batch == 0) return RR_OK;
    if (rope && dims->total_tokens > 0) {
        if (!aligned16(rope)) return fail(RR_ERR_INVALID_ARG, "rope table must be 16-byte aligned");
        if (rope_max_pos <= 0) return fail(RR_ERR_INVALID_ARG, "rope_max_pos must be positive");
    }
    if (!page_table || !prefix_lens || !suffix_lens) return fail(RR_ERR_INVALID_ARG, "null lens or page table");
    if (dims->total_tokens > 0 && (!k_new || !v_new || !k_pool || !v_pool))
        return fail(RR_ERR_INVALID_ARG, "null K/V pointer");
    if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(k_pool) || !aligned16(v_pool))
        return fail(RR_ERR_INVALID_ARG, "K/V pointers must be 16-byte aligned");
    if (!aligned4(page_table) || !aligned4(prefix_lens) || !aligned4(suffix_lens))
        return fail(RR_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
    Device* d = nullptr;
    if ((rc = current_device(&d, nullptr))) return rc;
    rr::AppendArgs a{};
    a.k_new = static_cast<const uint4*>(k_new);
    a.v_new = static_cast<const uint4*>(v_new);
    a.k_pool = static_cast<uint4*>(k_pool);
    a.v_pool = static_cast<uint4*>(v_pool);
    a.page_table = page_table;
    a.prefix = prefix_lens;
    a.suffix = suffix_lens;
    a.err = d->err;
    a.T = dims->total_tokens;
    a.num_pages = dims->num_pages;
    a.B = dims->batch;
    a.max_pages = dims->max_pages;
    a.ps = dims->page_size;
    a.row16 = dims->num_kv_heads * dims->head_dim * 2 / 16;
    if (rope) {
        a.rope = reinterpret_cast<const float2*>(rope);
        a.rope_max_pos = rope_max_pos;
        a.hkv = dims->num_kv_heads;
        a.d16 = dims->head_dim / 16;
    }
    cudaError_t e = cudaSuccess;
    if (dims->batch <= rr::kAppendSelfLensMaxB) {  // one kernel: it checks and sums the lengths itself
        a.self_lens = 1;
        e = rr::launch_kv_append(a, d->sm_count, stream);
        if (e != cudaSuccess) return cuda_fail(e, "kv_append kernel launch");
        return RR_OK;
    }
    const Layout L = layout_for(dims->batch, 0);
    if ((rc = ensure_ws(*d, L.total))) return rc;
    uint8_t* ws = static_cast<uint8_t*>(d->ws);

    rr::SchedArgs s{};
    s.prefix = prefix_lens;
    s.suffix = suffix_lens;
    s.B = dims->batch;
    s.Hkv = dims->num_kv_heads;
    s.unit_tokens = 1;
    s.T = dims->total_tokens;
    s.max_pages = dims->max_pages;
    s.ps = dims->page_size;
    s.max_units = 0;
    s.build_units = 0;
    s.cu = reinterpret_cast<int32_t*>(ws + L.off_cu);
    s.unit_off = reinterpret_cast<int32_t*>(ws + L.off_unit_off);
    s.units = nullptr;
    s.item_slot = nullptr;
    s.split_units = nullptr;
    s.n_split = reinterpret_cast<int32_t*>(ws) + 2;
    s.split_grid = 0;
    s.n_units = reinterpret_cast<int32_t*>(ws);
    s.lens_ok = reinterpret_cast<int32_t*>(ws) + 1;
    s.err = d->err;
    e = rr::launch_sched(s, stream);
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");
    if (dims->total_tokens == 0) return RR_OK;

    a.cu = s.cu;
    a.lens_ok = s.lens_ok;
    e = rr::launch_kv_append(a, d->sm_count, stream);
    if (e != cudaSuccess) return cuda_fail(e, "kv_append kernel launch");
    return RR_OK;
}

}  // namespace

extern "C" {

int rr_kv_append(const void* k_new, const void* v_new, void* k_pool, void* v_pool, const int32_t* page_table,
                 const int32_t* prefix_lens, const int32_t* suffix_lens, const rr_dims* dims, cudaStream_t stream) {
    return append_impl(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, dims, stream, nullptr, 0);
}

int rr_rope_table(float* table, int32_t max_pos, int32_t head_dim, double base, cudaStream_t stream) {
    g_msg[0] = 0;
    if (max_pos < 0) return fail(RR_ERR_INVALID_ARG, "max_pos must be >= 0");
    if (head_dim != 64 && head_dim != 128) return fail(RR_ERR_UNSUPPORTED, "head_dim %d unsupported (64 or 128)", head_dim);
    if (!(base > 1.0)) return fail(RR_ERR_INVALID_ARG, "base must be > 1");
    if (max_pos == 0) return RR_OK;
    if (!table || !aligned16(table)) return fail(RR_ERR_INVALID_ARG, "table must be a 16-byte aligned device pointer");
    Device* d = nullptr;
    int rc = current_device(&d, nullptr);
    if (rc) return rc;
    cudaError_t e = rr::launch_rope_table(reinterpret_cast<float2*>(table), max_pos, head_dim, base, d->sm_count, stream);
    if (e != cudaSuccess) return cuda_fail(e, "rope table kernel launch");
    return RR_OK;
}

int rr_kv_append_rope(const void* k_new, const void* v_new, void* k_pool, void* v_pool, const int32_t* page_table,
                      const int32_t* prefix_lens, const int32_t* suffix_lens, const rr_dims* dims,
                      const float* rope_table, int32_t rope_max_pos, cudaStream_t stream) {
    if (!rope_table) return fail(RR_ERR_INVALID_ARG, "null rope table");
    return append_impl(k_new, v_new, k_pool, v_pool, page_table, prefix_lens, suffix_lens, dims, stream, rope_table,
                       rope_max_pos);
}

int rr_extend_attention_rope(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                             const int32_t* prefix_lens, const int32_t* suffix_lens, void* out, const rr_dims* dims,
                             float softmax_scale, const float* rope_table, int32_t rope_max_pos,
                             cudaStream_t stream) {
    if (!rope_table) return fail(RR_ERR_INVALID_ARG, "null rope table");
    return attention_impl(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, nullptr, out, dims, softmax_scale,
                          stream, false, nullptr, nullptr, rope_table, rope_max_pos);
}

int rr_extend_step_rope(const void* q, const void* k_new, const void* v_new, void* k_pool, void* v_pool,
                        const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens, void* out,
                        const rr_dims* dims, float softmax_scale, const float* rope_table, int32_t rope_max_pos,
                        cudaStream_t stream) {
    if (!rope_table) return fail(RR_ERR_INVALID_ARG, "null rope table");
    const bool any = dims && dims->total_tokens > 0;
    if (any && (!k_new || !v_new)) return fail(RR_ERR_INVALID_ARG, "null k_new / v_new");
    return attention_impl(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, nullptr, out, dims, softmax_scale,
                          stream, false, any ? k_new : nullptr, any ? v_new : nullptr, rope_table, rope_max_pos);
}

int rr_extend_attention(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                        const int32_t* prefix_lens, const int32_t* suffix_lens, void* out, const rr_dims* dims,
                        float softmax_scale, cudaStream_t stream) {
    return attention_impl(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, nullptr, out, dims, softmax_scale,
                          stream, false);
}

int rr_decode_attention(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                        const int32_t* kv_lens, void* out, const rr_dims* dims, float softmax_scale,
                        cudaStream_t stream) {
    return attention_impl(q, k_pool, v_pool, page_table, nullptr, nullptr, kv_lens, out, dims, softmax_scale, stream,
                          true);
}

int rr_decode_attention_shared(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                               const int32_t* kv_lens, int32_t shared_len, void* out, const rr_dims* dims,
                               float softmax_scale, cudaStream_t stream) {
    return decode_shared_impl(q, k_pool, v_pool, page_table, kv_lens, shared_len, out, dims, softmax_scale, stream);
}

int rr_extend_attention_shared(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                               const int32_t* prefix_lens, const int32_t* suffix_lens, int32_t shared_len, void* out,
                               const rr_dims* dims, float softmax_scale, cudaStream_t stream) {
    return extend_shared_impl(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, shared_len, out, dims,
                              softmax_scale, stream);
}

int rr_decode_attention_rope(const void* q, const void* k_pool, const void* v_pool, const int32_t* page_table,
                             const int32_t* kv_lens, void* out, const rr_dims* dims, float softmax_scale,
                             const float* rope_table, int32_t rope_max_pos, cudaStream_t stream) {
    if (!rope_table) return fail(RR_ERR_INVALID_ARG, "null rope table");
    return attention_impl(q, k_pool, v_pool, page_table, nullptr, nullptr, kv_lens, out, dims, softmax_scale, stream,
                          true, nullptr, nullptr, rope_table, rope_max_pos);
}

int rr_extend_step(const void* q, const void* k_new, const void* v_new, void* k_pool, void* v_pool,
                   const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens, void* out,
                   const rr_dims* dims, float softmax_scale, cudaStream_t stream) {
    if (dims && dims->total_tokens > 0 && (!k_new || !v_new))
        return fail(RR_ERR_INVALID_ARG, "null k_new / v_new");
    return attention_impl(q, k_pool, v_pool, page_table, prefix_lens, suffix_lens, nullptr, out, dims, softmax_scale,
                          stream, false, dims && dims->total_tokens > 0 ? k_new : nullptr,
                          dims && dims->total_tokens > 0 ? v_new : nullptr);
}

int rr_validate_page_table(const int32_t* page_table, const int32_t* prefix_lens, const int32_t* suffix_lens,
                           const rr_dims* dims) {
    g_msg[0] = 0;
    if (!dims) return fail(RR_ERR_INVALID_ARG, "dims is null");
    if (dims->batch > 0 && (!page_table || !prefix_lens || !suffix_lens))
        return fail(RR_ERR_INVALID_ARG, "null host array");
    const int64_t ps = dims->page_size, np = dims->num_pages;
    if (ps <= 0 || np < 0 || dims->max_pages < 0) return fail(RR_ERR_INVALID_ARG, "bad dims");
    int64_t T = 0;
    // owner[p]: -1 unused, else (agent << 1) | (page holds suffix positions)
    std::vector<int64_t> owner((size_t)np, -1);
    std::vector<uint8_t> shared_read((size_t)np, 0);
    for (int32_t b = 0; b < dims->batch; ++b) {
        const int64_t P = prefix_lens[b], S = suffix_lens[b];
        if (P < 0 || S < 0 || P + S > (int64_t)dims->max_pages * ps)
            return fail(RR_ERR_LENS, "agent %d: bad lengths (prefix %lld, suffix %lld)", b, (long long)P,
                        (long long)S);
        T += S;
        const int64_t n = (P + S + ps - 1) / ps;
        for (int64_t i = 0; i < n; ++i) {
            const int64_t p = page_table[(int64_t)b * dims->max_pages + i];
            if (p < 0 || p >= np) return fail(RR_ERR_OOB, "agent %d: page %lld of logical page %lld outside the pool",
                                              b, (long long)p, (long long)i);
            const bool writes = (i + 1) * ps > P && S > 0;  // holds at least one suffix position
            if (writes) {
                if (owner[(size_t)p] != -1 || shared_read[(size_t)p])
                    return fail(RR_ERR_OVERLAP, "agent %d: suffix page %lld is also used elsewhere", b, (long long)p);
                owner[(size_t)p] = ((int64_t)b << 1) | 1;
            } else {
                if (owner[(size_t)p] != -1 && (owner[(size_t)p] & 1))
                    return fail(RR_ERR_OVERLAP, "agent %d: prefix page %lld is another agent's suffix page", b,
                                (long long)p);
                shared_read[(size_t)p] = 1;
            }
        }
    }
    if (T != dims->total_tokens)
        return fail(RR_ERR_LENS, "sum of suffix lengths %lld != total_tokens %lld", (long long)T,
                    (long long)dims->total_tokens);
    return RR_OK;
}

int rr_get_device_error(cudaStream_t stream) {
    Device* d = nullptr;
    int rc = current_device(&d, nullptr);
    if (rc) return rc;
    cudaError_t e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int32_t v = 0;
    e = cudaMemcpy(&v, d->err, sizeof v, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy(error word)");
    e = cudaMemset(d->err, 0, sizeof v);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemset(error word)");
    return v;
}

void rr_shutdown(void) {
    for (int i = 0; i < kMaxDevices; ++i) {
        Device& d = g_dev[i];
        std::lock_guard<std::mutex> lk(d.mu);
        if (!d.init) continue;
        int prev = 0;
        cudaGetDevice(&prev);
        cudaSetDevice(i);
        if (d.ws) cudaFree(d.ws);
        if (d.err) cudaFree(d.err);
        d.ws = nullptr;
        d.err = nullptr;
        d.ws_bytes = 0;
        d.init = false;
        cudaSetDevice(prev);
    }
}

}  // extern "C"

// ---------------------------------------------------------------------------
// rr_extend_attention_noalloc: the same extend attention, with its schedule
// scratch in a fixed static device array instead of the growable workspace.
//
// For callers that must not allocate device memory during a call: code that
// runs inside a memory-budgeted serving loop or a custom allocator that owns
// every device byte, or that cannot tolerate the implicit device
// synchronisation of cudaMalloc/cudaFree.  The array below is part of the
// library image: every GPU that loads librr.so holds it until process exit.
namespace {

constexpr int32_t kNoAllocMaxBatch = 4096;    // agents per call
constexpr int64_t kNoAllocMaxUnits = 65536;   // schedule work units per call
constexpr size_t kNoAllocOffCu = 256;         // [0] n_units, [1] lens_ok, [2] spare error word, [3] n_split
constexpr size_t kNoAllocOffUnitOff = kNoAllocOffCu + ((size_t)(kNoAllocMaxBatch + 1) * 4 + 255) / 256 * 256;
constexpr size_t kNoAllocOffUnits = kNoAllocOffUnitOff + ((size_t)(kNoAllocMaxBatch + 1) * 4 + 255) / 256 * 256;
constexpr size_t kNoAllocOffSlot = kNoAllocOffUnits + (size_t)kNoAllocMaxUnits * 16;
constexpr size_t kNoAllocBytes = kNoAllocOffSlot + (size_t)kNoAllocMaxUnits * 4;
static_assert(kNoAllocBytes == 1344256, "the static scratch size stated in rr.h (1,344,256 bytes, ~1.28 MiB)");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

struct NoAllocDevice {
    std::mutex mu;
    bool ready = false;
    void* scratch = nullptr;  // device address of g_noalloc_scratch on this device
    int sm_count = 0;
};
NoAllocDevice g_noalloc[kMaxDevices];

// One-time set-up per device, with that device current: the device address of
// the static array (its host-side name is only a stand-in) and the SM count.
int noalloc_setup(void** scratch, int* sm_count) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(RR_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
    NoAllocDevice& d = g_noalloc[dev];
    std::lock_guard<std::mutex> lk(d.mu);
    if (!d.ready) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) return cuda_fail(e, "cudaGetSymbolAddress(static scratch)");
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        d.scratch = p;
        d.sm_count = sms;
        d.ready = true;
    }
    *scratch = d.scratch;
    *sm_count = d.sm_count;
    return RR_OK;
}

}  // namespace

extern "C" int rr_extend_attention_noalloc(const void* q, const void* k_pool, const void* v_pool,
                                           const int32_t* page_table, const int32_t* prefix_lens,
                                           const int32_t* suffix_lens, void* out, const rr_dims* dims,
                                           float softmax_scale, int32_t* device_error, cudaStream_t stream) {
    g_msg[0] = 0;
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (dims->total_tokens == 0 && dims->batch == 0) return RR_OK;
    if (!page_table || !prefix_lens || !suffix_lens) return fail(RR_ERR_INVALID_ARG, "null lens or page table");
    if (dims->total_tokens > 0 && (!q || !k_pool || !v_pool || !out))
        return fail(RR_ERR_INVALID_ARG, "null q/pool/out pointer");
    if (!aligned16(q) || !aligned16(k_pool) || !aligned16(v_pool) || !aligned16(out))
        return fail(RR_ERR_INVALID_ARG, "q, pools and out must be 16-byte aligned");
    if (!aligned4(page_table) || !aligned4(prefix_lens) || !aligned4(suffix_lens) || !aligned4(device_error))
        return fail(RR_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
    if (dims->total_tokens > 0 && dims->num_pages == 0) return fail(RR_ERR_INVALID_ARG, "empty pool");
    const int Hq = dims->num_q_heads, Hkv = dims->num_kv_heads, D = dims->head_dim, ps = dims->page_size;
    const int G = Hq / Hkv;
    const int tq = rr::kBM / G;
    const int unit_tokens = rr::kNQ * tq;
    const int64_t T = dims->total_tokens, B = dims->batch;
    const int64_t max_units = (int64_t)Hkv * (T / unit_tokens + B + 1);
    if (B > kNoAllocMaxBatch)
        return fail(RR_ERR_UNSUPPORTED, "batch %lld exceeds the static scratch limit of %d agents", (long long)B,
                    kNoAllocMaxBatch);
    if (max_units > kNoAllocMaxUnits)
        return fail(RR_ERR_UNSUPPORTED,
                    "batch needs up to %lld work units; the static scratch holds %lld (fewer suffix tokens per call)",
                    (long long)max_units, (long long)kNoAllocMaxUnits);

    void* scratch = nullptr;
    int sm_count = 0;
    if ((rc = noalloc_setup(&scratch, &sm_count))) return rc;
    if ((rc = get_encoder())) return rc;
    uint8_t* ws = static_cast<uint8_t*>(scratch);
    int32_t* err = device_error ? device_error : reinterpret_cast<int32_t*>(ws) + 2;

    rr::SchedArgs s{};
    s.prefix = prefix_lens;
    s.suffix = suffix_lens;
    s.B = (int32_t)B;
    s.Hkv = Hkv;
    s.unit_tokens = unit_tokens;
    s.T = T;
    s.max_pages = dims->max_pages;
    s.ps = ps;
    s.max_units = max_units;
    s.build_units = 1;
    s.cu = reinterpret_cast<int32_t*>(ws + kNoAllocOffCu);
    s.unit_off = reinterpret_cast<int32_t*>(ws + kNoAllocOffUnitOff);
    s.units = reinterpret_cast<int4*>(ws + kNoAllocOffUnits);
    s.item_slot = reinterpret_cast<int32_t*>(ws + kNoAllocOffSlot);
    s.split_units = nullptr;                       // no split-K: the partial buffers would not fit
    s.n_split = reinterpret_cast<int32_t*>(ws) + 3;
    s.split_grid = 0;
    s.n_units = reinterpret_cast<int32_t*>(ws);
    s.lens_ok = reinterpret_cast<int32_t*>(ws) + 1;
    s.err = err;
    cudaError_t e = rr::launch_sched(s, stream);
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");
    if (T == 0) return RR_OK;

    rr::AttnArgs a;
    memset(&a, 0, sizeof a);
    if ((rc = encode_3d(&a.tm_q, q, (uint64_t)D, (uint64_t)Hq, (uint64_t)T, (uint64_t)D * 2, (uint64_t)Hq * D * 2, 64,
                        (uint32_t)G, (uint32_t)tq)))
        return rc;
    const uint64_t rows = (uint64_t)dims->num_pages * (uint64_t)ps;
    if ((rc = encode_2d(&a.tm_k, k_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
    if ((rc = encode_2d(&a.tm_v, v_pool, (uint64_t)Hkv * D, rows, (uint64_t)Hkv * D * 2, 64, (uint32_t)ps))) return rc;
    a.page_table = page_table;
    a.prefix = prefix_lens;
    a.suffix = suffix_lens;
    a.cu = s.cu;
    a.units = s.units;
    a.n_units = s.n_units;
    a.item_slot = s.item_slot;
    a.part_o = nullptr;
    a.part_ml = nullptr;
    a.err = err;
    a.out = out;
    a.num_pages = dims->num_pages;
    a.Hq = Hq;
    a.G = G;
    a.ps = ps;
    a.max_pages = dims->max_pages;
    a.tq = tq;
    a.oob_row = (int32_t)rows;
    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / sqrtf((float)D);
    a.scale_log2 = scale * 1.4426950408889634f;
    a.wait_limit = rr::wait_limit_cycles();
    a.wait_hint_ns = (uint32_t)std::min<long long>(200000, std::max<long long>(1, a.wait_limit / 4));
    const int64_t grid = std::min<int64_t>((int64_t)sm_count, max_units);
    e = rr::launch_extend_attention(a, D, (int)std::max<int64_t>(grid, 1), stream);
    if (e != cudaSuccess) return cuda_fail(e, "extend attention kernel launch");
    return RR_OK;
}

// ---------------------------------------------------------------------------
// rr_tensor forms of the extend step's two calls: check every argument's rank, element type, shape and
// strides on the host, derive rr_dims from the shapes and forward to the plain call.
namespace {

const char* dtype_name(int32_t d) {
    return d == RR_DTYPE_BF16 ? "bf16" : d == RR_DTYPE_I32 ? "int32" : "unknown";
}

int check_tensor(const rr_tensor* t, const char* name, int ndim, int32_t dtype) {
    if (!t) return fail(RR_ERR_INVALID_ARG, "%s: null rr_tensor", name);
    if (t->ndim != ndim) return fail(RR_ERR_INVALID_ARG, "%s: %d dimensions, expected %d", name, t->ndim, ndim);
    if (t->dtype != dtype)
        return fail(RR_ERR_UNSUPPORTED, "%s: dtype %d (%s), expected %s", name, t->dtype, dtype_name(t->dtype),
                    dtype_name(dtype));
    int64_t n = 1;
    for (int i = 0; i < ndim; ++i) {
        if (t->shape[i] < 0) return fail(RR_ERR_INVALID_ARG, "%s: negative extent %lld in dimension %d", name,
                                         (long long)t->shape[i], i);
        n *= t->shape[i];
    }
    if (n == 0) return RR_OK;  // an empty tensor has no layout to check
    if (!t->data) return fail(RR_ERR_INVALID_ARG, "%s: null data pointer", name);
    int64_t expect = 1;
    for (int i = ndim - 1; i >= 0; --i) {
        if (t->shape[i] != 1 && t->stride[i] != expect)
            return fail(RR_ERR_UNSUPPORTED, "%s: stride %lld in dimension %d, expected %lld (row-major contiguous)",
                        name, (long long)t->stride[i], i, (long long)expect);
        expect *= t->shape[i];
    }
    return RR_OK;
}

int same_dim(const rr_tensor* a, int ia, const char* na, const rr_tensor* b, int ib, const char* nb) {
    if (a->shape[ia] != b->shape[ib])
        return fail(RR_ERR_INVALID_ARG, "%s dimension %d (%lld) differs from %s dimension %d (%lld)", na, ia,
                    (long long)a->shape[ia], nb, ib, (long long)b->shape[ib]);
    return RR_OK;
}

int fits_i32(int64_t x, const char* what) {
    if (x > INT32_MAX) return fail(RR_ERR_INVALID_ARG, "%s %lld exceeds int32", what, (long long)x);
    return RR_OK;
}

// Shared checks of the pools, page table and lengths; fills every field of d except num_q_heads and
// total_tokens.
int check_pool_args(const rr_tensor* k_pool, const rr_tensor* v_pool, const rr_tensor* page_table,
                    const rr_tensor* prefix_lens, const rr_tensor* suffix_lens, rr_dims* d) {
    int rc;
    if ((rc = check_tensor(k_pool, "k_pool", 4, RR_DTYPE_BF16))) return rc;
    if ((rc = check_tensor(v_pool, "v_pool", 4, RR_DTYPE_BF16))) return rc;
    for (int i = 0; i < 4; ++i)
        if ((rc = same_dim(k_pool, i, "k_pool", v_pool, i, "v_pool"))) return rc;
    if ((rc = check_tensor(page_table, "page_table", 2, RR_DTYPE_I32))) return rc;
    if ((rc = check_tensor(prefix_lens, "prefix_lens", 1, RR_DTYPE_I32))) return rc;
    if ((rc = check_tensor(suffix_lens, "suffix_lens", 1, RR_DTYPE_I32))) return rc;
    if ((rc = same_dim(prefix_lens, 0, "prefix_lens", page_table, 0, "page_table"))) return rc;
    if ((rc = same_dim(suffix_lens, 0, "suffix_lens", page_table, 0, "page_table"))) return rc;
    if ((rc = fits_i32(page_table->shape[0], "batch"))) return rc;
    if ((rc = fits_i32(page_table->shape[1], "max_pages"))) return rc;
    if ((rc = fits_i32(k_pool->shape[1], "page_size"))) return rc;
    if ((rc = fits_i32(k_pool->shape[2], "num_kv_heads"))) return rc;
    if ((rc = fits_i32(k_pool->shape[3], "head_dim"))) return rc;
    d->batch = (int32_t)page_table->shape[0];
    d->max_pages = (int32_t)page_table->shape[1];
    d->num_pages = k_pool->shape[0];
    d->page_size = (int32_t)k_pool->shape[1];
    d->num_kv_heads = (int32_t)k_pool->shape[2];
    d->head_dim = (int32_t)k_pool->shape[3];
    return RR_OK;
}

}  // namespace

extern "C" int rr_kv_append_tensors(const rr_tensor* k_new, const rr_tensor* v_new, const rr_tensor* k_pool,
                                    const rr_tensor* v_pool, const rr_tensor* page_table,
                                    const rr_tensor* prefix_lens, const rr_tensor* suffix_lens,
                                    cudaStream_t stream) {
    g_msg[0] = 0;
    rr_dims d{};
    int rc;
    if ((rc = check_pool_args(k_pool, v_pool, page_table, prefix_lens, suffix_lens, &d))) return rc;
    if ((rc = check_tensor(k_new, "k_new", 3, RR_DTYPE_BF16))) return rc;
    if ((rc = check_tensor(v_new, "v_new", 3, RR_DTYPE_BF16))) return rc;
    for (int i = 0; i < 3; ++i)
        if ((rc = same_dim(k_new, i, "k_new", v_new, i, "v_new"))) return rc;
    if ((rc = same_dim(k_new, 1, "k_new", k_pool, 2, "k_pool"))) return rc;
    if ((rc = same_dim(k_new, 2, "k_new", k_pool, 3, "k_pool"))) return rc;
    d.num_q_heads = d.num_kv_heads;  // no queries in the append; any multiple of Hkv passes the dims check
    d.total_tokens = k_new->shape[0];
    return rr_kv_append(k_new->data, v_new->data, k_pool->data, v_pool->data,
                        static_cast<const int32_t*>(page_table->data), static_cast<const int32_t*>(prefix_lens->data),
                        static_cast<const int32_t*>(suffix_lens->data), &d, stream);
}

extern "C" int rr_extend_attention_tensors(const rr_tensor* q, const rr_tensor* k_pool, const rr_tensor* v_pool,
                                           const rr_tensor* page_table, const rr_tensor* prefix_lens,
                                           const rr_tensor* suffix_lens, const rr_tensor* out, float softmax_scale,
                                           cudaStream_t stream) {
    g_msg[0] = 0;
    rr_dims d{};
    int rc;
    if ((rc = check_pool_args(k_pool, v_pool, page_table, prefix_lens, suffix_lens, &d))) return rc;
    if ((rc = check_tensor(q, "q", 3, RR_DTYPE_BF16))) return rc;
    if ((rc = check_tensor(out, "out", 3, RR_DTYPE_BF16))) return rc;
    for (int i = 0; i < 3; ++i)
        if ((rc = same_dim(q, i, "q", out, i, "out"))) return rc;
    if ((rc = same_dim(q, 2, "q", k_pool, 3, "k_pool"))) return rc;
    if ((rc = fits_i32(q->shape[1], "num_q_heads"))) return rc;
    d.num_q_heads = (int32_t)q->shape[1];
    d.total_tokens = q->shape[0];
    return rr_extend_attention(q->data, k_pool->data, v_pool->data, static_cast<const int32_t*>(page_table->data),
                               static_cast<const int32_t*>(prefix_lens->data),
                               static_cast<const int32_t*>(suffix_lens->data), out->data, &d, softmax_scale, stream);
}
