// capi.cu -- the extern "C" entry points declared in include/cadkv.h.
//
// Host side only: argument validation, workspace carving, TMA tensor-map
// encoding and kernel launches.  Every numeric step runs in the kernels of
// decode_attention.cu and prefix_stage.cu.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "internal.h"

using namespace cadkv;

struct cadkv_pool {
    int num_layers = 0, num_pages = 0, page_size = 0, num_kv_heads = 0, head_dim = 0;
    int device = 0;
    void *owned = nullptr;          // single allocation holding all pages, if owned
    void **dev_layer_ptrs = nullptr;  // device array [2 * num_layers]: K pointers then V
    std::vector<void *> k, v;
};

namespace {

constexpr int kAbiVersion = (1 << 16) | 2;

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

size_t align_up_host(size_t x, size_t a) { return (x + a - 1) / a * a; }

int device_sms()
{
    static std::mutex mu;
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0)
        return CADKV_ERR_CUDA;
    if (dev < 64) {
        std::lock_guard<std::mutex> lock(mu);
        if (cache[dev] > 0)
            return cache[dev];
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        return CADKV_ERR_CUDA;
    if (dev < 64) {
        std::lock_guard<std::mutex> lock(mu);
        cache[dev] = sms;
    }
    return sms;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled_fn()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

// Tensor map over one layer's pages.  Preferred (D = 128): a 4-D view
// {64 columns, 16 tokens, 2 column halves, page-heads} with strides
// {256 B, 128 B, 16*D*2 B} and box {64, 16, 2, 1}, so one TMA op moves a whole
// 4 KB (page, head) block and lands it as [half][token][64] -- two 16 x 128 B
// panels, 128-byte swizzled so that ldmatrix reads are bank-conflict free.
// Fallback (and D = 64): a 2-D view [rows = page-heads * 16][D] with a
// 16 x 64 box, one op per 64-column panel.  *whole_block reports which.
int encode_pages_map(CUtensorMap *map, const void *pages, int num_pages, int num_kv_heads,
                     int head_dim, bool allow_whole, int *whole_block)
{
    EncodeTiledFn fn = encode_tiled_fn();
    if (!fn)
        return CADKV_ERR_CUDA;
    const cuuint64_t page_heads = (cuuint64_t)num_pages * num_kv_heads;
    if (head_dim == 128 && allow_whole) {
        const cuuint64_t dims[4] = {64, (cuuint64_t)kPageSize, 2, page_heads};
        const cuuint64_t strides[3] = {(cuuint64_t)head_dim * 2, 128,
                                       (cuuint64_t)kPageSize * head_dim * 2};
        const cuuint32_t box[4] = {64, (cuuint32_t)kPageSize, 2, 1};
        const cuuint32_t elem[4] = {1, 1, 1, 1};
        CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(pages), dims,
                        strides, box, elem, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r == CUDA_SUCCESS) {
            *whole_block = 1;
            return CADKV_OK;
        }
    }
    *whole_block = 0;
    const cuuint64_t dims[2] = {(cuuint64_t)head_dim, page_heads * kPageSize};
    const cuuint64_t strides[1] = {(cuuint64_t)head_dim * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)kPageSize};
    const cuuint32_t elem[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(pages), dims,
                    strides, box, elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? CADKV_OK : CADKV_ERR_CUDA;
}

// encode_pages_map through a small per-thread cache: a serving loop calls
// decode attention with the same page pools over and over, and encoding a
// tensor map costs host time on every call.  A map depends only on its inputs
// (the pool pointer and geometry), so equal inputs give an equal map.
int encode_pages_map_cached(CUtensorMap *map, const void *pages, int num_pages, int num_kv_heads,
                            int head_dim, bool allow_whole, int *whole_block)
{
    struct Entry {
        const void *pages;
        int num_pages, num_kv_heads, head_dim, allow_whole, whole;
        CUtensorMap map;
    };
    constexpr int kEntries = 8;
    thread_local Entry cache[kEntries] = {};
    thread_local int next = 0;
    for (int i = 0; i < kEntries; ++i) {
        const Entry &e = cache[i];
        if (e.pages == pages && e.num_pages == num_pages && e.num_kv_heads == num_kv_heads &&
            e.head_dim == head_dim && e.allow_whole == (int)allow_whole) {
            *map = e.map;
            *whole_block = e.whole;
            return CADKV_OK;
        }
    }
    const int rc = encode_pages_map(map, pages, num_pages, num_kv_heads, head_dim, allow_whole,
                                    whole_block);
    if (rc == CADKV_OK) {
        Entry &e = cache[next];
        next = (next + 1) % kEntries;
        e.pages = pages;
        e.num_pages = num_pages;
        e.num_kv_heads = num_kv_heads;
        e.head_dim = head_dim;
        e.allow_whole = (int)allow_whole;
        e.whole = *whole_block;
        e.map = *map;
    }
    return rc;
}

struct DecodeShape {
    int batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages;
};

int check_decode_shape(const DecodeShape &s)
{
    if (s.batch < 0 || s.num_q_heads <= 0 || s.num_kv_heads <= 0 || s.max_pages < 0 ||
        s.head_dim <= 0 || s.page_size <= 0)
        return CADKV_ERR_SHAPE;
    if (s.num_q_heads % s.num_kv_heads != 0)
        return CADKV_ERR_SHAPE;
    if (s.num_q_heads / s.num_kv_heads > kMaxGroup)
        return CADKV_ERR_UNSUPPORTED;
    if (s.head_dim != 64 && s.head_dim != 128)
        return CADKV_ERR_UNSUPPORTED;
    if (s.page_size != kPageSize)
        return CADKV_ERR_UNSUPPORTED;
    if ((long long)s.max_pages * kPageSize > INT32_MAX)
        return CADKV_ERR_SHAPE;
    return CADKV_OK;
}

int workspace_carve(const DecodeShape &s, void *workspace, size_t workspace_bytes, int sms,
                    DecodeWorkspaceLayout *L)
{
    *L = decode_workspace_layout(s.batch, s.num_kv_heads, s.num_q_heads / s.num_kv_heads,
                                 s.head_dim, sms);
    if (!workspace || !aligned(workspace, kWorkspaceAlign) || workspace_bytes < L->total)
        return CADKV_ERR_WORKSPACE;
    return CADKV_OK;
}

// Threads of the planner launch: small batches without a fused append are
// planned by a CTA small enough to share an SM with an attention CTA.
int plan_threads(int batch, bool append)
{
    return !append && batch <= kSmallPlanMaxBatch ? kPlanThreadsSmall : kPlanThreads;
}

// New-token rows written into the pool before attention (decode_attention_append).
struct AppendArgs {
    const void *k_new, *v_new;
    void *k_pages, *v_pages;
    const int32_t *block_table;
};

int plan_impl(const int32_t *context_lens, void *out, float *lse, const DecodeShape &s,
              int slice_pages, void *workspace, size_t workspace_bytes, cudaStream_t stream,
              const AppendArgs *append = nullptr, bool describe_first = false)
{
    int rc = check_decode_shape(s);
    if (rc != CADKV_OK)
        return rc;
    if (s.batch == 0)
        return CADKV_OK;
    if (!context_lens || !out)
        return CADKV_ERR_INVALID;
    if (!aligned(out, 16) || !aligned(context_lens, 4) || (lse && !aligned(lse, 4)))
        return CADKV_ERR_INVALID;
    if (slice_pages < 0)
        return CADKV_ERR_INVALID;
    const int sms = device_sms();
    if (sms < 0)
        return sms;
    DecodeWorkspaceLayout L;
    rc = workspace_carve(s, workspace, workspace_bytes, sms, &L);
    if (rc != CADKV_OK)
        return rc;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    PlanParams p{};
    p.context_lens = context_lens;
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.lse = lse;
    p.hdr = reinterpret_cast<WorkspaceHeader *>(ws);
    p.page_prefix = reinterpret_cast<long long *>(ws + L.page_prefix);
    p.unit_counter = reinterpret_cast<int *>(ws + L.unit_counter);
    p.first_seg = ws + L.first_seg;
    p.describe_first = describe_first ? 1 : 0;
    p.batch = s.batch;
    p.num_q_heads = s.num_q_heads;
    p.num_kv_heads = s.num_kv_heads;
    p.head_dim = s.head_dim;
    p.max_pages = s.max_pages;
    p.slice_cap = L.slice_cap;
    p.slice_pages = slice_pages;
    p.threads = plan_threads(s.batch, append != nullptr);
    if (append) {
        p.k_new = static_cast<const __nv_bfloat16 *>(append->k_new);
        p.v_new = static_cast<const __nv_bfloat16 *>(append->v_new);
        p.k_pages = static_cast<__nv_bfloat16 *>(append->k_pages);
        p.v_pages = static_cast<__nv_bfloat16 *>(append->v_pages);
        p.block_table = append->block_table;
        p.num_pages = s.num_pages;
    }
    return launch_plan(p, stream) == cudaSuccess ? CADKV_OK : CADKV_ERR_CUDA;
}

int check_run_args(const void *q, const void *k_pages, const void *v_pages,
                   const int32_t *block_table, const int32_t *context_lens, const void *out,
                   const float *lse, const DecodeShape &s)
{
    if (!q || !k_pages || !v_pages || !block_table || !context_lens || !out)
        return CADKV_ERR_INVALID;
    if (!aligned(q, 16) || !aligned(k_pages, 16) || !aligned(v_pages, 16) || !aligned(out, 16) ||
        !aligned(block_table, 4) || !aligned(context_lens, 4) || (lse && !aligned(lse, 4)))
        return CADKV_ERR_INVALID;
    if (s.num_pages <= 0)
        return CADKV_ERR_SHAPE;
    if ((long long)s.num_pages * s.num_kv_heads * kPageSize > INT32_MAX)
        return CADKV_ERR_UNSUPPORTED;
    return CADKV_OK;
}

int run_impl(const void *q, const void *k_pages, const void *v_pages,
             const int32_t *block_table, const int32_t *context_lens, void *out, float *lse,
             const DecodeShape &s, void *workspace, size_t workspace_bytes, cudaStream_t stream)
{
    int rc = check_decode_shape(s);
    if (rc != CADKV_OK)
        return rc;
    if (s.batch == 0)
        return CADKV_OK;
    rc = check_run_args(q, k_pages, v_pages, block_table, context_lens, out, lse, s);
    if (rc != CADKV_OK)
        return rc;
    const int sms = device_sms();
    if (sms < 0)
        return sms;
    DecodeWorkspaceLayout L;
    rc = workspace_carve(s, workspace, workspace_bytes, sms, &L);
    if (rc != CADKV_OK)
        return rc;
    CUtensorMap kmap, vmap;
    int k_whole = 0, v_whole = 0;
    if (encode_pages_map_cached(&kmap, k_pages, s.num_pages, s.num_kv_heads, s.head_dim, true,
                                &k_whole) != CADKV_OK ||
        encode_pages_map_cached(&vmap, v_pages, s.num_pages, s.num_kv_heads, s.head_dim, true,
                                &v_whole) != CADKV_OK)
        return CADKV_ERR_CUDA;
    if (k_whole != v_whole) {  // both maps must use the same box shape
        if (encode_pages_map_cached(&kmap, k_pages, s.num_pages, s.num_kv_heads, s.head_dim,
                                    false, &k_whole) != CADKV_OK ||
            encode_pages_map_cached(&vmap, v_pages, s.num_pages, s.num_kv_heads, s.head_dim,
                                    false, &v_whole) != CADKV_OK)
            return CADKV_ERR_CUDA;
    }
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    AttnParams p{};
    p.q = static_cast<const __nv_bfloat16 *>(q);
    p.block_table = block_table;
    p.context_lens = context_lens;
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.lse = lse;
    p.hdr = reinterpret_cast<WorkspaceHeader *>(ws);
    p.page_prefix = reinterpret_cast<const long long *>(ws + L.page_prefix);
    p.first_seg = ws + L.first_seg;
    p.unit_counter = reinterpret_cast<int *>(ws + L.unit_counter);
    p.part_lse = reinterpret_cast<float *>(ws + L.part_lse);
    p.part_o = reinterpret_cast<float *>(ws + L.part_o);
    p.batch = s.batch;
    p.num_q_heads = s.num_q_heads;
    p.num_kv_heads = s.num_kv_heads;
    p.group = s.num_q_heads / s.num_kv_heads;
    p.max_pages = s.max_pages;
    p.num_pages = s.num_pages;
    p.whole_page_box = k_whole && v_whole;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)s.head_dim));
    return launch_attention(p, kmap, vmap, s.head_dim, sms, stream) == cudaSuccess ? CADKV_OK
                                                                                    : CADKV_ERR_CUDA;
}

int read_status(const void *workspace, cudaStream_t stream)
{
    if (!workspace)
        return CADKV_ERR_INVALID;
    int status = 0;
    if (cudaMemcpyAsync(&status, workspace, sizeof(int), cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return CADKV_ERR_CUDA;
    return status;
}

// Persistent CTAs of the prefill kernel: one per SM of the current device (an
// upper bound when no device answers, so that a size query never comes short).
int prefill_ctas()
{
    const int sms = device_sms();
    return sms > 0 ? sms : 256;
}

struct PrefillWorkspaceLayout {
    size_t item_prefix, merge_counter, partial_lambda, partial_o, total;
};

PrefillWorkspaceLayout prefill_workspace_layout(int batch, int ctas)
{
    PrefillWorkspaceLayout L{};
    size_t off = align_up_host(sizeof(WorkspaceHeader), kWorkspaceAlign);
    L.item_prefix = off;
    off += align_up_host((size_t)(batch + 1) * sizeof(long long), kWorkspaceAlign);
    L.merge_counter = off;
    off += align_up_host((size_t)ctas * sizeof(int), kWorkspaceAlign);
    const size_t slots = (size_t)2 * ctas * 256;
    L.partial_lambda = off;
    off += align_up_host(slots * sizeof(float), kWorkspaceAlign);
    L.partial_o = off;
    off += align_up_host(slots * 128 * sizeof(float), kWorkspaceAlign);
    L.total = off;
    return L;
}

int stage_impl(const cadkv_pool *pool, const int32_t *block_table, int max_pages,
               const int32_t *context_lens, int batch, int layer_begin, int layer_end,
               const void *rows, const int64_t *offsets, void *workspace,
               size_t workspace_bytes, cudaStream_t stream, int to_pool)
{
    if (!pool)
        return CADKV_ERR_INVALID;
    if (batch < 0 || max_pages < 0 || layer_begin < 0 || layer_end > pool->num_layers ||
        layer_begin > layer_end)
        return CADKV_ERR_SHAPE;
    if ((long long)max_pages * kPageSize > INT32_MAX)
        return CADKV_ERR_SHAPE;
    if (batch == 0 || layer_begin == layer_end)
        return CADKV_OK;
    if (!block_table || !context_lens || !rows)
        return CADKV_ERR_INVALID;
    if (!aligned(rows, 16) || !aligned(block_table, 4) || !aligned(context_lens, 4) ||
        (offsets && !aligned(offsets, 8)))
        return CADKV_ERR_INVALID;
    const StageWorkspaceLayout L = stage_workspace_layout(batch);
    if (!workspace || !aligned(workspace, kWorkspaceAlign) || workspace_bytes < L.total)
        return CADKV_ERR_WORKSPACE;
    // The staged rows may be device memory or page-locked host memory that the
    // device can address (then the copy kernel reads or writes host memory
    // directly over the CPU-GPU link); pageable host memory is refused.
    cudaPointerAttributes attr{};
    if (cudaPointerGetAttributes(&attr, rows) != cudaSuccess) {
        cudaGetLastError();
        return CADKV_ERR_INVALID;
    }
    if (attr.type == cudaMemoryTypeUnregistered ||
        (attr.type == cudaMemoryTypeHost && attr.devicePointer == nullptr))
        return CADKV_ERR_INVALID;
    const void *dev_rows = attr.type == cudaMemoryTypeHost ? attr.devicePointer : rows;
    if (!aligned(dev_rows, 16))
        return CADKV_ERR_INVALID;
    const int sms = device_sms();
    if (sms < 0)
        return sms;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    StageParams p{};
    p.layer_k = pool->dev_layer_ptrs;
    p.layer_v = pool->dev_layer_ptrs + pool->num_layers;
    p.block_table = block_table;
    p.context_lens = context_lens;
    p.rows = const_cast<void *>(dev_rows);
    p.row_offsets = reinterpret_cast<const long long *>(offsets);
    p.hdr = reinterpret_cast<WorkspaceHeader *>(ws);
    p.page_prefix = reinterpret_cast<long long *>(ws + L.page_prefix);
    p.token_prefix = reinterpret_cast<long long *>(ws + L.token_prefix);
    p.unit_prefix = reinterpret_cast<long long *>(ws + L.unit_prefix);
    p.batch = batch;
    p.max_pages = max_pages;
    p.num_pages = pool->num_pages;
    p.num_kv_heads = pool->num_kv_heads;
    p.head_dim = pool->head_dim;
    p.layer_begin = layer_begin;
    p.layer_end = layer_end;
    p.to_pool = to_pool;
    return launch_stage(p, sms, stream) == cudaSuccess ? CADKV_OK : CADKV_ERR_CUDA;
}

}  // namespace

extern "C" {

const char *kv_status_string(int status)
{
    switch (status) {
    case CADKV_OK: return "ok";
    case CADKV_ERR_INVALID: return "invalid argument (null or misaligned pointer, bad value)";
    case CADKV_ERR_SHAPE: return "inconsistent sizes or context length out of range";
    case CADKV_ERR_CUDA: return "CUDA call failed";
    case CADKV_ERR_UNSUPPORTED: return "unsupported head_dim, page_size or head group";
    case CADKV_ERR_OOB: return "block-table entry outside the KV pool";
    case CADKV_ERR_TIMEOUT: return "device-side wait timed out";
    case CADKV_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    default: return "unknown status";
    }
}

int cadkv_abi_version(void) { return kAbiVersion; }

int cadkv_device_sms(void) { return device_sms(); }

int kv_pool_create(cadkv_pool **out, int num_layers, int num_pages, int page_size,
                   int num_kv_heads, int head_dim, void *const *k_layers, void *const *v_layers)
{
    if (!out)
        return CADKV_ERR_INVALID;
    *out = nullptr;
    if (num_layers <= 0 || num_pages <= 0 || num_kv_heads <= 0)
        return CADKV_ERR_SHAPE;
    if (page_size != kPageSize || (head_dim != 64 && head_dim != 128))
        return CADKV_ERR_UNSUPPORTED;
    if ((k_layers == nullptr) != (v_layers == nullptr))
        return CADKV_ERR_INVALID;
    if (k_layers)
        for (int l = 0; l < num_layers; ++l)
            if (!k_layers[l] || !v_layers[l] || !aligned(k_layers[l], 16) ||
                !aligned(v_layers[l], 16))
                return CADKV_ERR_INVALID;
    cadkv_pool *pool = new (std::nothrow) cadkv_pool;
    if (!pool)
        return CADKV_ERR_INVALID;
    try {
        pool->k.resize(num_layers);
        pool->v.resize(num_layers);
    } catch (...) {
        delete pool;
        return CADKV_ERR_INVALID;
    }
    pool->num_layers = num_layers;
    pool->num_pages = num_pages;
    pool->page_size = page_size;
    pool->num_kv_heads = num_kv_heads;
    pool->head_dim = head_dim;
    cudaGetDevice(&pool->device);
    const size_t layer_bytes = (size_t)num_pages * num_kv_heads * page_size * head_dim * 2;
    if (k_layers) {
        for (int l = 0; l < num_layers; ++l) {
            pool->k[l] = k_layers[l];
            pool->v[l] = v_layers[l];
        }
    } else {
        if (cudaMalloc(&pool->owned, layer_bytes * 2 * num_layers) != cudaSuccess) {
            delete pool;
            return CADKV_ERR_CUDA;
        }
        for (int l = 0; l < num_layers; ++l) {
            pool->k[l] = static_cast<uint8_t *>(pool->owned) + (size_t)(2 * l) * layer_bytes;
            pool->v[l] = static_cast<uint8_t *>(pool->owned) + (size_t)(2 * l + 1) * layer_bytes;
        }
    }
    std::vector<void *> ptrs(2 * (size_t)num_layers);
    for (int l = 0; l < num_layers; ++l) {
        ptrs[l] = pool->k[l];
        ptrs[num_layers + l] = pool->v[l];
    }
    if (cudaMalloc(&pool->dev_layer_ptrs, ptrs.size() * sizeof(void *)) != cudaSuccess ||
        cudaMemcpy(pool->dev_layer_ptrs, ptrs.data(), ptrs.size() * sizeof(void *),
                   cudaMemcpyHostToDevice) != cudaSuccess) {
        if (pool->dev_layer_ptrs)
            cudaFree(pool->dev_layer_ptrs);
        if (pool->owned)
            cudaFree(pool->owned);
        delete pool;
        return CADKV_ERR_CUDA;
    }
    *out = pool;
    return CADKV_OK;
}

int kv_pool_destroy(cadkv_pool *pool)
{
    if (!pool)
        return CADKV_OK;
    int rc = CADKV_OK;
    if (pool->dev_layer_ptrs && cudaFree(pool->dev_layer_ptrs) != cudaSuccess)
        rc = CADKV_ERR_CUDA;
    if (pool->owned && cudaFree(pool->owned) != cudaSuccess)
        rc = CADKV_ERR_CUDA;
    delete pool;
    return rc;
}

int kv_pool_layer(const cadkv_pool *pool, int layer, void **k_pages, void **v_pages)
{
    if (!pool || layer < 0 || layer >= pool->num_layers)
        return CADKV_ERR_INVALID;
    if (k_pages)
        *k_pages = pool->k[layer];
    if (v_pages)
        *v_pages = pool->v[layer];
    return CADKV_OK;
}

int kv_pool_geometry(const cadkv_pool *pool, int *num_layers, int *num_pages, int *page_size,
                     int *num_kv_heads, int *head_dim)
{
    if (!pool)
        return CADKV_ERR_INVALID;
    if (num_layers)
        *num_layers = pool->num_layers;
    if (num_pages)
        *num_pages = pool->num_pages;
    if (page_size)
        *page_size = pool->page_size;
    if (num_kv_heads)
        *num_kv_heads = pool->num_kv_heads;
    if (head_dim)
        *head_dim = pool->head_dim;
    return CADKV_OK;
}

size_t decode_attention_workspace_size(int batch, int num_q_heads, int num_kv_heads,
                                       int head_dim, int max_pages)
{
    const DecodeShape s{batch, num_q_heads, num_kv_heads, head_dim, kPageSize, 1, max_pages};
    if (check_decode_shape(s) != CADKV_OK)
        return 0;
    const int sms = device_sms();
    if (sms < 0)
        return 0;
    return decode_workspace_layout(batch, num_kv_heads, num_q_heads / num_kv_heads, head_dim, sms)
        .total;
}

int decode_attention_plan(const int32_t *context_lens, void *out, float *lse, int batch,
                          int num_q_heads, int num_kv_heads, int head_dim, int max_pages,
                          int slice_pages, void *workspace, size_t workspace_bytes,
                          cadkv_stream_t stream)
{
    const DecodeShape s{batch, num_q_heads, num_kv_heads, head_dim, kPageSize, 1, max_pages};
    return plan_impl(context_lens, out, lse, s, slice_pages, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream), nullptr, true);
}

int decode_attention_run(const void *q, const void *k_pages, const void *v_pages,
                         const int32_t *block_table, const int32_t *context_lens, void *out,
                         float *lse, int batch, int num_q_heads, int num_kv_heads, int head_dim,
                         int page_size, int num_pages, int max_pages, void *workspace,
                         size_t workspace_bytes, cadkv_stream_t stream)
{
    const DecodeShape s{batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages};
    return run_impl(q, k_pages, v_pages, block_table, context_lens, out, lse, s, workspace,
                    workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int decode_attention_split(const void *q, const void *k_pages, const void *v_pages,
                           const int32_t *block_table, const int32_t *context_lens, void *out,
                           float *lse, int batch, int num_q_heads, int num_kv_heads,
                           int head_dim, int page_size, int num_pages, int max_pages,
                           int slice_pages, void *workspace, size_t workspace_bytes,
                           cadkv_stream_t stream)
{
    const DecodeShape s{batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages};
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // Validate everything the run needs before launching the planner.
    int rc = check_decode_shape(s);
    if (rc != CADKV_OK)
        return rc;
    if (batch == 0)
        return CADKV_OK;
    rc = check_run_args(q, k_pages, v_pages, block_table, context_lens, out, lse, s);
    if (rc != CADKV_OK)
        return rc;
    rc = plan_impl(context_lens, out, lse, s, slice_pages, workspace, workspace_bytes, st);
    if (rc != CADKV_OK)
        return rc;
    return run_impl(q, k_pages, v_pages, block_table, context_lens, out, lse, s, workspace,
                    workspace_bytes, st);
}

int decode_attention(const void *q, const void *k_pages, const void *v_pages,
                     const int32_t *block_table, const int32_t *context_lens, void *out,
                     float *lse, int batch, int num_q_heads, int num_kv_heads, int head_dim,
                     int page_size, int num_pages, int max_pages, void *workspace,
                     size_t workspace_bytes, cadkv_stream_t stream)
{
    return decode_attention_split(q, k_pages, v_pages, block_table, context_lens, out, lse,
                                  batch, num_q_heads, num_kv_heads, head_dim, page_size,
                                  num_pages, max_pages, 0, workspace, workspace_bytes, stream);
}

int decode_attention_status(const void *workspace, cadkv_stream_t stream)
{
    return read_status(workspace, reinterpret_cast<cudaStream_t>(stream));
}

size_t prefill_attention_workspace_size(int batch)
{
    if (batch < 0)
        return 0;
    return prefill_workspace_layout(batch, prefill_ctas()).total;
}

int prefill_attention(const void *q, const int64_t *q_offsets, const void *k_pages,
                      const void *v_pages, const int32_t *block_table,
                      const int32_t *context_lens, void *out, float *lse, int batch,
                      int total_q, int num_q_heads, int num_kv_heads, int head_dim,
                      int page_size, int num_pages, int max_pages, void *workspace,
                      size_t workspace_bytes, cadkv_stream_t stream)
{
    if (batch < 0 || total_q < 0 || num_q_heads <= 0 || num_kv_heads <= 0 || max_pages < 0 ||
        num_pages <= 0 || num_q_heads % num_kv_heads != 0)
        return CADKV_ERR_SHAPE;
    const int group = num_q_heads / num_kv_heads;
    if (head_dim != 128 || page_size != kPageSize || group > kMaxGroup)
        return CADKV_ERR_UNSUPPORTED;
    if ((long long)num_pages * num_kv_heads * kPageSize > INT32_MAX ||
        (long long)max_pages * kPageSize > INT32_MAX)
        return CADKV_ERR_UNSUPPORTED;
    if (batch == 0 || total_q == 0)
        return CADKV_OK;
    if (!q || !q_offsets || !k_pages || !v_pages || !block_table || !context_lens || !out)
        return CADKV_ERR_INVALID;
    if (!aligned(q, 16) || !aligned(k_pages, 16) || !aligned(v_pages, 16) || !aligned(out, 16) ||
        !aligned(q_offsets, 8) || !aligned(block_table, 4) || !aligned(context_lens, 4) ||
        (lse && !aligned(lse, 4)))
        return CADKV_ERR_INVALID;
    if (!workspace || !aligned(workspace, kWorkspaceAlign) ||
        workspace_bytes < prefill_attention_workspace_size(batch))
        return CADKV_ERR_WORKSPACE;
    EncodeTiledFn fn = encode_tiled_fn();
    if (!fn)
        return CADKV_ERR_CUDA;
    // Q viewed as {D, Hq, T}: box {64, G, floor(128/G)} = up to 128 rows (token-major,
    // head-minor)
    CUtensorMap qmap, kmap, vmap;
    {
        const cuuint64_t dims[3] = {(cuuint64_t)head_dim, (cuuint64_t)num_q_heads,
                                    (cuuint64_t)total_q};
        const cuuint64_t strides[2] = {(cuuint64_t)head_dim * 2,
                                       (cuuint64_t)num_q_heads * head_dim * 2};
        const cuuint32_t box[3] = {64, (cuuint32_t)group, (cuuint32_t)(128 / group)};
        const cuuint32_t elem[3] = {1, 1, 1};
        if (fn(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(q), dims, strides, box,
               elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return CADKV_ERR_CUDA;
    }
    // K: 2-D boxes of one 64-column panel (its operand is panel-major); V: whole
    // 4 KB (page, head) blocks through the 4-D view, which the kernel requires
    int k_whole = 0, v_whole = 0;
    if (encode_pages_map(&kmap, k_pages, num_pages, num_kv_heads, head_dim, false, &k_whole) !=
            CADKV_OK ||
        encode_pages_map(&vmap, v_pages, num_pages, num_kv_heads, head_dim, true, &v_whole) !=
            CADKV_OK)
        return CADKV_ERR_CUDA;
    if (!v_whole)
        return CADKV_ERR_UNSUPPORTED;
    if (!prefill_register_split_fits())
        return CADKV_ERR_UNSUPPORTED;
    const int ctas = prefill_ctas();
    const PrefillWorkspaceLayout L = prefill_workspace_layout(batch, ctas);
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    PrefillParams p{};
    p.q_offsets = reinterpret_cast<const long long *>(q_offsets);
    p.context_lens = context_lens;
    p.block_table = block_table;
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.lse = lse;
    p.hdr = reinterpret_cast<WorkspaceHeader *>(ws);
    p.item_prefix = reinterpret_cast<long long *>(ws + L.item_prefix);
    p.merge_counter = reinterpret_cast<int *>(ws + L.merge_counter);
    p.partial_lambda = reinterpret_cast<float *>(ws + L.partial_lambda);
    p.partial_o = reinterpret_cast<float *>(ws + L.partial_o);
    p.num_ctas = ctas;
    p.total_q = total_q;
    p.batch = batch;
    p.num_q_heads = num_q_heads;
    p.num_kv_heads = num_kv_heads;
    p.group = group;
    p.max_pages = max_pages;
    p.num_pages = num_pages;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)head_dim));
    return launch_prefill(p, qmap, kmap, vmap, reinterpret_cast<cudaStream_t>(stream)) ==
                   cudaSuccess
               ? CADKV_OK
               : CADKV_ERR_CUDA;
}

int prefill_attention_status(const void *workspace, cadkv_stream_t stream)
{
    return read_status(workspace, reinterpret_cast<cudaStream_t>(stream));
}

int decode_attention_append(const void *q, const void *k_new, const void *v_new, void *k_pages,
                            void *v_pages, const int32_t *block_table,
                            const int32_t *context_lens, void *out, float *lse, int batch,
                            int num_q_heads, int num_kv_heads, int head_dim, int page_size,
                            int num_pages, int max_pages, void *workspace,
                            size_t workspace_bytes, cadkv_stream_t stream)
{
    const DecodeShape s{batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages};
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int rc = check_decode_shape(s);
    if (rc != CADKV_OK)
        return rc;
    if (batch == 0)
        return CADKV_OK;
    rc = check_run_args(q, k_pages, v_pages, block_table, context_lens, out, lse, s);
    if (rc != CADKV_OK)
        return rc;
    if (!k_new || !v_new || !aligned(k_new, 16) || !aligned(v_new, 16))
        return CADKV_ERR_INVALID;
    const AppendArgs append{k_new, v_new, k_pages, v_pages, block_table};
    rc = plan_impl(context_lens, out, lse, s, 0, workspace, workspace_bytes, st, &append);
    if (rc != CADKV_OK)
        return rc;
    return run_impl(q, k_pages, v_pages, block_table, context_lens, out, lse, s, workspace,
                    workspace_bytes, st);
}

}  // extern "C"

// Scratch of decode_attention_noalloc: one array per device, never allocated
// at call time.  Host code may only use its device address, obtained with
// cudaGetSymbolAddress while that device is current (the name itself is a
// host-side stand-in).
static __device__ __align__(256) unsigned char g_noalloc_scratch[CADKV_NOALLOC_SCRATCH_BYTES];

namespace {

using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);

// Process-unique id of the CUDA context current on this thread, or 0 when no
// context is current or the driver cannot tell.
unsigned long long current_context_id()
{
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *a = nullptr, *b = nullptr;
        cudaDriverEntryPointQueryResult qa{}, qb{};
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &a, 12000, cudaEnableDefault,
                                             &qa) == cudaSuccess &&
            qa == cudaDriverEntryPointSuccess &&
            cudaGetDriverEntryPointByVersion("cuCtxGetId", &b, 12000, cudaEnableDefault, &qb) ==
                cudaSuccess &&
            qb == cudaDriverEntryPointSuccess) {
            get_current = reinterpret_cast<CtxGetCurrentFn>(a);
            get_id = reinterpret_cast<CtxGetIdFn>(b);
        }
    });
    if (!get_current || !get_id)
        return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
        return 0;
    return id;
}

// Device address of g_noalloc_scratch in the current device's context.  It is
// looked up (cudaGetSymbolAddress, with that device current) on the first
// call in a context and cached with the context's id; a call from another
// context of the same device -- after cudaDeviceReset, or under a context the
// caller made current -- looks it up again, so a cached address is never used
// in a context it does not belong to.
int noalloc_scratch(void **ptr)
{
    struct Entry {
        unsigned long long ctx;
        void *ptr;
    };
    static std::mutex mu;
    static Entry cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
        return CADKV_ERR_CUDA;
    std::lock_guard<std::mutex> lock(mu);
    unsigned long long ctx = current_context_id();
    if (ctx != 0 && cache[dev].ctx == ctx && cache[dev].ptr) {
        *ptr = cache[dev].ptr;
        return CADKV_OK;
    }
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
        return CADKV_ERR_CUDA;
    if (ctx == 0)  // the lookup above made the device's primary context current
        ctx = current_context_id();
    cache[dev].ctx = ctx;
    cache[dev].ptr = ctx != 0 ? p : nullptr;  // without a context id, never reuse
    *ptr = p;
    return CADKV_OK;
}

}  // namespace

extern "C" {

int decode_attention_noalloc(const void *q, const void *k_pages, const void *v_pages,
                             const int32_t *block_table, const int32_t *context_lens, void *out,
                             float *lse, int batch, int num_q_heads, int num_kv_heads,
                             int head_dim, int page_size, int num_pages, int max_pages,
                             cadkv_stream_t stream)
{
    const DecodeShape s{batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages};
    int rc = check_decode_shape(s);
    if (rc != CADKV_OK)
        return rc;
    if (batch == 0)
        return CADKV_OK;
    rc = check_run_args(q, k_pages, v_pages, block_table, context_lens, out, lse, s);
    if (rc != CADKV_OK)
        return rc;
    const int sms = device_sms();
    if (sms < 0)
        return sms;
    const size_t need = decode_workspace_layout(batch, num_kv_heads, num_q_heads / num_kv_heads,
                                                head_dim, sms)
                            .total;
    if (need > (size_t)CADKV_NOALLOC_SCRATCH_BYTES)
        return CADKV_ERR_WORKSPACE;
    void *scratch = nullptr;
    rc = noalloc_scratch(&scratch);
    if (rc != CADKV_OK)
        return rc;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    rc = plan_impl(context_lens, out, lse, s, 0, scratch, CADKV_NOALLOC_SCRATCH_BYTES, st);
    if (rc != CADKV_OK)
        return rc;
    return run_impl(q, k_pages, v_pages, block_table, context_lens, out, lse, s, scratch,
                    CADKV_NOALLOC_SCRATCH_BYTES, st);
}

int decode_attention_noalloc_status(cadkv_stream_t stream)
{
    void *scratch = nullptr;
    const int rc = noalloc_scratch(&scratch);
    if (rc != CADKV_OK)
        return rc;
    // the status word is the first field of the workspace header at the array's start
    return read_status(scratch, reinterpret_cast<cudaStream_t>(stream));
}

size_t kv_prefix_stage_workspace_size(int batch)
{
    if (batch < 0)
        return 0;
    return stage_workspace_layout(batch).total;
}

int kv_prefix_stage(const cadkv_pool *pool, const int32_t *block_table, int max_pages,
                    const int32_t *context_lens, int batch, int layer_begin, int layer_end,
                    void *dst, const int64_t *dst_offsets, void *workspace,
                    size_t workspace_bytes, cadkv_stream_t stream)
{
    return stage_impl(pool, block_table, max_pages, context_lens, batch, layer_begin, layer_end,
                      dst, dst_offsets, workspace, workspace_bytes,
                      reinterpret_cast<cudaStream_t>(stream), 0);
}

int kv_prefix_load(const cadkv_pool *pool, const int32_t *block_table, int max_pages,
                   const int32_t *context_lens, int batch, int layer_begin, int layer_end,
                   const void *src, const int64_t *src_offsets, void *workspace,
                   size_t workspace_bytes, cadkv_stream_t stream)
{
    return stage_impl(pool, block_table, max_pages, context_lens, batch, layer_begin, layer_end,
                      src, src_offsets, workspace, workspace_bytes,
                      reinterpret_cast<cudaStream_t>(stream), 1);
}

int kv_prefix_stage_status(const void *workspace, cadkv_stream_t stream)
{
    return read_status(workspace, reinterpret_cast<cudaStream_t>(stream));
}

int cadkv_wait_selftest(long long limit_ns, void *workspace, size_t workspace_bytes,
                        cadkv_stream_t stream)
{
    if (limit_ns <= 0 || limit_ns > 2000000000ll)
        return CADKV_ERR_INVALID;
    if (!workspace || !aligned(workspace, kWorkspaceAlign) ||
        workspace_bytes < sizeof(WorkspaceHeader))
        return CADKV_ERR_WORKSPACE;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    WorkspaceHeader *hdr = static_cast<WorkspaceHeader *>(workspace);
    if (cudaMemsetAsync(hdr, 0, sizeof(WorkspaceHeader), s) != cudaSuccess)
        return CADKV_ERR_CUDA;
    return launch_wait_selftest(hdr, (unsigned long long)limit_ns, s) == cudaSuccess ? CADKV_OK
                                                                                       : CADKV_ERR_CUDA;
}

int cadkv_hbm_read_probe(const void *buf, size_t bytes, unsigned long long *sink,
                         cadkv_stream_t stream)
{
    if (!buf || !sink || !aligned(buf, 16) || !aligned(sink, 8) || bytes % 16 != 0)
        return CADKV_ERR_INVALID;
    if (bytes == 0)
        return CADKV_OK;
    const int sms = device_sms();
    if (sms < 0)
        return sms;
    return launch_hbm_read(buf, bytes, sink, sms, reinterpret_cast<cudaStream_t>(stream)) ==
                   cudaSuccess
               ? CADKV_OK
               : CADKV_ERR_CUDA;
}

}  // extern "C"
