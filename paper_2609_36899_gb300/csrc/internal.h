// internal.h -- types shared by the host launchers and the kernels.
#pragma once

#include <atomic>
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "cadkv.h"

namespace cadkv {

// Raises a kernel's dynamic shared-memory limit to `bytes`, once per device:
// the attribute belongs to the device's context, and host threads may launch
// concurrently.  `done` keeps one bit per device id below 64.
template <typename Kernel>
inline cudaError_t ensure_smem_limit(Kernel *kernel, int bytes, std::atomic<uint64_t> &done)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    const uint64_t bit = dev >= 0 && dev < 64 ? 1ull << dev : 0;
    if (bit && (done.load(std::memory_order_acquire) & bit))
        return cudaSuccess;
    e = cudaFuncSetAttribute(reinterpret_cast<const void *>(kernel),
                             cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && bit)
        done.fetch_or(bit, std::memory_order_release);
    return e;
}


constexpr int kPageSize = 16;      // tokens per KV page
constexpr int kMaxGroup = 8;       // query heads per KV head handled by one tile
constexpr int kNumConsumerWarps = 8;
constexpr int kAttnThreads = (kNumConsumerWarps + 1) * 32;
constexpr int kSegRing = 16;       // segment descriptors in flight per CTA (two per consumer
                                   // warp in the per-warp mode)
constexpr int kSlicesPerCta = 4;   // dynamic work slices per persistent CTA
constexpr int kMinSlicePages = 16; // auto slicing never cuts finer than this
constexpr long long kOneSliceMaxPerCta = 4096;  // page-heads per CTA up to which auto
                                                // slicing gives each CTA a single slice
constexpr size_t kWorkspaceAlign = 256;
// Batches up to this size are planned by a 256-thread CTA (kPlanThreadsSmall)
// instead of 1024: it fits on an SM beside an attention CTA, so the planner of
// the next decode step can launch while this step's attention kernel still
// runs and wait there, and no attention CTA waits for an SM behind it.
constexpr int kSmallPlanMaxBatch = 2048;
// Per-warp mode: when the (trajectory, KV head) units are short, every consumer
// warp streams a slice of its own (kNumConsumerWarps slices per CTA) and ends
// its segments alone, instead of eight warps sharing each segment and merging
// at its end.  Taken automatically when units average at most
// kWarpModeMaxAvgPages pages and every warp slice gets at least
// kWarpModeMinSlicePages page-heads.
constexpr long long kWarpModeMaxAvgPages = 48;
constexpr long long kWarpModeMinSlicePages = 4;

// Work slices T of W flattened page-heads: one equal slice per CTA while a CTA
// would hold at most kOneSliceMaxPerCta page-heads, up to kSlicesPerCta per CTA
// above that, or ceil(W / slice_pages) when forced, never more than slice_cap
// and never fewer than one.
__host__ __device__ inline long long plan_num_slices(long long W, int slice_pages, int slice_cap)
{
    const long long unit = slice_pages > 0 ? slice_pages : kMinSlicePages;
    long long T = (W + unit - 1) / unit;
    const long long ctas = slice_cap / kSlicesPerCta;
    const long long cap = (slice_pages > 0 || W > kOneSliceMaxPerCta * ctas) ? slice_cap : ctas;
    if (T > cap)
        T = cap;
    if (T < 1)
        T = 1;
    return T;
}

// Header at the start of a decode-attention or staging workspace.
struct alignas(64) WorkspaceHeader {
    int status;            // first device-side error code, 0 = none
    int slice_counter;     // next work slice to hand out
    int num_slices;        // T: slices of the flattened work sequence
    int exit_counter;      // decode: CTAs done fetching slices (reset by the last one)
    long long total_work;  // W: page-heads (decode), copy units (staging), work units (prefill)
    long long total_items; // prefill: work items
    long long dp_items;    // prefill: items run whole (the rest are split)
    long long pieces;      // prefill: pieces per split item
    long long first_segs;  // decode: CTAs whose first segment the planner described (0: none)
    int warp_mode;         // decode: 1 = per-warp slices (kNumConsumerWarps per CTA)
    int pad1;
};

// Byte offsets of the decode-attention workspace regions.
// Bytes of the planner's description of one attention CTA's first segment.
constexpr size_t kFirstSegBytes = 64;

struct DecodeWorkspaceLayout {
    size_t page_prefix;   // int64 [batch + 1]
    size_t first_seg;     // kFirstSegBytes x #SM: each CTA's first segment, as planned
    size_t unit_counter;  // int32 [batch * Hkv]
    size_t part_lse;      // fp32  [capacity][G]
    size_t part_o;        // fp32  [capacity][G][D]
    size_t total;
    int capacity;         // partial slots = batch * Hkv + the most slices of either mode
    int slice_cap;
};

DecodeWorkspaceLayout decode_workspace_layout(int batch, int num_kv_heads, int group,
                                              int head_dim, int num_sms);

struct PlanParams {
    const int *context_lens;
    __nv_bfloat16 *out;
    float *lse;
    WorkspaceHeader *hdr;
    long long *page_prefix;
    int *unit_counter;
    void *first_seg;    // [slice_cap / kSlicesPerCta] first-segment records
    int describe_first; // 1: write them (a plan that may serve several runs)
    int batch, num_q_heads, num_kv_heads, head_dim, max_pages;
    int slice_cap;      // upper bound on slices (partial capacity)
    int slice_pages;    // forced slice length in pages, 0 = automatic
    // Optional fused KV append (CTAs 1.. of the planner launch): the new
    // token's rows k_new/v_new [batch][Hkv][D] go to position n_b - 1.
    const __nv_bfloat16 *k_new, *v_new;  // null: no append
    __nv_bfloat16 *k_pages, *v_pages;
    const int *block_table;
    int num_pages;
    int threads;        // threads per CTA: kPlanThreadsSmall for small batches without a
                        // fused append (the append CTAs need kPlanThreads)
};

constexpr int kAppendRowsPerCta = 32;  // one warp per (trajectory, KV head)
constexpr int kPlanThreads = 1024;
constexpr int kPlanThreadsSmall = 256;

struct AttnParams {
    const __nv_bfloat16 *q;
    const int *block_table;
    const int *context_lens;
    __nv_bfloat16 *out;
    float *lse;
    WorkspaceHeader *hdr;
    const long long *page_prefix;
    const void *first_seg;  // the planner's first-segment records (valid: hdr->first_segs)
    int *unit_counter;
    float *part_lse;
    float *part_o;
    int batch, num_q_heads, num_kv_heads, group, max_pages, num_pages;
    int whole_page_box;  // 1: the tensor maps copy a whole (page, head) block per TMA op
    float scale_log2;    // log2(e) / sqrt(D)
};

cudaError_t launch_plan(const PlanParams &p, cudaStream_t stream);  // + append CTAs if k_new
cudaError_t launch_attention(const AttnParams &p, const CUtensorMap &kmap,
                             const CUtensorMap &vmap, int head_dim, int grid,
                             cudaStream_t stream);
size_t attention_smem_bytes(int head_dim);

// ---------------------------------------------------------------- prefill

struct PrefillParams {
    const long long *q_offsets;  // device [batch + 1]
    const int *context_lens;
    const int *block_table;
    __nv_bfloat16 *out;          // [T][Hq][D]
    float *lse;                  // [T][Hq], nullable
    WorkspaceHeader *hdr;        // total_work = work units; slice_counter = next unit
    long long *item_prefix;      // [batch + 1] work items of trajectories before b
    int *merge_counter;          // [num_ctas] pieces done of split item i
    float *partial_lambda;       // [2 * num_ctas][256] log2-lse of a piece's rows
    float *partial_o;            // [2 * num_ctas][128][256] O / l of a piece's rows, column-major
    long long total_q;           // rows of q / out; offsets beyond it are rejected
    int batch, num_q_heads, num_kv_heads, group, max_pages, num_pages, num_ctas;
    float scale_log2;
};

size_t prefill_smem_bytes();
bool prefill_register_split_fits();  // the kernel's launch registers cover its setmaxnreg split
cudaError_t launch_prefill(const PrefillParams &p, const CUtensorMap &qmap, const CUtensorMap &kmap,
                           const CUtensorMap &vmap, cudaStream_t stream);

// ---------------------------------------------------------------- staging

struct StageParams {
    const void *const *layer_k;  // device array [num_layers] of K page pointers
    const void *const *layer_v;  // device array [num_layers] of V page pointers
    const int *block_table;
    const int *context_lens;
    void *rows;                  // staged rows (dst of stage, src of load)
    const long long *row_offsets;  // nullable
    WorkspaceHeader *hdr;
    long long *page_prefix;      // [B + 1]
    long long *token_prefix;     // [B + 1]
    long long *unit_prefix;      // [B + 1]
    int batch, max_pages, num_pages, num_kv_heads, head_dim;
    int layer_begin, layer_end;
    int to_pool;                 // 0: pool -> rows (stage), 1: rows -> pool (load)
};

struct StageWorkspaceLayout {
    size_t page_prefix, token_prefix, unit_prefix, total;
};
StageWorkspaceLayout stage_workspace_layout(int batch);

cudaError_t launch_stage(const StageParams &p, int num_sms, cudaStream_t stream);

cudaError_t launch_wait_selftest(WorkspaceHeader *hdr, unsigned long long limit_ns,
                                 cudaStream_t stream);
cudaError_t launch_hbm_read(const void *src, size_t bytes, unsigned long long *sink,
                            int num_sms, cudaStream_t stream);

}  // namespace cadkv
