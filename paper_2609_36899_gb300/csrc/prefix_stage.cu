// prefix_stage.cu -- paged-KV prefix staging (gather) and loading (scatter).
//
// Late-bound KV preparation (Sec. 4.4) snapshots a departing trajectory's KV
// state: its blocks, scattered over the paged pool, are copied into one
// contiguous buffer per trajectory (phase 1), and a destination later
// materialises that prefix in its own pool (phase 3).  Both directions are a
// pure bit copy bound by HBM read + write bandwidth.
//
// Work unit = (trajectory b, row (layer, K|V, KV head), chunk of kPagesPerUnit
// pages).  One (page, head) block is 16 tokens x D bf16 = 4 KB contiguous at
// D = 128 (head-major pool), and its staged image is also contiguous, so a
// warp moves each block with 16-byte loads and stores, all loads of a unit in
// flight before the first store.  A prep kernel computes the per-trajectory
// prefix sums (pages, tokens, units) once; the copy kernel's warps stride over
// units and find their trajectory by binary search in shared memory.
#include "internal.h"
#include "ptx.cuh"

namespace cadkv {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kPagesPerUnit = 2;
constexpr int kCopyThreads = 256;
constexpr int kCopyCtasPerSm = 4;
constexpr int kSmemPrefix = 4096;  // trajectories whose unit prefix is cached in smem

__host__ __device__ constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Exclusive block scan of one value per thread (1024 threads); returns the
// exclusive prefix and adds the block total to *carry (shared).
__device__ long long block_exclusive_scan(long long v, long long *warp_sums, long long *carry)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    long long x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long u = __shfl_up_sync(kFull, x, o);
        if (lane >= o)
            x += u;
    }
    if (lane == 31)
        warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        long long w = warp_sums[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long u = __shfl_up_sync(kFull, w, o);
            if (lane >= o)
                w += u;
        }
        warp_sums[lane] = w;
    }
    __syncthreads();
    const long long c = *carry;
    const long long incl = c + x + (warp > 0 ? warp_sums[warp - 1] : 0);
    __syncthreads();
    if (tid == 1023)
        *carry = incl;
    __syncthreads();
    return incl - v;
}

__global__ void __launch_bounds__(1024, 1) stage_prep_kernel(const StageParams p)
{
    __shared__ long long warp_sums[32];
    __shared__ long long carry[3];
    const int tid = threadIdx.x;
    const int rows = (p.layer_end - p.layer_begin) * 2 * p.num_kv_heads;
    const int max_len = p.max_pages * kPageSize;
    if (tid == 0) {
        p.hdr->status = 0;
        carry[0] = carry[1] = carry[2] = 0;
    }
    __syncthreads();
    for (int base = 0; base < p.batch; base += 1024) {
        const int b = base + tid;
        long long n = 0;
        if (b < p.batch) {
            n = p.context_lens[b];
            if (n < 0 || n > max_len) {
                record_status(&p.hdr->status, CADKV_ERR_SHAPE);
                n = 0;
            }
        }
        const long long pages = (n + kPageSize - 1) / kPageSize;
        const long long units = (long long)rows * ((pages + kPagesPerUnit - 1) / kPagesPerUnit);
        const long long ep = block_exclusive_scan(pages, warp_sums, &carry[0]);
        const long long et = block_exclusive_scan(n, warp_sums, &carry[1]);
        const long long eu = block_exclusive_scan(units, warp_sums, &carry[2]);
        if (b < p.batch) {
            p.page_prefix[b] = ep;
            p.token_prefix[b] = et;
            p.unit_prefix[b] = eu;
        }
    }
    if (tid == 0) {
        p.page_prefix[p.batch] = carry[0];
        p.token_prefix[p.batch] = carry[1];
        p.unit_prefix[p.batch] = carry[2];
        p.hdr->total_work = carry[2];
    }
}

// Largest b in [0, batch) with prefix[b] <= u (prefix non-decreasing, prefix[0] = 0).
__device__ __forceinline__ int find_trajectory(const long long *prefix, int batch, long long u)
{
    int lo = 0, hi = batch - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (prefix[mid] <= u)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

template <int D>
__global__ void __launch_bounds__(kCopyThreads) stage_copy_kernel(const StageParams p)
{
    constexpr int kVecPerPage = kPageSize * D / 8;      // 16-byte vectors per (page, head)
    constexpr int kVecPerLane = kVecPerPage / 32;
    __shared__ long long unit_prefix_s[kSmemPrefix + 1];
    const bool cached = p.batch + 1 <= kSmemPrefix + 1;
    if (cached)
        for (int i = threadIdx.x; i <= p.batch; i += blockDim.x)
            unit_prefix_s[i] = p.unit_prefix[i];
    __syncthreads();
    const long long *uprefix = cached ? unit_prefix_s : p.unit_prefix;

    const long long total = p.unit_prefix[p.batch];
    const int lane = threadIdx.x & 31;
    const long long warp_id = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long num_warps = ((long long)gridDim.x * blockDim.x) >> 5;
    const int rows = (p.layer_end - p.layer_begin) * 2 * p.num_kv_heads;
    const int hkv = p.num_kv_heads;

    for (long long u = warp_id; u < total; u += num_warps) {
        const int b = find_trajectory(uprefix, p.batch, u);
        const long long n = p.token_prefix[b + 1] - p.token_prefix[b];
        const long long pages = p.page_prefix[b + 1] - p.page_prefix[b];
        const long long chunks = (pages + kPagesPerUnit - 1) / kPagesPerUnit;
        const long long local = u - uprefix[b];
        const int row = (int)(local / chunks);
        const int chunk = (int)(local % chunks);
        const int lrel = row / (2 * hkv);
        const int kv = (row / hkv) & 1;
        const int h = row % hkv;
        const int layer = p.layer_begin + lrel;
        const long long off = p.row_offsets ? p.row_offsets[b]
                                            : (long long)rows * D * p.token_prefix[b];
        if (off & 7) {  // staged rows must start on a 16-byte boundary
            if (lane == 0)
                record_status(&p.hdr->status, CADKV_ERR_INVALID);
            continue;
        }
        __nv_bfloat16 *pool = reinterpret_cast<__nv_bfloat16 *>(
            const_cast<void *>(kv ? p.layer_v[layer] : p.layer_k[layer]));
        __nv_bfloat16 *staged = reinterpret_cast<__nv_bfloat16 *>(p.rows) + off + (long long)row * n * D;

        const int j0 = chunk * kPagesPerUnit;
        uint4 buf[kPagesPerUnit][kVecPerLane];
        uint4 *dstp[kPagesPerUnit];
        int nvec[kPagesPerUnit];
#pragma unroll
        for (int q = 0; q < kPagesPerUnit; ++q) {
            const int j = j0 + q;
            nvec[q] = 0;
            dstp[q] = nullptr;
            if (j < pages) {
                int phys = p.block_table[(long long)b * p.max_pages + j];
                if (phys < 0 || phys >= p.num_pages) {
                    if (lane == 0)
                        record_status(&p.hdr->status, CADKV_ERR_OOB);
                    continue;
                }
                const long long valid = n - (long long)j * kPageSize;
                nvec[q] = (int)((valid < kPageSize ? valid : kPageSize) * D / 8);
                uint4 *pool_blk = reinterpret_cast<uint4 *>(pool + ((long long)phys * hkv + h) * kPageSize * D);
                uint4 *row_blk = reinterpret_cast<uint4 *>(staged + (long long)j * kPageSize * D);
                const uint4 *srcp = p.to_pool ? row_blk : pool_blk;
                dstp[q] = p.to_pool ? pool_blk : row_blk;
#pragma unroll
                for (int v = 0; v < kVecPerLane; ++v) {
                    const int idx = lane + 32 * v;
                    if (idx < nvec[q])
                        buf[q][v] = __ldcs(srcp + idx);
                }
            }
        }
#pragma unroll
        for (int q = 0; q < kPagesPerUnit; ++q) {
#pragma unroll
            for (int v = 0; v < kVecPerLane; ++v) {
                const int idx = lane + 32 * v;
                if (idx < nvec[q])
                    __stcs(dstp[q] + idx, buf[q][v]);
            }
        }
    }
}

}  // namespace

StageWorkspaceLayout stage_workspace_layout(int batch)
{
    StageWorkspaceLayout L{};
    size_t off = align_up(sizeof(WorkspaceHeader), kWorkspaceAlign);
    const size_t arr = align_up((size_t)(batch + 1) * sizeof(long long), kWorkspaceAlign);
    L.page_prefix = off;
    L.token_prefix = off + arr;
    L.unit_prefix = off + 2 * arr;
    L.total = off + 3 * arr;
    return L;
}

cudaError_t launch_stage(const StageParams &p, int num_sms, cudaStream_t stream)
{
    stage_prep_kernel<<<1, 1024, 0, stream>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    const int grid = num_sms * kCopyCtasPerSm;
    if (p.head_dim == 128)
        stage_copy_kernel<128><<<grid, kCopyThreads, 0, stream>>>(p);
    else
        stage_copy_kernel<64><<<grid, kCopyThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace cadkv
