// decode_attention.cu -- batched paged-KV decode attention for sm_103a.
//
// One decode step of scaled dot-product attention (one query token per
// trajectory) over a paged KV cache.  The decode step is the memory-bound
// phase the paper's scheduler reshapes (Sec. 2.3, Sec. 3.1); attention and the
// paged cache themselves come from the paper's inference backend (Sec. 5).
//
// Design (GB300-first):
//  * Work = the flattened sequence of (trajectory b, KV head g, page j)
//    "page-heads", ordered b-major.  A planner kernel computes the page prefix
//    sum over trajectories; the sequence is cut into T equal slices.  In a
//    persistent grid (one CTA per SM) CTA i starts on slice i and pulls any
//    further slice from an atomic counter.  Equal
//    slices balance HBM bytes, not trajectories, so a few 128K-token tails and
//    hundreds of 2K-token trajectories both keep every SM streaming.
//  * Inside a CTA one producer warp issues TMA copies (cp.async.bulk.tensor,
//    128-byte swizzle) of each page-head's K and V block (16 tokens x D bf16,
//    contiguous in the head-major pool) into a ring of shared-memory stages
//    guarded by mbarriers, plus a 1-D bulk copy of the G query rows of every
//    new segment.  Each KV page is read from HBM exactly once per KV head:
//    all G query heads of the group share it (grouped-query attention).
//  * Eight consumer warps take pages round-robin (four could not keep up
//    with HBM on every SM).  Per page a warp computes
//    S^T = K Q^T with mma.sync m16n8k16 (16 tokens x 8 query heads), runs the
//    online softmax in registers (warp shuffles for the per-head max), turns
//    P^T into the B operand with movmatrix, and accumulates O^T += V^T P^T.
//  * At the end of a segment the warps merge their (m, l, O) in shared memory.
//    A trajectory-head that lies inside one slice is written straight to
//    `out`; otherwise the slice writes a partial (o, log2-sum-exp) and the CTA
//    that delivers a unit's last partial merges all of them in slice order
//    (deterministic), so no separate merge kernel runs.  One release/acquire
//    atomic per partial orders the partials; its result is read only after the
//    CTA's next segment, so the warps do not stall on it.
//  * Every wait is bounded (kWaitLimitNs); on timeout the kernel records
//    CADKV_ERR_TIMEOUT, drains its own copies and returns.
#include <cfloat>
#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace cadkv {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kIssueGroup = 8;  // pages the producer warp issues in parallel (<= stages)
constexpr float kLn2 = 0.6931471805599453f;

__host__ __device__ constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ------------------------------------------------------------------ work slices

// One segment: the part of a (trajectory, KV head) unit inside one work slice.
struct SegDesc {
    int b, kvh, page_begin, num_pages;  // num_pages < 0: no more work
    int n, slot, count, unit;
    int first, pad[3];
};

// The planner's description of an attention CTA's first segment (slice i is
// CTA i's first), so that the CTA starts streaming without working it out.
struct FirstSeg {
    SegDesc d;     // d.num_pages = 0: the slice is empty
    long long s1;  // end of the slice
    long long se;  // end of the segment: where the slice's next segment starts
};
static_assert(sizeof(FirstSeg) == kFirstSegBytes, "first-segment record size");

__device__ __forceinline__ long long slice_begin(long long s, long long W, long long T)
{
    return s * W / T;
}

// Index of the slice containing flattened position x.
__device__ __forceinline__ int slice_of(long long x, long long W, long long T)
{
    return (int)(((x + 1) * T + W - 1) / W - 1);
}

// The segment of slice `slice` (which ends at s1) that starts at flattened
// position x inside trajectory b, whose page-heads are [pb0 * Hkv, pb1 * Hkv);
// se receives where it ends.  d.n is left for the caller.
__device__ __forceinline__ SegDesc describe_segment(long long x, int b, long long pb0, long long pb1,
                                                    long long s1, int slice, long long W,
                                                    long long T, int Hkv, long long &se)
{
    const long long pages_b = pb1 - pb0;
    const long long base = pb0 * Hkv;
    const long long rel = x - base;
    const int kvh = rel <= 0xffffffffLL ? (int)((unsigned)rel / (unsigned)pages_b)
                                        : (int)(rel / pages_b);
    const long long us = base + kvh * pages_b, ue = us + pages_b;
    se = ue < s1 ? ue : s1;
    // x lies in slice `slice`: a unit that starts at x, or ends by s1, needs no search
    const int first = us == x ? slice : slice_of(us, W, T);
    const int last = ue <= s1 ? slice : slice_of(ue - 1, W, T);
    SegDesc d;
    d.b = b;
    d.kvh = kvh;
    d.page_begin = (int)(x - us);
    d.num_pages = (int)(se - x);
    d.n = 0;
    d.count = last - first + 1;
    d.unit = b * Hkv + kvh;
    d.slot = d.count == 1 ? -1 : d.unit + slice;
    d.first = first;
    d.pad[0] = d.pad[1] = d.pad[2] = 0;
    return d;
}

// ------------------------------------------------------------------ planner

// CTAs 1.. of the planner launch: write each trajectory's new-token K and V
// rows into slot (n_b - 1) % 16 of page block_table[b][(n_b - 1) / 16].  One
// warp per (trajectory, KV head); lanes 0-15 copy K, lanes 16-31 copy V, 16
// bytes each.  Invalid lengths or pages are skipped here: CTA 0 flags bad
// lengths, and the attention kernel flags the bad page when it reads it.
__device__ __forceinline__ void append_rows(const PlanParams &p)
{
    const int lane = threadIdx.x & 31;
    const int row = (blockIdx.x - 1) * kAppendRowsPerCta + (threadIdx.x >> 5);
    if (row >= p.batch * p.num_kv_heads)
        return;
    const int b = row / p.num_kv_heads, g = row % p.num_kv_heads;
    const int n = p.context_lens[b];
    if (n < 1 || n > p.max_pages * kPageSize)
        return;
    const int phys = p.block_table[(size_t)b * p.max_pages + (n - 1) / kPageSize];
    if (phys < 0 || phys >= p.num_pages)
        return;
    const int slot = (n - 1) % kPageSize;
    const bool is_v = lane >= 16;
    const uint4 *src = reinterpret_cast<const uint4 *>((is_v ? p.v_new : p.k_new) +
                                                       (size_t)row * p.head_dim);
    uint4 *dst = reinterpret_cast<uint4 *>(
        (is_v ? p.v_pages : p.k_pages) +
        (((size_t)phys * p.num_kv_heads + g) * kPageSize + slot) * p.head_dim);
    for (int c = lane & 15; c < p.head_dim / 8; c += 16)
        dst[c] = src[c];
}

__global__ void __launch_bounds__(kPlanThreads, 1) plan_kernel(const PlanParams p)
{
    // This grid is launched programmatically, so it may start while the previous
    // kernel on the stream (often the last decode step's attention kernel, which
    // lets it launch as soon as it starts) is still running: nothing is read or
    // written here before that kernel's writes are visible.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    // Now let the attention kernel launch: it sets up its shared memory and then
    // waits (griddepcontrol.wait) for this whole grid to finish before it reads
    // anything the planner or the append CTAs write.  Triggered before the wait
    // above, its CTAs took the SMs of the previous step's CTAs as they left and
    // the small-batch steps ran slower (29.5 against 27.3 us for 32 x 1,024
    // tokens in a CUDA graph).
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (blockIdx.x > 0) {
        append_rows(p);
        return;
    }
    __shared__ long long warp_sums[32];
    __shared__ long long carry_s;
    // small batches: the page prefix and clamped lengths also in shared memory,
    // for describing the attention CTAs' first segments below
    __shared__ long long s_prefix[kSmallPlanMaxBatch + 1];
    __shared__ int s_len[kSmallPlanMaxBatch];
    const bool small = p.describe_first && p.batch <= kSmallPlanMaxBatch;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nthreads = blockDim.x, nwarps = nthreads >> 5;
    const int max_len = p.max_pages * kPageSize;
    if (tid == 0) {
        p.hdr->status = 0;
        carry_s = 0;
    }
    __syncthreads();

    for (int base = 0; base < p.batch; base += nthreads) {
        const int b = base + tid;
        long long pages = 0;
        int n = 0;
        if (b < p.batch) {
            n = p.context_lens[b];
            if (n < 0 || n > max_len) {
                record_status(&p.hdr->status, CADKV_ERR_SHAPE);
                n = 0;
            }
            pages = (n + kPageSize - 1) / kPageSize;
            if (n == 0) {  // empty trajectory: out = 0, lse = -inf
                uint4 *row = reinterpret_cast<uint4 *>(p.out + (size_t)b * p.num_q_heads * p.head_dim);
                const int vecs = p.num_q_heads * p.head_dim / 8;
                for (int v = 0; v < vecs; ++v)
                    row[v] = make_uint4(0, 0, 0, 0);
                if (p.lse)
                    for (int h = 0; h < p.num_q_heads; ++h)
                        p.lse[(size_t)b * p.num_q_heads + h] = -INFINITY;
            }
        }
        // block-wide inclusive scan of `pages`
        long long v = pages;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            long long u = __shfl_up_sync(kFull, v, o);
            if (lane >= o)
                v += u;
        }
        if (lane == 31)
            warp_sums[warp] = v;
        __syncthreads();
        if (warp == 0) {
            long long w = lane < nwarps ? warp_sums[lane] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                long long u = __shfl_up_sync(kFull, w, o);
                if (lane >= o)
                    w += u;
            }
            warp_sums[lane] = w;  // inclusive over warps
        }
        __syncthreads();
        const long long carry = carry_s;
        const long long incl = carry + v + (warp > 0 ? warp_sums[warp - 1] : 0);
        if (b < p.batch) {
            p.page_prefix[b] = incl - pages;
            if (small) {
                s_prefix[b] = incl - pages;
                s_len[b] = n;  // the clamped length (0 when out of range)
            }
        }
        __syncthreads();
        if (tid == nthreads - 1)
            carry_s = incl;
        __syncthreads();
    }
    for (int i = tid; i < p.batch * p.num_kv_heads; i += nthreads)
        p.unit_counter[i] = 0;
    const long long total = carry_s;
    const int Hkv = p.num_kv_heads;
    const long long W = total * Hkv;
    // Dynamic slices (several per CTA) absorb per-SM speed differences, but
    // each costs a start-up chain of dependent loads (slice, trajectory,
    // table) and a pipeline fill; below ~4K page-heads per CTA that cost wins,
    // so automatic slicing gives each CTA one equal slice there.
    const long long ctas = p.slice_cap / kSlicesPerCta;
    // Short units (automatic slicing only): one slice per consumer warp, each
    // warp on its own (see kWarpModeMaxAvgPages).
    const long long units = (long long)p.batch * Hkv;
    const long long warp_slices = ctas * kNumConsumerWarps;
    const bool warp_mode = p.slice_pages == 0 && W <= kWarpModeMaxAvgPages * units &&
                           W >= kWarpModeMinSlicePages * warp_slices;
    const long long T = warp_mode ? warp_slices : plan_num_slices(W, p.slice_pages, p.slice_cap);
    // Describe each attention CTA's first segment (its first slice is slice
    // blockIdx.x), as its producer warp would: the CTA then loads one record
    // instead of searching the prefix and dividing before its first copy.  This
    // costs the planner about as much as it saves one attention launch, so only
    // a plan made to serve several launches (decode_attention_plan) does it.
    const long long nrec = small && !warp_mode ? (T < ctas ? T : ctas) : 0;
    if (small && tid == 0)
        s_prefix[p.batch] = total;
    __syncthreads();
    for (long long i = tid; i < nrec; i += nthreads) {
        FirstSeg f;
        const long long s0 = slice_begin(i, W, T), s1 = slice_begin(i + 1, W, T);
        f.s1 = s1;
        if (s0 >= s1) {
            f.d = SegDesc{};
            f.d.num_pages = 0;
            f.se = s0;
        } else {
            // largest b with s_prefix[b] <= s0 / Hkv (a trajectory with pages)
            const long long v = s0 / Hkv;
            int lo = 0, hi = p.batch - 1;
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (s_prefix[mid] <= v)
                    lo = mid;
                else
                    hi = mid - 1;
            }
            f.d = describe_segment(s0, lo, s_prefix[lo], s_prefix[lo + 1], s1, (int)i, W, T, Hkv,
                                   f.se);
            f.d.n = s_len[lo];
        }
        reinterpret_cast<FirstSeg *>(p.first_seg)[i] = f;
    }
    if (tid == 0) {
        p.page_prefix[p.batch] = total;
        p.hdr->total_work = W;
        p.hdr->num_slices = (int)T;
        p.hdr->slice_counter = 0;
        p.hdr->exit_counter = 0;
        p.hdr->first_segs = nrec;
        p.hdr->warp_mode = warp_mode ? 1 : 0;
    }
}

// ------------------------------------------------------------------ attention

template <int D>
struct AttnConfig {
    static constexpr int kStages = D == 128 ? 16 : 32;
    static constexpr int kBoxes = D / 64;                    // 64-element (128 B) TMA boxes per row
    static constexpr int kBoxBytes = kPageSize * 128;        // 16 rows x 128 B
    static constexpr int kKBytes = kBoxes * kBoxBytes;       // one page-head of K
    static constexpr int kStageBytes = 2 * kKBytes;          // K + V
    static constexpr int kQBytes = kMaxGroup * D * 2;        // one segment's query rows (padded)
    static constexpr int kMergeStride = D + 4;               // floats per merge row (bank spread)
    static constexpr size_t kStagesOff = 0;
    static constexpr size_t kQOff = kStagesOff + (size_t)kStages * kStageBytes;
    static constexpr size_t kMergeOOff = kQOff + (size_t)kSegRing * kQBytes;
    static constexpr size_t kMergeMLOff =
        kMergeOOff + (size_t)kNumConsumerWarps * kMaxGroup * kMergeStride * 4;
    static constexpr size_t kDescOff = kMergeMLOff + (size_t)kNumConsumerWarps * kMaxGroup * 2 * 4;
    static constexpr size_t kBarOff = align_up(kDescOff + (size_t)kSegRing * sizeof(SegDesc), 8);
    static constexpr int kNumBars = 2 * kStages + 2 * kSegRing + 1;
    static constexpr size_t kFlagOff = kBarOff + (size_t)kNumBars * 8;
    static constexpr size_t kBytes = kFlagOff + 16 + 1024;  // + slack for 1024-B alignment
};

// A small-batch planner CTA (kPlanThreadsSmall threads) must fit on an SM beside an
// attention CTA, so that the next step's planner can launch while this step's
// attention kernel runs (see plan_kernel): shared memory of both, plus the 1 KB the
// hardware reserves per CTA, within the SM's 228 KB.
constexpr size_t kPlanSmemBytes = (size_t)(kSmallPlanMaxBatch + 1) * sizeof(long long) +
                                  (size_t)kSmallPlanMaxBatch * sizeof(int) +
                                  32 * sizeof(long long) + sizeof(long long);
static_assert(AttnConfig<128>::kBytes + kPlanSmemBytes + 2 * 1024 <= 228 * 1024,
              "the planner no longer fits beside an attention CTA");
static_assert(AttnConfig<64>::kBytes <= AttnConfig<128>::kBytes, "D = 128 is the larger");

// One page-head of a segment for one warp: S^T = K Q^T (16 tokens x 8 query
// heads, mma.sync m16n8k16), online softmax over the page's valid tokens, and
// O^T += V^T P^T.  kbase: the stage's K block (V follows it); tokens at or past
// `valid` are masked and their V rows zeroed (they may hold NaN).
template <int D>
__device__ __forceinline__ void attend_page(uint32_t kbase, int valid,
                                            const uint32_t (&qf)[D / 16][2], float scale_log2,
                                            float &m0, float &m1, float &l0, float &l1,
                                            float (&o)[D / 16][4], int lane)
{
    using C = AttnConfig<D>;
    const int g = lane >> 2, t = lane & 3;    // mma fragment coordinates
    const int mi = lane >> 3, rr = lane & 7;  // ldmatrix: matrix index, row in matrix
    const uint32_t vbase = kbase + C::kKBytes;

    // ---- S^T (16 tokens x 8 heads) = K (16 x D) . Q^T (D x 8)
    float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
    {
        const int row = (mi & 1) * 8 + rr;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
            const int chunk = 2 * kk + (mi >> 1);
            const uint32_t addr = kbase + (chunk >> 3) * C::kBoxBytes + row * 128 +
                                  (((chunk & 7) ^ rr) << 4);
            uint32_t a0, a1, a2, a3;
            ldmatrix_x4(addr, a0, a1, a2, a3);
            if (kk & 1)
                mma_bf16_m16n8k16(sb, a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
            else
                mma_bf16_m16n8k16(sa, a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
        }
    }
    // s[0]: (token g, head 2t)  s[1]: (g, 2t+1)  s[2]: (g+8, 2t)  s[3]: (g+8, 2t+1)
    float s[4];
#pragma unroll
    for (int e = 0; e < 4; ++e)
        s[e] = (sa[e] + sb[e]) * scale_log2;
    if (valid < kPageSize) {
        if (g >= valid) {
            s[0] = -INFINITY;
            s[1] = -INFINITY;
        }
        if (g + 8 >= valid) {
            s[2] = -INFINITY;
            s[3] = -INFINITY;
        }
    }
    float mx0 = fmaxf(s[0], s[2]), mx1 = fmaxf(s[1], s[3]);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(kFull, mx0, off));
        mx1 = fmaxf(mx1, __shfl_xor_sync(kFull, mx1, off));
    }
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float alpha0 = exp2_approx(m0 - mn0), alpha1 = exp2_approx(m1 - mn1);
    m0 = mn0;
    m1 = mn1;
    const float p0 = exp2_approx(s[0] - mn0), p1 = exp2_approx(s[1] - mn1);
    const float p2 = exp2_approx(s[2] - mn0), p3 = exp2_approx(s[3] - mn1);
    l0 = l0 * alpha0 + (p0 + p2);
    l1 = l1 * alpha1 + (p1 + p3);
#pragma unroll
    for (int mt = 0; mt < D / 16; ++mt) {
        o[mt][0] *= alpha0;
        o[mt][1] *= alpha1;
        o[mt][2] *= alpha0;
        o[mt][3] *= alpha1;
    }
    // P^T as the B operand: transpose the two 8x8 (token x head) blocks.
    const uint32_t pb0 = movmatrix_trans(pack_bf16x2(p0, p1));
    const uint32_t pb1 = movmatrix_trans(pack_bf16x2(p2, p3));
    uint32_t mask_lo = 0xffffffffu, mask_hi = 0xffffffffu;
    if (valid < kPageSize) {  // zero value rows past n (they may hold NaN)
        mask_lo = (2 * t < valid ? 0x0000ffffu : 0u) | (2 * t + 1 < valid ? 0xffff0000u : 0u);
        mask_hi = (2 * t + 8 < valid ? 0x0000ffffu : 0u) | (2 * t + 9 < valid ? 0xffff0000u : 0u);
    }
    // ---- O^T (D x 8) += V^T (D x 16 tokens) . P^T (16 x 8)
    {
        const int row = (mi >> 1) * 8 + rr;
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
            const int chunk = 2 * mt + (mi & 1);
            const uint32_t addr = vbase + (chunk >> 3) * C::kBoxBytes + row * 128 +
                                  (((chunk & 7) ^ rr) << 4);
            uint32_t a0, a1, a2, a3;
            ldmatrix_x4_trans(addr, a0, a1, a2, a3);
            a0 &= mask_lo;
            a1 &= mask_lo;
            a2 &= mask_hi;
            a3 &= mask_hi;
            mma_bf16_m16n8k16(o[mt], a0, a1, a2, a3, pb0, pb1);
        }
    }
}

// Largest b in [0, batch) with prefix[b] <= v, given prefix non-decreasing,
// prefix[0] = 0 <= v < prefix[batch].  Whole warp cooperates (32-way search).
__device__ __forceinline__ int warp_find_trajectory(const long long *prefix, int batch,
                                                    long long v, int lane)
{
    int lo = 0, hi = batch - 1;
    while (lo < hi) {
        const int span = hi - lo + 1;
        const int step = (span + 31) / 32;
        const int idx = lo + lane * step;
        const bool pred = idx <= hi && prefix[idx] <= v;
        const unsigned ballot = __ballot_sync(kFull, pred);
        const int last = 31 - __clz(ballot);  // lane 0 always true (prefix[lo] <= v)
        lo = lo + last * step;
        hi = min(hi, lo + step - 1);
    }
    return lo;
}

// All consumer threads (8 warps, 256 threads) arrive and wait; bounded, abort-aware.
__device__ __forceinline__ bool consumer_sync(uint64_t *bar, uint32_t &phase, volatile int *abort)
{
    mbar_arrive(bar);
    const bool ok = mbar_wait(bar, phase, abort);
    phase ^= 1u;
    return __all_sync(kFull, ok);
}

template <int D>
__global__ void __launch_bounds__(kAttnThreads, 1)
    decode_attention_kernel(const AttnParams p, const __grid_constant__ CUtensorMap kmap,
                            const __grid_constant__ CUtensorMap vmap)
{
    using C = AttnConfig<D>;
    constexpr int S = C::kStages;
    static_assert(kIssueGroup <= S, "a parallel issue group must not reuse a stage");
    // The next decode step's planner may launch now: it waits (griddepcontrol.wait)
    // for this whole grid before it touches memory, so its launch latency hides
    // behind this step instead of following it.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // Page i of a segment goes to consumer warp i % kNumConsumerWarps and lands in
    // stage (k + i) % S.  With S a multiple of the warp count, the next use of a
    // stage within a segment belongs to the warp that released its last use, so
    // no warp can wait on a stage two phases ahead, where a parity wait would
    // match the stale phase (the end-of-segment barrier covers segment borders).
    static_assert(S % kNumConsumerWarps == 0, "each stage must be reused by the warp that released it");
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(align_up(reinterpret_cast<size_t>(smem_raw), 1024));
    uint8_t *stages = smem + C::kStagesOff;
    __nv_bfloat16 *qbuf = reinterpret_cast<__nv_bfloat16 *>(smem + C::kQOff);
    float *merge_o = reinterpret_cast<float *>(smem + C::kMergeOOff);
    float *merge_m = reinterpret_cast<float *>(smem + C::kMergeMLOff);
    float *merge_l = merge_m + kNumConsumerWarps * kMaxGroup;
    SegDesc *desc = reinterpret_cast<SegDesc *>(smem + C::kDescOff);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::kBarOff);
    uint64_t *full_bar = bars;
    uint64_t *empty_bar = bars + S;
    uint64_t *seg_full = bars + 2 * S;
    uint64_t *seg_empty = seg_full + kSegRing;
    uint64_t *cons_bar = seg_empty + kSegRing;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + C::kFlagOff);
    volatile int *is_last_flag = abort_flag + 1;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = p.group;
    const int Hkv = p.num_kv_heads;

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int r = 0; r < kSegRing; ++r) {
            mbar_init(&seg_full[r], 1);
            mbar_init(&seg_empty[r], kNumConsumerWarps);
        }
        mbar_init(cons_bar, kNumConsumerWarps * 32);
        *abort_flag = 0;
        *is_last_flag = 0;
        fence_mbarrier_init();
    }
    // Query rows G..7 of every segment slot stay zero (TMA writes rows < G).
    for (int i = tid; i < kSegRing * kMaxGroup * D / 8; i += kAttnThreads) {
        const int row = (i / (D / 8)) % kMaxGroup;
        if (row >= G)
            reinterpret_cast<uint4 *>(qbuf)[i] = make_uint4(0, 0, 0, 0);
    }
    __syncthreads();
    // Everything above overlaps the planner (programmatic dependent launch);
    // from here on the planner's and the append CTAs' writes are visible.
    asm volatile("griddepcontrol.wait;" ::: "memory");

    const long long W = p.hdr->total_work;
    const int T = p.hdr->num_slices;
    const bool warp_mode = p.hdr->warp_mode != 0;

    if (warp == kNumConsumerWarps) {
        // ============================ producer warp ============================
        if (warp_mode)  // every consumer warp loads its own pages
            return;
        if (lane == 0) {
            prefetch_tensor_map(&kmap);
            prefetch_tensor_map(&vmap);
        }
        const uint64_t policy = l2_evict_first_policy();
        const uint32_t q_bytes = (uint32_t)(G * D * 2);
        uint32_t kp = 0;  // page-heads issued
        uint32_t sp = 0;  // segments issued
        bool ok = true;
        // The planner's description of this CTA's first segment, when it wrote one
        // (small batches): the first copies then need no prefix search and no
        // divisions here.
        const bool have_rec = (long long)blockIdx.x < p.hdr->first_segs;
        FirstSeg rec;
        if (have_rec)
            rec = reinterpret_cast<const FirstSeg *>(p.first_seg)[blockIdx.x];
        // Slice i < grid is CTA i's first; later slices come from the counter.
        int slice = blockIdx.x;
        for (bool initial = true; ok; initial = false) {
            if (!initial) {
                if (lane == 0)
                    slice = (int)gridDim.x + atomicAdd(&p.hdr->slice_counter, 1);
                slice = __shfl_sync(kFull, slice, 0);
            }
            if (slice >= T) {
                // This CTA fetches no more slices.  The last CTA to get here puts the
                // slice counter back to zero, so that the next attention launch over
                // the same plan starts from a clean counter (acq_rel: every other
                // CTA's fetches happened before its increment).
                if (lane == 0) {
                    int old;
                    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], 1;"
                                 : "=r"(old) : "l"(&p.hdr->exit_counter) : "memory");
                    if (old == (int)gridDim.x - 1) {
                        p.hdr->slice_counter = 0;
                        p.hdr->exit_counter = 0;
                    }
                }
                break;
            }
            bool use_rec = initial && have_rec;
            long long x = 0, s1;
            int b;
            if (use_rec) {
                if (rec.d.num_pages <= 0)
                    continue;  // an empty slice
                s1 = rec.s1;
                b = rec.d.b;
            } else {
                const long long s0 = slice_begin(slice, W, T);
                s1 = slice_begin(slice + 1, W, T);
                if (s0 >= s1)
                    continue;
                b = warp_find_trajectory(p.page_prefix, p.batch, s0 / Hkv, lane);
                x = s0;
            }
            while (use_rec || x < s1) {
                SegDesc d;
                long long se;
                int max_n = 0;  // > 0: d.n still to be read (and clamped to this)
                if (use_rec) {
                    d = rec.d;
                    se = rec.se;
                    use_rec = false;
                } else {
                    const long long pb0 = p.page_prefix[b], pb1 = p.page_prefix[b + 1];
                    if (x >= pb1 * Hkv) {
                        ++b;
                        continue;
                    }
                    d = describe_segment(x, b, pb0, pb1, s1, slice, W, T, Hkv, se);
                    max_n = (int)((pb1 - pb0) * kPageSize);
                }
                const int npg = d.num_pages;
                const int kvh = d.kvh;
                const int *bt_row = p.block_table + (size_t)d.b * p.max_pages + d.page_begin;
                // Block-table entries come 32 at a time, one chunk ahead of use; the
                // first chunk's load is issued before the length's, so that the two
                // latencies overlap.
                int next_phys = lane < npg ? __ldg(bt_row + lane) : 0;

                const uint32_t r = sp % kSegRing;
                if (sp >= kSegRing) {
                    ok = mbar_wait(&seg_empty[r], ((sp / kSegRing) + 1) & 1, abort_flag);
                    ok = __all_sync(kFull, ok);
                    if (!ok)
                        break;
                }
                if (lane == 0) {
                    if (max_n > 0) {
                        const int n = p.context_lens[d.b];
                        d.n = n < max_n ? n : max_n;
                    }
                    desc[r] = d;
                    mbar_arrive_expect_tx(&seg_full[r], q_bytes);
                    bulk_load(qbuf + (size_t)r * kMaxGroup * D,
                              p.q + ((size_t)d.b * p.num_q_heads + (size_t)kvh * G) * D, q_bytes,
                              &seg_full[r]);
                }
                ++sp;

                for (int c = 0; c < npg && ok; c += 32) {
                    int phys = next_phys;
                    if (c + 32 + lane < npg)
                        next_phys = __ldg(bt_row + c + 32 + lane);
                    if (c + lane < npg) {
                        if (phys < 0 || phys >= p.num_pages) {
                            record_status(&p.hdr->status, CADKV_ERR_OOB);
                            phys = 0;
                        }
                    }
                    const int cnt = min(32, npg - c);
                    // Issue kIssueGroup pages at once, one lane per page: each lane
                    // waits for its own stage to be released and starts its own
                    // copies, so the mbarrier and TMA-issue latencies of a group
                    // overlap instead of adding up page after page.
                    for (int i0 = 0; i0 < cnt; i0 += kIssueGroup) {
                        const int gcnt = min(kIssueGroup, cnt - i0);
                        const int ph = __shfl_sync(kFull, phys, (i0 + lane) & 31);
                        const uint32_t kl = kp + lane;
                        const uint32_t st = kl % S;
                        bool lok = true;
                        if (lane < gcnt) {
                            if (kl >= (uint32_t)S)
                                lok = mbar_wait(&empty_bar[st], ((kl / S) + 1) & 1, abort_flag);
                            if (lok) {
                                uint8_t *kdst = stages + (size_t)st * C::kStageBytes;
                                uint8_t *vdst = kdst + C::kKBytes;
                                const int ph_head = ph * Hkv + kvh;
                                mbar_arrive_expect_tx(&full_bar[st], C::kStageBytes);
                                if (C::kBoxes > 1 && p.whole_page_box) {
                                    // one 4 KB op per block: box {64 cols, 16 tokens, 2 halves}
                                    tma_load_4d(kdst, &kmap, 0, 0, 0, ph_head, &full_bar[st], policy);
                                    tma_load_4d(vdst, &vmap, 0, 0, 0, ph_head, &full_bar[st], policy);
                                } else {
#pragma unroll
                                    for (int bx = 0; bx < C::kBoxes; ++bx) {
                                        tma_load_2d(kdst + bx * C::kBoxBytes, &kmap, bx * 64,
                                                    ph_head * kPageSize, &full_bar[st], policy);
                                        tma_load_2d(vdst + bx * C::kBoxBytes, &vmap, bx * 64,
                                                    ph_head * kPageSize, &full_bar[st], policy);
                                    }
                                }
                            }
                        }
                        ok = __all_sync(kFull, lok);
                        if (!ok) {
                            // copies this group did start must land before we leave
                            if (lane < gcnt && lok) {
                                volatile int never = 0;
                                mbar_wait(&full_bar[st], (kl / S) & 1, &never);
                            }
                            break;
                        }
                        kp += gcnt;
                    }
                }
                if (!ok)
                    break;
                x = se;
            }
        }
        // End-of-work sentinel.
        if (ok) {
            const uint32_t r = sp % kSegRing;
            if (sp >= kSegRing) {
                ok = mbar_wait(&seg_empty[r], ((sp / kSegRing) + 1) & 1, abort_flag);
                ok = __all_sync(kFull, ok);
            }
            if (ok && lane == 0) {
                desc[r].num_pages = -1;
                mbar_arrive(&seg_full[r]);
            }
            if (ok)
                ++sp;  // the sentinel occupies a ring slot like any segment
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
        }
        // Drain: every copy this warp issued must land before the CTA exits.
        if (lane == 0) {
            const uint32_t k_lo = kp > (uint32_t)S ? kp - S : 0;
            for (uint32_t k = k_lo; k < kp; ++k) {
                volatile int never = 0;
                mbar_wait(&full_bar[k % S], (k / S) & 1, &never);
            }
            const uint32_t s_lo = sp > (uint32_t)kSegRing ? sp - kSegRing : 0;
            for (uint32_t s = s_lo; s < sp; ++s) {
                volatile int never = 0;
                mbar_wait(&seg_full[s % kSegRing], (s / kSegRing) & 1, &never);
            }
        }
        return;
    }

    // ================================ consumer warps ================================
    const int g = lane >> 2, t = lane & 3;          // mma fragment coordinates
    const int ct = tid;                             // consumer thread 0..255
    uint32_t k = 0, sc = 0, cphase = 0;
    bool ok = true;
    SegDesc pd{};         // the last partial whose unit may still need its merge
    bool pending = false;
    int pend_old = 0;     // thread 0: the unit counter before pd's partial was counted
    // The CTA that completes a unit merges its partials in slice order.
    auto merge_unit = [&](const SegDesc &u, int first, int stride) {
        const int slot0 = u.unit + u.first;
        for (int it = first; it < G * (D / 8); it += stride) {
            const int h = it / (D / 8), d0 = (it % (D / 8)) * 8;
            // One pass in slice order, rescaling the running sum as the max grows.
            float M = -INFINITY, L = 0.f;
            float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
            for (int s2 = 0; s2 < u.count; ++s2) {
                const size_t sl = (size_t)(slot0 + s2);
                const float lse_s = __ldcg(p.part_lse + sl * G + h);
                const float4 *src = reinterpret_cast<const float4 *>(p.part_o + (sl * G + h) * D + d0);
                const float4 u0 = __ldcg(src), u1 = __ldcg(src + 1);
                const float Mn = fmaxf(M, lse_s);
                const float a = exp2_approx(M - Mn), w = exp2_approx(lse_s - Mn);
                M = Mn;
                L = L * a + w;
                acc[0] = acc[0] * a + w * u0.x;
                acc[1] = acc[1] * a + w * u0.y;
                acc[2] = acc[2] * a + w * u0.z;
                acc[3] = acc[3] * a + w * u0.w;
                acc[4] = acc[4] * a + w * u1.x;
                acc[5] = acc[5] * a + w * u1.y;
                acc[6] = acc[6] * a + w * u1.z;
                acc[7] = acc[7] * a + w * u1.w;
            }
            const float inv = 1.f / L;
            uint4 packed;
            packed.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
            packed.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
            packed.z = pack_bf16x2(acc[4] * inv, acc[5] * inv);
            packed.w = pack_bf16x2(acc[6] * inv, acc[7] * inv);
            const size_t row = (size_t)u.b * p.num_q_heads + u.kvh * G + h;
            *reinterpret_cast<uint4 *>(p.out + row * D + d0) = packed;
            if (d0 == 0 && p.lse)
                p.lse[row] = (M + __log2f(L)) * kLn2;
        }
    };
    auto resolve_pending = [&]() -> bool {
        if (ct == 0)
            *is_last_flag = (pend_old == pd.count - 1) ? 1 : 0;
        if (!consumer_sync(cons_bar, cphase, abort_flag))
            return false;
        if (*is_last_flag) {
            merge_unit(pd, ct, kNumConsumerWarps * 32);
            // every partial of the unit has been counted: clear its counter for
            // the next attention launch over the same plan
            if (ct == 0)
                p.unit_counter[pd.unit] = 0;
        }
        pending = false;
        return true;
    };

    // Trajectories without pages (n_b = 0, or a length outside [0, 16 * max_pages],
    // which the planner reports) get out = 0 and lse = -inf here, each by one
    // thread: trajectory b by CTA b % grid.  The planner writes the same rows; with
    // this, every attention launch completes its own outputs, so one plan can serve
    // several launches (the layers of one decode step).
    {
        const int max_len = p.max_pages * kPageSize;
        const int ncand = ((int)blockIdx.x < p.batch)
                              ? (p.batch - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x
                              : 0;
        for (int c = ct; c < ncand; c += kNumConsumerWarps * 32) {
            const int b = (int)blockIdx.x + c * (int)gridDim.x;
            const int n = p.context_lens[b];
            if (n <= 0 || n > max_len) {
                uint4 *row = reinterpret_cast<uint4 *>(p.out + (size_t)b * p.num_q_heads * D);
                for (int v = 0; v < p.num_q_heads * D / 8; ++v)
                    row[v] = make_uint4(0, 0, 0, 0);
                if (p.lse)
                    for (int h = 0; h < p.num_q_heads; ++h)
                        p.lse[(size_t)b * p.num_q_heads + h] = -INFINITY;
            }
        }
    }

    if (warp_mode) {
        // ======================== per-warp mode (short units) ========================
        // Warp w of CTA c streams slice c * 8 + w alone, with its own stages
        // (w + 8 m, m < S / 8), its own two query slots (w and w + 8) and its own
        // merge tile, and ends each segment alone: no CTA barrier.  Lane 0 issues
        // the copies, at most S / 8 pages and one segment ahead of the warp's
        // consumption; each stage is used by this warp only, in order.
        constexpr int R = S / kNumConsumerWarps;
        static_assert(kSegRing >= 2 * kNumConsumerWarps, "two query slots per warp");
        const long long slice = (long long)blockIdx.x * kNumConsumerWarps + warp;
        if (slice >= T)
            return;
        const long long s0 = slice_begin(slice, W, T), s1 = slice_begin(slice + 1, W, T);
        if (s0 >= s1)
            return;
        if (lane == 0) {
            prefetch_tensor_map(&kmap);
            prefetch_tensor_map(&vmap);
        }
        const uint64_t policy = l2_evict_first_policy();
        const uint32_t q_bytes = (uint32_t)(G * D * 2);
        float *tile = merge_o + (size_t)warp * kMaxGroup * C::kMergeStride;
        float *tile_lse = merge_m + warp * kMaxGroup;

        int bcur = warp_find_trajectory(p.page_prefix, p.batch, s0 / Hkv, lane);
        // The segment that starts at flattened position x (trajectories without
        // pages are skipped); se receives where it ends.
        auto describe_at = [&](long long x, long long &se) -> SegDesc {
            for (;;) {
                const long long pb0 = p.page_prefix[bcur], pb1 = p.page_prefix[bcur + 1];
                if (x >= pb1 * Hkv) {
                    ++bcur;
                    continue;
                }
                SegDesc d = describe_segment(x, bcur, pb0, pb1, s1, (int)slice, W, T, Hkv, se);
                const int n = p.context_lens[bcur];
                const int max_n = (int)((pb1 - pb0) * kPageSize);
                d.n = n < max_n ? n : max_n;
                return d;
            }
        };
        uint32_t jw = 0, jc = 0;  // pages issued / consumed by this warp
        uint32_t ki = 0, kc = 0;  // ordinals of the segments being issued / consumed
        long long di_se, dc_se;
        SegDesc di = describe_at(s0, di_se);
        SegDesc dc = di;
        dc_se = di_se;
        int ii = 0;     // next page of di to issue
        int cb = 0;     // first page of di whose table entry `chunk` holds
        int chunk = 0;  // lane l: physical page of di's page cb + l
        auto load_chunk = [&]() {
            chunk = 0;
            if (cb + lane < di.num_pages) {
                chunk = __ldg(p.block_table + (size_t)di.b * p.max_pages + di.page_begin + cb + lane);
                if (chunk < 0 || chunk >= p.num_pages) {
                    record_status(&p.hdr->status, CADKV_ERR_OOB);
                    chunk = 0;
                }
            }
        };
        auto load_q = [&](const SegDesc &d, uint32_t ord) {
            if (lane == 0) {
                const int slot = warp + kNumConsumerWarps * (int)(ord & 1u);
                // the slot's previous query rows were read (generic proxy) before
                // this copy (async proxy) overwrites them
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                mbar_arrive_expect_tx(&seg_full[slot], q_bytes);
                bulk_load(qbuf + (size_t)slot * kMaxGroup * D,
                          p.q + ((size_t)d.b * p.num_q_heads + (size_t)d.kvh * G) * D, q_bytes,
                          &seg_full[slot]);
            }
        };
        auto issue_more = [&]() {
            while (jw - jc < (uint32_t)R) {
                if (ii == di.num_pages) {
                    if (ki != kc || di_se >= s1)
                        break;  // already one segment ahead, or the slice ends here
                    di = describe_at(di_se, di_se);
                    ++ki;
                    ii = 0;
                    cb = 0;
                    load_chunk();
                    load_q(di, ki);
                }
                if (ii - cb == 32) {
                    cb += 32;
                    load_chunk();
                }
                const int phys = __shfl_sync(kFull, chunk, ii - cb);
                // stage of page jw: its previous use (page jw - R) is consumed
                const uint32_t st = warp + kNumConsumerWarps * (jw % R);
                if (lane == 0) {
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    uint8_t *kdst = stages + (size_t)st * C::kStageBytes;
                    uint8_t *vdst = kdst + C::kKBytes;
                    const int ph_head = phys * Hkv + di.kvh;
                    mbar_arrive_expect_tx(&full_bar[st], C::kStageBytes);
                    if (C::kBoxes > 1 && p.whole_page_box) {
                        tma_load_4d(kdst, &kmap, 0, 0, 0, ph_head, &full_bar[st], policy);
                        tma_load_4d(vdst, &vmap, 0, 0, 0, ph_head, &full_bar[st], policy);
                    } else {
#pragma unroll
                        for (int bx = 0; bx < C::kBoxes; ++bx) {
                            tma_load_2d(kdst + bx * C::kBoxBytes, &kmap, bx * 64,
                                        ph_head * kPageSize, &full_bar[st], policy);
                            tma_load_2d(vdst + bx * C::kBoxBytes, &vmap, bx * 64,
                                        ph_head * kPageSize, &full_bar[st], policy);
                        }
                    }
                }
                ++jw;
                ++ii;
            }
        };

        load_chunk();
        load_q(di, 0);
        issue_more();
        bool wok = true;
        for (;;) {
            const int qslot = warp + kNumConsumerWarps * (int)(kc & 1u);
            wok = __all_sync(kFull, mbar_wait(&seg_full[qslot], (kc >> 1) & 1u, abort_flag));
            if (!wok)
                break;
            uint32_t qf[D / 16][2];
            {
                const __nv_bfloat16 *qs = qbuf + (size_t)qslot * kMaxGroup * D + g * D + 2 * t;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    qf[kk][0] = *reinterpret_cast<const uint32_t *>(qs + 16 * kk);
                    qf[kk][1] = *reinterpret_cast<const uint32_t *>(qs + 16 * kk + 8);
                }
            }
            float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
            float o[D / 16][4];
#pragma unroll
            for (int mt = 0; mt < D / 16; ++mt)
                o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
            for (int i = 0; i < dc.num_pages; ++i) {
                const uint32_t st = warp + kNumConsumerWarps * (jc % R);
                wok = __all_sync(kFull, mbar_wait(&full_bar[st], (jc / R) & 1u, abort_flag));
                if (!wok)
                    break;
                const int valid = min(kPageSize, dc.n - (dc.page_begin + i) * kPageSize);
                attend_page<D>(smem_addr(stages + (size_t)st * C::kStageBytes), valid, qf,
                               p.scale_log2, m0, m1, l0, l1, o, lane);
                __syncwarp();
                ++jc;
                issue_more();
            }
            if (!wok)
                break;

            // ---- the segment's result, from this warp alone
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                l0 += __shfl_xor_sync(kFull, l0, off);
                l1 += __shfl_xor_sync(kFull, l1, off);
            }
            {
                const float inv0 = 1.f / l0, inv1 = 1.f / l1;
#pragma unroll
                for (int mt = 0; mt < D / 16; ++mt) {
                    tile[(2 * t) * C::kMergeStride + 16 * mt + g] = o[mt][0] * inv0;
                    tile[(2 * t + 1) * C::kMergeStride + 16 * mt + g] = o[mt][1] * inv1;
                    tile[(2 * t) * C::kMergeStride + 16 * mt + g + 8] = o[mt][2] * inv0;
                    tile[(2 * t + 1) * C::kMergeStride + 16 * mt + g + 8] = o[mt][3] * inv1;
                }
                if (g == 0) {
                    tile_lse[2 * t] = m0 + __log2f(l0);
                    tile_lse[2 * t + 1] = m1 + __log2f(l1);
                }
            }
            __syncwarp();
            const bool partial = dc.slot >= 0;
            for (int it = lane; it < G * (D / 8); it += 32) {
                const int h = it / (D / 8), d0 = (it % (D / 8)) * 8;
                const float *src = tile + h * C::kMergeStride + d0;
                const float lse2 = tile_lse[h];
                if (!partial) {
                    uint4 packed;
                    packed.x = pack_bf16x2(src[0], src[1]);
                    packed.y = pack_bf16x2(src[2], src[3]);
                    packed.z = pack_bf16x2(src[4], src[5]);
                    packed.w = pack_bf16x2(src[6], src[7]);
                    const size_t row = (size_t)dc.b * p.num_q_heads + dc.kvh * G + h;
                    *reinterpret_cast<uint4 *>(p.out + row * D + d0) = packed;
                    if (d0 == 0 && p.lse)
                        p.lse[row] = lse2 * kLn2;
                } else {
                    float4 *dst = reinterpret_cast<float4 *>(p.part_o + ((size_t)dc.slot * G + h) * D + d0);
                    dst[0] = make_float4(src[0], src[1], src[2], src[3]);
                    dst[1] = make_float4(src[4], src[5], src[6], src[7]);
                    if (d0 == 0)
                        p.part_lse[(size_t)dc.slot * G + h] = lse2;
                }
            }
            __syncwarp();  // the tile is rewritten by the next segment; the partial is complete
            if (partial) {
                // count this partial (release: the warp's stores above, ordered by
                // the warp barrier); the warp that completes the unit merges it
                int old = 0;
                if (lane == 0)
                    asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], 1;"
                                 : "=r"(old) : "l"(&p.unit_counter[dc.unit]) : "memory");
                old = __shfl_sync(kFull, old, 0);
                if (old == dc.count - 1) {
                    __syncwarp();
                    merge_unit(dc, lane, 32);
                    if (lane == 0)
                        p.unit_counter[dc.unit] = 0;
                }
            }

            // ---- on to the next segment (the issuing side may have described it)
            if (ki == kc) {
                if (dc_se >= s1)
                    break;
                di = describe_at(dc_se, di_se);
                ++ki;
                ii = 0;
                cb = 0;
                load_chunk();
                load_q(di, ki);
            }
            dc = di;
            dc_se = di_se;
            ++kc;
            issue_more();
        }
        if (!wok) {
            if (lane == 0) {
                *abort_flag = 1;
                record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
                // every copy this warp started must land before it leaves
                for (uint32_t j = jc; j < jw; ++j) {
                    volatile int never = 0;
                    mbar_wait(&full_bar[warp + kNumConsumerWarps * (j % R)], (j / R) & 1u, &never);
                }
                for (uint32_t o2 = kc; o2 <= ki; ++o2) {
                    volatile int never = 0;
                    mbar_wait(&seg_full[warp + kNumConsumerWarps * (int)(o2 & 1u)], (o2 >> 1) & 1u,
                              &never);
                }
            }
        }
        return;
    }

    for (;;) {
        const uint32_t r = sc % kSegRing;
        ok = __all_sync(kFull, mbar_wait(&seg_full[r], (sc / kSegRing) & 1, abort_flag));
        if (!ok)
            break;
        const SegDesc d = desc[r];
        if (d.num_pages < 0)
            break;

        // B operand of S^T = K Q^T: b0 = Q[g][16kk + 2t .. +1], b1 = Q[g][16kk + 8 + 2t .. +1]
        uint32_t qf[D / 16][2];
        {
            const __nv_bfloat16 *qs = qbuf + (size_t)r * kMaxGroup * D + g * D + 2 * t;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                qf[kk][0] = *reinterpret_cast<const uint32_t *>(qs + 16 * kk);
                qf[kk][1] = *reinterpret_cast<const uint32_t *>(qs + 16 * kk + 8);
            }
        }
        __syncwarp();
        if (lane == 0)
            mbar_arrive(&seg_empty[r]);
        ++sc;

        float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
        float o[D / 16][4];
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt)
            o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;

        const int npg = d.num_pages;
        // Page i of a segment always goes to warp i % kNumConsumerWarps, whatever
        // the CTA did before, so the summation order (and the result) is
        // deterministic.
        for (int i = warp; i < npg; i += kNumConsumerWarps) {
            const uint32_t kk_idx = k + i;
            const uint32_t st = kk_idx % S;
            ok = __all_sync(kFull, mbar_wait(&full_bar[st], (kk_idx / S) & 1, abort_flag));
            if (!ok)
                break;
            const int valid = min(kPageSize, d.n - (d.page_begin + i) * kPageSize);
            attend_page<D>(smem_addr(stages + (size_t)st * C::kStageBytes), valid, qf,
                           p.scale_log2, m0, m1, l0, l1, o, lane);
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&empty_bar[st]);
        }
        if (!ok)
            break;
        k += npg;

        // ---- per-warp totals: l summed over the 8 lanes sharing t
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            l0 += __shfl_xor_sync(kFull, l0, off);
            l1 += __shfl_xor_sync(kFull, l1, off);
        }
        {
            float *mo = merge_o + (size_t)warp * kMaxGroup * C::kMergeStride;
#pragma unroll
            for (int mt = 0; mt < D / 16; ++mt) {
                mo[(2 * t) * C::kMergeStride + 16 * mt + g] = o[mt][0];
                mo[(2 * t + 1) * C::kMergeStride + 16 * mt + g] = o[mt][1];
                mo[(2 * t) * C::kMergeStride + 16 * mt + g + 8] = o[mt][2];
                mo[(2 * t + 1) * C::kMergeStride + 16 * mt + g + 8] = o[mt][3];
            }
            if (g == 0) {
                merge_m[warp * kMaxGroup + 2 * t] = m0;
                merge_m[warp * kMaxGroup + 2 * t + 1] = m1;
                merge_l[warp * kMaxGroup + 2 * t] = l0;
                merge_l[warp * kMaxGroup + 2 * t + 1] = l1;
            }
        }
        ok = consumer_sync(cons_bar, cphase, abort_flag);
        if (!ok)
            break;

        // ---- combine the warps; write the result or this slice's partial
        const bool partial = d.slot >= 0;
        const int q_head0 = d.kvh * G;
        for (int it = ct; it < G * (D / 8); it += kNumConsumerWarps * 32) {
            const int h = it / (D / 8), d0 = (it % (D / 8)) * 8;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kNumConsumerWarps; ++w)
                M = fmaxf(M, merge_m[w * kMaxGroup + h]);
            float L = 0.f, acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int w = 0; w < kNumConsumerWarps; ++w) {
                const float sc_w = exp2_approx(merge_m[w * kMaxGroup + h] - M);
                L += merge_l[w * kMaxGroup + h] * sc_w;
                const float *src = merge_o + ((size_t)w * kMaxGroup + h) * C::kMergeStride + d0;
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    acc[e] += src[e] * sc_w;
            }
            const float inv = 1.f / L;
            const float lse2 = M + __log2f(L);
            if (!partial) {
                uint4 packed;
                packed.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
                packed.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
                packed.z = pack_bf16x2(acc[4] * inv, acc[5] * inv);
                packed.w = pack_bf16x2(acc[6] * inv, acc[7] * inv);
                const size_t row = (size_t)d.b * p.num_q_heads + q_head0 + h;
                *reinterpret_cast<uint4 *>(p.out + row * D + d0) = packed;
                if (d0 == 0 && p.lse)
                    p.lse[row] = lse2 * kLn2;
            } else {
                float4 *dst = reinterpret_cast<float4 *>(p.part_o + ((size_t)d.slot * G + h) * D + d0);
                dst[0] = make_float4(acc[0] * inv, acc[1] * inv, acc[2] * inv, acc[3] * inv);
                dst[1] = make_float4(acc[4] * inv, acc[5] * inv, acc[6] * inv, acc[7] * inv);
                if (d0 == 0)
                    p.part_lse[(size_t)d.slot * G + h] = lse2;
            }
        }
        ok = consumer_sync(cons_bar, cphase, abort_flag);
        if (!ok)
            break;
        // the previous partial's counter update has long completed: merge its
        // unit now if this CTA delivered that unit's last partial
        if (pending) {
            ok = resolve_pending();
            if (!ok)
                break;
        }
        if (!partial)
            continue;

        // ---- count this partial; whether it completes the unit is read after
        // the next segment (or at the end), so the warps go straight on to it
        if (ct == 0) {
            // acq_rel at GPU scope: releases this CTA's partial stores (ordered
            // before it by the barrier above) and acquires every earlier slice's
            asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], 1;"
                         : "=r"(pend_old) : "l"(&p.unit_counter[d.unit]) : "memory");
        }
        pd = d;
        pending = true;
    }
    if (ok && pending)
        ok = resolve_pending();
    if (!ok && lane == 0) {
        *abort_flag = 1;
        record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
    }
}

template <int D>
cudaError_t launch_attention_d(const AttnParams &p, const CUtensorMap &kmap,
                               const CUtensorMap &vmap, int grid, cudaStream_t stream)
{
    static std::atomic<uint64_t> configured{0};
    const size_t smem = AttnConfig<D>::kBytes;
    cudaError_t e = ensure_smem_limit(decode_attention_kernel<D>, (int)smem, configured);
    if (e != cudaSuccess)
        return e;
    // Programmatic dependent launch: may start while the planner still runs.
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decode_attention_kernel<D>, p, kmap, vmap);
}

}  // namespace

DecodeWorkspaceLayout decode_workspace_layout(int batch, int num_kv_heads, int group,
                                              int head_dim, int num_sms)
{
    DecodeWorkspaceLayout L{};
    L.slice_cap = num_sms * kSlicesPerCta;
    L.capacity = batch * num_kv_heads +
                 num_sms * (kSlicesPerCta > kNumConsumerWarps ? kSlicesPerCta : kNumConsumerWarps);
    size_t off = align_up(sizeof(WorkspaceHeader), kWorkspaceAlign);
    L.page_prefix = off;
    off = align_up(off + (size_t)(batch + 1) * sizeof(long long), kWorkspaceAlign);
    L.first_seg = off;
    off = align_up(off + (size_t)num_sms * kFirstSegBytes, kWorkspaceAlign);
    L.unit_counter = off;
    off = align_up(off + (size_t)batch * num_kv_heads * sizeof(int), kWorkspaceAlign);
    L.part_lse = off;
    off = align_up(off + (size_t)L.capacity * group * sizeof(float), kWorkspaceAlign);
    L.part_o = off;
    off = align_up(off + (size_t)L.capacity * group * head_dim * sizeof(float), kWorkspaceAlign);
    L.total = off;
    return L;
}

cudaError_t launch_plan(const PlanParams &p, cudaStream_t stream)
{
    const int append_ctas =
        p.k_new ? (p.batch * p.num_kv_heads + kAppendRowsPerCta - 1) / kAppendRowsPerCta : 0;
    // Programmatic launch: the planner's start overlaps the previous kernel's
    // tail; it waits for that kernel's writes before touching memory.
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(1 + append_ctas);
    cfg.blockDim = dim3(p.threads > 0 ? p.threads : kPlanThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, plan_kernel, p);
}

size_t attention_smem_bytes(int head_dim)
{
    return head_dim == 128 ? AttnConfig<128>::kBytes : AttnConfig<64>::kBytes;
}

cudaError_t launch_attention(const AttnParams &p, const CUtensorMap &kmap,
                             const CUtensorMap &vmap, int head_dim, int grid,
                             cudaStream_t stream)
{
    if (head_dim == 128)
        return launch_attention_d<128>(p, kmap, vmap, grid, stream);
    return launch_attention_d<64>(p, kmap, vmap, grid, stream);
}

}  // namespace cadkv
