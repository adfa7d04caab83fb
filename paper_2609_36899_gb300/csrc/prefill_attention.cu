// prefill_attention.cu -- chunked (re-)prefill attention over the paged KV pool
// on the 5th-generation tensor cores (tcgen05, accumulators in TMEM).
//
// When prepared KV state cannot be used, the destination recomputes the
// prefix (Sec. 4.4, the fallback of late-bound KV preparation): each
// trajectory's last C_b tokens attend causally over its paged KV.  Unlike the
// decode step this is a dense contraction, so it runs on tcgen05.mma:
//
//  * A work item is (trajectory b, KV head g, query block of two 128-row
//    tiles A and B).  A row is a (query token, query head of group g) pair,
//    token-major, so the G heads sharing a KV head share every K/V tile (GQA),
//    and tiles A and B share each K/V tile: every K/V byte brought into shared
//    memory feeds twice the MMA work.
//  * Persistent CTAs, one per SM, pull work units in order from a counter:
//    first whole items (so the query blocks of a (trajectory, KV head) run
//    side by side and share its K/V through L2), then the items of the last
//    partial wave cut into pieces of their key tiles, about one per CTA, so
//    that the CTAs that finish first take the remaining work and no SM idles
//    through a last partial wave.  Each piece stores its rows' O / l and
//    log2-lse; the CTA that completes an item last merges its pieces in piece
//    order (deterministic).  Within a CTA the producer warp fetches the units
//    and hands them to the other warps through a small ring; every ring and
//    barrier phase counts the CTA's key tiles or units, so the pipelines run
//    on from one unit to the next.
//  * Warp 2 loads each segment's two Q tiles (3-D tensor map, two 64-column
//    panels each, 128-byte swizzle) once the previous segment's S MMAs are
//    done.  Warp 0 streams K and V tiles of 128 keys (8 pages, issued from 32
//    lanes at once) into a 3-stage K ring and a 2-stage V ring; K is released
//    as soon as both S MMAs have read it, so it is loaded a tile ahead of V.
//    The SM's TMA box rate bounds this kernel (~98 cycles per swizzled 2 KB box,
//    ~144 per 4 KB box, measured), so V comes as one 4 KB box per (page, KV head)
//    block, landing page-major, which its MN-major operand descriptor allows;
//    K's K-major operand needs all 128 keys of a 64-column panel at one
//    stride, so it keeps two 2 KB boxes per page.
//  * Warp 1 (MMA issuer, one lane) keeps S_A, S_B, O_A, O_B in TMEM (4 x 128
//    fp32 columns).  Per key tile j it issues S_X = Q_X K_j^T and, once the
//    softmax has turned S_X into P_X, O_X += P_X V_j with P_X read straight
//    from TMEM (the MMA form whose A operand lives in tensor memory) and V as
//    an MN-major operand from the swizzled stage.  Tiles A and B alternate, so
//    the tensor cores work on one tile while the softmax works on the other.
//  * Warps 4-7 (tile A) and 8-11 (tile B): one query row per thread = one TMEM
//    lane (setmaxnreg gives them 192 registers, the control warps 120).  The
//    row's 128 scores come in one burst of tcgen05.ld, causal mask only on
//    tiles that cross the diagonal.  P = 2^(s - m) is taken against the running
//    max m without a max pass while every P stays below 2^8 (the tile's row sum
//    bounds them); otherwise, and on a row's first tile, the max is taken, m
//    moves and O is rescaled in TMEM (warp-uniform decisions, since tcgen05.ld/st
//    are warp-collective).  P is packed to bf16 and stored with tcgen05.st over
//    the S columns already consumed.  At the end of a segment: O / l and lse,
//    or the piece's partial row.
//  * All waits are bounded; on timeout the kernel records CADKV_ERR_TIMEOUT,
//    waits for its own copies and MMAs, frees TMEM and returns.
#include <cfloat>
#include <cmath>

#include <type_traits>

#include "internal.h"
#include "ptx.cuh"

namespace cadkv {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kRows = 128;               // query rows per tile = MMA M
constexpr int kTiles = 2;                // query tiles per CTA (A and B)
constexpr int kKeys = 128;               // keys per tile = MMA N of QK^T, K of PV
constexpr int kD = 128;                  // head_dim
constexpr int kPanel = 16384;            // 128 rows x 128 B (one 64-column panel)
constexpr int kTileBytes = 2 * kPanel;   // 128 rows x 128 columns bf16
constexpr int kPageBlock = kPageSize * kD * 2;  // one (page, head) block: 4 KB
constexpr int kSoftmaxThreads = 128 * kTiles;   // one warpgroup per query tile
// Warpgroup 0: K/V producer (warp 0), MMA issuer (1), Q loader (2), spare (3);
// warpgroups 1 and 2: softmax of query tiles A and B.
constexpr int kQLoaderWarp = 2;
constexpr int kFirstSoftmaxWarp = 4;
constexpr int kPrefillThreads = 128 + kSoftmaxThreads;
// registers per thread after the split (launch: 168 for 384 threads; the
// sum 128 * 120 + 256 * 192 equals the 384 * 168 the CTA holds).  The softmax
// threads hold a row's 128 scores plus the segment state and spill below 192;
// the control warps need far fewer.
constexpr int kControlRegs = 120;
constexpr int kSoftmaxRegs = 192;
static_assert(128 * kControlRegs + kSoftmaxThreads * kSoftmaxRegs <= kPrefillThreads * 168,
              "register split exceeds the launch allocation");
constexpr float kMaxP = 256.f;  // P against a stale row max stays below 2^8
constexpr int kKStages = 3;              // K is freed early (after S), so it runs further ahead
constexpr int kVStages = 2;
constexpr int kUnitRing = 4;                 // work units handed from the producer to the other warps
constexpr int kUnitReaders = 2 + kSoftmaxThreads / 32;  // Q loader, MMA issuer, softmax warps
constexpr int kMaxPieces = 16;

// A run of key tiles [kt0, kt1) of one work item.
struct Segment {
    long long q0;            // first query row of trajectory b
    int b, g, qt;            // trajectory, KV head, query block
    int kt0, kt1, num_kt;    // this run, and the item's key tile count
    int i0, valid_tokens, chunk_start, pos_max, last_page;
    int split;               // index of the split item, or -1 for a whole item
    int piece;               // piece of the split item
};

struct PrefillSmem {
    uint8_t q[kTiles][kTileBytes];
    uint8_t k[kKStages][kTileBytes];
    uint8_t v[kVStages][kTileBytes];
    uint64_t q_full, q_empty, s_full[kTiles], p_full[kTiles], o_done[kTiles], k_full[kKStages],
        k_empty[kKStages], v_full[kVStages], v_empty[kVStages], mma_done, part_written,
        merge_decided, unit_full[kUnitRing], unit_empty[kUnitRing];
    uint32_t tmem_base;
    int abort;
    int merge_last;
    Segment unit_seg[kUnitRing];  // work units decoded by the producer warp
    int unit_end[kUnitRing];      // 1: no more work
};

__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = (uint64_t)((saddr & 0x3FFFF) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;  // fixed 0b001
    d |= (uint64_t)2 << 61;  // 128-byte swizzle
    return d;
}

// kind::f16 instruction descriptor: bf16 A/B, fp32 D, M x N, operand majors.
__device__ __forceinline__ uint32_t idesc_bf16(int m, int n, int a_mn, int b_mn)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) |
           ((uint32_t)b_mn << 16) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

// D (TMEM) = A (smem descriptor) * B (smem descriptor) [+ D]
__device__ __forceinline__ void umma_ss(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                        uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}

// D (TMEM) = A (TMEM: one row per lane, two bf16 per column) * B (smem) [+ D]
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b,
                                        uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void umma_commit(uint64_t *bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_addr(bar))
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

#define CADKV_TMEM_LD32(taddr, r)                                                                   \
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,"   \
                 "%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,"  \
                 "%31}, [%32];"                                                                   \
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),          \
                   "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),        \
                   "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]),    \
                   "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),    \
                   "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),    \
                   "=r"(r[30]), "=r"(r[31])                                                       \
                 : "r"(taddr))

#define CADKV_TMEM_ST32(taddr, r)                                                                   \
    asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,"    \
                 "%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,"  \
                 "%30,%31,%32};" ::"r"(taddr),                                                    \
                 "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]),       \
                 "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]),   \
                 "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]),            \
                 "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]),            \
                 "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])             \
                 : "memory")

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// ------------------------------------------------------------------ work split

// Key tiles of query block qt of a trajectory whose chunk of C tokens ends at
// position n - 1; block qt holds chunk tokens [qt * tpi, min((qt + 1) * tpi, C)).
__device__ __forceinline__ int block_key_tiles(int n, int C, int tpi, int qt)
{
    const int end = n - C + min((qt + 1) * tpi, C);  // one past the block's last position
    return (end + kKeys - 1) / kKeys;
}


// Work item i: trajectory b, KV head g, query block qt (items are ordered by
// trajectory, then KV head, then query block), all its key tiles.
__device__ Segment item_segment(const PrefillParams &p, long long i, int tokens_per_tile)
{
    Segment s;
    int lo_b = 0, hi_b = p.batch - 1;
    while (lo_b < hi_b) {  // largest b with item_prefix[b] <= i: never an empty trajectory
        const int mid = (lo_b + hi_b + 1) >> 1;
        if (p.item_prefix[mid] <= i)
            lo_b = mid;
        else
            hi_b = mid - 1;
    }
    s.b = lo_b;
    s.q0 = p.q_offsets[s.b];
    const int C = (int)(p.q_offsets[s.b + 1] - s.q0);
    const int n = p.context_lens[s.b];
    const int tpi = kTiles * tokens_per_tile;
    const int qblocks = (C + tpi - 1) / tpi;
    const int local = (int)(i - p.item_prefix[s.b]);
    s.g = local / qblocks;
    s.qt = local - s.g * qblocks;
    s.num_kt = block_key_tiles(n, C, tpi, s.qt);
    s.kt0 = 0;
    s.kt1 = s.num_kt;
    s.i0 = s.qt * tpi;
    s.valid_tokens = min(tpi, C - s.i0);
    s.chunk_start = n - C;
    s.pos_max = s.chunk_start + s.i0 + s.valid_tokens - 1;
    s.last_page = s.pos_max / kPageSize;
    s.split = -1;
    s.piece = 0;
    return s;
}

// Piece k of an item of nk key tiles split `pieces` ways: tiles
// [k nk / pieces, (k + 1) nk / pieces); empty when nk < pieces for some k.
__device__ __forceinline__ int piece_begin(int k, int nk, int pieces)
{
    return (int)((long long)k * nk / pieces);
}

// Work unit u: items [0, dp_items) whole, then piece (u - dp_items) % pieces
// of split item dp_items + (u - dp_items) / pieces.  False for an empty piece.
__device__ bool unit_segment(const PrefillParams &p, long long dp_items, int pieces, long long u,
                             int tokens_per_tile, Segment &s)
{
    if (u < dp_items) {
        s = item_segment(p, u, tokens_per_tile);
        return true;
    }
    const long long v = u - dp_items;
    const int split = (int)(v / pieces), k = (int)(v - (long long)split * pieces);
    s = item_segment(p, dp_items + split, tokens_per_tile);
    s.kt0 = piece_begin(k, s.num_kt, pieces);
    s.kt1 = piece_begin(k + 1, s.num_kt, pieces);
    s.split = split;
    s.piece = k;
    return s.kt0 < s.kt1;
}

// The CTA's k-th segment as the producer warp decoded and published it
// (bounded wait); false at the end of the work or when the wait gave up.  The
// caller releases the ring slot once it has read it.
__device__ __forceinline__ bool read_segment(PrefillSmem &sm, long long k, volatile int *abort_flag,
                                             bool &ok, Segment &sg)
{
    const int slot = (int)(k % kUnitRing);
    ok = mbar_wait(&sm.unit_full[slot], (uint32_t)(k / kUnitRing) & 1, abort_flag);
    if (!ok || sm.unit_end[slot])
        return false;
    sg = sm.unit_seg[slot];
    return true;
}

// ------------------------------------------------------------------ planner

// In-place exclusive scan of a[0..n) by one 1024-thread block; a[n] = total.
__device__ void block_exclusive_scan(long long *a, int n, long long *warp_sums, long long *carry)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0)
        *carry = 0;
    __syncthreads();
    for (int base = 0; base < n; base += 1024) {
        const int i = base + tid;
        const long long x = i < n ? a[i] : 0;
        long long v = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long u = __shfl_up_sync(kFull, v, o);
            if (lane >= o)
                v += u;
        }
        if (lane == 31)
            warp_sums[warp] = v;
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
        const long long incl = *carry + v + (warp > 0 ? warp_sums[warp - 1] : 0);
        if (i < n)
            a[i] = incl - x;
        __syncthreads();
        if (tid == 1023)
            *carry = incl;
        __syncthreads();
    }
    if (tid == 0)
        a[n] = *carry;
    __syncthreads();
}

__global__ void __launch_bounds__(1024, 1) prefill_plan_kernel(const PrefillParams p)
{
    __shared__ long long warp_sums[32];
    __shared__ long long carry_s;
    // Let the attention kernel launch now: it sets up its barriers and tensor
    // memory, then waits (griddepcontrol.wait) for this grid before it reads
    // anything written here.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int tid = threadIdx.x;
    if (tid == 0) {
        p.hdr->status = 0;
        p.hdr->slice_counter = 0;  // next work unit
    }
    for (int i = tid; i < p.num_ctas; i += 1024)
        p.merge_counter[i] = 0;
    const int tpi = kTiles * (kRows / p.group);
    for (int b = tid; b < p.batch; b += 1024) {  // work items per trajectory
        const long long qa = p.q_offsets[b], qb = p.q_offsets[b + 1];
        const long long c = qb - qa;
        const int n = p.context_lens[b];
        long long qblocks = 0;
        if (qa < 0 || qb > p.total_q || c < 0 || n < 0 || c > n || n > p.max_pages * kPageSize)
            record_status(&p.hdr->status, CADKV_ERR_SHAPE);
        else
            qblocks = (c + tpi - 1) / tpi;
        p.item_prefix[b] = (long long)p.num_kv_heads * qblocks;
    }
    __syncthreads();
    block_exclusive_scan(p.item_prefix, p.batch, warp_sums, &carry_s);
    // The items of the last partial wave (all of them when there are fewer
    // items than CTAs) are cut into pieces; sum their key tiles in parallel.
    __shared__ unsigned long long tail_tiles_s;
    if (tid == 0)
        tail_tiles_s = 0;
    __syncthreads();
    const long long items = p.item_prefix[p.batch];
    const long long split = items >= p.num_ctas ? items % p.num_ctas : items;
    for (long long i = items - split + tid; i < items; i += 1024) {
        int lo_b = 0, hi_b = p.batch - 1;
        while (lo_b < hi_b) {
            const int mid = (lo_b + hi_b + 1) >> 1;
            if (p.item_prefix[mid] <= i)
                lo_b = mid;
            else
                hi_b = mid - 1;
        }
        const int C = (int)(p.q_offsets[lo_b + 1] - p.q_offsets[lo_b]);
        const int qblocks = (C + tpi - 1) / tpi;
        const int qt = (int)((i - p.item_prefix[lo_b]) % qblocks);
        atomicAdd(&tail_tiles_s, (unsigned long long)block_key_tiles(p.context_lens[lo_b], C, tpi, qt));
    }
    __syncthreads();
    if (tid == 0) {
        // All pieces run in one round (split * pieces <= P): a second round, or
        // merging many pieces, costs more than it balances.  At least 16 key
        // tiles per piece.
        long long pieces = 1;
        if (split > 0) {
            const long long per_item = (long long)tail_tiles_s / split;
            pieces = min((long long)kMaxPieces, max(1ll, (long long)p.num_ctas / split));
            pieces = min(pieces, max(1ll, per_item / 16));
        }
        p.hdr->total_items = items;
        p.hdr->dp_items = items - split;
        p.hdr->pieces = pieces;
        p.hdr->total_work = items - split + split * pieces;  // work units
    }
}

// ------------------------------------------------------------------ attention

__global__ void __launch_bounds__(kPrefillThreads, 1)
    prefill_attention_kernel(const PrefillParams p, const __grid_constant__ CUtensorMap qmap,
                             const __grid_constant__ CUtensorMap kmap,
                             const __grid_constant__ CUtensorMap vmap)
{
    extern __shared__ uint8_t smem_raw[];
    PrefillSmem &sm = *reinterpret_cast<PrefillSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = p.group;
    // a tile holds floor(128 / G) whole tokens (all G heads of each); for G that
    // does not divide 128 the last 128 mod G rows are padding, never written out
    const int tokens_per_tile = kRows / G;
    const int rows_used = tokens_per_tile * G;

    if (tid == 0) {
        mbar_init(&sm.q_full, 1);
        mbar_init(&sm.q_empty, 1);
        for (int t = 0; t < kTiles; ++t) {
            mbar_init(&sm.s_full[t], 1);
            mbar_init(&sm.p_full[t], 128);
            mbar_init(&sm.o_done[t], 1);
        }
        for (int s = 0; s < kKStages; ++s) {
            mbar_init(&sm.k_full[s], 1);
            mbar_init(&sm.k_empty[s], 1);
        }
        for (int s = 0; s < kVStages; ++s) {
            mbar_init(&sm.v_full[s], 1);
            mbar_init(&sm.v_empty[s], 1);
        }
        mbar_init(&sm.mma_done, 1);
        mbar_init(&sm.part_written, kSoftmaxThreads);
        mbar_init(&sm.merge_decided, 1);
        for (int i = 0; i < kUnitRing; ++i) {
            mbar_init(&sm.unit_full[i], 1);
            mbar_init(&sm.unit_empty[i], kUnitReaders);
        }
        sm.abort = 0;
        sm.merge_last = 0;
        fence_mbarrier_init();
    }
    if (rows_used < kRows) {
        // padding rows of both Q tiles: zero them so the MMAs read finite values
        // (the Q copies never write them)
        const int pad = kRows - rows_used;
        for (int i = tid; i < kTiles * 2 * pad * 8; i += kPrefillThreads) {
            const int t = i / (2 * pad * 8), h = (i / (pad * 8)) % 2, r = rows_used + (i / 8) % pad;
            reinterpret_cast<uint4 *>(sm.q[t] + h * kPanel + r * 128)[i % 8] = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(
                         smem_addr(&sm.tmem_base))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem_base;
    // columns: S_A [0,128), S_B [128,256), O_A [256,384), O_B [384,512); P_X is
    // written over the first 64 columns of S_X (two bf16 per column).
    volatile int *abort_flag = &sm.abort;
    // Everything above overlaps the planner (programmatic dependent launch);
    // from here on its writes are visible.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long long units = p.hdr->total_work, dp_items = p.hdr->dp_items;
    const int pieces = (int)p.hdr->pieces;
    if (blockIdx.x < units) {  // uniform across the CTA
    // Registers move from the control warpgroup to the softmax warpgroups,
    // which hold a row's 128 scores plus the segment state; each warpgroup
    // changes its allocation at the top of its own branch.
    if (warp < kFirstSoftmaxWarp) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kControlRegs));
    if (warp == 0) {
        // ============================ K/V producer ============================
        bool ok = true;
        // every (trajectory, KV head)'s K/V is re-read by all its query blocks
        const uint64_t policy = l2_evict_last_policy();
        if (lane == 0) {
            prefetch_tensor_map(&kmap);
            prefetch_tensor_map(&vmap);
        }
        // Step J of a segment issues its K_J (lanes 0-15) and V_{J-1} (lanes
        // 16-31): K is freed right after the S MMAs while V waits for PV, so each
        // stream is gated only by its own ring and K runs a tile ahead.  Page =
        // (lane / 2) % 8; a K box is the 64-column panel lane % 2 of it, a V box
        // the whole 4 KB block (issued by the even lane).
        const int op = lane >> 4, pg = (lane >> 1) & 7, hh = lane & 1;
        int nk = 0, nv = 0;  // K and V tiles this CTA has loaded
        for (long long k = 0; ok; ++k) {
            // fetch the CTA's next non-empty work unit, decode it once and hand
            // the segment to the other warps
            const int slot = (int)(k % kUnitRing);
            if (lane == 0) {
                if (k >= kUnitRing)
                    ok = mbar_wait(&sm.unit_empty[slot], (uint32_t)((k / kUnitRing) + 1) & 1, abort_flag);
                int end = 1;
                while (ok) {
                    const long long u = atomicAdd(&p.hdr->slice_counter, 1);
                    if (u >= units)
                        break;
                    if (unit_segment(p, dp_items, pieces, u, tokens_per_tile, sm.unit_seg[slot])) {
                        end = 0;
                        break;
                    }
                }
                sm.unit_end[slot] = end;
                mbar_arrive(&sm.unit_full[slot]);
            }
            __syncwarp();
            ok = __shfl_sync(kFull, ok ? 1 : 0, 0) != 0;
            if (!ok || sm.unit_end[slot])
                break;
            const Segment sg = sm.unit_seg[slot];
            const int nseg = sg.kt1 - sg.kt0;
            for (int J = 0; J <= nseg && ok; ++J) {
                const bool do_k = J < nseg, do_v = J > 0;
                const int ktk = sg.kt0 + J, ktv = ktk - 1;
                const int pages_k = do_k ? min(kKeys / kPageSize, sg.last_page + 1 - ktk * (kKeys / kPageSize)) : 0;
                const int pages_v = do_v ? min(kKeys / kPageSize, sg.last_page + 1 - ktv * (kKeys / kPageSize)) : 0;
                const int sk = nk % kKStages, sv = nv % kVStages;
                if (lane == 0) {
                    if (do_k) {
                        if (nk >= kKStages)
                            ok = mbar_wait(&sm.k_empty[sk], (uint32_t)((nk / kKStages) + 1) & 1, abort_flag);
                        if (ok)
                            mbar_arrive_expect_tx(&sm.k_full[sk], (uint32_t)pages_k * kPageBlock);
                    }
                    if (do_v && ok) {
                        if (nv >= kVStages)
                            ok = mbar_wait(&sm.v_empty[sv], (uint32_t)((nv / kVStages) + 1) & 1, abort_flag);
                        if (ok)
                            mbar_arrive_expect_tx(&sm.v_full[sv], (uint32_t)pages_v * kPageBlock);
                    }
                }
                ok = __shfl_sync(kFull, ok ? 1 : 0, 0) != 0;
                if (!ok)
                    break;
                const int kt = op == 0 ? ktk : ktv;
                const int pages = op == 0 ? pages_k : pages_v;
                // V as whole 4 KB (page, head) blocks: one box per page (lane hh == 0),
                // landing page-major ([page][half][16][128 B])
                if ((op == 0 ? do_k : do_v) && pg < pages && (op == 0 || hh == 0)) {
                    int phys = p.block_table[(size_t)sg.b * p.max_pages + kt * (kKeys / kPageSize) + pg];
                    if (phys < 0 || phys >= p.num_pages) {
                        record_status(&p.hdr->status, CADKV_ERR_OOB);
                        phys = 0;
                    }
                    const int y = (phys * p.num_kv_heads + sg.g) * kPageSize;
                    if (op == 1)
                        tma_load_4d(sm.v[sv] + pg * kPageBlock, &vmap, 0, 0, 0, phys * p.num_kv_heads + sg.g,
                                    &sm.v_full[sv], policy);
                    else
                        tma_load_2d(sm.k[sk] + hh * kPanel + pg * 2048, &kmap, hh * 64, y, &sm.k_full[sk],
                                    policy);
                }
                nk += do_k;
                nv += do_v;
            }
        }
        if (lane == 0) {
            if (!ok) {
                *abort_flag = 1;
                record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
            }
            // every copy this warp started must land before the CTA exits
            volatile int never = 0;
            for (int j = max(0, nk - kKStages); j < nk; ++j)
                mbar_wait(&sm.k_full[j % kKStages], (uint32_t)(j / kKStages) & 1, &never);
            for (int j = max(0, nv - kVStages); j < nv; ++j)
                mbar_wait(&sm.v_full[j % kVStages], (uint32_t)(j / kVStages) & 1, &never);
        }
        __syncwarp();
    } else if (warp == kQLoaderWarp) {
        // ============================ Q loader ============================
        if (lane == 0) {
            prefetch_tensor_map(&qmap);
            bool ok = true;
            int seg = 0;
            for (long long k = 0; ok; ++k) {
                Segment sg;
                const bool work = read_segment(sm, k, abort_flag, ok, sg);
                mbar_arrive(&sm.unit_empty[k % kUnitRing]);
                if (!work)
                    break;
                // the previous segment's S MMAs must be done with the Q tiles
                if (seg > 0)
                    ok = mbar_wait(&sm.q_empty, (uint32_t)(seg - 1) & 1, abort_flag);
                if (!ok)
                    break;
                mbar_arrive_expect_tx(&sm.q_full, kTiles * 2 * rows_used * 128);
                for (int t = 0; t < kTiles; ++t) {
                    const int qy = (int)(sg.q0 + sg.i0 + t * tokens_per_tile);
                    for (int h = 0; h < 2; ++h)
                        tma_load_3d(sm.q[t] + h * kPanel, &qmap, h * 64, sg.g * G, qy, &sm.q_full);
                }
                ++seg;
            }
            if (!ok) {
                *abort_flag = 1;
                record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
            }
            volatile int never = 0;
            if (seg > 0)  // the last Q copy this lane started lands before the CTA exits
                mbar_wait(&sm.q_full, (uint32_t)(seg - 1) & 1, &never);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ============================ MMA issuer ============================
        {
            const uint32_t id_qk = idesc_bf16(kRows, kKeys, 0, 0);
            const uint32_t id_pv = idesc_bf16(kRows, kD, 0, 1);
            // The issuing lane shares its SM sub-partition with softmax warps, so
            // every instruction it spends between MMAs can leave the tensor pipe
            // idle.  All operand descriptors share one high word (stride, fixed
            // bits, swizzle); their low words are computed here once and the
            // issue loop below only offsets them: the ring stages are kTileBytes apart.
            // (One step body for every stage keeps the issuing lane's code small.)
            const uint32_t d_hi = (uint32_t)(desc_sw128(smem_addr(sm.q[0]), 16, 1024) >> 32);
            uint32_t q_lo[kTiles][kD / 16], k_lo[1][kD / 16], v_lo[1][kKeys / 16];
#pragma unroll
            for (int k = 0; k < kD / 16; ++k) {
                const int off = (k >> 2) * kPanel + (k & 3) * 32;
#pragma unroll
                for (int t = 0; t < kTiles; ++t)
                    q_lo[t][k] = (uint32_t)desc_sw128(smem_addr(sm.q[t] + off), 16, 1024);
                k_lo[0][k] = (uint32_t)desc_sw128(smem_addr(sm.k[0] + off), 16, 1024);
            }
#pragma unroll
            for (int k = 0; k < kKeys / 16; ++k)
                // keys 16k .. 16k+15 = page k of the page-major V stage: its two
                // 64-column halves are 2 KB apart (LBO), 8-key groups 1 KB (SBO)
                v_lo[0][k] = (uint32_t)desc_sw128(smem_addr(sm.v[0] + k * kPageBlock), 2048, 1024);
            if (lane == 0) {
            auto desc = [&](uint32_t lo_word) { return ((uint64_t)d_hi << 32) | lo_word; };
            constexpr uint32_t kStage16 = kTileBytes >> 4;  // one ring stage in descriptor units
            auto issue_s = [&](int t, uint32_t koff) {  // S_t = Q_t K^T from the K stage at koff
#pragma unroll
                for (int k = 0; k < kD / 16; ++k)
                    umma_ss(tmem + t * kRows, desc(q_lo[t][k]), desc(k_lo[0][k] + koff), id_qk, k > 0);
                umma_commit(&sm.s_full[t]);
            };
            auto issue_pv = [&](int t, bool first, uint32_t voff) {  // O_t += P_t V, P_t from TMEM
#pragma unroll
                for (int k = 0; k < kKeys / 16; ++k)  // keys 16k .. 16k+15 = P columns 8k ..
                    umma_ts(tmem + 256 + t * kRows, tmem + t * kRows + 8 * k, desc(v_lo[0][k] + voff), id_pv,
                            (!first || k > 0) ? 1u : 0u);
            };
            bool ok = true;
            // one key tile, the CTA's n-th, j-th of a segment of nseg tiles: V in V
            // stage sv = n % 2, the next tile's K in K stage sk1 = (n + 1) % 3;
            // ph_p = n & 1, ph_v = (n / 2) & 1 and ph_k1 = ((n + 1) / 3) & 1 are the phases
            auto step = [&](uint32_t ph_p, uint32_t ph_v, uint32_t ph_k1, int j, int nseg, int sv, int sk1) {
                const bool more = j + 1 < nseg;
                const uint32_t voff = (uint32_t)sv * kStage16, koff = (uint32_t)sk1 * kStage16;
                // tile A: PV_A once P_A is in TMEM, then the next S_A over it
                ok = mbar_wait(&sm.p_full[0], ph_p, abort_flag) &&
                     mbar_wait(&sm.v_full[sv], ph_v, abort_flag) &&
                     (!more || mbar_wait(&sm.k_full[sk1], ph_k1, abort_flag));
                if (!ok)
                    return;
                tc_fence_after();
                issue_pv(0, j == 0, voff);
                if (!more)
                    umma_commit(&sm.o_done[0]);
                if (more)
                    issue_s(0, koff);
                // tile B likewise; then this V and the next K are no longer needed
                ok = mbar_wait(&sm.p_full[1], ph_p, abort_flag);
                if (!ok)
                    return;
                tc_fence_after();
                issue_pv(1, j == 0, voff);
                if (!more)
                    umma_commit(&sm.o_done[1]);
                umma_commit(&sm.v_empty[sv]);
                if (more) {
                    issue_s(1, koff);
                    umma_commit(&sm.k_empty[sk1]);
                    if (j + 2 == nseg)  // that was the segment's last S: Q is free
                        umma_commit(&sm.q_empty);
                }
            };
            long long n0 = 0;  // key tiles of this CTA before the current segment
            int seg = 0;
            for (long long k = 0; ok; ++k) {
                Segment sg;
                const bool work = read_segment(sm, k, abort_flag, ok, sg);
                mbar_arrive(&sm.unit_empty[k % kUnitRing]);
                if (!work)
                    break;
                const int nseg = sg.kt1 - sg.kt0;
                const int sk = (int)(n0 % kKStages);
                ok = mbar_wait(&sm.q_full, (uint32_t)seg & 1, abort_flag) &&
                     mbar_wait(&sm.k_full[sk], (uint32_t)(n0 / kKStages) & 1, abort_flag);
                if (!ok)
                    break;
                tc_fence_after();
                issue_s(0, (uint32_t)sk * kStage16);
                issue_s(1, (uint32_t)sk * kStage16);
                umma_commit(&sm.k_empty[sk]);
                if (nseg == 1)
                    umma_commit(&sm.q_empty);
                // ring phases of tile n0, then advanced one tile at a time (no
                // divisions on the issuing lane's path)
                uint32_t ph_p = (uint32_t)n0 & 1, ph_v = (uint32_t)(n0 / kVStages) & 1,
                         ph_k1 = (uint32_t)((n0 + 1) / kKStages) & 1;
                int sv = (int)(n0 & 1), sk1 = (int)((n0 + 1) % kKStages);
                for (int j = 0; j < nseg && ok; ++j) {
                    step(ph_p, ph_v, ph_k1, j, nseg, sv, sk1);
                    ph_p ^= 1;
                    ph_v ^= (uint32_t)sv;  // V stage 1 -> 0 wraps the ring
                    sv ^= 1;
                    sk1 = sk1 == kKStages - 1 ? 0 : sk1 + 1;
                    ph_k1 ^= sk1 == 0 ? 1u : 0u;  // the next K stage wrapped
                }
                n0 += nseg;
                ++seg;
            }
            if (!ok) {
                *abort_flag = 1;
                record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
            }
            // all MMAs this thread issued complete before TMEM is freed
            umma_commit(&sm.mma_done);
            volatile int never = 0;
            mbar_wait(&sm.mma_done, 0, &never);
            }
        }
        __syncwarp();
    }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kSoftmaxRegs));
        // ============================ softmax warps ============================
        const int t = (warp - kFirstSoftmaxWarp) >> 2;  // query tile: 0 (A) or 1 (B)
        const int row = 32 * (warp & 3) + lane;   // TMEM lane = row of the tile
        const int prow = t * kRows + row;         // row of the 256-row partial
        const uint32_t lane_base = (uint32_t)(32 * (warp & 3)) << 16;
        const uint32_t s_col = tmem + lane_base + t * kRows;
        const uint32_t o_col = tmem + lane_base + 256 + t * kRows;
        const int head = row % G;
        const int token = t * tokens_per_tile + row / G;  // within the query block
        const float scale = p.scale_log2;
        bool ok = true;
        long long n0 = 0;
        int seg = 0, pieces_done = 0;
        for (long long k = 0; ok; ++k) {
            bool got;
            Segment sg;
            const bool work = __all_sync(kFull, read_segment(sm, k, abort_flag, got, sg));
            ok = __all_sync(kFull, got);
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&sm.unit_empty[k % kUnitRing]);
            if (!work)
                break;
            const int nseg = sg.kt1 - sg.kt0;
            const bool row_valid = row < rows_used && token < sg.valid_tokens;
            const int pos_row = row_valid ? sg.chunk_start + sg.i0 + token : sg.pos_max;
            const int pos_min = sg.chunk_start + sg.i0 + t * tokens_per_tile;  // first row of the tile
            float m = -INFINITY, l = 0.f;
            for (int j = 0; j < nseg && ok; ++j) {
                const long long n = n0 + j;
                ok = __all_sync(kFull, mbar_wait(&sm.s_full[t], (uint32_t)n & 1, abort_flag));
                if (!ok)
                    break;
                tc_fence_after();
                const int kt = sg.kt0 + j;
                const int key0 = kt * kKeys;
                const bool full_tile = key0 + kKeys - 1 <= pos_min;  // no key masked for any row
                // the row's 128 scores in one burst of loads, one wait
                uint32_t r[kKeys];
                CADKV_TMEM_LD32(s_col + 0, r);
                CADKV_TMEM_LD32(s_col + 32, (r + 32));
                CADKV_TMEM_LD32(s_col + 64, (r + 64));
                CADKV_TMEM_LD32(s_col + 96, (r + 96));
                tmem_wait_ld();
                if (!full_tile) {  // causal mask on tiles that cross the diagonal
#pragma unroll
                    for (int e = 0; e < kKeys; ++e)
                        if (key0 + e > pos_row)
                            r[e] = __float_as_uint(-INFINITY);
                }
                // P = 2^(s*scale - m) against the running max m, without a max pass:
                // while every P stays below 2^8 (the tile's row sum bounds them) m is
                // kept; otherwise (and on a row's first tile) the max is taken, m
                // moves to it and P is recomputed.  Masked scores are -inf: P = 0.
                bool rescale = false;
                float alpha = 1.f;
                float lt = 0.f;
                bool fresh = __any_sync(kFull, !(m > -INFINITY));
                if (!fresh) {
                    const float m_use = m;
                    const uint64_t sc2 = ((uint64_t)__float_as_uint(scale) << 32) | __float_as_uint(scale);
                    const uint64_t nm2 = ((uint64_t)__float_as_uint(-m_use) << 32) | __float_as_uint(-m_use);
                    uint64_t l2 = 0;
#pragma unroll
                    for (int c2 = 0; c2 < 2; ++c2) {
                        uint32_t packed[32];
#pragma unroll
                        for (int e = 0; e < 64; e += 2) {
                            const uint64_t x = ((uint64_t)r[64 * c2 + e + 1] << 32) | r[64 * c2 + e];
                            uint64_t y;
                            asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(y) : "l"(x), "l"(sc2), "l"(nm2));
                            const float p0 = exp2_approx(__uint_as_float((uint32_t)y));
                            const float p1 = exp2_approx(__uint_as_float((uint32_t)(y >> 32)));
                            const uint64_t pp = ((uint64_t)__float_as_uint(p1) << 32) | __float_as_uint(p0);
                            asm("add.f32x2 %0, %1, %2;" : "=l"(l2) : "l"(l2), "l"(pp));
                            packed[e >> 1] = pack_bf16x2(p0, p1);
                        }
                        CADKV_TMEM_ST32(s_col + c2 * 32, packed);
                    }
                    lt = __uint_as_float((uint32_t)l2) + __uint_as_float((uint32_t)(l2 >> 32));
                    fresh = __any_sync(kFull, !(lt <= kMaxP));
                }
                if (fresh) {
                    float mx = -INFINITY;
#pragma unroll
                    for (int e = 0; e < kKeys; ++e)
                        mx = fmaxf(mx, __uint_as_float(r[e]));
                    const float m_new = fmaxf(m, mx * scale);
                    // a row whose keys so far are all masked keeps m = -inf, l = 0, P = 0
                    rescale = __any_sync(kFull, m_new > m);
                    alpha = (m_new > m && m_new > -INFINITY) ? exp2_approx(m - m_new) : 1.f;
                    l *= alpha;
                    m = fmaxf(m, m_new);
                    const float m_use = m > -INFINITY ? m : 0.f;
                    const uint64_t sc2 = ((uint64_t)__float_as_uint(scale) << 32) | __float_as_uint(scale);
                    const uint64_t nm2 = ((uint64_t)__float_as_uint(-m_use) << 32) | __float_as_uint(-m_use);
                    uint64_t l2 = 0;
#pragma unroll
                    for (int c2 = 0; c2 < 2; ++c2) {
                        uint32_t packed[32];
#pragma unroll
                        for (int e = 0; e < 64; e += 2) {
                            const uint64_t x = ((uint64_t)r[64 * c2 + e + 1] << 32) | r[64 * c2 + e];
                            uint64_t y;
                            asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(y) : "l"(x), "l"(sc2), "l"(nm2));
                            const float p0 = exp2_approx(__uint_as_float((uint32_t)y));
                            const float p1 = exp2_approx(__uint_as_float((uint32_t)(y >> 32)));
                            const uint64_t pp = ((uint64_t)__float_as_uint(p1) << 32) | __float_as_uint(p0);
                            asm("add.f32x2 %0, %1, %2;" : "=l"(l2) : "l"(l2), "l"(pp));
                            packed[e >> 1] = pack_bf16x2(p0, p1);
                        }
                        CADKV_TMEM_ST32(s_col + c2 * 32, packed);
                    }
                    lt = __uint_as_float((uint32_t)l2) + __uint_as_float((uint32_t)(l2 >> 32));
                }
                l += lt;
                // O_t is stable here (this S_t was issued after the previous PV_t)
                // and is not read again before the next PV_t, which waits for p_full.
                if (rescale && j > 0) {
                    for (int c = 0; c < 4; ++c) {
                        uint32_t o[32];
                        CADKV_TMEM_LD32(o_col + c * 32, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e)
                            o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                        CADKV_TMEM_ST32(o_col + c * 32, o);
                    }
                }
                tmem_wait_st();
                if (kt == sg.num_kt - 1 && t == 0) {
                    // Zero V rows past pos_max: those keys may hold NaN (slots past n_b,
                    // or pages never loaded) and 0 * NaN would poison the PV sums.
                    // PV_B of this tile is issued after PV_A, which waits for this.
                    const int sv = (int)(n % kVStages);
                    ok = __all_sync(kFull, mbar_wait(&sm.v_full[sv], (uint32_t)(n / kVStages) & 1, abort_flag));
                    if (!ok)
                        break;
                    if (key0 + row > sg.pos_max) {
                        for (int h = 0; h < 2; ++h) {
                            uint4 *rz = reinterpret_cast<uint4 *>(sm.v[sv] + (row >> 4) * kPageBlock +
                                                                  h * 2048 + (row & 15) * 128);
#pragma unroll
                            for (int c16 = 0; c16 < 8; ++c16)
                                rz[c16] = make_uint4(0, 0, 0, 0);
                        }
                    }
                    fence_proxy_async_smem();
                }
                tc_fence_before();
                mbar_arrive(&sm.p_full[t]);
            }
            // ---- end of segment: O / l -> out, lse; or the piece's partial row
            if (ok) {
                ok = __all_sync(kFull, mbar_wait(&sm.o_done[t], (uint32_t)seg & 1, abort_flag));
                tc_fence_after();
            }
            const bool whole = sg.kt0 == 0 && sg.kt1 == sg.num_kt;  // uniform across the CTA
            const size_t out_row = (size_t)(sg.q0 + sg.i0 + token) * p.num_q_heads + sg.g * G + head;
            if (ok && whole) {
                const float inv = 1.f / l;
                __nv_bfloat16 *orow = p.out + out_row * kD;
                for (int c = 0; c < 4; ++c) {
                    uint32_t o[32];
                    CADKV_TMEM_LD32(o_col + c * 32, o);
                    tmem_wait_ld();
                    if (row_valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(orow + c * 32);
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) {
                            uint4 v;
                            v.x = pack_bf16x2(__uint_as_float(o[8 * q4 + 0]) * inv, __uint_as_float(o[8 * q4 + 1]) * inv);
                            v.y = pack_bf16x2(__uint_as_float(o[8 * q4 + 2]) * inv, __uint_as_float(o[8 * q4 + 3]) * inv);
                            v.z = pack_bf16x2(__uint_as_float(o[8 * q4 + 4]) * inv, __uint_as_float(o[8 * q4 + 5]) * inv);
                            v.w = pack_bf16x2(__uint_as_float(o[8 * q4 + 6]) * inv, __uint_as_float(o[8 * q4 + 7]) * inv);
                            dst[q4] = v;
                        }
                    }
                }
                if (row_valid && p.lse)
                    p.lse[out_row] = (m + __log2f(l)) * kLn2;
            } else if (ok) {
                // A piece of a split item: its rows go to the piece's own slot.
                const int slot = sg.split * pieces + sg.piece;
                const float inv = l > 0.f ? 1.f / l : 0.f;
                // column-major ([column][row]): a warp's stores and the merge's loads
                // cover 32 consecutive rows of one column (coalesced)
                float *po = p.partial_o + (size_t)slot * kD * kSoftmaxThreads + prow;
                for (int c = 0; c < 4; ++c) {
                    uint32_t o[32];
                    CADKV_TMEM_LD32(o_col + c * 32, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        po[(size_t)(c * 32 + e) * kSoftmaxThreads] = __uint_as_float(o[e]) * inv;
                }
                p.partial_lambda[(size_t)slot * kSoftmaxThreads + prow] = l > 0.f ? m + __log2f(l) : -INFINITY;
                __threadfence();
                // the first softmax thread counts the piece once all 256 rows are out
                tc_fence_before();
                mbar_arrive(&sm.part_written);
                const int nonempty = min(sg.num_kt, pieces);  // pieces holding key tiles
                if (tid == 32 * kFirstSoftmaxWarp) {
                    ok = mbar_wait(&sm.part_written, (uint32_t)pieces_done & 1, abort_flag);
                    if (ok) {
                        __threadfence();
                        const int prev = atomicAdd(&p.merge_counter[sg.split], 1);
                        sm.merge_last = prev == nonempty - 1;  // every other piece is out
                        __threadfence();
                    }
                    mbar_arrive(&sm.merge_decided);
                }
                ok = ok && __all_sync(kFull, mbar_wait(&sm.merge_decided, (uint32_t)pieces_done & 1, abort_flag));
                ++pieces_done;
                if (ok && *reinterpret_cast<volatile int *>(&sm.merge_last)) {
                    // this CTA completes the item: merge the pieces in piece order
                    __threadfence();
                    float lam_max = -INFINITY;
                    for (int k2 = 0; k2 < pieces; ++k2) {
                        if (piece_begin(k2, sg.num_kt, pieces) == piece_begin(k2 + 1, sg.num_kt, pieces))
                            continue;
                        const int s2 = sg.split * pieces + k2;
                        lam_max = fmaxf(lam_max, __ldcg(p.partial_lambda + (size_t)s2 * kSoftmaxThreads + prow));
                    }
                    float wsum = 0.f;
                    for (int k2 = 0; k2 < pieces; ++k2) {
                        if (piece_begin(k2, sg.num_kt, pieces) == piece_begin(k2 + 1, sg.num_kt, pieces))
                            continue;
                        const int s2 = sg.split * pieces + k2;
                        const float lam = __ldcg(p.partial_lambda + (size_t)s2 * kSoftmaxThreads + prow);
                        wsum += lam > -INFINITY ? exp2_approx(lam - lam_max) : 0.f;
                    }
                    const float inv_w = 1.f / wsum;
                    for (int c = 0; c < 4; ++c) {  // 32 columns at a time
                        float acc[32];
#pragma unroll
                        for (int d = 0; d < 32; ++d)
                            acc[d] = 0.f;
                        for (int k2 = 0; k2 < pieces; ++k2) {
                            if (piece_begin(k2, sg.num_kt, pieces) == piece_begin(k2 + 1, sg.num_kt, pieces))
                                continue;
                            const int s2 = sg.split * pieces + k2;
                            const float lam = __ldcg(p.partial_lambda + (size_t)s2 * kSoftmaxThreads + prow);
                            const float w = lam > -INFINITY ? exp2_approx(lam - lam_max) : 0.f;
                            const float *src =
                                p.partial_o + ((size_t)s2 * kD + c * 32) * kSoftmaxThreads + prow;
                            float v[32];
#pragma unroll
                            for (int e = 0; e < 32; ++e)  // all 32 loads in flight at once
                                v[e] = __ldcg(src + (size_t)e * kSoftmaxThreads);
#pragma unroll
                            for (int e = 0; e < 32; ++e)
                                acc[e] += w * v[e];
                        }
                        if (row_valid) {
                            uint4 *dst = reinterpret_cast<uint4 *>(p.out + out_row * kD + c * 32);
#pragma unroll
                            for (int q8 = 0; q8 < 4; ++q8) {
                                uint4 v;
                                v.x = pack_bf16x2(acc[8 * q8 + 0] * inv_w, acc[8 * q8 + 1] * inv_w);
                                v.y = pack_bf16x2(acc[8 * q8 + 2] * inv_w, acc[8 * q8 + 3] * inv_w);
                                v.z = pack_bf16x2(acc[8 * q8 + 4] * inv_w, acc[8 * q8 + 5] * inv_w);
                                v.w = pack_bf16x2(acc[8 * q8 + 6] * inv_w, acc[8 * q8 + 7] * inv_w);
                                dst[q8] = v;
                            }
                        }
                    }
                    if (row_valid) {
                        if (p.lse)
                            p.lse[out_row] = (lam_max + __log2f(wsum)) * kLn2;
                    }
                }
            }
            n0 += nseg;
            ++seg;
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
        }
    }

    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
    }
}

}  // namespace

size_t prefill_smem_bytes() { return sizeof(PrefillSmem) + 1024; }

// setmaxnreg.inc waits until the CTA has the registers it asks for, and it only
// has what it was launched with: a build whose launch allocation is below the
// split would wait forever, so it is refused before launch.
bool prefill_register_split_fits()
{
    static std::atomic<int> fits{-1};
    int f = fits.load();
    if (f < 0) {
        cudaFuncAttributes a{};
        f = cudaFuncGetAttributes(&a, prefill_attention_kernel) == cudaSuccess &&
                    128 * kControlRegs + kSoftmaxThreads * kSoftmaxRegs <= kPrefillThreads * a.numRegs
                ? 1
                : 0;
        fits.store(f);
    }
    return f == 1;
}

cudaError_t launch_prefill(const PrefillParams &p, const CUtensorMap &qmap, const CUtensorMap &kmap,
                           const CUtensorMap &vmap, cudaStream_t stream)
{
    static std::atomic<uint64_t> configured{0};
    const size_t smem = prefill_smem_bytes();
    cudaError_t e = ensure_smem_limit(prefill_attention_kernel, (int)smem, configured);
    if (e != cudaSuccess)
        return e;
    prefill_plan_kernel<<<1, 1024, 0, stream>>>(p);
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    // Programmatic dependent launch: the attention kernel's prologue overlaps the planner.
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(p.num_ctas);
    cfg.blockDim = dim3(kPrefillThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, prefill_attention_kernel, p, qmap, kmap, vmap);
}

}  // namespace cadkv
