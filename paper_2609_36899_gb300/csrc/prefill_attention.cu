// prefill_attention.cu -- chunked (re-)prefill attention over the paged KV pool
// on the 5th-generation tensor cores (tcgen05, accumulators in TMEM).
//
// When prepared KV state cannot be used, the destination recomputes the
// prefix (Sec. 4.4, the fallback of late-bound KV preparation): each
// trajectory's last C_b tokens attend causally over its paged KV.  Unlike the
// decode step this is a dense contraction, so it runs on tcgen05.mma:
//
//  * One CTA per work item (trajectory b, KV head g, 256 query rows).  A row
//    is a (query token, query head of group g) pair, token-major, so the G
//    heads sharing a KV head share every K/V tile (GQA).  The 256 rows form
//    two 128-row tiles, A and B, that share each K/V tile: every K/V byte
//    brought into shared memory feeds twice the MMA work.
//  * Warp 0 (TMA producer) loads the two Q tiles once (3-D tensor map, two
//    64-column panels each, 128-byte swizzle) and streams K and V tiles of 128
//    keys (8 pages, two 2 KB boxes per page and operand, issued from 32 lanes
//    at once) into a 3-stage K ring and a 2-stage V ring; K is released as
//    soon as both S MMAs have read it, so it is loaded a tile ahead of V.
//  * Warp 1 (MMA issuer, one lane) keeps S_A, S_B, O_A, O_B in TMEM (4 x 128
//    fp32 columns).  Per key tile j it issues S_X = Q_X K_j^T and, once the
//    softmax has turned S_X into P_X, O_X += P_X V_j with P_X read straight
//    from TMEM (the MMA form whose A operand lives in tensor memory) and V as
//    an MN-major operand from the swizzled stage.  Tiles A and B alternate, so
//    the tensor cores work on one tile while the softmax works on the other.
//  * Warps 2-5 (tile A) and 6-9 (tile B): one query row per thread = one TMEM
//    lane.  The row's 128 scores come in one burst of tcgen05.ld, causal mask
//    only on tiles that cross the diagonal, running max with lazy O rescaling
//    (only when the max grows by more than 2^8; the decision is warp-uniform
//    since tcgen05.ld/st are warp-collective), P = 2^(s - m) packed to bf16
//    and stored with tcgen05.st over the S columns already consumed.  Finally
//    O / l and lse.
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
constexpr int kItemRows = kRows * kTiles;
constexpr int kKeys = 128;               // keys per tile = MMA N of QK^T, K of PV
constexpr int kD = 128;                  // head_dim
constexpr int kPanel = 16384;            // 128 rows x 128 B (one 64-column panel)
constexpr int kTileBytes = 2 * kPanel;   // 128 rows x 128 columns bf16
constexpr int kPageBlock = kPageSize * kD * 2;  // one (page, head) block: 4 KB
constexpr int kSoftmaxThreads = 128 * kTiles;   // one warpgroup per query tile
constexpr int kPrefillThreads = 64 + kSoftmaxThreads;  // producer, MMA, softmax
constexpr float kRescaleThreshold = 8.0f;  // log2 units
constexpr int kKStages = 3;              // K is freed early (after S), so it runs further ahead
constexpr int kVStages = 2;

struct PrefillSmem {
    uint8_t q[kTiles][kTileBytes];
    uint8_t k[kKStages][kTileBytes];
    uint8_t v[kVStages][kTileBytes];
    uint64_t q_full, s_full[kTiles], p_full[kTiles], o_done[kTiles], k_full[kKStages],
        k_empty[kKStages], v_full[kVStages], v_empty[kVStages], mma_done;
    uint32_t tmem_base;
    int abort;
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

#define CADKV_TMEM_ST16(taddr, r)                                                                   \
    asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,"    \
                 "%11,%12,%13,%14,%15,%16};" ::"r"(taddr),                                        \
                 "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]),       \
                 "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]),   \
                 "r"(r[14]), "r"(r[15])                                                           \
                 : "memory")

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// ------------------------------------------------------------------ planner

__global__ void __launch_bounds__(1024, 1) prefill_plan_kernel(const PrefillParams p)
{
    __shared__ long long warp_sums[32];
    __shared__ long long carry_s;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        p.hdr->status = 0;
        carry_s = 0;
    }
    __syncthreads();
    for (int base = 0; base < p.batch; base += 1024) {
        const int b = base + tid;
        long long items = 0;
        if (b < p.batch) {
            const long long qa = p.q_offsets[b], qb = p.q_offsets[b + 1];
            const long long c = qb - qa;
            const int n = p.context_lens[b];
            if (qa < 0 || qb > p.total_q || c < 0 || n < 0 || c > n ||
                n > p.max_pages * kPageSize) {
                record_status(&p.hdr->status, CADKV_ERR_SHAPE);
            } else {
                const long long tpi = prefill_tokens_per_item(p.group);
                items = (long long)p.num_kv_heads * ((c + tpi - 1) / tpi);
            }
        }
        long long v = items;
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
        const long long incl = carry_s + v + (warp > 0 ? warp_sums[warp - 1] : 0);
        if (b < p.batch)
            p.item_prefix[b] = incl - items;
        __syncthreads();
        if (tid == 1023)
            carry_s = incl;
        __syncthreads();
    }
    if (tid == 0) {
        p.item_prefix[p.batch] = carry_s;
        p.hdr->total_work = carry_s;
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
    const long long total = p.hdr->total_work;
    const long long item = blockIdx.x;
    if (item >= total)
        return;  // uniform across the CTA, before any barrier or TMEM use

    // ---- decode the work item: (trajectory b, KV head g, 256-row query block qt)
    int lo = 0, hi = p.batch - 1;
    while (lo < hi) {  // largest b with item_prefix[b] <= item
        const int mid = (lo + hi + 1) >> 1;
        if (p.item_prefix[mid] <= item)
            lo = mid;
        else
            hi = mid - 1;
    }
    const int b = lo;
    const int G = p.group;
    // a tile holds floor(128 / G) whole tokens (all G heads of each); for G that
    // does not divide 128 the last 128 mod G rows are padding, never written out
    const int tokens_per_tile = kRows / G;
    const int rows_used = tokens_per_tile * G;
    const long long q0 = p.q_offsets[b];
    const int chunk = (int)(p.q_offsets[b + 1] - q0);
    const int n = p.context_lens[b];
    const int qblocks = (chunk + kTiles * tokens_per_tile - 1) / (kTiles * tokens_per_tile);
    const int local = (int)(item - p.item_prefix[b]);
    const int g = local / qblocks;
    const int qt = qblocks - 1 - local % qblocks;  // heaviest blocks first
    const int i0 = qt * kTiles * tokens_per_tile;  // first token of tile A
    const int valid_tokens = min(kTiles * tokens_per_tile, chunk - i0);
    const int chunk_start = n - chunk;
    const int pos_max = chunk_start + i0 + valid_tokens - 1;
    const int num_kt = (pos_max + 1 + kKeys - 1) / kKeys;
    const int last_page = pos_max / kPageSize;  // inclusive

    if (tid == 0) {
        mbar_init(&sm.q_full, 1);
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
        sm.abort = 0;
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

    if (warp == 0) {
        // ============================ TMA producer ============================
        bool ok = true;
        // every (trajectory, KV head)'s K/V is re-read by all its query-block CTAs
        const uint64_t policy = l2_evict_last_policy();
        if (lane == 0) {
            prefetch_tensor_map(&qmap);
            prefetch_tensor_map(&kmap);
            prefetch_tensor_map(&vmap);
            mbar_arrive_expect_tx(&sm.q_full, kTiles * 2 * rows_used * 128);
            for (int t = 0; t < kTiles; ++t) {
                const int qy = (int)(q0 + i0 + t * tokens_per_tile);
                for (int h = 0; h < 2; ++h)
                    tma_load_3d(sm.q[t] + h * kPanel, &qmap, h * 64, g * G, qy, &sm.q_full);
            }
        }
        // Step J issues K_J (lanes 0-15) and V_{J-1} (lanes 16-31): K is freed
        // right after the S MMAs while V waits for PV, so each stream is gated
        // only by its own ring and K runs a tile ahead.  Box = one 64-column
        // panel of one page: page = (lane / 2) % 8, panel = lane % 2.
        const int op = lane >> 4, pg = (lane >> 1) & 7, hh = lane & 1;
        int issued_k = 0, issued_v = 0;
        for (int J = 0; J <= num_kt && ok; ++J) {
            const int jk = J, jv = J - 1;
            const bool do_k = jk < num_kt, do_v = jv >= 0;
            const int pages_k = do_k ? min(kKeys / kPageSize, last_page + 1 - jk * (kKeys / kPageSize)) : 0;
            const int pages_v = do_v ? min(kKeys / kPageSize, last_page + 1 - jv * (kKeys / kPageSize)) : 0;
            if (lane == 0) {
                if (do_k) {
                    const int sk = jk % kKStages;
                    if (jk >= kKStages)
                        ok = mbar_wait(&sm.k_empty[sk], ((jk / kKStages) + 1) & 1, abort_flag);
                    if (ok)
                        mbar_arrive_expect_tx(&sm.k_full[sk], (uint32_t)pages_k * kPageBlock);
                }
                if (do_v && ok) {
                    const int sv = jv % kVStages;
                    if (jv >= kVStages)
                        ok = mbar_wait(&sm.v_empty[sv], ((jv / kVStages) + 1) & 1, abort_flag);
                    if (ok)
                        mbar_arrive_expect_tx(&sm.v_full[sv], (uint32_t)pages_v * kPageBlock);
                }
            }
            ok = __shfl_sync(kFull, ok ? 1 : 0, 0) != 0;
            if (!ok)
                break;
            const int jt = op == 0 ? jk : jv;
            const int pages = op == 0 ? pages_k : pages_v;
            if ((op == 0 ? do_k : do_v) && pg < pages) {
                int phys = p.block_table[(size_t)b * p.max_pages + jt * (kKeys / kPageSize) + pg];
                if (phys < 0 || phys >= p.num_pages) {
                    record_status(&p.hdr->status, CADKV_ERR_OOB);
                    phys = 0;
                }
                const int y = (phys * p.num_kv_heads + g) * kPageSize;
                uint8_t *dst = (op == 0 ? sm.k[jt % kKStages] : sm.v[jt % kVStages]) + hh * kPanel + pg * 2048;
                tma_load_2d(dst, op == 0 ? &kmap : &vmap, hh * 64, y,
                            op == 0 ? &sm.k_full[jt % kKStages] : &sm.v_full[jt % kVStages], policy);
            }
            issued_k += do_k;
            issued_v += do_v;
        }
        if (lane == 0) {
            if (!ok) {
                *abort_flag = 1;
                record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
            }
            // every copy this warp started must land before the CTA exits
            volatile int never = 0;
            mbar_wait(&sm.q_full, 0, &never);
            for (int j = max(0, issued_k - kKStages); j < issued_k; ++j)
                mbar_wait(&sm.k_full[j % kKStages], (j / kKStages) & 1, &never);
            for (int j = max(0, issued_v - kVStages); j < issued_v; ++j)
                mbar_wait(&sm.v_full[j % kVStages], (j / kVStages) & 1, &never);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ============================ MMA issuer ============================
        if (lane == 0) {
            const uint32_t id_qk = idesc_bf16(kRows, kKeys, 0, 0);
            const uint32_t id_pv = idesc_bf16(kRows, kD, 0, 1);
            // The issuing lane shares its SM sub-partition with softmax warps, so
            // every instruction it spends between MMAs can leave the tensor pipe
            // idle.  All operand descriptors share one high word (stride, fixed
            // bits, swizzle); their low words are computed here once and the
            // issue loop below, unrolled over the ring stages, only selects them.
            const uint32_t d_hi = (uint32_t)(desc_sw128(smem_addr(sm.q[0]), 16, 1024) >> 32);
            uint32_t q_lo[kTiles][kD / 16], k_lo[kKStages][kD / 16], v_lo[kVStages][kKeys / 16];
#pragma unroll
            for (int k = 0; k < kD / 16; ++k) {
                const int off = (k >> 2) * kPanel + (k & 3) * 32;
#pragma unroll
                for (int t = 0; t < kTiles; ++t)
                    q_lo[t][k] = (uint32_t)desc_sw128(smem_addr(sm.q[t] + off), 16, 1024);
#pragma unroll
                for (int st = 0; st < kKStages; ++st)
                    k_lo[st][k] = (uint32_t)desc_sw128(smem_addr(sm.k[st] + off), 16, 1024);
            }
#pragma unroll
            for (int k = 0; k < kKeys / 16; ++k)
#pragma unroll
                for (int st = 0; st < kVStages; ++st)
                    v_lo[st][k] = (uint32_t)desc_sw128(smem_addr(sm.v[st] + k * 2048), kPanel, 1024);
            auto desc = [&](uint32_t lo) { return ((uint64_t)d_hi << 32) | lo; };
            auto issue_s = [&](int t, auto stage) {  // S_t = Q_t K^T from K stage `stage`
                constexpr int st = decltype(stage)::value;
#pragma unroll
                for (int k = 0; k < kD / 16; ++k)
                    umma_ss(tmem + t * kRows, desc(q_lo[t][k]), desc(k_lo[st][k]), id_qk, k > 0);
                umma_commit(&sm.s_full[t]);
            };
            auto issue_pv = [&](int t, bool first, auto stage) {  // O_t += P_t V, P_t from TMEM
                constexpr int st = decltype(stage)::value;
#pragma unroll
                for (int k = 0; k < kKeys / 16; ++k)  // keys 16k .. 16k+15 = P columns 8k ..
                    umma_ts(tmem + 256 + t * kRows, tmem + t * kRows + 8 * k, desc(v_lo[st][k]), id_pv,
                            (!first || k > 0) ? 1u : 0u);
                umma_commit(&sm.o_done[t]);
            };
            using S0 = std::integral_constant<int, 0>;
            using S1 = std::integral_constant<int, 1>;
            using S2 = std::integral_constant<int, 2>;
            static_assert(kKStages == 3 && kVStages == 2, "the issue loop is unrolled over 6 tiles");
            bool ok = mbar_wait(&sm.q_full, 0, abort_flag) && mbar_wait(&sm.k_full[0], 0, abort_flag);
            if (ok) {
                tc_fence_after();
                issue_s(0, S0{});
                issue_s(1, S0{});
                umma_commit(&sm.k_empty[0]);
            }
            // one key tile: V_j in V stage sv, K_{j+1} in K stage sk1
            auto step = [&](int j, auto sv_c, auto sk1_c) {
                constexpr int sv = decltype(sv_c)::value, sk1 = decltype(sk1_c)::value;
                const bool more = j + 1 < num_kt;
                // tile A: PV_A(j) once P_A(j) is in TMEM, then S_A(j+1) over it
                ok = mbar_wait(&sm.p_full[0], j & 1, abort_flag) &&
                     mbar_wait(&sm.v_full[sv], (j / kVStages) & 1, abort_flag) &&
                     (!more || mbar_wait(&sm.k_full[sk1], ((j + 1) / kKStages) & 1, abort_flag));
                if (!ok)
                    return;
                tc_fence_after();
                issue_pv(0, j == 0, sv_c);
                if (more)
                    issue_s(0, sk1_c);
                // tile B likewise; then V_j and K_{j+1} are no longer needed
                ok = mbar_wait(&sm.p_full[1], j & 1, abort_flag);
                if (!ok)
                    return;
                tc_fence_after();
                issue_pv(1, j == 0, sv_c);
                umma_commit(&sm.v_empty[sv]);
                if (more) {
                    issue_s(1, sk1_c);
                    umma_commit(&sm.k_empty[sk1]);
                }
            };
            for (int j0 = 0; j0 < num_kt && ok; j0 += 6) {
                // (j mod 2, (j + 1) mod 3) for j = j0 .. j0 + 5, j0 a multiple of 6
                step(j0, S0{}, S1{});
                if (ok && j0 + 1 < num_kt) step(j0 + 1, S1{}, S2{});
                if (ok && j0 + 2 < num_kt) step(j0 + 2, S0{}, S0{});
                if (ok && j0 + 3 < num_kt) step(j0 + 3, S1{}, S1{});
                if (ok && j0 + 4 < num_kt) step(j0 + 4, S0{}, S2{});
                if (ok && j0 + 5 < num_kt) step(j0 + 5, S1{}, S0{});
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
        __syncwarp();
    } else {
        // ============================ softmax warps ============================
        const int t = (warp - 2) >> 2;            // query tile: 0 (A) or 1 (B)
        const int row = 32 * (warp & 3) + lane;   // TMEM lane = row of the tile
        const uint32_t lane_base = (uint32_t)(32 * (warp & 3)) << 16;
        const uint32_t s_col = tmem + lane_base + t * kRows;
        const uint32_t o_col = tmem + lane_base + 256 + t * kRows;
        const int token = t * tokens_per_tile + row / G, head = row % G;
        const bool row_valid = row < rows_used && token < valid_tokens;
        const int pos_row = row_valid ? chunk_start + i0 + token : pos_max;
        const int pos_min = chunk_start + i0 + t * tokens_per_tile;  // first row of the tile
        const float scale = p.scale_log2;
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < num_kt && ok; ++j) {
            ok = __all_sync(kFull, mbar_wait(&sm.s_full[t], j & 1, abort_flag));
            if (!ok)
                break;
            tc_fence_after();
            const int key0 = j * kKeys;
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
            float mx = -INFINITY;
#pragma unroll
            for (int e = 0; e < kKeys; ++e)
                mx = fmaxf(mx, __uint_as_float(r[e]));
            const float m_new = fmaxf(m, mx * scale);
            // Lazy rescaling: keep the stale max unless some lane's grew past the
            // threshold; the decision is warp-uniform (tcgen05.ld/st are collective).
            const bool rescale = __any_sync(kFull, m_new > m + kRescaleThreshold);
            const float alpha = rescale ? exp2_approx(m - m_new) : 1.f;  // 0 on the first tile
            if (rescale) {
                l *= alpha;
                m = m_new;
            }
            // P = 2^(s*scale - m) as bf16 pairs, over S columns already read
            // (masked scores are -inf, so their P is exactly 0)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t packed[16];
#pragma unroll
                for (int e = 0; e < 32; e += 2) {
                    const float p0 = exp2_approx(__uint_as_float(r[32 * c + e]) * scale - m);
                    const float p1 = exp2_approx(__uint_as_float(r[32 * c + e + 1]) * scale - m);
                    l += p0 + p1;
                    packed[e >> 1] = pack_bf16x2(p0, p1);
                }
                CADKV_TMEM_ST16(s_col + c * 16, packed);
            }
            // O_t is stable here (S_t(j) was issued after PV_t(j-1)) and is not read
            // again before PV_t(j), which waits for this tile's p_full.
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
            if (j == num_kt - 1 && t == 0) {
                // Zero V rows past pos_max: those keys may hold NaN (slots past n_b,
                // or pages never loaded) and 0 * NaN would poison the PV sums.
                ok = __all_sync(kFull, mbar_wait(&sm.v_full[j % kVStages], (j / kVStages) & 1, abort_flag));
                if (!ok)
                    break;
                if (key0 + row > pos_max) {
                    for (int h = 0; h < 2; ++h) {
                        uint4 *rz = reinterpret_cast<uint4 *>(sm.v[j % kVStages] + h * kPanel + row * 128);
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
        // ---- epilogue: O / l -> out, lse
        if (ok) {
            ok = __all_sync(kFull, mbar_wait(&sm.o_done[t], (num_kt - 1) & 1, abort_flag));
            tc_fence_after();
        }
        if (ok) {
            const float inv = 1.f / l;
            __nv_bfloat16 *orow = p.out + ((size_t)(q0 + i0 + token) * p.num_q_heads + g * G + head) * kD;
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
                p.lse[(size_t)(q0 + i0 + token) * p.num_q_heads + g * G + head] =
                    (m + __log2f(l)) * kLn2;
        }
        if (!ok && lane == 0) {
            *abort_flag = 1;
            record_status(&p.hdr->status, CADKV_ERR_TIMEOUT);
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

__host__ __device__ long long prefill_tokens_per_item(int group) { return (long long)kTiles * (kRows / group); }

cudaError_t launch_prefill(const PrefillParams &p, const CUtensorMap &qmap, const CUtensorMap &kmap,
                           const CUtensorMap &vmap, int grid, cudaStream_t stream)
{
    static bool configured = false;
    const size_t smem = prefill_smem_bytes();
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(prefill_attention_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess)
            return e;
        configured = true;
    }
    prefill_plan_kernel<<<1, 1024, 0, stream>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || grid == 0)
        return e;
    prefill_attention_kernel<<<grid, kPrefillThreads, smem, stream>>>(p, qmap, kmap, vmap);
    return cudaGetLastError();
}

}  // namespace cadkv
