/*
 * cadkv.h -- C ABI of libcadkv.so: batched paged-KV decode attention and
 * paged-KV prefix staging on one NVIDIA GB300 (sm_103a).
 *
 * Where the operations come from.  The paper (CadenceRL, a rollout scheduler
 * for asynchronous RL post-training) reshapes the resident batch of every
 * rollout worker.  What that reshaping speeds up is the autoregressive decode
 * step, whose cost is the per-trajectory KV-cache traffic through HBM
 * (Sec. 2.3, Sec. 3.1: as the batch shrinks and contexts grow, KV traffic
 * approaches the memory-bandwidth limit).  The paper takes attention and the
 * paged KV cache from its inference backend (Sec. 5, vLLM with PagedAttention)
 * and prints no formula; this library computes standard scaled dot-product
 * attention for one query token per trajectory over that trajectory's pages:
 *
 *     g = h / G,  G = Hq / Hkv                 (grouped-query attention)
 *     s_t = q[b,h,:] . K[block_table[b][t/P], g, t%P, :] / sqrt(D),  t < n_b
 *     out[b,h,:] = sum_t softmax(s)_t V[block_table[b][t/P], g, t%P, :]
 *     lse[b,h]   = ln sum_t exp(s_t)
 *
 * Prefix staging is phase 1 of the paper's late-bound KV preparation
 * (Sec. 4.4): when a trajectory departs a worker, its KV blocks are gathered
 * from the paged pool into one contiguous per-trajectory buffer (which is then
 * shipped to host memory).  Phase 3 of Sec. 4.4, materialising a staged prefix
 * in a destination pool, is kv_prefix_load.
 *
 * Conventions for every entry point
 * ---------------------------------
 * - Every tensor argument is a DEVICE pointer owned by the caller, unless a
 *   comment says "host".  The library never frees caller memory.  A pool made
 *   with NULL layer pointers owns the pages it allocated and frees them in
 *   kv_pool_destroy.
 * - bf16 is the IEEE bfloat16 bit layout (uint16 storage).
 * - KV pages: per layer, K and V are each [num_pages][Hkv][P][D] bf16,
 *   row-major ("head-major inside a page": one (page, head) block of P*D
 *   elements is contiguous).  P (page_size) must be 16.  D (head_dim) must be
 *   64 or 128.  G = Hq / Hkv must divide exactly and be 1..8.
 * - block_table: int32 [batch][max_pages]; entry j of row b is the physical
 *   page holding tokens 16j .. 16j+15 of trajectory b.  Only the first
 *   ceil(n_b / 16) entries of a row are read.  context_lens: int32 [batch].
 * - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *   stream) and never synchronise, except the *_status functions, which
 *   synchronise `stream` to read the device status word.
 * - Errors found on the host are returned synchronously and nothing is
 *   launched.  Errors that depend on device-resident data (a context length
 *   outside [0, 16*max_pages], a block-table entry outside [0, num_pages), a
 *   device wait that gave up) never fault: the offending trajectory is treated
 *   as empty or its page is replaced by page 0, the result is unspecified for
 *   it, and the code is recorded in a status word inside the workspace, read
 *   back by decode_attention_status / kv_prefix_stage_status.
 * - All pointers must be 16-byte aligned.
 */
#ifndef CADKV_H
#define CADKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st *cadkv_stream_t;

enum cadkv_status {
    CADKV_OK = 0,
    CADKV_ERR_INVALID = -1,     /* null or misaligned pointer, bad argument   */
    CADKV_ERR_SHAPE = -2,       /* sizes disagree; context length out of range */
    CADKV_ERR_CUDA = -3,        /* a CUDA runtime/driver call failed          */
    CADKV_ERR_UNSUPPORTED = -4, /* head_dim, page_size or group not supported */
    CADKV_ERR_OOB = -5,         /* block-table entry outside the pool         */
    CADKV_ERR_TIMEOUT = -6,     /* a bounded device-side wait gave up         */
    CADKV_ERR_WORKSPACE = -7    /* workspace missing or too small             */
};

/* Static English text for a status code (never NULL). */
const char *kv_status_string(int status);

/* ABI version of this header: (major << 16) | minor. */
int cadkv_abi_version(void);

/* Number of SMs the library sizes its persistent grids for on the current
 * device, or a negative status. */
int cadkv_device_sms(void);

/* ------------------------------------------------------------------------ */
/* Paged KV pool (Sec. 2.3 / Sec. 5: the backend's paged KV cache; the       */
/* paper's KV headroom of Sec. 4.1 is counted in these pages).               */
/* ------------------------------------------------------------------------ */

typedef struct cadkv_pool cadkv_pool;

/*
 * Describe (or allocate) a paged KV pool of num_layers layers.
 * k_layers, v_layers: HOST arrays of num_layers device pointers, each to a
 * [num_pages][num_kv_heads][page_size][head_dim] bf16 block owned by the
 * caller; or both NULL, in which case the pool allocates (uninitialised) pages
 * with cudaMalloc on the current device and owns them.
 * On success *pool receives an opaque handle.  Returns CADKV_OK or an error.
 */
int kv_pool_create(cadkv_pool **pool, int num_layers, int num_pages, int page_size,
                   int num_kv_heads, int head_dim, void *const *k_layers,
                   void *const *v_layers);

/* Free the handle (and pages it allocated).  NULL is accepted. */
int kv_pool_destroy(cadkv_pool *pool);

/* Device pointers of one layer's K and V pages (host outputs). */
int kv_pool_layer(const cadkv_pool *pool, int layer, void **k_pages, void **v_pages);

/* Geometry of the pool (host outputs; any may be NULL). */
int kv_pool_geometry(const cadkv_pool *pool, int *num_layers, int *num_pages,
                     int *page_size, int *num_kv_heads, int *head_dim);

/* ------------------------------------------------------------------------ */
/* Decode attention                                                         */
/* ------------------------------------------------------------------------ */

/*
 * Bytes of workspace decode_attention needs for this problem on the current
 * device (partial results of split trajectories, a page prefix sum, arrival
 * counters and the status word).  Returns 0 on invalid sizes.
 */
size_t decode_attention_workspace_size(int batch, int num_q_heads, int num_kv_heads,
                                       int head_dim, int max_pages);

/*
 * One decode step of attention for `batch` trajectories (one query token each):
 * the bandwidth-bound step of autoregressive rollout (Sec. 2.3, Sec. 3.1),
 * with the attention operator and paged KV cache of the paper's inference
 * backend (Sec. 5), as written out at the top of this file.
 *   q            bf16 [batch][num_q_heads][head_dim]
 *   k_pages      bf16 [num_pages][num_kv_heads][16][head_dim]   (one layer)
 *   v_pages      bf16 [num_pages][num_kv_heads][16][head_dim]
 *   block_table  int32 [batch][max_pages]
 *   context_lens int32 [batch]; n_b = 0 gives out = 0 and lse = -inf
 *   out          bf16 [batch][num_q_heads][head_dim]       (written)
 *   lse          fp32 [batch][num_q_heads], natural log of sum exp(s_t);
 *                may be NULL
 *   workspace    >= decode_attention_workspace_size(...) bytes, 256-byte
 *                aligned, caller-owned; contents need no initialisation; one
 *                workspace must not be used by two calls that may overlap on
 *                the GPU.
 * Launches a planner kernel and one persistent attention kernel on `stream`.
 * The split-KV partials of trajectories spread over several CTAs are merged
 * inside the attention kernel by whichever CTA finishes a trajectory's last
 * piece, so no third launch is needed.
 */
int decode_attention(const void *q, const void *k_pages, const void *v_pages,
                     const int32_t *block_table, const int32_t *context_lens,
                     void *out, float *lse, int batch, int num_q_heads,
                     int num_kv_heads, int head_dim, int page_size, int num_pages,
                     int max_pages, void *workspace, size_t workspace_bytes,
                     cadkv_stream_t stream);

/*
 * decode_attention with the work split forced: `slice_pages` > 0 cuts the
 * flattened (trajectory, KV head, page) sequence into slices of at most that
 * many pages (one slice per CTA task), 0 chooses automatically.  The result
 * equals decode_attention's within floating-point tolerance for any value;
 * the tests use it to check split-count invariance.
 */
int decode_attention_split(const void *q, const void *k_pages, const void *v_pages,
                           const int32_t *block_table, const int32_t *context_lens,
                           void *out, float *lse, int batch, int num_q_heads,
                           int num_kv_heads, int head_dim, int page_size,
                           int num_pages, int max_pages, int slice_pages,
                           void *workspace, size_t workspace_bytes,
                           cadkv_stream_t stream);

/*
 * The two launches of decode_attention, exposed separately so a caller can
 * time or graph-capture them apart.  decode_attention_run must follow
 * decode_attention_plan on the same stream with the same context_lens,
 * sizes and workspace.
 *
 * One plan serves several runs.  The plan depends only on the lengths, so a
 * decode step of an L-layer model plans once and runs once per layer, each
 * run with that layer's q, k_pages, v_pages, block_table (same width), out
 * and lse, one after another on the stream: every run leaves the workspace's
 * counters as the plan left them, and writes all of its outputs (out = 0 and
 * lse = -inf for trajectories without pages) itself.  Plan again when the
 * lengths change, when another problem used the workspace, or after a run
 * whose status word reports an error.  The status word keeps the first error
 * of any run since the plan.
 */
int decode_attention_plan(const int32_t *context_lens, void *out, float *lse,
                          int batch, int num_q_heads, int num_kv_heads,
                          int head_dim, int max_pages, int slice_pages,
                          void *workspace, size_t workspace_bytes,
                          cadkv_stream_t stream);
int decode_attention_run(const void *q, const void *k_pages, const void *v_pages,
                         const int32_t *block_table, const int32_t *context_lens,
                         void *out, float *lse, int batch, int num_q_heads,
                         int num_kv_heads, int head_dim, int page_size,
                         int num_pages, int max_pages, void *workspace,
                         size_t workspace_bytes, cadkv_stream_t stream);

/*
 * The whole decode step of one layer: first append each trajectory's new-token
 * key and value, then attend.  n_b = context_lens[b] counts the new token, so
 * k_new[b][h][:] and v_new[b][h][:] (bf16 [batch][num_kv_heads][head_dim]) are
 * written to token position n_b - 1 -- page block_table[b][(n_b - 1) / 16],
 * slot (n_b - 1) % 16 -- of k_pages / v_pages, which are modified in place;
 * trajectories with n_b = 0 append nothing.  Then exactly decode_attention
 * over the updated pages.  The append runs in extra CTAs of the planner
 * launch, so the step is still two launches.  (Sec. 2.3: every decode step
 * extends each trajectory's KV cache by one token before attending over it.)
 * A bad last page is reported as CADKV_ERR_OOB in the status word, and the
 * row is not written.
 */
int decode_attention_append(const void *q, const void *k_new, const void *v_new,
                            void *k_pages, void *v_pages, const int32_t *block_table,
                            const int32_t *context_lens, void *out, float *lse, int batch,
                            int num_q_heads, int num_kv_heads, int head_dim, int page_size,
                            int num_pages, int max_pages, void *workspace,
                            size_t workspace_bytes, cadkv_stream_t stream);

/*
 * Synchronise `stream` and return the device status word the last call that
 * used `workspace` left (CADKV_OK, CADKV_ERR_SHAPE, CADKV_ERR_OOB or
 * CADKV_ERR_TIMEOUT), or CADKV_ERR_CUDA if the copy failed.
 */
int decode_attention_status(const void *workspace, cadkv_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Chunked (re-)prefill attention (Sec. 4.4: the fallback when prepared KV   */
/* state cannot be used and the destination recomputes the prefix)           */
/* ------------------------------------------------------------------------ */

/* Bytes of workspace prefill_attention needs for `batch` trajectories on the
 * current device (it holds, besides per-trajectory counts, partial rows for
 * two pieces per SM: about 0.26 MB per SM). */
size_t prefill_attention_workspace_size(int batch);

/*
 * Causal attention of each trajectory's last C_b tokens over its paged KV.
 *   q          bf16 [total_q][num_q_heads][head_dim]; trajectory b owns rows
 *              q_offsets[b] .. q_offsets[b+1]-1 (C_b of them)
 *   q_offsets  device int64 [batch + 1], q_offsets[0] = 0, non-decreasing,
 *              q_offsets[batch] = total_q
 *   k_pages, v_pages, block_table, context_lens: as decode_attention; the K/V
 *              of the C_b query tokens are already in the pool, at positions
 *              n_b - C_b .. n_b - 1 (so C_b <= n_b)
 *   out        bf16 [total_q][num_q_heads][head_dim]
 *   lse        fp32 [total_q][num_q_heads] or NULL
 * Query row i of trajectory b sits at position p = n_b - C_b + i and attends
 * to keys 0 .. p:  out = softmax_t<=p(q . K_t / sqrt(D)) V,  lse = ln sum exp.
 * Runs on the tcgen05 tensor cores (accumulators in TMEM) with one
 * persistent CTA per SM pulling work items (trajectory, KV head, block of 2 x
 * 128 (query token, head) rows); the items of the last partial wave are cut
 * into pieces of their key tiles whose partial rows are merged, in a fixed
 * order, by the CTA that completes the item.  The workspace must not be used
 * by two calls in flight at once.
 * Supported: head_dim 128, page_size 16, G = Hq / Hkv in 1..8 (the Qwen3
 * models of Sec. 6 have G = 4, 5 and 8); anything else returns
 * CADKV_ERR_UNSUPPORTED, as does a driver that cannot describe V as whole
 * 4 KB (page, KV head) blocks (a 4-D tensor map: V is loaded one block per
 * TMA box), or a build whose kernel was given fewer registers per thread at
 * launch than its warp roles divide among themselves (checked once, before
 * the first launch).
 * A trajectory with C_b > n_b or n_b out of range is skipped (its rows are
 * not written) and CADKV_ERR_SHAPE lands in the status word.
 */
int prefill_attention(const void *q, const int64_t *q_offsets, const void *k_pages,
                      const void *v_pages, const int32_t *block_table,
                      const int32_t *context_lens, void *out, float *lse, int batch,
                      int total_q, int num_q_heads, int num_kv_heads, int head_dim,
                      int page_size, int num_pages, int max_pages, void *workspace,
                      size_t workspace_bytes, cadkv_stream_t stream);

/* As decode_attention_status, for a prefill workspace. */
int prefill_attention_status(const void *workspace, cadkv_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Prefix staging (Sec. 4.4, phase 1) and its inverse (Sec. 4.4, phase 3)    */
/* ------------------------------------------------------------------------ */

/* Bytes of workspace kv_prefix_stage / kv_prefix_load need for `batch`. */
size_t kv_prefix_stage_workspace_size(int batch);

/*
 * Gather the first n_b tokens of layers [layer_begin, layer_end) of every
 * trajectory b from the pool into contiguous rows (Sec. 4.4, late-bound KV
 * preparation: the departing trajectory's prefix is snapshotted):
 *   dst[off_b + (((l - layer_begin)*2 + kv)*Hkv + h)*n_b*D + t*D + d]
 *       = (kv == 0 ? K : V)_l[block_table[b][t/16]][h][t%16][d]
 * off_b = dst_offsets[b] (device int64 [batch], elements, multiples of 8) or,
 * when dst_offsets is NULL, (layer_end - layer_begin)*2*Hkv*D*sum_{b'<b} n_b'.
 * A bit-exact copy: every bf16 pattern, NaN payloads included, is preserved.
 * Elements of dst outside the rows are not written.
 * dst (host or device): device memory, or page-locked host memory the device
 * can address (cudaHostAlloc / cudaHostRegister; a pinned torch tensor).  With
 * host memory the kernel writes the rows straight over the CPU-GPU link
 * (NVLink-C2C on Grace systems), so a snapshot reaches host memory in one pass
 * with no device-side staging buffer.  Pageable host memory: CADKV_ERR_INVALID.
 * The caller keeps dst alive until the stream reaches the call.
 */
int kv_prefix_stage(const cadkv_pool *pool, const int32_t *block_table, int max_pages,
                    const int32_t *context_lens, int batch, int layer_begin,
                    int layer_end, void *dst, const int64_t *dst_offsets,
                    void *workspace, size_t workspace_bytes, cadkv_stream_t stream);

/*
 * Inverse of kv_prefix_stage: write staged rows `src` (same layout and
 * offsets) into the pool pages named by block_table.  Slots of a last page
 * past n_b are not written.  Pages named twice give an unspecified result.
 * src may be page-locked host memory, as dst of kv_prefix_stage: a prefix
 * kept in host memory is loaded into a destination pool in one pass.
 */
int kv_prefix_load(const cadkv_pool *pool, const int32_t *block_table, int max_pages,
                   const int32_t *context_lens, int batch, int layer_begin,
                   int layer_end, const void *src, const int64_t *src_offsets,
                   void *workspace, size_t workspace_bytes, cadkv_stream_t stream);

/* As decode_attention_status, for a staging/load workspace. */
int kv_prefix_stage_status(const void *workspace, cadkv_stream_t stream);

/*
 * Self-test of the failure path (no counterpart in the paper).  Every device
 * wait in this library is bounded; when one gives up, the kernel records
 * CADKV_ERR_TIMEOUT in its workspace status word, waits (bounded) for its own
 * copies, frees its tensor memory and returns, so the CUDA context stays
 * usable.  This call runs exactly that path on purpose: one CTA holds tensor
 * memory and waits, with the library's bounded wait, on a barrier phase that
 * nothing ever completes; after limit_ns (1 ns .. 2 s) it records the timeout
 * and returns.  Afterwards kv_prefix_stage_status(workspace, stream) reads
 * CADKV_ERR_TIMEOUT.  workspace: device, at least 64 bytes, 256-byte aligned.
 */
int cadkv_wait_selftest(long long limit_ns, void *workspace, size_t workspace_bytes,
                        cadkv_stream_t stream);

/*
 * Measuring aid (no counterpart in the paper): read `bytes` (a multiple of 16)
 * of device memory `buf` with 16-byte streaming loads and XOR them into the
 * device word *sink (8-byte aligned; the caller zeroes it).  The only DRAM
 * traffic is the read, so bytes / time is the read-bandwidth ceiling that the
 * read-dominated decode-attention stream is compared with.
 */
int cadkv_hbm_read_probe(const void *buf, size_t bytes, unsigned long long *sink,
                         cadkv_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Decode attention without caller-provided scratch                          */
/* ------------------------------------------------------------------------ */

/* Size of the scratch array decode_attention_noalloc uses (32 MiB). */
#define CADKV_NOALLOC_SCRATCH_BYTES (32u << 20)

/*
 * decode_attention for callers that cannot allocate device memory when they
 * call it.  (The paper has no counterpart; this is a library convenience.)
 * Examples: a serving engine that reserved nearly all HBM for its KV cache at
 * start-up, so a cudaMalloc at call time would fail or fragment that pool; or
 * a plugin that has no handle on its host framework's allocator and must not
 * call cudaMalloc/cudaFree itself (cudaFree also synchronises the device).
 *
 * Arguments and results are those of decode_attention without the workspace:
 * the caller still passes every input and output.  The scratch space the
 * computation needs (page prefix sums, arrival counters, split partials) lives
 * in one file-scope device array of CADKV_NOALLOC_SCRATCH_BYTES, which every
 * GPU that loads the library holds until the process exits.  Nothing is
 * allocated: no cudaMalloc, no cudaFree, no allocating library routine.
 *
 * - The first call in a device's context looks up that context's address of
 *   the array (cudaGetSymbolAddress, with the device current) and caches it
 *   with the context's id; make that first call before any stream capture on
 *   the device.  A call made in another context of the same device (after
 *   cudaDeviceReset, or under a context the caller made current) looks the
 *   address up again: a cached address is tied to its context.
 * - A problem whose scratch would exceed CADKV_NOALLOC_SCRATCH_BYTES is
 *   rejected with CADKV_ERR_WORKSPACE before anything is launched (the
 *   requirement is decode_attention_workspace_size() of the same sizes).
 * - Every call on a device shares the one array, and the array keeps the last
 *   call's contents; each call's planner clears what must start at zero
 *   (status word, work counter, arrival counters) itself.  Calls whose
 *   kernels may overlap on the GPU (different streams without ordering) race
 *   on the array and give wrong results: order them on one stream.
 * - The device status word of the last call (bad block-table entries, lengths
 *   beyond the table, timeouts) is read by decode_attention_noalloc_status.
 */
int decode_attention_noalloc(const void *q, const void *k_pages, const void *v_pages,
                             const int32_t *block_table, const int32_t *context_lens,
                             void *out, float *lse, int batch, int num_q_heads,
                             int num_kv_heads, int head_dim, int page_size, int num_pages,
                             int max_pages, cadkv_stream_t stream);

/*
 * Device status word of the last decode_attention_noalloc call on the current
 * device's context, as decode_attention_status reads it from a workspace:
 * synchronises `stream` (pass the stream of that call), returns 0 or the first
 * CADKV_ERR_* the kernels recorded (CADKV_ERR_OOB, CADKV_ERR_SHAPE,
 * CADKV_ERR_TIMEOUT), or CADKV_ERR_CUDA if the copy fails.  The next call
 * clears the word, so read it before calling again.
 */
int decode_attention_noalloc_status(cadkv_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* CADKV_H */
