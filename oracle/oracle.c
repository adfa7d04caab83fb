/*
 * oracle.c -- plain fp64 CPU oracle for the decode step's hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load this file's library.  The product
 * (libcadkv.so and its Python binding) never calls, links or imports it, and
 * this file includes nothing from the product.
 *
 * What it computes
 * ----------------
 * 1. oracle_decode_attention: one decode step of attention over a paged KV
 *    cache.  The paper (Sec. 2.3 and Sec. 3.1) places this step at the centre
 *    of rollout cost: every decode step reads each resident trajectory's KV
 *    cache, so the step is bound by memory bandwidth.  The paper takes the
 *    attention operator and the paged cache from its inference backend
 *    (Sec. 5, vLLM/PagedAttention) and never writes the formula; this oracle
 *    writes out the standard scaled dot-product attention for one query token:
 *
 *        g          = h / G                      (G = Hq / Hkv, GQA grouping)
 *        K_t, V_t   = row of page block_table[b][t / P], slot t % P, head g
 *        s_t        = (q_{b,h} . K_t) / sqrt(D)       for t = 0 .. n_b - 1
 *        m          = max_t s_t
 *        l          = sum_t exp(s_t - m)
 *        out[b,h,:] = sum_t exp(s_t - m) V_t / l
 *        lse[b,h]   = m + ln l                   (natural log of sum exp s_t)
 *
 *    Inputs are bf16 bit patterns, widened exactly to double.  It is a plain
 *    two-pass computation over the logical token order: no blocking, no
 *    splitting, no online rescaling.  A trajectory with n_b = 0 yields
 *    out = 0 and lse = -inf.
 *
 * 2. oracle_prefix_stage: the snapshot step of late-bound KV preparation
 *    (Sec. 4.4, phase 1): a departing trajectory's KV blocks, scattered over
 *    the paged pool, are copied into one contiguous per-trajectory buffer.
 *    For trajectory b, layer l in [layer_begin, layer_end), kv in {K, V},
 *    KV head h and token t < n_b:
 *
 *        dst[off_b + (((l - layer_begin) * 2 + kv) * Hkv + h) * n_b * D
 *                  + t * D + d]
 *            = pool_kv[l][block_table[b][t / P]][h][t % P][d]
 *
 *    with off_b = (layer_end - layer_begin) * 2 * Hkv * D * sum_{b' < b} n_b'
 *    unless explicit offsets are given.  It is a bit copy.
 *
 * 3. oracle_prefix_load: the inverse, phase 3 of Sec. 4.4: a staged
 *    contiguous prefix is written back into a (possibly different) paged pool
 *    following a destination block table.  Token slots of the last page past
 *    n_b are left untouched.
 *
 * 4. oracle_kv_append: the step that precedes attention in every decode step
 *    (Sec. 2.3: each step appends the new token's key and value to the
 *    trajectory's KV cache): for every trajectory with n_b >= 1 and KV head h,
 *    the new token's rows k_new[b][h][:] and v_new[b][h][:] are written to
 *    token position n_b - 1, i.e. page block_table[b][(n_b - 1) / P], slot
 *    (n_b - 1) % P.  Trajectories with n_b = 0 append nothing.
 *
 * 5. oracle_prefill_attention: chunked prefill (re-prefill) attention over the
 *    paged pool -- the fallback of Sec. 4.4 when prepared KV state cannot be
 *    used and the destination recomputes the prefix.  Trajectory b contributes
 *    its last C_b = q_offsets[b+1] - q_offsets[b] tokens as queries; their K
 *    and V are already in the pool, so query i of b sits at absolute position
 *    p = n_b - C_b + i and attends causally to keys t = 0 .. p:
 *
 *        s_t = (q_{row,h} . K_t) / sqrt(D)   for t <= p
 *        out[row,h,:] = sum_{t<=p} exp(s_t - m) V_t / sum_{t<=p} exp(s_t - m)
 *        lse[row,h]   = m + ln sum_{t<=p} exp(s_t - m)
 *
 *    with row = q_offsets[b] + i, g = h / G as above.  Requires C_b <= n_b.
 *
 * Pool layout: per layer, K and V are each [num_pages][Hkv][P][D] bf16
 * (head-major inside a page); layers are stacked with stride
 * num_pages * Hkv * P * D elements.
 *
 * Return codes: 0 on success, -1 on a bad argument (null pointer, bad size),
 * -2 on a context length outside [0, max_pages * P], -5 on a block-table entry
 * outside [0, num_pages).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double widen_bf16(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static void set_threads(int num_threads)
{
#ifdef _OPENMP
    if (num_threads > 0)
        omp_set_num_threads(num_threads);
#else
    (void)num_threads;
#endif
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

static int check_lengths(const int32_t *block_table, const int32_t *context_lens,
                         int64_t batch, int64_t page_size, int64_t num_pages,
                         int64_t max_pages)
{
    for (int64_t b = 0; b < batch; ++b) {
        int64_t n = context_lens[b];
        if (n < 0 || n > max_pages * page_size)
            return -2;
        int64_t pages = (n + page_size - 1) / page_size;
        for (int64_t j = 0; j < pages; ++j) {
            int64_t phys = block_table[b * max_pages + j];
            if (phys < 0 || phys >= num_pages)
                return -5;
        }
    }
    return 0;
}

/*
 * Attention for the (b, h) pairs listed in rows[] (row = b * Hq + h), or for
 * every pair when rows is NULL.  out is [num_rows][D] (or [B][Hq][D]), lse is
 * [num_rows] (or [B][Hq]).
 */
int oracle_decode_attention(const uint16_t *q, const uint16_t *k_pages,
                            const uint16_t *v_pages, const int32_t *block_table,
                            const int32_t *context_lens, int64_t batch,
                            int64_t num_q_heads, int64_t num_kv_heads,
                            int64_t head_dim, int64_t page_size,
                            int64_t num_pages, int64_t max_pages,
                            const int64_t *rows, int64_t num_rows,
                            double *out, double *lse, int num_threads)
{
    if (!q || !k_pages || !v_pages || !block_table || !context_lens || !out || !lse)
        return -1;
    if (batch < 0 || num_q_heads <= 0 || num_kv_heads <= 0 || head_dim <= 0 ||
        page_size <= 0 || num_pages < 0 || max_pages < 0)
        return -1;
    if (num_q_heads % num_kv_heads != 0)
        return -1;
    int rc = check_lengths(block_table, context_lens, batch, page_size, num_pages,
                           max_pages);
    if (rc != 0)
        return rc;
    if (!rows)
        num_rows = batch * num_q_heads;
    for (int64_t i = 0; rows && i < num_rows; ++i)
        if (rows[i] < 0 || rows[i] >= batch * num_q_heads)
            return -1;

    const int64_t group = num_q_heads / num_kv_heads;
    const double scale = 1.0 / sqrt((double)head_dim);
    set_threads(num_threads);

#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t i = 0; i < num_rows; ++i) {
        const int64_t row = rows ? rows[i] : i;
        const int64_t b = row / num_q_heads;
        const int64_t h = row % num_q_heads;
        const int64_t g = h / group;
        const int64_t n = context_lens[b];
        double *o = out + i * head_dim;
        for (int64_t d = 0; d < head_dim; ++d)
            o[d] = 0.0;
        if (n == 0) {
            lse[i] = -INFINITY;
            continue;
        }
        double *s = (double *)malloc((size_t)n * sizeof(double));
        const uint16_t *qv = q + (b * num_q_heads + h) * head_dim;

        /* pass 1: scaled scores over the logical token sequence */
        double m = -INFINITY;
        for (int64_t t = 0; t < n; ++t) {
            const int64_t phys = block_table[b * max_pages + t / page_size];
            const int64_t slot = t % page_size;
            const uint16_t *kv =
                k_pages + ((phys * num_kv_heads + g) * page_size + slot) * head_dim;
            double dot = 0.0;
            for (int64_t d = 0; d < head_dim; ++d)
                dot += widen_bf16(qv[d]) * widen_bf16(kv[d]);
            s[t] = dot * scale;
            if (s[t] > m)
                m = s[t];
        }

        /* pass 2: softmax weights and the weighted sum of value rows */
        double l = 0.0;
        for (int64_t t = 0; t < n; ++t) {
            const int64_t phys = block_table[b * max_pages + t / page_size];
            const int64_t slot = t % page_size;
            const uint16_t *vv =
                v_pages + ((phys * num_kv_heads + g) * page_size + slot) * head_dim;
            const double w = exp(s[t] - m);
            l += w;
            for (int64_t d = 0; d < head_dim; ++d)
                o[d] += w * widen_bf16(vv[d]);
        }
        for (int64_t d = 0; d < head_dim; ++d)
            o[d] /= l;
        lse[i] = m + log(l);
        free(s);
    }
    return 0;
}

static int64_t packed_offset(const int32_t *context_lens, int64_t b, int64_t row_elems)
{
    int64_t tokens = 0;
    for (int64_t i = 0; i < b; ++i)
        tokens += context_lens[i];
    return tokens * row_elems;
}

/*
 * k_pool / v_pool: [num_layers][num_pages][Hkv][P][D] bf16 bits.
 * dst: bf16 bits; dst_offsets: [B] element offsets, or NULL for packed.
 */
int oracle_prefix_stage(const uint16_t *k_pool, const uint16_t *v_pool,
                        int64_t num_layers, int64_t num_pages, int64_t num_kv_heads,
                        int64_t page_size, int64_t head_dim,
                        const int32_t *block_table, int64_t max_pages,
                        const int32_t *context_lens, int64_t batch,
                        int64_t layer_begin, int64_t layer_end, uint16_t *dst,
                        const int64_t *dst_offsets, int num_threads)
{
    if (!k_pool || !v_pool || !block_table || !context_lens || !dst)
        return -1;
    if (layer_begin < 0 || layer_end > num_layers || layer_begin > layer_end)
        return -1;
    int rc = check_lengths(block_table, context_lens, batch, page_size, num_pages,
                           max_pages);
    if (rc != 0)
        return rc;
    const int64_t layers = layer_end - layer_begin;
    const int64_t layer_stride = num_pages * num_kv_heads * page_size * head_dim;
    set_threads(num_threads);

#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t b = 0; b < batch; ++b) {
        const int64_t n = context_lens[b];
        const int64_t off = dst_offsets ? dst_offsets[b]
                                        : packed_offset(context_lens, b,
                                                        layers * 2 * num_kv_heads * head_dim);
        for (int64_t l = layer_begin; l < layer_end; ++l) {
            for (int64_t kv = 0; kv < 2; ++kv) {
                const uint16_t *pool = (kv == 0 ? k_pool : v_pool) + l * layer_stride;
                for (int64_t h = 0; h < num_kv_heads; ++h) {
                    uint16_t *row = dst + off +
                                    (((l - layer_begin) * 2 + kv) * num_kv_heads + h) * n * head_dim;
                    for (int64_t t = 0; t < n; ++t) {
                        const int64_t phys = block_table[b * max_pages + t / page_size];
                        const int64_t slot = t % page_size;
                        const uint16_t *src =
                            pool + ((phys * num_kv_heads + h) * page_size + slot) * head_dim;
                        for (int64_t d = 0; d < head_dim; ++d)
                            row[t * head_dim + d] = src[d];
                    }
                }
            }
        }
    }
    return 0;
}

/*
 * Inverse of oracle_prefix_stage: src holds staged rows in the layout above;
 * each token t < n_b is written to pool_kv[l][block_table[b][t / P]][h][t % P].
 */
int oracle_prefix_load(uint16_t *k_pool, uint16_t *v_pool, int64_t num_layers,
                       int64_t num_pages, int64_t num_kv_heads, int64_t page_size,
                       int64_t head_dim, const int32_t *block_table,
                       int64_t max_pages, const int32_t *context_lens,
                       int64_t batch, int64_t layer_begin, int64_t layer_end,
                       const uint16_t *src, const int64_t *src_offsets)
{
    if (!k_pool || !v_pool || !block_table || !context_lens || !src)
        return -1;
    if (layer_begin < 0 || layer_end > num_layers || layer_begin > layer_end)
        return -1;
    int rc = check_lengths(block_table, context_lens, batch, page_size, num_pages,
                           max_pages);
    if (rc != 0)
        return rc;
    const int64_t layers = layer_end - layer_begin;
    const int64_t layer_stride = num_pages * num_kv_heads * page_size * head_dim;
    for (int64_t b = 0; b < batch; ++b) {
        const int64_t n = context_lens[b];
        const int64_t off = src_offsets ? src_offsets[b]
                                        : packed_offset(context_lens, b,
                                                        layers * 2 * num_kv_heads * head_dim);
        for (int64_t l = layer_begin; l < layer_end; ++l)
            for (int64_t kv = 0; kv < 2; ++kv) {
                uint16_t *pool = (kv == 0 ? k_pool : v_pool) + l * layer_stride;
                for (int64_t h = 0; h < num_kv_heads; ++h) {
                    const uint16_t *row = src + off +
                                          (((l - layer_begin) * 2 + kv) * num_kv_heads + h) * n * head_dim;
                    for (int64_t t = 0; t < n; ++t) {
                        const int64_t phys = block_table[b * max_pages + t / page_size];
                        const int64_t slot = t % page_size;
                        uint16_t *d = pool + ((phys * num_kv_heads + h) * page_size + slot) * head_dim;
                        memcpy(d, row + t * head_dim, (size_t)head_dim * sizeof(uint16_t));
                    }
                }
            }
    }
    return 0;
}

/*
 * k_new, v_new: [B][Hkv][D] bf16 bits; k_pages, v_pages: [num_pages][Hkv][P][D]
 * (one layer), updated in place.
 */
int oracle_kv_append(uint16_t *k_pages, uint16_t *v_pages, const uint16_t *k_new,
                     const uint16_t *v_new, const int32_t *block_table,
                     const int32_t *context_lens, int64_t batch, int64_t num_kv_heads,
                     int64_t head_dim, int64_t page_size, int64_t num_pages,
                     int64_t max_pages)
{
    if (!k_pages || !v_pages || !k_new || !v_new || !block_table || !context_lens)
        return -1;
    int rc = check_lengths(block_table, context_lens, batch, page_size, num_pages,
                           max_pages);
    if (rc != 0)
        return rc;
    for (int64_t b = 0; b < batch; ++b) {
        const int64_t n = context_lens[b];
        if (n == 0)
            continue;
        const int64_t t = n - 1;
        const int64_t phys = block_table[b * max_pages + t / page_size];
        const int64_t slot = t % page_size;
        for (int64_t h = 0; h < num_kv_heads; ++h) {
            const int64_t dst = ((phys * num_kv_heads + h) * page_size + slot) * head_dim;
            const int64_t src = (b * num_kv_heads + h) * head_dim;
            for (int64_t d = 0; d < head_dim; ++d) {
                k_pages[dst + d] = k_new[src + d];
                v_pages[dst + d] = v_new[src + d];
            }
        }
    }
    return 0;
}

/*
 * q: [T][Hq][D] bf16 bits, T = q_offsets[batch]; out: [T][Hq][D]; lse: [T][Hq].
 */
int oracle_prefill_attention(const uint16_t *q, const int64_t *q_offsets,
                             const uint16_t *k_pages, const uint16_t *v_pages,
                             const int32_t *block_table, const int32_t *context_lens,
                             int64_t batch, int64_t num_q_heads, int64_t num_kv_heads,
                             int64_t head_dim, int64_t page_size, int64_t num_pages,
                             int64_t max_pages, double *out, double *lse, int num_threads)
{
    if (!q || !q_offsets || !k_pages || !v_pages || !block_table || !context_lens || !out ||
        !lse)
        return -1;
    if (batch < 0 || num_q_heads <= 0 || num_kv_heads <= 0 || head_dim <= 0 ||
        page_size <= 0 || num_q_heads % num_kv_heads != 0)
        return -1;
    int rc = check_lengths(block_table, context_lens, batch, page_size, num_pages,
                           max_pages);
    if (rc != 0)
        return rc;
    if (q_offsets[0] != 0)
        return -1;
    for (int64_t b = 0; b < batch; ++b) {
        const int64_t chunk = q_offsets[b + 1] - q_offsets[b];
        if (chunk < 0 || chunk > context_lens[b])
            return -2;
    }
    const int64_t total = q_offsets[batch];
    const int64_t group = num_q_heads / num_kv_heads;
    const double scale = 1.0 / sqrt((double)head_dim);
    set_threads(num_threads);

#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t i = 0; i < total * num_q_heads; ++i) {
        const int64_t row = i / num_q_heads;
        const int64_t h = i % num_q_heads;
        int64_t b = 0;
        while (q_offsets[b + 1] <= row)
            ++b;
        const int64_t chunk = q_offsets[b + 1] - q_offsets[b];
        const int64_t pos = context_lens[b] - chunk + (row - q_offsets[b]);
        const int64_t n = pos + 1;                /* keys 0 .. pos */
        const int64_t g = h / group;
        const uint16_t *qv = q + (row * num_q_heads + h) * head_dim;
        double *o = out + i * head_dim;
        double *s = (double *)malloc((size_t)n * sizeof(double));

        double m = -INFINITY;
        for (int64_t t = 0; t < n; ++t) {
            const int64_t phys = block_table[b * max_pages + t / page_size];
            const uint16_t *kv =
                k_pages + ((phys * num_kv_heads + g) * page_size + t % page_size) * head_dim;
            double dot = 0.0;
            for (int64_t d = 0; d < head_dim; ++d)
                dot += widen_bf16(qv[d]) * widen_bf16(kv[d]);
            s[t] = dot * scale;
            if (s[t] > m)
                m = s[t];
        }
        for (int64_t d = 0; d < head_dim; ++d)
            o[d] = 0.0;
        double l = 0.0;
        for (int64_t t = 0; t < n; ++t) {
            const int64_t phys = block_table[b * max_pages + t / page_size];
            const uint16_t *vv =
                v_pages + ((phys * num_kv_heads + g) * page_size + t % page_size) * head_dim;
            const double w = exp(s[t] - m);
            l += w;
            for (int64_t d = 0; d < head_dim; ++d)
                o[d] += w * widen_bf16(vv[d]);
        }
        for (int64_t d = 0; d < head_dim; ++d)
            o[d] /= l;
        lse[i] = m + log(l);
        free(s);
    }
    return 0;
}
