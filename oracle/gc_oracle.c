/*
 * Float64 CPU oracle for prefix-reuse prefill (paged KV restore, KV append,
 * causal GQA attention of the new tokens over [cached prefix ++ new tokens]).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA path; it is written from the
 * definitions in the paper (Sec. 2.1 "LLM Serving Process": the KV cache
 * stores the keys and values of processed tokens for reuse; Sec. 2.2
 * "Caching for LLM Serving", Fig. 2a: on a cache hit the cached KV of the
 * context is loaded and stitched with the new tokens' KV, and both are
 * processed together).  Because reuse must give exactly what a full
 * recomputation gives, every function here is the plain definition, not an
 * approximation:
 *
 *   restore   pool[l][kv][block_ids[i]] = host_src[i][l][kv]        (copy)
 *   append    pool[layer][kv][bt[b][pos/ps]][g][pos%ps] = new[t][g],
 *             pos = prefix_len[b] + t                                (copy)
 *   attention O[b,h,i] = sum_{j <= P_b + i} softmax_j(scale * q.k_j) v_j,
 *             kv head g = h / (Hq/Hkv), keys read through block table b.
 *
 * Layouts (all row-major; bf16 values are passed as their uint16 bit
 * patterns and widened to double exactly):
 *   pool      [L][2][num_pages][Hkv][ps][d]     (K plane 0, V plane 1)
 *   host_src  [n_blocks][L][2][Hkv][ps][d]      (one cached page per block)
 *   q         [T_new][Hq][d]     k_new, v_new  [T_new][Hkv][d]
 *   block_table [batch][max_blocks]   cu_new_lens [batch+1]
 *
 * Parity status: every function below is pinned by the CPU tests
 * (closed forms, invariants, brute force, the dense second path).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR_ARG 1
#define OR_ERR_RANGE 2
#define OR_ERR_OOM 3

/* bf16 bit pattern -> double.  A bf16 value is the upper half of a binary32
 * value, so widening through float is exact. */
static double bf16_to_double(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

double oracle_bf16_to_double(uint16_t bits) { return bf16_to_double(bits); }

static size_t pool_index(int L, int Hkv, int ps, int d, int num_pages, int l, int kv,
                         int page, int g, int slot, int c) {
    (void)L;
    return (((((size_t)l * 2 + kv) * num_pages + page) * Hkv + g) * ps + slot) * d + c;
}

/* ---------------------------------------------------------------- restore */
/* Sec. 2.2, Fig. 2a step 2: load the cached context KV.  Block i of the
 * staging image is copied into page block_ids[i] of every (layer, K/V)
 * plane; nothing else in the pool changes.  Element-wise loops on purpose. */
int oracle_kv_restore(uint16_t *pool, int L, int Hkv, int ps, int d, int num_pages,
                      const uint16_t *host_src, const int32_t *block_ids, int n_blocks) {
    if (n_blocks < 0 || L <= 0 || Hkv <= 0 || ps <= 0 || d <= 0 || num_pages <= 0)
        return OR_ERR_ARG;
    for (int i = 0; i < n_blocks; ++i)
        if (block_ids[i] < 0 || block_ids[i] >= num_pages) return OR_ERR_RANGE;
    for (int i = 0; i < n_blocks; ++i) {
        int page = block_ids[i];
        for (int l = 0; l < L; ++l)
            for (int kv = 0; kv < 2; ++kv)
                for (int g = 0; g < Hkv; ++g)
                    for (int s = 0; s < ps; ++s)
                        for (int c = 0; c < d; ++c) {
                            size_t src = (((((size_t)i * L + l) * 2 + kv) * Hkv + g) * ps + s) * d + c;
                            pool[pool_index(L, Hkv, ps, d, num_pages, l, kv, page, g, s, c)] = host_src[src];
                        }
    }
    return OR_OK;
}

/* Inverse map, used by the pins: read page block_ids[i] of every plane back
 * into a staging image laid out like host_src. */
int oracle_kv_gather_blocks(const uint16_t *pool, int L, int Hkv, int ps, int d, int num_pages,
                            const int32_t *block_ids, int n_blocks, uint16_t *dst) {
    for (int i = 0; i < n_blocks; ++i) {
        int page = block_ids[i];
        if (page < 0 || page >= num_pages) return OR_ERR_RANGE;
        for (int l = 0; l < L; ++l)
            for (int kv = 0; kv < 2; ++kv)
                for (int g = 0; g < Hkv; ++g)
                    for (int s = 0; s < ps; ++s)
                        for (int c = 0; c < d; ++c) {
                            size_t o = (((((size_t)i * L + l) * 2 + kv) * Hkv + g) * ps + s) * d + c;
                            dst[o] = pool[pool_index(L, Hkv, ps, d, num_pages, l, kv, page, g, s, c)];
                        }
    }
    return OR_OK;
}

/* ------------------------------------------------------ 8-bit cache tier */
/* An 8-bit copy of the cached pages for the cache tier (the 70B runs of
 * Sec. 6.1 use INT8; an 8-bit image halves the bytes the tier stores and
 * the host link carries).  Symmetric absmax INT8 with one scale per
 * (block, layer, plane, kv head) group of ps*d values:
 *   amax = max |x| over the group's finite values
 *   s    = amax / 127                      (stored, binary32)
 *   c    = clamp(round_half_even(x * (127 / amax)), -127, 127), 0 for NaN
 *          (all codes 0 when amax is 0)
 *   x'   = bf16_round_half_even(c * s)     (restore)
 * The code is an integer decided by floating point, so it is decided here
 * in binary32 like the kernel does (x * inv and 127 / amax each rounded
 * once), not in float64.
 * Image chunk of one (block, layer, plane): Hkv binary32 scales, zero padding
 * to a multiple of 16 bytes, then the codes [Hkv][ps][d] as int8; the image
 * is [n_blocks][L][2][chunk]. */
size_t oracle_q8_chunk_bytes(int Hkv, int ps, int d) {
    size_t hdr = ((size_t)Hkv * 4 + 15) / 16 * 16;
    return hdr + (size_t)Hkv * ps * d;
}

static float bf16_to_float(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* binary32 -> bf16 bits, round half to even (finite inputs only here). */
static uint16_t float_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7fffu + lsb;
    return (uint16_t)(u >> 16);
}

static int8_t q8_code(float x, float inv) {
    if (isnan(x)) return 0;
    float v = x * inv;
    if (isnan(v)) return 0;          /* inf * 0 when amax is 0 */
    if (v > 127.0f) v = 127.0f;
    if (v < -127.0f) v = -127.0f;
    return (int8_t)rintf(v);         /* default rounding: half to even */
}

int oracle_kv_save_q8(const uint16_t *pool, int L, int Hkv, int ps, int d, int num_pages,
                      const int32_t *block_ids, int n_blocks, int layer_begin, int layer_count,
                      uint8_t *dst) {
    if (layer_begin < 0 || layer_count < 0 || layer_begin + layer_count > L) return OR_ERR_ARG;
    size_t chunk = oracle_q8_chunk_bytes(Hkv, ps, d);
    size_t hdr = chunk - (size_t)Hkv * ps * d;
    size_t group = (size_t)ps * d;
    for (int i = 0; i < n_blocks; ++i) {
        int page = block_ids[i];
        if (page < 0 || page >= num_pages) return OR_ERR_RANGE;
        for (int l = layer_begin; l < layer_begin + layer_count; ++l)
            for (int kv = 0; kv < 2; ++kv) {
                uint8_t *c = dst + (((size_t)i * L + l) * 2 + kv) * chunk;
                memset(c, 0, hdr);
                for (int g = 0; g < Hkv; ++g) {
                    const uint16_t *x = pool + pool_index(L, Hkv, ps, d, num_pages, l, kv, page, g, 0, 0);
                    float amax = 0.0f;
                    for (size_t e = 0; e < group; ++e) {
                        float a = fabsf(bf16_to_float(x[e]));
                        if (isfinite(a) && a > amax) amax = a;
                    }
                    float scale = amax / 127.0f;
                    float inv = amax > 0.0f ? 127.0f / amax : 0.0f;
                    memcpy(c + (size_t)g * 4, &scale, 4);
                    int8_t *codes = (int8_t *)(c + hdr) + (size_t)g * group;
                    for (size_t e = 0; e < group; ++e) codes[e] = q8_code(bf16_to_float(x[e]), inv);
                }
            }
    }
    return OR_OK;
}

int oracle_kv_restore_q8(uint16_t *pool, int L, int Hkv, int ps, int d, int num_pages,
                         const uint8_t *src, const int32_t *block_ids, int n_blocks,
                         int layer_begin, int layer_count) {
    if (layer_begin < 0 || layer_count < 0 || layer_begin + layer_count > L) return OR_ERR_ARG;
    size_t chunk = oracle_q8_chunk_bytes(Hkv, ps, d);
    size_t hdr = chunk - (size_t)Hkv * ps * d;
    size_t group = (size_t)ps * d;
    for (int i = 0; i < n_blocks; ++i)
        if (block_ids[i] < 0 || block_ids[i] >= num_pages) return OR_ERR_RANGE;
    for (int i = 0; i < n_blocks; ++i)
        for (int l = layer_begin; l < layer_begin + layer_count; ++l)
            for (int kv = 0; kv < 2; ++kv) {
                const uint8_t *c = src + (((size_t)i * L + l) * 2 + kv) * chunk;
                for (int g = 0; g < Hkv; ++g) {
                    float scale;
                    memcpy(&scale, c + (size_t)g * 4, 4);
                    const int8_t *codes = (const int8_t *)(c + hdr) + (size_t)g * group;
                    uint16_t *y = pool + pool_index(L, Hkv, ps, d, num_pages, l, kv, block_ids[i], g, 0, 0);
                    for (size_t e = 0; e < group; ++e)
                        y[e] = float_to_bf16_rne((float)codes[e] * scale);
                }
            }
    return OR_OK;
}

/* ----------------------------------------------------------------- append */
/* Sec. 2.2: stitch the new tokens' KV after the cached prefix.  Token t of
 * request b sits at absolute position prefix_lens[b] + t of its sequence. */
int oracle_kv_append(uint16_t *pool, int L, int Hkv, int ps, int d, int num_pages, int layer,
                     const uint16_t *k_new, const uint16_t *v_new, const int32_t *block_table,
                     int max_blocks, const int32_t *prefix_lens, const int32_t *cu_new_lens,
                     int batch) {
    if (layer < 0 || layer >= L || batch < 0) return OR_ERR_ARG;
    for (int b = 0; b < batch; ++b) {
        int n_b = cu_new_lens[b + 1] - cu_new_lens[b];
        for (int t = 0; t < n_b; ++t) {
            int pos = prefix_lens[b] + t;
            int blk = pos / ps;
            if (blk >= max_blocks) return OR_ERR_RANGE;
            int page = block_table[(size_t)b * max_blocks + blk];
            if (page < 0 || page >= num_pages) return OR_ERR_RANGE;
            int slot = pos % ps;
            size_t row = (size_t)(cu_new_lens[b] + t);
            for (int g = 0; g < Hkv; ++g)
                for (int c = 0; c < d; ++c) {
                    size_t src = (row * Hkv + g) * d + c;
                    pool[pool_index(L, Hkv, ps, d, num_pages, layer, 0, page, g, slot, c)] = k_new[src];
                    pool[pool_index(L, Hkv, ps, d, num_pages, layer, 1, page, g, slot, c)] = v_new[src];
                }
        }
    }
    return OR_OK;
}

/* ------------------------------------------------------------- attention */
typedef struct {
    const uint16_t *q, *pool;
    const int32_t *block_table, *prefix_lens, *cu_new_lens;
    int L, Hkv, ps, d, num_pages, layer, max_blocks, batch, Hq;
    double scale;
    double *out;            /* [T_new][Hq][d] or [n_rows][d] */
    const int32_t *rows;    /* NULL: all rows; else [n_rows][3] = (b, h, i) */
    int n_rows;
    int status;
} attn_job;

/* Block-table gather of request b, kv head g: K[j], V[j] for j < T,
 * widened to double.  Returns OR_ERR_RANGE on a page outside the pool. */
static int gather_request(const attn_job *J, int b, int g, int T, double *K, double *V) {
    for (int j = 0; j < T; ++j) {
        int blk = j / J->ps;
        if (blk >= J->max_blocks) return OR_ERR_RANGE;
        int page = J->block_table[(size_t)b * J->max_blocks + blk];
        if (page < 0 || page >= J->num_pages) return OR_ERR_RANGE;
        int slot = j % J->ps;
        for (int c = 0; c < J->d; ++c) {
            K[(size_t)j * J->d + c] = bf16_to_double(J->pool[pool_index(
                J->L, J->Hkv, J->ps, J->d, J->num_pages, J->layer, 0, page, g, slot, c)]);
            V[(size_t)j * J->d + c] = bf16_to_double(J->pool[pool_index(
                J->L, J->Hkv, J->ps, J->d, J->num_pages, J->layer, 1, page, g, slot, c)]);
        }
    }
    return OR_OK;
}

/* One attention row, straight from the softmax definition:
 *   s_j = scale * sum_c q_c k_jc,  m = max_j s_j,  w_j = exp(s_j - m),
 *   out = sum_j w_j v_j / sum_j w_j,  over keys j < n_keys.
 * If wn is not NULL it receives the normalised weights w_j / sum w. */
static void attend_row(const double *q, const double *K, const double *V, int n_keys, int d,
                       double scale, double *s, double *out, double *wn) {
    double m = -INFINITY;
    for (int j = 0; j < n_keys; ++j) {
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += q[c] * K[(size_t)j * d + c];
        s[j] = scale * acc;
        if (s[j] > m) m = s[j];
    }
    double sum = 0.0;
    for (int j = 0; j < n_keys; ++j) {
        s[j] = exp(s[j] - m);
        sum += s[j];
    }
    for (int c = 0; c < d; ++c) out[c] = 0.0;
    for (int j = 0; j < n_keys; ++j)
        for (int c = 0; c < d; ++c) out[c] += s[j] * V[(size_t)j * d + c];
    for (int c = 0; c < d; ++c) out[c] /= sum;
    if (wn)
        for (int j = 0; j < n_keys; ++j) wn[j] = s[j] / sum;
}

static int request_total_len(const attn_job *J, int b) {
    return J->prefix_lens[b] + (J->cu_new_lens[b + 1] - J->cu_new_lens[b]);
}

static void load_q(const attn_job *J, size_t row, int h, double *qd) {
    for (int c = 0; c < J->d; ++c)
        qd[c] = bf16_to_double(J->q[(row * J->Hq + h) * J->d + c]);
}

/* Work item = (request b, kv head g): gather once, then every q head of the
 * group and every new-token row of the request. */
static int run_group(attn_job *J, int b, int g) {
    int G = J->Hq / J->Hkv;
    int P = J->prefix_lens[b];
    int n = J->cu_new_lens[b + 1] - J->cu_new_lens[b];
    int T = P + n;
    if (n <= 0) return OR_OK;
    double *K = malloc(sizeof(double) * (size_t)T * J->d);
    double *V = malloc(sizeof(double) * (size_t)T * J->d);
    double *s = malloc(sizeof(double) * (size_t)T);
    double *qd = malloc(sizeof(double) * (size_t)J->d);
    if (!K || !V || !s || !qd) { free(K); free(V); free(s); free(qd); return OR_ERR_OOM; }
    int st = gather_request(J, b, g, T, K, V);
    for (int hh = 0; st == OR_OK && hh < G; ++hh) {
        int h = g * G + hh;
        for (int i = 0; i < n; ++i) {
            size_t row = (size_t)(J->cu_new_lens[b] + i);
            load_q(J, row, h, qd);
            /* causal, bottom-right aligned: new row i sits at position P + i */
            attend_row(qd, K, V, P + i + 1, J->d, J->scale, s, J->out + (row * J->Hq + h) * J->d, NULL);
        }
    }
    free(K); free(V); free(s); free(qd);
    return st;
}

/* Sampled row (b, h, i): exact over all its keys. */
static int run_row(attn_job *J, int r) {
    int b = J->rows[3 * r], h = J->rows[3 * r + 1], i = J->rows[3 * r + 2];
    if (b < 0 || b >= J->batch || h < 0 || h >= J->Hq) return OR_ERR_ARG;
    int G = J->Hq / J->Hkv;
    int P = J->prefix_lens[b];
    int n = J->cu_new_lens[b + 1] - J->cu_new_lens[b];
    if (i < 0 || i >= n) return OR_ERR_ARG;
    int nk = P + i + 1;
    double *K = malloc(sizeof(double) * (size_t)nk * J->d);
    double *V = malloc(sizeof(double) * (size_t)nk * J->d);
    double *s = malloc(sizeof(double) * (size_t)nk);
    double *qd = malloc(sizeof(double) * (size_t)J->d);
    if (!K || !V || !s || !qd) { free(K); free(V); free(s); free(qd); return OR_ERR_OOM; }
    int st = gather_request(J, b, h / G, nk, K, V);
    if (st == OR_OK) {
        load_q(J, (size_t)(J->cu_new_lens[b] + i), h, qd);
        attend_row(qd, K, V, nk, J->d, J->scale, s, J->out + (size_t)r * J->d, NULL);
    }
    free(K); free(V); free(s); free(qd);
    return st;
}

typedef struct {
    attn_job *J;
    int first, last; /* item range */
    int status;
} worker_arg;

static void *worker(void *p) {
    worker_arg *w = p;
    w->status = OR_OK;
    for (int it = w->first; it < w->last && w->status == OR_OK; ++it) {
        if (w->J->rows) w->status = run_row(w->J, it);
        else w->status = run_group(w->J, it / w->J->Hkv, it % w->J->Hkv);
    }
    return NULL;
}

static int run_parallel(attn_job *J, int n_items, int nthreads) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > n_items) nthreads = n_items > 0 ? n_items : 1;
    pthread_t *th = malloc(sizeof(pthread_t) * nthreads);
    worker_arg *wa = malloc(sizeof(worker_arg) * nthreads);
    if (!th || !wa) { free(th); free(wa); return OR_ERR_OOM; }
    int st = OR_OK;
    int started = 0;
    for (int t = 0; t < nthreads; ++t) {
        wa[t].J = J;
        wa[t].first = (int)((long long)n_items * t / nthreads);
        wa[t].last = (int)((long long)n_items * (t + 1) / nthreads);
        wa[t].status = OR_OK;
        if (nthreads == 1) { worker(&wa[t]); continue; }
        if (pthread_create(&th[t], NULL, worker, &wa[t]) != 0) { st = OR_ERR_OOM; break; }
        started++;
    }
    for (int t = 0; t < started; ++t) pthread_join(th[t], NULL);
    if (st == OR_OK)
        for (int t = 0; t < nthreads; ++t)
            if (wa[t].status != OR_OK) { st = wa[t].status; break; }
    free(th); free(wa);
    return st;
}

static int check_shapes(int L, int Hkv, int ps, int d, int num_pages, int layer, int batch, int Hq) {
    if (L <= 0 || Hkv <= 0 || ps <= 0 || d <= 0 || num_pages <= 0 || batch < 0 || Hq <= 0)
        return OR_ERR_ARG;
    if (layer < 0 || layer >= L || Hq % Hkv != 0) return OR_ERR_ARG;
    return OR_OK;
}

/* Full prefix-reuse attention: out[T_new][Hq][d] in double. */
int oracle_prefix_attn(const uint16_t *q, const uint16_t *pool, int L, int Hkv, int ps, int d,
                       int num_pages, int layer, const int32_t *block_table, int max_blocks,
                       const int32_t *prefix_lens, const int32_t *cu_new_lens, int batch, int Hq,
                       double scale, double *out, int nthreads) {
    int st = check_shapes(L, Hkv, ps, d, num_pages, layer, batch, Hq);
    if (st) return st;
    attn_job J = {q, pool, block_table, prefix_lens, cu_new_lens, L, Hkv, ps, d, num_pages,
                  layer, max_blocks, batch, Hq, scale, out, NULL, 0, OR_OK};
    for (int b = 0; b < batch; ++b)
        if (prefix_lens[b] < 0 || cu_new_lens[b + 1] < cu_new_lens[b]) return OR_ERR_ARG;
    (void)request_total_len;
    return run_parallel(&J, batch * Hkv, nthreads);
}

/* Sampled rows: rows[n_rows][3] = (b, h, i); out[n_rows][d]. */
int oracle_prefix_attn_rows(const uint16_t *q, const uint16_t *pool, int L, int Hkv, int ps, int d,
                            int num_pages, int layer, const int32_t *block_table, int max_blocks,
                            const int32_t *prefix_lens, const int32_t *cu_new_lens, int batch, int Hq,
                            double scale, const int32_t *rows, int n_rows, double *out,
                            int nthreads) {
    int st = check_shapes(L, Hkv, ps, d, num_pages, layer, batch, Hq);
    if (st) return st;
    attn_job J = {q, pool, block_table, prefix_lens, cu_new_lens, L, Hkv, ps, d, num_pages,
                  layer, max_blocks, batch, Hq, scale, out, rows, n_rows, OR_OK};
    return run_parallel(&J, n_rows, nthreads);
}

/* Normalised softmax weights of one row (b, h, i): w[P_b + i + 1]. */
int oracle_prefix_attn_row_weights(const uint16_t *q, const uint16_t *pool, int L, int Hkv, int ps,
                                   int d, int num_pages, int layer, const int32_t *block_table,
                                   int max_blocks, const int32_t *prefix_lens,
                                   const int32_t *cu_new_lens, int batch, int Hq, double scale,
                                   int b, int h, int i, double *w, double *out_row) {
    int st = check_shapes(L, Hkv, ps, d, num_pages, layer, batch, Hq);
    if (st) return st;
    attn_job J = {q, pool, block_table, prefix_lens, cu_new_lens, L, Hkv, ps, d, num_pages,
                  layer, max_blocks, batch, Hq, scale, NULL, NULL, 0, OR_OK};
    if (b < 0 || b >= batch || h < 0 || h >= Hq) return OR_ERR_ARG;
    int n = cu_new_lens[b + 1] - cu_new_lens[b];
    if (i < 0 || i >= n) return OR_ERR_ARG;
    int nk = prefix_lens[b] + i + 1;
    double *K = malloc(sizeof(double) * (size_t)nk * d);
    double *V = malloc(sizeof(double) * (size_t)nk * d);
    double *s = malloc(sizeof(double) * (size_t)nk);
    double *qd = malloc(sizeof(double) * (size_t)d);
    if (!K || !V || !s || !qd) { free(K); free(V); free(s); free(qd); return OR_ERR_OOM; }
    st = gather_request(&J, b, h / (Hq / Hkv), nk, K, V);
    if (st == OR_OK) {
        load_q(&J, (size_t)(cu_new_lens[b] + i), h, qd);
        attend_row(qd, K, V, nk, d, scale, s, out_row, w);
    }
    free(K); free(V); free(s); free(qd);
    return st;
}

/* ----------------------------------------------- dense second path (no paging) */
/* Plain causal self-attention over a dense sequence, written separately from
 * the paged path so that the two can pin each other: q [T][Hq][d],
 * k, v [T][Hkv][d], row t attends keys 0..t.  out [T][Hq][d] in double. */
typedef struct {
    const uint16_t *q, *k, *v;
    int T, Hq, Hkv, d;
    double scale;
    double *out;
    int h0, h1;
    int status;
} dense_arg;

static void *dense_worker(void *p) {
    dense_arg *a = p;
    int G = a->Hq / a->Hkv;
    double *sc = malloc(sizeof(double) * (size_t)(a->T > 0 ? a->T : 1));
    if (!sc) { a->status = OR_ERR_OOM; return NULL; }
    for (int h = a->h0; h < a->h1; ++h) {
        int g = h / G;
        for (int t = 0; t < a->T; ++t) {
            double mx = -INFINITY;
            for (int j = 0; j <= t; ++j) {
                double dot = 0.0;
                for (int c = 0; c < a->d; ++c)
                    dot += bf16_to_double(a->q[((size_t)t * a->Hq + h) * a->d + c]) *
                           bf16_to_double(a->k[((size_t)j * a->Hkv + g) * a->d + c]);
                sc[j] = a->scale * dot;
                mx = sc[j] > mx ? sc[j] : mx;
            }
            double den = 0.0;
            for (int j = 0; j <= t; ++j) den += exp(sc[j] - mx);
            for (int c = 0; c < a->d; ++c) {
                double num = 0.0;
                for (int j = 0; j <= t; ++j)
                    num += exp(sc[j] - mx) * bf16_to_double(a->v[((size_t)j * a->Hkv + g) * a->d + c]);
                a->out[((size_t)t * a->Hq + h) * a->d + c] = num / den;
            }
        }
    }
    free(sc);
    a->status = OR_OK;
    return NULL;
}

int oracle_full_causal_attn(const uint16_t *q, const uint16_t *k, const uint16_t *v, int T, int Hq,
                            int Hkv, int d, double scale, double *out, int nthreads) {
    if (T < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || Hq % Hkv) return OR_ERR_ARG;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > Hq) nthreads = Hq;
    pthread_t th[256];
    dense_arg a[256];
    if (nthreads > 256) nthreads = 256;
    int started = 0, st = OR_OK;
    for (int t = 0; t < nthreads; ++t) {
        a[t] = (dense_arg){q, k, v, T, Hq, Hkv, d, scale, out, Hq * t / nthreads,
                           Hq * (t + 1) / nthreads, OR_OK};
        if (nthreads == 1) { dense_worker(&a[t]); continue; }
        /* only threads that were created are joined */
        if (pthread_create(&th[t], NULL, dense_worker, &a[t]) != 0) { st = OR_ERR_OOM; break; }
        started++;
    }
    for (int t = 0; t < started; ++t) pthread_join(th[t], NULL);
    if (st != OR_OK) return st;
    for (int t = 0; t < nthreads; ++t)
        if (a[t].status) return a[t].status;
    return OR_OK;
}
