/*
 * gc.h — C ABI of libgc: prefix-reuse prefill on one GB300 GPU (sm_103a).
 *
 * The operation is the data-plane step of context caching described in
 * arXiv 2505.23970, Sec. 2.2 ("Caching for LLM Serving", Fig. 2a): when a
 * request's context is found in the cache, its KV cache is loaded back into
 * GPU memory, the KV of the new tokens is stitched after it, and the new
 * tokens are prefilled against [cached context ++ new tokens] instead of
 * recomputing the whole context.  Sec. 2.1 defines the KV cache as the keys
 * and values of processed tokens kept for reuse.  The calls below are that
 * step:
 *
 *   gc_kv_restore           cached pages (pinned host or device staging)
 *                           -> paged HBM KV pool                  (load)
 *   gc_kv_save              paged HBM KV pool -> pinned host / device
 *                           staging image; the inverse of restore  (save)
 *   gc_kv_restore_layers,   the same for a range of layers, for restores
 *   gc_kv_save_layers       and saves pipelined with per-layer compute
 *   gc_kv_save_q8,          the same with an 8-bit (INT8 + scales) image
 *   gc_kv_restore_q8        in the cache tier
 *   gc_kv_append            new tokens' K,V -> pool slots after each
 *                           request's cached prefix                (stitch)
 *   gc_prefix_prefill_attn  causal GQA attention of the new tokens over
 *                           the pool through a block table         (prefill)
 *   gc_paged_decode_attn    the same for one new token per request,
 *                           split over key ranges                  (decode)
 *
 * Conventions for every call
 *  - All device work is ordered on the caller's stream; no call synchronises
 *    the device except gc_kv_pool_check().
 *  - Every array argument is borrowed: no call keeps a pointer after it
 *    returns, but asynchronous work reads it later in stream order, so the
 *    caller keeps it alive and unchanged until the stream has passed it (the
 *    same rule as cudaMemcpyAsync).
 *  - Host-side argument checks (null pointers, negative sizes, unsupported
 *    shapes) fail with a status before anything is launched; the message is
 *    available from gc_last_error() on the same thread.
 *  - Indices that live in device memory (block ids, block tables, lengths)
 *    are checked by the kernels: a bad one is skipped (never dereferenced)
 *    and its error code is recorded in the pool's device status word, read
 *    and cleared by gc_kv_pool_check().
 *  - Zero sizes (n_blocks = 0, batch = 0, a request with no new tokens) are
 *    valid no-ops.
 *  - A pool handle is not thread-safe; distinct pools are independent.
 *    Attention calls on one pool must not run concurrently on the GPU: they
 *    share the work counter in the pool's control block.
 *  - bf16 is the only element type.  All tensors are dense and row-major.
 *
 * Layouts (element = bf16 unless stated)
 *   pool       [L][2][num_pages][Hkv][ps][d]    plane 0 = K, plane 1 = V
 *   host_src   [n_blocks][L][2][Hkv][ps][d]     one cached page per block
 *   q, out     [T_new][Hq][d]                   new tokens of all requests,
 *                                               packed request after request
 *   k_new, v_new [T_new][Hkv][d]
 *   block_table  int32 [batch][max_blocks_per_seq]: page of each block of
 *                each request's sequence (prefix pages first)
 *   prefix_lens  int32 [batch]   cached prefix length P_b of each request
 *   new_lens     int32 [batch]   new-token count n_b of each request
 *   cu_new_lens  int32 [batch+1] exclusive prefix sum of new_lens
 *                (cu_new_lens[0] = 0, cu_new_lens[batch] = T_new)
 */
#ifndef GC_H_
#define GC_H_

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h> /* cudaStream_t */

#if defined(__GNUC__)
#define GC_API __attribute__((visibility("default")))
#else
#define GC_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum gc_status {
  GC_OK = 0,
  GC_ERR_INVALID_ARG = 1,  /* null pointer, negative size, inconsistent shape */
  GC_ERR_OUT_OF_RANGE = 2, /* a block id / page / layer outside the pool    */
  GC_ERR_OOM = 3,          /* device allocation failed                       */
  GC_ERR_CUDA = 4,         /* a CUDA runtime call or launch failed           */
  GC_ERR_UNSUPPORTED = 5,  /* valid request this build has no kernel for     */
  GC_ERR_TIMEOUT = 6       /* a device-side wait gave up (kernel returned)   */
} gc_status;

/* Opaque pool handle, owned by the library. */
typedef struct gc_kv_pool gc_kv_pool;

typedef struct gc_pool_config {
  int32_t num_layers;   /* L >= 1                                   */
  int32_t num_kv_heads; /* Hkv >= 1                                 */
  int32_t head_dim;     /* d: 64 or 128                             */
  int32_t page_size;    /* ps tokens per page: 16, 32, 64 or 128    */
  int32_t num_pages;    /* pages per (layer, K/V) plane, >= 1       */
} gc_pool_config;

/* Device bytes a pool of this shape needs: the KV planes
 * (L*2*num_pages*Hkv*ps*d*2 bytes, rounded up to 256) plus a 2048-byte
 * control block (device status word, attention work counter, decode merge
 * counters).
 * Returns 0 for an invalid configuration. */
GC_API size_t gc_kv_pool_bytes(const gc_pool_config* cfg);

/* Create a paged KV pool on the current CUDA device.
 *   dev_mem == NULL: the library allocates gc_kv_pool_bytes(cfg) bytes with
 *                    cudaMalloc and frees them in gc_kv_pool_destroy.
 *   dev_mem != NULL: caller-owned device memory of dev_bytes >=
 *                    gc_kv_pool_bytes(cfg) bytes, 256-byte aligned; the
 *                    library never frees it.
 * The KV planes are not initialised; the control block is cleared.
 * Errors: GC_ERR_INVALID_ARG, GC_ERR_UNSUPPORTED (d or ps), GC_ERR_OOM,
 * GC_ERR_CUDA. */
GC_API gc_status gc_kv_pool_create(const gc_pool_config* cfg, void* dev_mem, size_t dev_bytes,
                            gc_kv_pool** out);

/* Destroy a pool (NULL is a no-op).  Frees library-owned memory only.  The
 * caller must make sure no stream still uses the pool. */
GC_API gc_status gc_kv_pool_destroy(gc_kv_pool* pool);

/* Device address and byte size of the KV planes (control block excluded). */
GC_API gc_status gc_kv_pool_data(const gc_kv_pool* pool, void** dev_ptr, size_t* bytes);

/* Synchronise `stream`, then read and clear the pool's device status word:
 * *device_status receives GC_OK or the first error a kernel recorded since
 * the last check (GC_ERR_OUT_OF_RANGE for a bad device-side index,
 * GC_ERR_TIMEOUT for a device wait that gave up); after an error the
 * control block's decode merge counters are cleared too.  The return value
 * reports failures of the check itself (GC_ERR_CUDA). */
GC_API gc_status gc_kv_pool_check(gc_kv_pool* pool, cudaStream_t stream, int32_t* device_status);

/* gc_kv_restore flags */
#define GC_RESTORE_SRC_DEVICE 1u /* host_src is device memory (already staged) */
#define GC_RESTORE_VECTOR 2u     /* 16-byte vector-copy kernel instead of bulk copies */
#define GC_RESTORE_LAYER_MAJOR 4u /* image is [L][n_blocks][2][Hkv][ps][d] (see below) */

/* Restore cached prefix pages into the pool (Sec. 2.2, Fig. 2a: on a hit
 * the cached KV of the context is loaded instead of recomputed).
 * For i < n_blocks and every layer l and plane kv:
 *     pool[l][kv][block_ids[i]] <- host_src[i][l][kv]
 * a byte-exact copy of Hkv*ps*d*2 bytes; no other page changes.
 *   host_src   [n_blocks][L][2][Hkv][ps][d] bf16.  Pinned host memory
 *              (cudaHostAlloc / cudaHostRegister), or device memory when
 *              flags has GC_RESTORE_SRC_DEVICE.
 *   block_ids  int32 [n_blocks], DEVICE memory.  Ids outside
 *              [0, num_pages) are skipped and recorded as
 *              GC_ERR_OUT_OF_RANGE in the status word.  Duplicate ids give
 *              an unspecified choice between the duplicates' contents.
 *   dev_staging  NULL: the kernel reads host_src directly over the
 *              host-device link (zero copy).  Otherwise device memory of at
 *              least n_blocks*L*2*Hkv*ps*d*2 bytes: host_src is first copied
 *              there with one cudaMemcpyAsync, then scattered.  Ignored with
 *              GC_RESTORE_SRC_DEVICE.
 * Errors: GC_ERR_INVALID_ARG (null/negative, or host_src not pinned on the
 * zero-copy path), GC_ERR_CUDA. */
GC_API gc_status gc_kv_restore(gc_kv_pool* pool, const void* host_src, const int32_t* block_ids,
                        int32_t n_blocks, cudaStream_t stream, void* dev_staging, uint32_t flags);

/* Restore layers [layer_begin, layer_begin + layer_count) of the cached
 * pages only: the same map as gc_kv_restore restricted to those layers
 * (gc_kv_restore is layer_begin 0, layer_count L).  A serving loop calls
 * it once per layer on a side stream, each call followed by an event that
 * the layer's compute waits on, so the restore of later layers overlaps the
 * attention of earlier ones (Sec. 2.2, Fig. 2b: loading the cached KV
 * costs far less time than recomputing it, so the load can hide behind the
 * prefill of the new tokens).
 *   host_src, dev_staging  the whole image [n_blocks][L][2][Hkv][ps][d] and
 *              a device buffer of the same size, as for gc_kv_restore; only
 *              the slices of the chosen layers are read (and, on the staged
 *              path, copied into the same offsets of dev_staging with one
 *              cudaMemcpy2DAsync), so calls for disjoint layer ranges touch
 *              disjoint bytes and may run on different streams.
 *   GC_RESTORE_LAYER_MAJOR  (any restore or save call, with the matching
 *              GC_SAVE_LAYER_MAJOR) the image is laid out [L][n_blocks][2]
 *              [Hkv][ps][d] instead: element (i, l, kv) of the map above sits
 *              at chunk (l*n_blocks + i)*2 + kv.  A layer range is then one
 *              contiguous span and the staged path copies it with one
 *              cudaMemcpyAsync; for the block-major image the strided 2-D
 *              copy of one layer runs at about a third of the contiguous
 *              copy's rate on a GB300 host link, so per-layer callers should
 *              keep their cache images layer-major.
 * Errors: as gc_kv_restore; GC_ERR_OUT_OF_RANGE for a layer range outside
 * [0, L) (layer_count 0 is a no-op). */
GC_API gc_status gc_kv_restore_layers(gc_kv_pool* pool, const void* host_src,
                                      const int32_t* block_ids, int32_t n_blocks,
                                      int32_t layer_begin, int32_t layer_count,
                                      cudaStream_t stream, void* dev_staging, uint32_t flags);

/* gc_kv_stage_layers flag: the images are the 8-bit cache tier's
 * (chunks of gc_kv_q8_chunk_bytes instead of Hkv*ps*d*2 bytes) */
#define GC_STAGE_Q8 8u

/* The host -> device leg of a staged restore on its own (Sec. 2.2: the
 * cached context KV is loaded from the cache tier before the prefill uses
 * it): copies layers [layer_begin, layer_begin + layer_count) of a pinned
 * host image into the same offsets of a device image of the same layout.
 * The scatter into the pool is then gc_kv_restore_layers (or
 * gc_kv_restore_q8) with GC_RESTORE_SRC_DEVICE on that device image.  With
 * the two legs apart, a serving loop can issue every layer's copy on a copy
 * stream, back to back so the host link never waits for a scatter, and run
 * each layer's scatter on the compute stream right before that layer's
 * append and attention, once the layer's copy has landed (an event).
 *   host_src   the whole image, pinned host memory: bf16
 *              [n_blocks][L][2][Hkv][ps][d], or with GC_STAGE_Q8 the 8-bit
 *              image [n_blocks][L][2][gc_kv_q8_chunk_bytes]; with
 *              GC_RESTORE_LAYER_MAJOR the layer-major layouts [L][n_blocks]...
 *   dev_image  device memory of the whole image's size (16-byte aligned);
 *              only the chosen layers' slices are written.
 *   Nothing is launched: the copies are cudaMemcpyAsync (one per call for a
 *   layer-major image or all layers; one cudaMemcpy2DAsync of the strided
 *   slices otherwise).  The pool is only read for its geometry.
 * Errors: GC_ERR_INVALID_ARG (null/negative, unknown flags, host_src not
 * pinned, dev_image misaligned), GC_ERR_OUT_OF_RANGE (layer range outside
 * [0, L)), GC_ERR_CUDA. */
GC_API gc_status gc_kv_stage_layers(const gc_kv_pool* pool, const void* host_src,
                                    void* dev_image, int32_t n_blocks, int32_t layer_begin,
                                    int32_t layer_count, cudaStream_t stream, uint32_t flags);

/* gc_kv_save flags */
#define GC_SAVE_DST_DEVICE 1u /* host_dst is device memory (gather only) */
#define GC_SAVE_VECTOR 2u     /* 16-byte vector-copy kernel instead of bulk copies */
#define GC_SAVE_LAYER_MAJOR 4u /* image is [L][n_blocks][2][Hkv][ps][d] */

/* Save pool pages to the cache tier (Sec. 2.2, Fig. 2a step 1: once a
 * request has been processed its KV is saved to storage); the inverse of
 * gc_kv_restore.  For i < n_blocks and every layer l and plane kv:
 *     host_dst[i][l][kv] <- pool[l][kv][block_ids[i]]
 * a byte-exact copy of Hkv*ps*d*2 bytes per (i, l, kv).
 *   host_dst   [n_blocks][L][2][Hkv][ps][d] bf16.  Pinned host memory, or
 *              device memory when flags has GC_SAVE_DST_DEVICE.  The caller
 *              reads it after the stream has passed the call.
 *   block_ids  int32 [n_blocks], DEVICE memory.  Ids outside [0, num_pages)
 *              are skipped and recorded as GC_ERR_OUT_OF_RANGE in the status
 *              word: their chunk of the written image (host_dst, or
 *              dev_staging on the staged path, which is then copied to
 *              host_dst whole) is not written.
 *   dev_staging  NULL: the kernel writes host_dst directly over the
 *              host-device link (zero copy).  Otherwise device memory of at
 *              least n_blocks*L*2*Hkv*ps*d*2 bytes: the pages are gathered
 *              there, then copied to host_dst with one cudaMemcpyAsync.
 *              Ignored with GC_SAVE_DST_DEVICE.
 * Errors: GC_ERR_INVALID_ARG (null/negative, unaligned, or host_dst not
 * pinned), GC_ERR_CUDA. */
GC_API gc_status gc_kv_save(gc_kv_pool* pool, void* host_dst, const int32_t* block_ids,
                            int32_t n_blocks, cudaStream_t stream, void* dev_staging,
                            uint32_t flags);

/* Save layers [layer_begin, layer_begin + layer_count) of the pages only:
 * gc_kv_save restricted to those layers, written into the same offsets of
 * the whole image [n_blocks][L][2][Hkv][ps][d] (host_dst, and dev_staging
 * on the staged path, are whole-image buffers; other layers' bytes are not
 * written).  Lets a request's KV be offloaded layer by layer as each layer
 * finishes (Sec. 2.2, Fig. 2a step 1).
 * Errors: as gc_kv_save; GC_ERR_OUT_OF_RANGE for a layer range outside
 * [0, L) (layer_count 0 is a no-op). */
GC_API gc_status gc_kv_save_layers(gc_kv_pool* pool, void* host_dst, const int32_t* block_ids,
                                   int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                                   cudaStream_t stream, void* dev_staging, uint32_t flags);

/* ---- 8-bit cache tier.  The 70B runs of Sec. 6.1 use INT8; keeping the
 * cached KV in 8 bits halves what the cache tier stores (the storage whose
 * embodied carbon Sec. 3.2, Eq. 4 charges per allocated byte) and what the
 * host link carries on a restore.  The pool stays bf16.
 * Quantisation is symmetric absmax INT8 with one binary32 scale per
 * (block, layer, plane kv, kv head g) group of ps*d values x:
 *     amax = max |x| over the group's finite values
 *     s    = amax / 127
 *     c    = clamp(round_half_even(x * (127 / amax)), -127, 127)
 *            (c = 0 for NaN x; every c = 0 when amax = 0)
 * each product and quotient rounded once in binary32; restore writes
 *     pool value = bf16_round_half_even(c * s).
 * Image: [n_blocks][L][2][chunk] (or [L][n_blocks][2][chunk] with the
 * LAYER_MAJOR flag), chunk = gc_kv_q8_chunk_bytes(cfg) bytes: Hkv binary32
 * scales, zero bytes up to a multiple of 16, then codes [Hkv][ps][d] int8.
 * Both calls take the same layer range, source / destination modes
 * (pinned host through dev_staging, zero copy with dev_staging NULL, or a
 * device image with GC_RESTORE_SRC_DEVICE / GC_SAVE_DST_DEVICE), block-id
 * checks and errors as gc_kv_restore_layers / gc_kv_save_layers; the
 * *_VECTOR flags do not apply. */
GC_API size_t gc_kv_q8_chunk_bytes(const gc_pool_config* cfg);  /* 0 if invalid */

/* Quantise pages block_ids[i], layers [layer_begin, layer_begin+layer_count),
 * into the 8-bit image (chunks of other layers are not written). */
GC_API gc_status gc_kv_save_q8(gc_kv_pool* pool, void* dst, const int32_t* block_ids,
                               int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                               cudaStream_t stream, void* dev_staging, uint32_t flags);

/* Dequantise the 8-bit image's chunks of those layers into pool pages
 * block_ids[i]; no other page or layer changes. */
GC_API gc_status gc_kv_restore_q8(gc_kv_pool* pool, const void* src, const int32_t* block_ids,
                                  int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                                  cudaStream_t stream, void* dev_staging, uint32_t flags);

/* Append the new tokens' K and V after each request's cached prefix
 * (Sec. 2.2: the KV of the cached tokens and of the new tokens is stitched
 * into one sequence).  For request b, new token t < n_b and kv head g:
 *     pos = seq_lens[b] + t
 *     pool[layer][0][block_table[b][pos/ps]][g][pos%ps] <- k_new[cu_new_lens[b]+t][g]
 *     pool[layer][1][...same slot...]                   <- v_new[cu_new_lens[b]+t][g]
 *   k_new, v_new  [T_new][Hkv][d] bf16, device.
 *   block_table   int32 [batch][max_blocks_per_seq], device.
 *   seq_lens      int32 [batch], device: the write offset of each request,
 *                 i.e. its cached prefix length P_b.
 *   cu_new_lens   int32 [batch+1], device.
 * A token whose block index is >= max_blocks_per_seq or whose page is
 * outside the pool is skipped and recorded as GC_ERR_OUT_OF_RANGE.
 *   total_new_tokens  T_new = cu_new_lens[batch], passed from the host; it
 *                 sizes the grid and bounds every k_new / v_new row read.
 *                 A request whose rows would pass it is skipped and
 *                 recorded as GC_ERR_OUT_OF_RANGE.
 * Errors: GC_ERR_INVALID_ARG, GC_ERR_OUT_OF_RANGE (layer), GC_ERR_CUDA. */
GC_API gc_status gc_kv_append(gc_kv_pool* pool, const void* k_new, const void* v_new,
                       const int32_t* block_table, const int32_t* seq_lens, cudaStream_t stream,
                       int32_t layer, const int32_t* cu_new_lens, int32_t batch,
                       int32_t max_blocks_per_seq, int32_t total_new_tokens);

/* Prefill of the new tokens over [cached prefix ++ new tokens] (Sec. 2.2:
 * the cached and new tokens' KV are processed together; Sec. 2.1: prefill).
 * For request b, q head h and new row i < n_b, with g = h / (Hq/Hkv),
 * P = prefix_lens[b] and keys j read through block_table[b]:
 *     out[cu_new_lens[b]+i][h] = sum_{j <= P+i} softmax_j(softmax_scale *
 *                                   q[cu_new_lens[b]+i][h] . k_j) v_j
 * i.e. causal attention bottom-right aligned: new row i sits at absolute
 * position P+i.  The result equals the corresponding rows of a full causal
 * prefill of the concatenated sequence.  Keys at positions >= P_b + n_b are
 * never used, whatever their contents (NaN included).
 *   q, out      [T_new][Hq][d] bf16, device (out is written for valid rows
 *               only).  Accumulation is fp32, P is rounded to bf16 before
 *               the PV product, out is rounded to nearest even.
 *   prefix_lens, new_lens  int32 [batch], device.  cu_new_lens int32
 *               [batch+1], device, consistent with new_lens.
 *   num_q_heads Hq, a multiple of the pool's Hkv with Hq/Hkv in
 *               {1,2,4,8,16}.
 *   total_new_tokens  T_new = cu_new_lens[batch], passed from the host; it
 *               bounds every q / out row access.  A request whose rows would
 *               pass it is skipped and recorded as GC_ERR_OUT_OF_RANGE.
 *   Kernels: head_dim 128 runs on pairs of SMs (tcgen05 cta_group::2, each
 *   K/V tile split between the two SMs); head_dim 64 runs one work item per
 *   SM.  Both compute the same operation to the same tolerance.
 *   Size limit: the kernel numbers its work items (a kv head of a request
 *   and 256 of its q rows) with 32-bit ints, so T_new * (Hq/Hkv) + 256 and
 *   Hkv * (T_new * (Hq/Hkv) / 256 + batch) + 2 * (SM count) must both stay
 *   at or below 2^31 - 1; a larger call fails with GC_ERR_UNSUPPORTED before
 *   anything is launched.
 * Errors: GC_ERR_INVALID_ARG, GC_ERR_OUT_OF_RANGE (layer),
 * GC_ERR_UNSUPPORTED (head grouping, size limit), GC_ERR_CUDA. */
GC_API gc_status gc_prefix_prefill_attn(const void* q, const gc_kv_pool* pool, const int32_t* block_table,
                                 const int32_t* prefix_lens, const int32_t* new_lens, void* out,
                                 cudaStream_t stream, int32_t layer, const int32_t* cu_new_lens,
                                 int32_t batch, int32_t max_blocks_per_seq, int32_t num_q_heads,
                                 float softmax_scale, int32_t total_new_tokens);

/* Same operation, arguments and result as gc_prefix_prefill_attn, for
 * callers that cannot allocate device memory.  The paper has no counterpart:
 * this entry point serves code that runs inside a device-memory budget it
 * does not control, for example a plugin living in a framework whose caching
 * allocator has reserved the GPU's memory, or a runtime that forbids
 * allocation while it serves.  Such a caller creates its pool in memory it
 * already owns (gc_kv_pool_create with dev_mem) and calls this function.
 *   It allocates nothing: the only scratch the kernel needs (its work-item
 *   counter) is a 256-byte array inside libgc's device image, which every GPU
 *   that loads the library holds until the process exits.  The first call on
 *   a device looks up the array's device address (cudaGetSymbolAddress) with
 *   that device current; make that first call before any stream capture.
 *   The address is kept per device and CUDA context: after a device reset
 *   (cudaDeviceReset) the next call finds a new context and looks it up
 *   again, so that call too should come before any stream capture.
 *   Each call clears the counter with a stream-ordered memset.
 *   All calls share the array, on every pool: two calls that overlap on the
 *   GPU race on it and give wrong results.  Serialise them.
 *   Limit: the size limit of gc_prefix_prefill_attn, i.e. at most
 *   2^31 - 1 - 2 * (SM count) work items,
 *   Hkv * (total_new_tokens * (Hq/Hkv) / 256 + batch), per call; larger
 *   calls fail with GC_ERR_UNSUPPORTED before anything is launched.
 *   The current device must be the pool's device (GC_ERR_INVALID_ARG).
 * Other errors as gc_prefix_prefill_attn. */
GC_API gc_status gc_prefix_prefill_attn_noalloc(const void* q, const gc_kv_pool* pool,
                                                const int32_t* block_table,
                                                const int32_t* prefix_lens,
                                                const int32_t* new_lens, void* out,
                                                cudaStream_t stream, int32_t layer,
                                                const int32_t* cu_new_lens, int32_t batch,
                                                int32_t max_blocks_per_seq, int32_t num_q_heads,
                                                float softmax_scale, int32_t total_new_tokens);

/* Prefill over a context whose cached pages stay in the 8-bit cache tier
 * (Sec. 6.1: the 70B runs keep the KV in INT8; Sec. 3.2: an 8-bit tier
 * halves what storage holds and what a restore moves).  The operation is
 * gc_kv_restore_q8 of the 8-bit pages into the pool followed by
 * gc_prefix_prefill_attn, but the pages are never written to the pool: the
 * kernel dequantises each one (x' = bf16_rne(c * s), the restore's
 * rounding) into the tile it would have loaded.  At head_dim 64 the result
 * is bit-identical to those two calls (both run on the one-SM kernel); at
 * head_dim 128 gc_prefix_prefill_attn runs on SM pairs, whose sums run in
 * another order, and the two agree within the attention tolerance.
 * Arguments as gc_prefix_prefill_attn, plus:
 *   q8_image   device memory, 16-byte aligned: the 8-bit image
 *              [n_image_blocks][L][2][gc_kv_q8_chunk_bytes], or with
 *              GC_RESTORE_LAYER_MAJOR in flags [L][n_image_blocks][2][...],
 *              as gc_kv_save_q8 writes it (e.g. staged by
 *              gc_kv_stage_layers with GC_STAGE_Q8).  Only the chunks of
 *              `layer` are read.
 *   q8_table   int32 [batch][max_blocks_per_seq], device: for page j of
 *              request b, an image block in [0, n_image_blocks) to read it
 *              from, or -1 to read pool page block_table[b][j] as
 *              gc_prefix_prefill_attn does (new tokens' pages, or pages
 *              already resident).  An entry >= n_image_blocks is skipped
 *              (the output of that request is then unspecified) and
 *              recorded as GC_ERR_OUT_OF_RANGE.
 *   n_image_blocks  blocks in the image (>= 0).
 *   flags      0 or GC_RESTORE_LAYER_MAJOR.
 * Both head sizes run on a 16-warp variant of the one-SM kernel: the
 * producer loads each image page's codes into the K/V ring (TMA) and a
 * fourth warpgroup dequantises them there, while the TMA unit loads the
 * pool pages.  Shared memory limits batch to 8192 as for
 * gc_prefix_prefill_attn.  Every work item dequantises its own copy of the
 * pages it reads, so with many new tokens per cached page the two-step path
 * (gc_kv_restore_q8, then gc_prefix_prefill_attn) is faster; this call
 * keeps no bf16 copy of the cached pages in the pool.
 * Errors: as gc_prefix_prefill_attn; GC_ERR_INVALID_ARG also for unknown
 * flags, a NULL q8_table (or q8_image with n_image_blocks > 0), a
 * misaligned q8_image. */
GC_API gc_status gc_prefix_prefill_attn_q8(const void* q, const gc_kv_pool* pool,
                                           const int32_t* block_table, const int32_t* prefix_lens,
                                           const int32_t* new_lens, void* out,
                                           cudaStream_t stream, int32_t layer,
                                           const int32_t* cu_new_lens, int32_t batch,
                                           int32_t max_blocks_per_seq, int32_t num_q_heads,
                                           float softmax_scale, int32_t total_new_tokens,
                                           const void* q8_image, const int32_t* q8_table,
                                           int32_t n_image_blocks, uint32_t flags);

/* Same operation and arguments as gc_prefix_prefill_attn, computed by a
 * plain CUDA-core kernel (one warp per row, fp32 throughout, no tensor
 * cores).  Slow; kept as an independent GPU cross-check of the indexing. */
GC_API gc_status gc_prefix_prefill_attn_simt(const void* q, const gc_kv_pool* pool,
                                      const int32_t* block_table, const int32_t* prefix_lens,
                                      const int32_t* new_lens, void* out, cudaStream_t stream,
                                      int32_t layer, const int32_t* cu_new_lens, int32_t batch,
                                      int32_t max_blocks_per_seq, int32_t num_q_heads,
                                      float softmax_scale, int32_t total_new_tokens);

/* Paged decode attention: one new token per request (Sec. 2.1: the decode
 * phase generates output tokens one at a time, and with the KV cache it is
 * bound by memory).  For request b, q head h and g = h / (Hq/Hkv):
 *     out[b][h] = sum_{j < seq_lens[b]} softmax_j(softmax_scale *
 *                                         q[b][h] . k_j) v_j
 * with k_j, v_j read from pool[layer] through block_table[b]; the new
 * token's own K/V must already be in the pool at position seq_lens[b] - 1
 * (gc_kv_append with one new token).  Equals gc_prefix_prefill_attn with
 * prefix_lens = seq_lens - 1 and one new token per request.
 *   q, out      [batch][Hq][d] bf16, device.  fp32 arithmetic, out rounded
 *               to nearest even.
 *   seq_lens    int32 [batch], device: context length T_b >= 1 including
 *               the new token; a request whose length is outside
 *               [1, max_blocks_per_seq*ps] is skipped (its out rows are not
 *               written) and recorded as GC_ERR_OUT_OF_RANGE.
 *   block_table int32 [batch][max_blocks_per_seq], device; a bad page is
 *               skipped (its keys left out) and recorded.
 *   workspace   device scratch for the partial results of requests split
 *               over several CTAs: gc_paged_decode_workspace_bytes(pool,
 *               batch, max_blocks_per_seq, num_q_heads) bytes (0: NULL is
 *               fine), owned by the caller, not used after the stream passes
 *               the call; no initial contents needed.  Calls sharing a
 *               workspace must not overlap on the GPU.
 * d = 128 with Hq/Hkv <= 16 runs on a transposed tensor-core kernel (keys on
 * the 128-row side of the MMA) that gives every SM an equal share of the K/V
 * tiles; a request cut between shares is combined by the last CTA to finish
 * it.  Other shapes run on the prefill kernel's tensor-core path in a decode
 * mode.  Calls on one pool must not overlap on the GPU with each other or
 * with gc_prefix_prefill_attn (they share counters in the pool's control
 * block).
 * Errors: GC_ERR_INVALID_ARG (null, unaligned, workspace too small),
 * GC_ERR_OUT_OF_RANGE (layer), GC_ERR_UNSUPPORTED (head grouping,
 * batch > 8192), GC_ERR_CUDA. */
GC_API size_t gc_paged_decode_workspace_bytes(const gc_kv_pool* pool, int32_t batch,
                                              int32_t max_blocks_per_seq, int32_t num_q_heads);
GC_API gc_status gc_paged_decode_attn(const void* q, const gc_kv_pool* pool,
                                      const int32_t* block_table, const int32_t* seq_lens,
                                      void* out, cudaStream_t stream, int32_t layer,
                                      int32_t batch, int32_t max_blocks_per_seq,
                                      int32_t num_q_heads, float softmax_scale, void* workspace,
                                      size_t workspace_bytes);

/* Paged decode attention with the cached pages read from the 8-bit cache
 * tier (Sec. 6.1: the 70B runs keep the KV in INT8; Sec. 2.1: decode is
 * bound by memory, and an 8-bit page is half the bytes).  The result is
 * exactly that of gc_kv_restore_q8 of the image pages into the pool followed
 * by gc_paged_decode_attn: the kernel dequantises each image page
 * (x' = bf16_rne(c * s), the restore's rounding) into the tile it would have
 * loaded, and the pool is never written.
 * Arguments as gc_paged_decode_attn, plus q8_image, q8_table, n_image_blocks
 * and flags as gc_prefix_prefill_attn_q8 (q8_table [batch][max_blocks_per_seq]:
 * an image block >= 0, or -1 for a pool page, e.g. the page the new token
 * was appended to).  Kernels: head_dim 128 runs the transposed decode kernel
 * with a converter warpgroup, head_dim 64 the decode mode of the 8-bit
 * prefill variant (gc_prefix_prefill_attn_q8); both dequantise with the
 * restore's rounding.
 * Errors: as gc_paged_decode_attn; GC_ERR_INVALID_ARG also for unknown flags, a NULL q8_table (or q8_image with
 * n_image_blocks > 0), a misaligned q8_image. */
GC_API gc_status gc_paged_decode_attn_q8(const void* q, const gc_kv_pool* pool,
                                         const int32_t* block_table, const int32_t* seq_lens,
                                         void* out, cudaStream_t stream, int32_t layer,
                                         int32_t batch, int32_t max_blocks_per_seq,
                                         int32_t num_q_heads, float softmax_scale,
                                         void* workspace, size_t workspace_bytes,
                                         const void* q8_image, const int32_t* q8_table,
                                         int32_t n_image_blocks, uint32_t flags);

/* Test hook, not part of the method (the paper has no counterpart): launches
 * one thread that waits on a device barrier nobody arrives at, with the same
 * bounded wait every libgc kernel uses.  After its limit (about 1.5 s) the
 * wait gives up, GC_ERR_TIMEOUT is recorded in the pool's status word (read
 * with gc_kv_pool_check) and the kernel returns, so the timeout path can be
 * exercised without hanging the GPU.  Errors: GC_ERR_INVALID_ARG, GC_ERR_CUDA. */
GC_API gc_status gc_selftest_wait_timeout(gc_kv_pool* pool, cudaStream_t stream);

/* Message of the last failing call on this thread ("" if none). */
GC_API const char* gc_last_error(void);

/* Static name of a status code. */
GC_API const char* gc_status_string(gc_status s);

#ifdef __cplusplus
}
#endif

#endif /* GC_H_ */
