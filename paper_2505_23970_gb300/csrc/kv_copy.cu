// Paged KV movement: restore (cached pages -> pool) and append (new tokens'
// K, V -> pool slots after each request's cached prefix).  Both are pure
// byte copies (Sec. 2.2: the cached KV is loaded, not recomputed, and the
// new tokens' KV is stitched after it), so the kernels are bandwidth-bound
// and bit-exact.
//
// Restore moves chunks of C = Hkv*ps*d*2 bytes: chunk (i, l, kv) of the
// staging image [n_blocks][L][2][chunk] goes to pool[l][kv][block_ids[i]],
// for the layers l of one contiguous range [layer0, layer0 + layers) (all L
// for a whole-request restore, one layer when restores are pipelined with
// the layers' compute).  A layer-major image [L][n_blocks][2][chunk] is
// also accepted (one contiguous span per layer range).
// Save (Sec. 2.2, Fig. 2a step 1: a processed request's KV is saved to the
// cache tier) is the same map run backwards: pool pages -> staging image.
// The bulk kernel streams 16 KB pieces global -> shared -> global with
// cp.async.bulk (one issuing thread per CTA, a ring of mbarrier-tracked
// stages); the vector kernel uses 16-byte loads/stores and is also the
// zero-copy path that reads pinned host memory directly.
#include "gc_internal.cuh"
#include "sm103_ptx.cuh"

namespace gc {
namespace {

constexpr int kPiece = 16384;   // bytes per bulk copy
constexpr int kStages = 6;      // pieces in flight per CTA
constexpr int kBulkCtasPerSm = 2;

struct RestoreGeom {
  uint64_t chunk_bytes;     // C
  uint32_t pieces;          // ceil(C / kPiece)
  int32_t L, num_pages;     // layers of the pool and of the image; pages of the pool
  int32_t layer0, layers;   // the layer range moved
  int32_t layer_major;      // image is [L][n_blocks][2][chunk] instead of [n_blocks][L][2][chunk]
  int32_t n_blocks;
  int32_t gather;           // 0: staging -> pool (restore), 1: pool -> staging (save)
};

// Index of chunk (block i, layer l, plane kv) in the staging image.
__device__ __forceinline__ uint64_t image_chunk(const RestoreGeom& g, int64_t i, int l, int kv) {
  const uint64_t il = g.layer_major ? static_cast<uint64_t>(l) * g.n_blocks + i
                                    : static_cast<uint64_t>(i) * g.L + l;
  return il * 2 + kv;
}

__device__ __forceinline__ bool piece_addr(const RestoreGeom& g, uint8_t* staging, uint8_t* pool,
                                           const int32_t* block_ids, int32_t* status, uint64_t u,
                                           const uint8_t** s_out, uint8_t** d_out,
                                           uint32_t* bytes) {
  const uint64_t c = u / g.pieces;
  const uint32_t piece = static_cast<uint32_t>(u - c * g.pieces);
  const int64_t i = static_cast<int64_t>(c / (2 * g.layers));
  const int lr = static_cast<int>((c / 2) % g.layers);
  const int l = g.layer0 + lr;
  const int kv = static_cast<int>(c % 2);
  const int32_t id = __ldg(block_ids + i);
  if (id < 0 || id >= g.num_pages) {
    if (piece == 0 && lr == 0 && kv == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
    return false;
  }
  const uint64_t off = static_cast<uint64_t>(piece) * kPiece;
  const uint64_t rem = g.chunk_bytes - off;
  *bytes = static_cast<uint32_t>(rem < kPiece ? rem : kPiece);
  uint8_t* stg = staging + image_chunk(g, i, l, kv) * g.chunk_bytes + off;
  uint8_t* pl = pool + ((static_cast<uint64_t>(l) * 2 + kv) * g.num_pages + id) * g.chunk_bytes + off;
  *s_out = g.gather ? pl : stg;
  *d_out = g.gather ? stg : pl;
  return true;
}

__global__ void __launch_bounds__(32) restore_bulk_kernel(uint8_t* __restrict__ staging,
                                                          uint8_t* __restrict__ pool,
                                                          const int32_t* __restrict__ block_ids,
                                                          RestoreGeom g, int32_t* status) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ uint64_t full[kStages];
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  for (int s = 0; s < kStages; ++s) ptx::mbar_init(&full[s], 1);
  abort_flag = 0;
  ptx::fence_barrier_init();

  const uint64_t units = static_cast<uint64_t>(g.n_blocks) * g.layers * 2 * g.pieces;
  uint64_t next = blockIdx.x;  // next candidate unit of this CTA
  uint8_t* dst_of[kStages];
  uint32_t bytes_of[kStages];

  // issue the load of this CTA's next valid unit into `slot`
  auto issue = [&](int slot) -> bool {
    while (next < units) {
      const uint8_t* s;
      uint8_t* d;
      uint32_t b;
      const bool ok = piece_addr(g, staging, pool, block_ids, status, next, &s, &d, &b);
      next += gridDim.x;
      if (!ok) continue;
      dst_of[slot] = d;
      bytes_of[slot] = b;
      ptx::mbar_arrive_expect_tx(&full[slot], b);
      ptx::bulk_load(smem + slot * kPiece, s, b, &full[slot]);
      return true;
    }
    return false;
  };

  int issued = 0;
  while (issued < kStages && issue(issued)) ++issued;
  bool ok = true;
  int consumed = 0;  // loads [0, consumed) have landed
  for (int k = 0; k < issued; ++k) {
    const int slot = k % kStages;
    if (!ptx::mbar_wait(&full[slot], (k / kStages) & 1, &abort_flag)) {
      ok = false;
      break;
    }
    consumed = k + 1;
    ptx::bulk_store(dst_of[slot], smem + slot * kPiece, bytes_of[slot]);
    ptx::bulk_commit();
    if (k >= 1) {
      ptx::bulk_wait_read<1>();  // store k-1 has finished reading its slot
      const int free_slot = (k - 1) % kStages;
      if (issue(free_slot)) ++issued;
    }
  }
  ptx::bulk_wait_all();
  if (!ok) {
    record_error(status, GC_ERR_TIMEOUT);
    // let the loads still in flight land before the CTA exits (bounded):
    // only loads [consumed, issued), at most kStages, one per slot
    for (int k = consumed; k < issued; ++k) {
      int dummy = 0;
      ptx::mbar_wait(&full[k % kStages], (k / kStages) & 1, &dummy);
    }
  }
}

__global__ void __launch_bounds__(256) restore_vector_kernel(uint4* __restrict__ staging,
                                                             uint8_t* __restrict__ pool,
                                                             const int32_t* __restrict__ block_ids,
                                                             RestoreGeom g, int32_t* status) {
  const uint64_t words_per_chunk = g.chunk_bytes / 16;
  const uint64_t total = static_cast<uint64_t>(g.n_blocks) * g.layers * 2 * words_per_chunk;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  constexpr int U = 4;
  for (uint64_t base = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; base < total;
       base += stride * U) {
    uint4 v[U];
    uint4* dst[U];  // destination word; the source was read into v
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const uint64_t w = base + k * stride;
      dst[k] = nullptr;
      if (w < total) {
        const uint64_t c = w / words_per_chunk;
        const uint64_t off = w - c * words_per_chunk;
        const int64_t i = static_cast<int64_t>(c / (2 * g.layers));
        const int lr = static_cast<int>((c / 2) % g.layers);
        const int l = g.layer0 + lr;
        const int kv = static_cast<int>(c % 2);
        const int32_t id = __ldg(block_ids + i);
        if (id < 0 || id >= g.num_pages) {
          if (off == 0 && lr == 0 && kv == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
          continue;
        }
        uint4* sw = staging + image_chunk(g, i, l, kv) * words_per_chunk + off;
        uint4* pl = reinterpret_cast<uint4*>(
                        pool + ((static_cast<uint64_t>(l) * 2 + kv) * g.num_pages + id) *
                                   g.chunk_bytes) +
                    off;
        if (g.gather) {
          v[k] = *pl;
          dst[k] = sw;
        } else {
          v[k] = *sw;
          dst[k] = pl;
        }
      }
    }
#pragma unroll
    for (int k = 0; k < U; ++k)
      if (dst[k]) *dst[k] = v[k];
  }
}

// ------------------------------------------------------------------ append
struct AppendGeom {
  int32_t Hkv, ps_shift, num_pages, n16, batch, max_blocks, layer, total_new;
};

__global__ void __launch_bounds__(256) append_kernel(const uint4* __restrict__ k_new,
                                                     const uint4* __restrict__ v_new,
                                                     uint8_t* __restrict__ pool,
                                                     const int32_t* __restrict__ block_table,
                                                     const int32_t* __restrict__ prefix_lens,
                                                     const int32_t* __restrict__ cu_new_lens,
                                                     AppendGeom g, int32_t* status) {
  const int ps = 1 << g.ps_shift;
  const uint64_t total = static_cast<uint64_t>(g.total_new) * 2 * g.Hkv * g.n16;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t w = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; w < total;
       w += stride) {
    const int c16 = static_cast<int>(w % g.n16);
    uint64_t rest = w / g.n16;
    const int h = static_cast<int>(rest % g.Hkv);
    rest /= g.Hkv;
    const int kv = static_cast<int>(rest % 2);
    const int t = static_cast<int>(rest / 2);
    // request b with cu[b] <= t < cu[b+1]: last b whose start is <= t
    int lo = 0, hi = g.batch;  // invariant: answer in [lo, hi)
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (__ldg(cu_new_lens + mid) <= t) lo = mid; else hi = mid;
    }
    const int b = lo;
    const int start = __ldg(cu_new_lens + b);
    const int end = __ldg(cu_new_lens + b + 1);
    if (t < start || t >= end || end > g.total_new) {
      record_error(status, GC_ERR_OUT_OF_RANGE);
      continue;
    }
    const int pos = __ldg(prefix_lens + b) + (t - start);
    const int blk = pos >> g.ps_shift;
    if (pos < 0 || blk >= g.max_blocks) {
      record_error(status, GC_ERR_OUT_OF_RANGE);
      continue;
    }
    const int page = __ldg(block_table + static_cast<int64_t>(b) * g.max_blocks + blk);
    if (page < 0 || page >= g.num_pages) {
      record_error(status, GC_ERR_OUT_OF_RANGE);
      continue;
    }
    const uint64_t row = ((((static_cast<uint64_t>(g.layer) * 2 + kv) * g.num_pages + page) * g.Hkv + h) *
                              ps + (pos & (ps - 1)));
    const uint4* src = (kv ? v_new : k_new) + (static_cast<uint64_t>(t) * g.Hkv + h) * g.n16 + c16;
    reinterpret_cast<uint4*>(pool)[row * g.n16 + c16] = __ldg(src);
  }
}

// Self-test of the bounded device wait every libgc kernel uses: one thread
// waits on a barrier nobody arrives at; the wait gives up after its cycle
// limit and the kernel records GC_ERR_TIMEOUT and returns.
__global__ void __launch_bounds__(32) selftest_timeout_kernel(int32_t* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  ptx::mbar_init(&bar, 1);
  abort_flag = 0;
  ptx::fence_barrier_init();
  if (!ptx::mbar_wait(&bar, 0, &abort_flag)) record_error(status, GC_ERR_TIMEOUT);
}

int ilog2(int x) {
  int s = 0;
  while ((1 << s) < x) ++s;
  return s;
}

}  // namespace

gc_status launch_selftest_timeout(const gc_kv_pool* pool, cudaStream_t stream) {
  selftest_timeout_kernel<<<1, 32, 0, stream>>>(pool->status);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_selftest_wait_timeout: launch");
  return GC_OK;
}

gc_status launch_restore_bulk(const gc_kv_pool* pool, uint8_t* staging,
                              const int32_t* block_ids, int32_t n_blocks, int32_t layer0,
                              int32_t layers, bool layer_major, bool gather,
                              cudaStream_t stream) {
  RestoreGeom g;
  g.gather = gather ? 1 : 0;
  g.chunk_bytes = page_bytes(pool->cfg);
  g.pieces = static_cast<uint32_t>((g.chunk_bytes + kPiece - 1) / kPiece);
  g.L = pool->cfg.num_layers;
  g.num_pages = pool->cfg.num_pages;
  g.n_blocks = n_blocks;
  g.layer0 = layer0;
  g.layers = layers;
  g.layer_major = layer_major ? 1 : 0;
  const uint64_t units = static_cast<uint64_t>(n_blocks) * layers * 2 * g.pieces;
  uint64_t grid = static_cast<uint64_t>(pool->num_sms) * kBulkCtasPerSm;
  if (grid > units) grid = units;
  const int smem = kStages * kPiece;
  cudaError_t ea =
      cudaFuncSetAttribute(restore_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (ea != cudaSuccess) return cuda_fail(ea, "gc_kv_restore: smem attribute");
  restore_bulk_kernel<<<static_cast<unsigned>(grid), 32, smem, stream>>>(staging, pool->data,
                                                                           block_ids, g,
                                                                           pool->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_kv_restore: bulk kernel launch");
  return GC_OK;
}

gc_status launch_restore_vector(const gc_kv_pool* pool, uint8_t* staging,
                                const int32_t* block_ids, int32_t n_blocks, int32_t layer0,
                                int32_t layers, bool layer_major, bool gather,
                                cudaStream_t stream) {
  RestoreGeom g;
  g.gather = gather ? 1 : 0;
  g.chunk_bytes = page_bytes(pool->cfg);
  g.pieces = 1;
  g.L = pool->cfg.num_layers;
  g.num_pages = pool->cfg.num_pages;
  g.n_blocks = n_blocks;
  g.layer0 = layer0;
  g.layers = layers;
  g.layer_major = layer_major ? 1 : 0;
  const uint64_t words = static_cast<uint64_t>(n_blocks) * layers * 2 * (g.chunk_bytes / 16);
  uint64_t grid = (words + 256 * 4 - 1) / (256 * 4);
  const uint64_t cap = static_cast<uint64_t>(pool->num_sms) * 8;
  if (grid > cap) grid = cap;
  restore_vector_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(
      reinterpret_cast<uint4*>(staging), pool->data, block_ids, g, pool->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_kv_restore: vector kernel launch");
  return GC_OK;
}

gc_status launch_append(const gc_kv_pool* pool, const void* k_new, const void* v_new,
                        const int32_t* block_table, const int32_t* prefix_lens,
                        const int32_t* cu_new_lens, int32_t batch, int32_t max_blocks,
                        int32_t layer, int32_t total_new_tokens, cudaStream_t stream) {
  AppendGeom g;
  g.Hkv = pool->cfg.num_kv_heads;
  g.ps_shift = ilog2(pool->cfg.page_size);
  g.num_pages = pool->cfg.num_pages;
  g.n16 = pool->cfg.head_dim * 2 / 16;
  g.batch = batch;
  g.max_blocks = max_blocks;
  g.layer = layer;
  g.total_new = total_new_tokens;
  const uint64_t words = static_cast<uint64_t>(total_new_tokens) * 2 * g.Hkv * g.n16;
  uint64_t grid = (words + 255) / 256;
  const uint64_t cap = static_cast<uint64_t>(pool->num_sms) * 16;
  if (grid > cap) grid = cap;
  append_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(
      static_cast<const uint4*>(k_new), static_cast<const uint4*>(v_new), pool->data, block_table,
      prefix_lens, cu_new_lens, g, pool->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_kv_append: kernel launch");
  return GC_OK;
}

}  // namespace gc
