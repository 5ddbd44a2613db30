// C ABI of libgc: pool management, host-side argument checks and dispatch to
// the CUDA kernels.  Nothing here computes on the host: every byte of the
// restore, append and attention results is produced by a kernel.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>

#include <nvtx3/nvToolsExt.h>

#include "gc_internal.cuh"

namespace {
thread_local char g_msg[512] = "";
// control block after the KV planes: status word, work counter (at 128 bytes),
// the decode merge counters (from 256 bytes)
constexpr size_t kTrailer = 2048;
}  // namespace

namespace gc {

gc_status fail(gc_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof g_msg, fmt, ap);
  va_end(ap);
  return s;
}

gc_status cuda_fail(cudaError_t e, const char* what) {
  return fail(e == cudaErrorMemoryAllocation ? GC_ERR_OOM : GC_ERR_CUDA, "%s: %s (%s)", what,
              cudaGetErrorName(e), cudaGetErrorString(e));
}

}  // namespace gc

using gc::fail;

// An NVTX range around every data-path call, so that profiler timelines show
// which libgc call each kernel belongs to (no cost without a profiler).
namespace {
struct Range {
  explicit Range(const char* name) { nvtxRangePushA(name); }
  ~Range() { nvtxRangePop(); }
};
}  // namespace

static bool pool_config_ok(const gc_pool_config* c) {
  return c && c->num_layers >= 1 && c->num_kv_heads >= 1 && c->head_dim >= 1 &&
         c->page_size >= 1 && c->num_pages >= 1;
}

static bool pool_config_supported(const gc_pool_config* c) {
  const bool d_ok = c->head_dim == 64 || c->head_dim == 128;
  const bool ps_ok = c->page_size == 16 || c->page_size == 32 || c->page_size == 64 ||
                     c->page_size == 128;
  return d_ok && ps_ok;
}

extern "C" {

const char* gc_last_error(void) { return g_msg; }

const char* gc_status_string(gc_status s) {
  switch (s) {
    case GC_OK: return "GC_OK";
    case GC_ERR_INVALID_ARG: return "GC_ERR_INVALID_ARG";
    case GC_ERR_OUT_OF_RANGE: return "GC_ERR_OUT_OF_RANGE";
    case GC_ERR_OOM: return "GC_ERR_OOM";
    case GC_ERR_CUDA: return "GC_ERR_CUDA";
    case GC_ERR_UNSUPPORTED: return "GC_ERR_UNSUPPORTED";
    case GC_ERR_TIMEOUT: return "GC_ERR_TIMEOUT";
  }
  return "GC_ERR_UNKNOWN";
}

size_t gc_kv_pool_bytes(const gc_pool_config* cfg) {
  if (!pool_config_ok(cfg)) return 0;
  const size_t planes = static_cast<size_t>(cfg->num_layers) * 2 * cfg->num_pages *
                        gc::page_bytes(*cfg);
  return ((planes + 255) / 256) * 256 + kTrailer;
}

gc_status gc_kv_pool_create(const gc_pool_config* cfg, void* dev_mem, size_t dev_bytes,
                            gc_kv_pool** out) {
  g_msg[0] = 0;
  if (!out) return fail(GC_ERR_INVALID_ARG, "gc_kv_pool_create: out is NULL");
  *out = nullptr;
  if (!pool_config_ok(cfg))
    return fail(GC_ERR_INVALID_ARG, "gc_kv_pool_create: invalid configuration");
  if (!pool_config_supported(cfg))
    return fail(GC_ERR_UNSUPPORTED,
                "gc_kv_pool_create: head_dim %d / page_size %d not supported "
                "(head_dim 64 or 128; page_size 16, 32, 64 or 128)",
                cfg->head_dim, cfg->page_size);
  const size_t need = gc_kv_pool_bytes(cfg);
  if (dev_mem) {
    if (dev_bytes < need)
      return fail(GC_ERR_INVALID_ARG, "gc_kv_pool_create: dev_bytes %zu < required %zu",
                  dev_bytes, need);
    if (reinterpret_cast<uintptr_t>(dev_mem) % 256)
      return fail(GC_ERR_INVALID_ARG, "gc_kv_pool_create: dev_mem not 256-byte aligned");
  }
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return gc::cuda_fail(e, "gc_kv_pool_create: device query");
  void* mem = dev_mem;
  void* owned = nullptr;
  if (!mem) {
    e = cudaMalloc(&mem, need);
    if (e == cudaErrorMemoryAllocation) {
      cudaGetLastError();  // not sticky: clear it so later calls are unaffected
      return fail(GC_ERR_OOM, "gc_kv_pool_create: cudaMalloc of %zu bytes failed", need);
    }
    if (e != cudaSuccess) return gc::cuda_fail(e, "gc_kv_pool_create: cudaMalloc");
    owned = mem;
  }
  auto* p = new (std::nothrow) gc_kv_pool;
  if (!p) {
    if (owned) cudaFree(owned);
    return fail(GC_ERR_OOM, "gc_kv_pool_create: host allocation");
  }
  p->cfg = *cfg;
  p->data = static_cast<uint8_t*>(mem);
  p->data_bytes = need - kTrailer;
  p->status = reinterpret_cast<int32_t*>(p->data + p->data_bytes);
  p->work_counter = p->status + 32;    // 128 bytes into the control block
  p->merge_counters = p->status + 64;  // 256 bytes in, kMergeCounters ints
  static_assert(256 + gc::kMergeCounters * 4 <= kTrailer, "control block too small");
  p->owned = owned;
  p->device = dev;
  p->num_sms = sms;
  e = cudaMemset(p->status, 0, kTrailer);
  if (e != cudaSuccess) {
    if (owned) cudaFree(owned);
    delete p;
    return gc::cuda_fail(e, "gc_kv_pool_create: clearing the status word");
  }
  // data_bytes reported to the caller excludes the alignment padding
  p->data_bytes = static_cast<size_t>(cfg->num_layers) * 2 * cfg->num_pages *
                  gc::page_bytes(*cfg);
  *out = p;
  return GC_OK;
}

gc_status gc_kv_pool_destroy(gc_kv_pool* pool) {
  g_msg[0] = 0;
  if (!pool) return GC_OK;
  if (pool->owned) {
    cudaError_t e = cudaFree(pool->owned);
    delete pool;
    if (e != cudaSuccess) return gc::cuda_fail(e, "gc_kv_pool_destroy: cudaFree");
    return GC_OK;
  }
  delete pool;
  return GC_OK;
}

gc_status gc_kv_pool_data(const gc_kv_pool* pool, void** dev_ptr, size_t* bytes) {
  g_msg[0] = 0;
  if (!pool || !dev_ptr || !bytes) return fail(GC_ERR_INVALID_ARG, "gc_kv_pool_data: NULL argument");
  *dev_ptr = pool->data;
  *bytes = pool->data_bytes;
  return GC_OK;
}

gc_status gc_kv_pool_check(gc_kv_pool* pool, cudaStream_t stream, int32_t* device_status) {
  g_msg[0] = 0;
  if (!pool || !device_status) return fail(GC_ERR_INVALID_ARG, "gc_kv_pool_check: NULL argument");
  int32_t host = 0;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e == cudaSuccess) e = cudaMemcpy(&host, pool->status, sizeof host, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemset(pool->status, 0, sizeof host);
  // a kernel that gave up on a wait may have left decode merge counters
  // raised: after any error, clear them (nothing runs on the pool now)
  if (e == cudaSuccess && host != GC_OK)
    e = cudaMemset(pool->merge_counters, 0, gc::kMergeCounters * sizeof(int32_t));
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return gc::cuda_fail(e, "gc_kv_pool_check");
  *device_status = host;
  return GC_OK;
}

namespace {

// Copy layers [lb, lb + lc) of every block between two whole images (same
// offsets on both sides).  Layer-major images [L][n][2][chunk], or a range
// of all layers: one contiguous copy.  Block-major images [n][L][2][chunk]:
// one strided 2-D copy (rows = blocks).
gc_status copy_layers(const char* who, void* dst, const void* src, int32_t n, int32_t L,
                      int32_t lb, int32_t lc, size_t layer_bytes, bool layer_major,
                      cudaMemcpyKind kind, cudaStream_t stream) {
  cudaError_t e;
  if (layer_major || lc == L) {
    const size_t off = layer_major ? static_cast<size_t>(lb) * n * layer_bytes : 0;
    const size_t len = static_cast<size_t>(lc) * n * layer_bytes;
    e = cudaMemcpyAsync(static_cast<uint8_t*>(dst) + off, static_cast<const uint8_t*>(src) + off,
                        len, kind, stream);
  } else {
    const size_t off = static_cast<size_t>(lb) * layer_bytes;
    const size_t pitch = static_cast<size_t>(L) * layer_bytes;
    const size_t width = static_cast<size_t>(lc) * layer_bytes;
    if (pitch <= 0x7fffffffu) {
      e = cudaMemcpy2DAsync(static_cast<uint8_t*>(dst) + off, pitch,
                            static_cast<const uint8_t*>(src) + off, pitch, width, n, kind, stream);
    } else {  // beyond the 2-D copy's pitch limit: one copy per block
      e = cudaSuccess;
      for (int32_t i = 0; i < n && e == cudaSuccess; ++i)
        e = cudaMemcpyAsync(static_cast<uint8_t*>(dst) + i * pitch + off,
                            static_cast<const uint8_t*>(src) + i * pitch + off, width, kind,
                            stream);
    }
  }
  if (e != cudaSuccess) return gc::cuda_fail(e, who);
  return GC_OK;
}

gc_status check_layers(const char* who, const gc_kv_pool* pool, int32_t lb, int32_t lc) {
  const int32_t L = pool->cfg.num_layers;
  if (lb < 0 || lc < 0 || lb > L || lc > L - lb)
    return fail(GC_ERR_OUT_OF_RANGE, "%s: layers [%d, %d + %d) outside [0, %d)", who, lb, lb, lc,
                L);
  return GC_OK;
}

gc_status restore_impl(const char* who, gc_kv_pool* pool, const void* host_src,
                       const int32_t* block_ids, int32_t n_blocks, int32_t lb, int32_t lc,
                       cudaStream_t stream, void* dev_staging, uint32_t flags) {
  g_msg[0] = 0;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (n_blocks < 0) return fail(GC_ERR_INVALID_ARG, "%s: n_blocks < 0", who);
  if (flags & ~(GC_RESTORE_SRC_DEVICE | GC_RESTORE_VECTOR | GC_RESTORE_LAYER_MAJOR))
    return fail(GC_ERR_INVALID_ARG, "%s: unknown flags 0x%x", who, flags);
  gc_status st = check_layers(who, pool, lb, lc);
  if (st != GC_OK) return st;
  if (n_blocks == 0 || lc == 0) return GC_OK;
  if (!host_src || !block_ids) return fail(GC_ERR_INVALID_ARG, "%s: host_src / block_ids is NULL", who);
  const size_t layer_bytes = 2 * gc::page_bytes(pool->cfg);
  const uint8_t* src = static_cast<const uint8_t*>(host_src);
  bool vector = (flags & GC_RESTORE_VECTOR) != 0;
  const bool lm = (flags & GC_RESTORE_LAYER_MAJOR) != 0;
  if (!(flags & GC_RESTORE_SRC_DEVICE)) {
    cudaPointerAttributes attr;
    cudaError_t e = cudaPointerGetAttributes(&attr, host_src);
    if (e != cudaSuccess || attr.type != cudaMemoryTypeHost) {
      cudaGetLastError();
      return fail(GC_ERR_INVALID_ARG,
                  "%s: host_src must be pinned host memory "
                  "(cudaHostAlloc / cudaHostRegister) unless GC_RESTORE_SRC_DEVICE is set", who);
    }
    if (dev_staging) {
      if (reinterpret_cast<uintptr_t>(dev_staging) % 16)
        return fail(GC_ERR_INVALID_ARG, "%s: dev_staging not 16-byte aligned", who);
      st = copy_layers(who, dev_staging, host_src, n_blocks, pool->cfg.num_layers, lb, lc,
                       layer_bytes, lm, cudaMemcpyHostToDevice, stream);
      if (st != GC_OK) return st;
      src = static_cast<const uint8_t*>(dev_staging);
    } else {
      // zero copy: the kernel reads the pinned buffer through its device alias
      void* dptr = attr.devicePointer;
      if (!dptr) return fail(GC_ERR_INVALID_ARG, "%s: host_src has no device mapping", who);
      src = static_cast<const uint8_t*>(dptr);
      vector = true;
    }
  }
  if (reinterpret_cast<uintptr_t>(src) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: source not 16-byte aligned", who);
  uint8_t* stg = const_cast<uint8_t*>(src);  // read only when restoring
  return vector
             ? gc::launch_restore_vector(pool, stg, block_ids, n_blocks, lb, lc, lm, false, stream)
             : gc::launch_restore_bulk(pool, stg, block_ids, n_blocks, lb, lc, lm, false, stream);
}

gc_status save_impl(const char* who, gc_kv_pool* pool, void* host_dst, const int32_t* block_ids,
                    int32_t n_blocks, int32_t lb, int32_t lc, cudaStream_t stream,
                    void* dev_staging, uint32_t flags) {
  g_msg[0] = 0;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (n_blocks < 0) return fail(GC_ERR_INVALID_ARG, "%s: n_blocks < 0", who);
  if (flags & ~(GC_SAVE_DST_DEVICE | GC_SAVE_VECTOR | GC_SAVE_LAYER_MAJOR))
    return fail(GC_ERR_INVALID_ARG, "%s: unknown flags 0x%x", who, flags);
  gc_status st = check_layers(who, pool, lb, lc);
  if (st != GC_OK) return st;
  if (n_blocks == 0 || lc == 0) return GC_OK;
  if (!host_dst || !block_ids) return fail(GC_ERR_INVALID_ARG, "%s: host_dst / block_ids is NULL", who);
  const size_t layer_bytes = 2 * gc::page_bytes(pool->cfg);
  bool vector = (flags & GC_SAVE_VECTOR) != 0;
  const bool lm = (flags & GC_SAVE_LAYER_MAJOR) != 0;
  if (flags & GC_SAVE_DST_DEVICE) {
    if (reinterpret_cast<uintptr_t>(host_dst) % 16)
      return fail(GC_ERR_INVALID_ARG, "%s: destination not 16-byte aligned", who);
    uint8_t* dst = static_cast<uint8_t*>(host_dst);
    return vector
               ? gc::launch_restore_vector(pool, dst, block_ids, n_blocks, lb, lc, lm, true, stream)
               : gc::launch_restore_bulk(pool, dst, block_ids, n_blocks, lb, lc, lm, true, stream);
  }
  cudaPointerAttributes attr;
  cudaError_t e = cudaPointerGetAttributes(&attr, host_dst);
  if (e != cudaSuccess || attr.type != cudaMemoryTypeHost) {
    cudaGetLastError();
    return fail(GC_ERR_INVALID_ARG,
                "%s: host_dst must be pinned host memory "
                "(cudaHostAlloc / cudaHostRegister) unless GC_SAVE_DST_DEVICE is set", who);
  }
  if (!dev_staging) {
    // zero copy: the kernel writes the pinned buffer through its device alias
    if (!attr.devicePointer) return fail(GC_ERR_INVALID_ARG, "%s: host_dst has no device mapping", who);
    if (reinterpret_cast<uintptr_t>(attr.devicePointer) % 16)
      return fail(GC_ERR_INVALID_ARG, "%s: host_dst not 16-byte aligned", who);
    return gc::launch_restore_vector(pool, static_cast<uint8_t*>(attr.devicePointer), block_ids,
                                     n_blocks, lb, lc, lm, true, stream);
  }
  if (reinterpret_cast<uintptr_t>(dev_staging) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: dev_staging not 16-byte aligned", who);
  uint8_t* stg = static_cast<uint8_t*>(dev_staging);
  st = vector ? gc::launch_restore_vector(pool, stg, block_ids, n_blocks, lb, lc, lm, true, stream)
              : gc::launch_restore_bulk(pool, stg, block_ids, n_blocks, lb, lc, lm, true, stream);
  if (st != GC_OK) return st;
  return copy_layers(who, host_dst, dev_staging, n_blocks, pool->cfg.num_layers, lb, lc,
                     layer_bytes, lm, cudaMemcpyDeviceToHost, stream);
}

// The 8-bit image: the same movement as restore / save (pinned host via a
// device staging copy, zero copy, or a device image), with the INT8 kernels.
gc_status restore_q8_impl(const char* who, gc_kv_pool* pool, const void* src_img,
                          const int32_t* block_ids, int32_t n_blocks, int32_t lb, int32_t lc,
                          cudaStream_t stream, void* dev_staging, uint32_t flags) {
  g_msg[0] = 0;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (n_blocks < 0) return fail(GC_ERR_INVALID_ARG, "%s: n_blocks < 0", who);
  if (flags & ~(GC_RESTORE_SRC_DEVICE | GC_RESTORE_LAYER_MAJOR))
    return fail(GC_ERR_INVALID_ARG, "%s: unknown flags 0x%x", who, flags);
  gc_status st = check_layers(who, pool, lb, lc);
  if (st != GC_OK) return st;
  if (n_blocks == 0 || lc == 0) return GC_OK;
  if (!src_img || !block_ids) return fail(GC_ERR_INVALID_ARG, "%s: image / block_ids is NULL", who);
  const bool lm = (flags & GC_RESTORE_LAYER_MAJOR) != 0;
  const size_t layer_bytes = 2 * gc::q8_chunk_bytes(pool->cfg);
  const uint8_t* src = static_cast<const uint8_t*>(src_img);
  if (!(flags & GC_RESTORE_SRC_DEVICE)) {
    cudaPointerAttributes attr;
    cudaError_t e = cudaPointerGetAttributes(&attr, src_img);
    if (e != cudaSuccess || attr.type != cudaMemoryTypeHost) {
      cudaGetLastError();
      return fail(GC_ERR_INVALID_ARG,
                  "%s: image must be pinned host memory unless GC_RESTORE_SRC_DEVICE is set", who);
    }
    if (dev_staging) {
      if (reinterpret_cast<uintptr_t>(dev_staging) % 16)
        return fail(GC_ERR_INVALID_ARG, "%s: dev_staging not 16-byte aligned", who);
      st = copy_layers(who, dev_staging, src_img, n_blocks, pool->cfg.num_layers, lb, lc,
                       layer_bytes, lm, cudaMemcpyHostToDevice, stream);
      if (st != GC_OK) return st;
      src = static_cast<const uint8_t*>(dev_staging);
    } else {
      if (!attr.devicePointer) return fail(GC_ERR_INVALID_ARG, "%s: image has no device mapping", who);
      src = static_cast<const uint8_t*>(attr.devicePointer);
    }
  }
  if (reinterpret_cast<uintptr_t>(src) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: image not 16-byte aligned", who);
  return gc::launch_restore_q8(pool, src, block_ids, n_blocks, lb, lc, lm, stream);
}

gc_status save_q8_impl(const char* who, gc_kv_pool* pool, void* dst_img, const int32_t* block_ids,
                       int32_t n_blocks, int32_t lb, int32_t lc, cudaStream_t stream,
                       void* dev_staging, uint32_t flags) {
  g_msg[0] = 0;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (n_blocks < 0) return fail(GC_ERR_INVALID_ARG, "%s: n_blocks < 0", who);
  if (flags & ~(GC_SAVE_DST_DEVICE | GC_SAVE_LAYER_MAJOR))
    return fail(GC_ERR_INVALID_ARG, "%s: unknown flags 0x%x", who, flags);
  gc_status st = check_layers(who, pool, lb, lc);
  if (st != GC_OK) return st;
  if (n_blocks == 0 || lc == 0) return GC_OK;
  if (!dst_img || !block_ids) return fail(GC_ERR_INVALID_ARG, "%s: image / block_ids is NULL", who);
  const bool lm = (flags & GC_SAVE_LAYER_MAJOR) != 0;
  const size_t layer_bytes = 2 * gc::q8_chunk_bytes(pool->cfg);
  if (flags & GC_SAVE_DST_DEVICE) {
    if (reinterpret_cast<uintptr_t>(dst_img) % 16)
      return fail(GC_ERR_INVALID_ARG, "%s: image not 16-byte aligned", who);
    return gc::launch_save_q8(pool, static_cast<uint8_t*>(dst_img), block_ids, n_blocks, lb, lc,
                              lm, stream);
  }
  cudaPointerAttributes attr;
  cudaError_t e = cudaPointerGetAttributes(&attr, dst_img);
  if (e != cudaSuccess || attr.type != cudaMemoryTypeHost) {
    cudaGetLastError();
    return fail(GC_ERR_INVALID_ARG,
                "%s: image must be pinned host memory unless GC_SAVE_DST_DEVICE is set", who);
  }
  if (!dev_staging) {
    if (!attr.devicePointer) return fail(GC_ERR_INVALID_ARG, "%s: image has no device mapping", who);
    if (reinterpret_cast<uintptr_t>(attr.devicePointer) % 16)
      return fail(GC_ERR_INVALID_ARG, "%s: image not 16-byte aligned", who);
    return gc::launch_save_q8(pool, static_cast<uint8_t*>(attr.devicePointer), block_ids, n_blocks,
                              lb, lc, lm, stream);
  }
  if (reinterpret_cast<uintptr_t>(dev_staging) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: dev_staging not 16-byte aligned", who);
  st = gc::launch_save_q8(pool, static_cast<uint8_t*>(dev_staging), block_ids, n_blocks, lb, lc,
                          lm, stream);
  if (st != GC_OK) return st;
  return copy_layers(who, dst_img, dev_staging, n_blocks, pool->cfg.num_layers, lb, lc,
                     layer_bytes, lm, cudaMemcpyDeviceToHost, stream);
}

}  // namespace

gc_status gc_kv_restore(gc_kv_pool* pool, const void* host_src, const int32_t* block_ids,
                        int32_t n_blocks, cudaStream_t stream, void* dev_staging, uint32_t flags) {
  Range range_("gc_kv_restore");
  return restore_impl("gc_kv_restore", pool, host_src, block_ids, n_blocks, 0,
                      pool ? pool->cfg.num_layers : 0, stream, dev_staging, flags);
}

gc_status gc_kv_restore_layers(gc_kv_pool* pool, const void* host_src, const int32_t* block_ids,
                               int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                               cudaStream_t stream, void* dev_staging, uint32_t flags) {
  Range range_("gc_kv_restore_layers");
  return restore_impl("gc_kv_restore_layers", pool, host_src, block_ids, n_blocks, layer_begin,
                      layer_count, stream, dev_staging, flags);
}

gc_status gc_kv_stage_layers(const gc_kv_pool* pool, const void* host_src, void* dev_image,
                             int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                             cudaStream_t stream, uint32_t flags) {
  Range range_("gc_kv_stage_layers");
  g_msg[0] = 0;
  const char* who = "gc_kv_stage_layers";
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (n_blocks < 0) return fail(GC_ERR_INVALID_ARG, "%s: n_blocks < 0", who);
  if (flags & ~(GC_RESTORE_LAYER_MAJOR | GC_STAGE_Q8))
    return fail(GC_ERR_INVALID_ARG, "%s: unknown flags 0x%x", who, flags);
  gc_status st = check_layers(who, pool, layer_begin, layer_count);
  if (st != GC_OK) return st;
  if (n_blocks == 0 || layer_count == 0) return GC_OK;
  if (!host_src || !dev_image) return fail(GC_ERR_INVALID_ARG, "%s: image is NULL", who);
  if (reinterpret_cast<uintptr_t>(dev_image) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: dev_image not 16-byte aligned", who);
  cudaPointerAttributes attr;
  cudaError_t e = cudaPointerGetAttributes(&attr, host_src);
  if (e != cudaSuccess || attr.type != cudaMemoryTypeHost) {
    cudaGetLastError();
    return fail(GC_ERR_INVALID_ARG, "%s: host_src must be pinned host memory", who);
  }
  const size_t layer_bytes =
      2 * ((flags & GC_STAGE_Q8) ? gc::q8_chunk_bytes(pool->cfg) : gc::page_bytes(pool->cfg));
  return copy_layers(who, dev_image, host_src, n_blocks, pool->cfg.num_layers, layer_begin,
                     layer_count, layer_bytes, (flags & GC_RESTORE_LAYER_MAJOR) != 0,
                     cudaMemcpyHostToDevice, stream);
}

gc_status gc_kv_save(gc_kv_pool* pool, void* host_dst, const int32_t* block_ids,
                     int32_t n_blocks, cudaStream_t stream, void* dev_staging, uint32_t flags) {
  Range range_("gc_kv_save");
  return save_impl("gc_kv_save", pool, host_dst, block_ids, n_blocks, 0,
                   pool ? pool->cfg.num_layers : 0, stream, dev_staging, flags);
}

gc_status gc_kv_save_layers(gc_kv_pool* pool, void* host_dst, const int32_t* block_ids,
                            int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                            cudaStream_t stream, void* dev_staging, uint32_t flags) {
  Range range_("gc_kv_save_layers");
  return save_impl("gc_kv_save_layers", pool, host_dst, block_ids, n_blocks, layer_begin,
                   layer_count, stream, dev_staging, flags);
}

size_t gc_kv_q8_chunk_bytes(const gc_pool_config* cfg) {
  if (!pool_config_ok(cfg)) return 0;
  return gc::q8_chunk_bytes(*cfg);
}

gc_status gc_kv_save_q8(gc_kv_pool* pool, void* dst, const int32_t* block_ids, int32_t n_blocks,
                        int32_t layer_begin, int32_t layer_count, cudaStream_t stream,
                        void* dev_staging, uint32_t flags) {
  Range range_("gc_kv_save_q8");
  return save_q8_impl("gc_kv_save_q8", pool, dst, block_ids, n_blocks, layer_begin, layer_count,
                      stream, dev_staging, flags);
}

gc_status gc_kv_restore_q8(gc_kv_pool* pool, const void* src, const int32_t* block_ids,
                           int32_t n_blocks, int32_t layer_begin, int32_t layer_count,
                           cudaStream_t stream, void* dev_staging, uint32_t flags) {
  Range range_("gc_kv_restore_q8");
  return restore_q8_impl("gc_kv_restore_q8", pool, src, block_ids, n_blocks, layer_begin,
                         layer_count, stream, dev_staging, flags);
}

gc_status gc_kv_append(gc_kv_pool* pool, const void* k_new, const void* v_new,
                       const int32_t* block_table, const int32_t* seq_lens, cudaStream_t stream,
                       int32_t layer, const int32_t* cu_new_lens, int32_t batch,
                       int32_t max_blocks_per_seq, int32_t total_new_tokens) {
  Range range_("gc_kv_append");
  g_msg[0] = 0;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "gc_kv_append: pool is NULL");
  if (batch < 0 || total_new_tokens < 0 || max_blocks_per_seq < 0)
    return fail(GC_ERR_INVALID_ARG, "gc_kv_append: negative size");
  if (layer < 0 || layer >= pool->cfg.num_layers)
    return fail(GC_ERR_OUT_OF_RANGE, "gc_kv_append: layer %d outside [0, %d)", layer,
                pool->cfg.num_layers);
  if (batch == 0 || total_new_tokens == 0) return GC_OK;
  if (!k_new || !v_new || !block_table || !seq_lens || !cu_new_lens)
    return fail(GC_ERR_INVALID_ARG, "gc_kv_append: NULL array argument");
  if (max_blocks_per_seq == 0)
    return fail(GC_ERR_INVALID_ARG, "gc_kv_append: max_blocks_per_seq is 0");
  if ((reinterpret_cast<uintptr_t>(k_new) | reinterpret_cast<uintptr_t>(v_new)) % 16)
    return fail(GC_ERR_INVALID_ARG, "gc_kv_append: k_new / v_new not 16-byte aligned");
  return gc::launch_append(pool, k_new, v_new, block_table, seq_lens, cu_new_lens, batch,
                           max_blocks_per_seq, layer, total_new_tokens, stream);
}

static gc_status attn_common(const char* who, const void* q, const gc_kv_pool* pool,
                             const int32_t* block_table, const int32_t* prefix_lens,
                             const int32_t* new_lens, void* out, int32_t layer,
                             const int32_t* cu_new_lens, int32_t batch,
                             int32_t max_blocks_per_seq, int32_t num_q_heads,
                             float softmax_scale, int32_t total_new_tokens, gc::AttnArgs* a,
                             bool* noop) {
  *noop = false;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (batch < 0 || total_new_tokens < 0 || max_blocks_per_seq < 0)
    return fail(GC_ERR_INVALID_ARG, "%s: negative size", who);
  if (layer < 0 || layer >= pool->cfg.num_layers)
    return fail(GC_ERR_OUT_OF_RANGE, "%s: layer %d outside [0, %d)", who, layer,
                pool->cfg.num_layers);
  const int hkv = pool->cfg.num_kv_heads;
  if (num_q_heads <= 0 || num_q_heads % hkv)
    return fail(GC_ERR_INVALID_ARG, "%s: num_q_heads %d not a multiple of num_kv_heads %d", who,
                num_q_heads, hkv);
  const int G = num_q_heads / hkv;
  if (G != 1 && G != 2 && G != 4 && G != 8 && G != 16)
    return fail(GC_ERR_UNSUPPORTED, "%s: q heads per kv head %d not in {1,2,4,8,16}", who, G);
  if (!(softmax_scale > 0.0f) || softmax_scale == __builtin_inff())
    return fail(GC_ERR_INVALID_ARG, "%s: softmax_scale must be positive and finite", who);
  if (batch > 8192) return fail(GC_ERR_UNSUPPORTED, "%s: batch %d > 8192", who, batch);
  if (batch == 0 || total_new_tokens == 0) {
    *noop = true;
    return GC_OK;
  }
  if (!q || !out || !block_table || !prefix_lens || !new_lens || !cu_new_lens)
    return fail(GC_ERR_INVALID_ARG, "%s: NULL array argument", who);
  if (max_blocks_per_seq == 0)
    return fail(GC_ERR_INVALID_ARG, "%s: max_blocks_per_seq is 0", who);
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out)) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: q / out not 16-byte aligned", who);
  *a = gc::AttnArgs{q, out, block_table, prefix_lens, new_lens, cu_new_lens, batch,
                    max_blocks_per_seq, layer, num_q_heads, total_new_tokens, softmax_scale};
  return GC_OK;
}

gc_status gc_prefix_prefill_attn(const void* q, const gc_kv_pool* pool, const int32_t* block_table,
                                 const int32_t* prefix_lens, const int32_t* new_lens, void* out,
                                 cudaStream_t stream, int32_t layer, const int32_t* cu_new_lens,
                                 int32_t batch, int32_t max_blocks_per_seq, int32_t num_q_heads,
                                 float softmax_scale, int32_t total_new_tokens) {
  Range range_("gc_prefix_prefill_attn");
  g_msg[0] = 0;
  gc::AttnArgs a;
  bool noop;
  gc_status s = attn_common("gc_prefix_prefill_attn", q, pool, block_table, prefix_lens, new_lens,
                            out, layer, cu_new_lens, batch, max_blocks_per_seq, num_q_heads,
                            softmax_scale, total_new_tokens, &a, &noop);
  if (s != GC_OK || noop) return s;
  return gc::launch_attn_tc(pool, a, stream);
}

gc_status gc_prefix_prefill_attn_noalloc(const void* q, const gc_kv_pool* pool,
                                         const int32_t* block_table, const int32_t* prefix_lens,
                                         const int32_t* new_lens, void* out, cudaStream_t stream,
                                         int32_t layer, const int32_t* cu_new_lens, int32_t batch,
                                         int32_t max_blocks_per_seq, int32_t num_q_heads,
                                         float softmax_scale, int32_t total_new_tokens) {
  Range range_("gc_prefix_prefill_attn_noalloc");
  g_msg[0] = 0;
  gc::AttnArgs a;
  bool noop;
  gc_status s = attn_common("gc_prefix_prefill_attn_noalloc", q, pool, block_table, prefix_lens,
                            new_lens, out, layer, cu_new_lens, batch, max_blocks_per_seq,
                            num_q_heads, softmax_scale, total_new_tokens, &a, &noop);
  if (s != GC_OK || noop) return s;
  return gc::launch_attn_tc_noalloc(pool, a, stream);
}

gc_status gc_prefix_prefill_attn_q8(const void* q, const gc_kv_pool* pool,
                                    const int32_t* block_table, const int32_t* prefix_lens,
                                    const int32_t* new_lens, void* out, cudaStream_t stream,
                                    int32_t layer, const int32_t* cu_new_lens, int32_t batch,
                                    int32_t max_blocks_per_seq, int32_t num_q_heads,
                                    float softmax_scale, int32_t total_new_tokens,
                                    const void* q8_image, const int32_t* q8_table,
                                    int32_t n_image_blocks, uint32_t flags) {
  Range range_("gc_prefix_prefill_attn_q8");
  g_msg[0] = 0;
  gc::AttnArgs a;
  bool noop;
  gc_status s = attn_common("gc_prefix_prefill_attn_q8", q, pool, block_table, prefix_lens,
                            new_lens, out, layer, cu_new_lens, batch, max_blocks_per_seq,
                            num_q_heads, softmax_scale, total_new_tokens, &a, &noop);
  if (s != GC_OK) return s;
  if (flags & ~GC_RESTORE_LAYER_MAJOR)
    return fail(GC_ERR_INVALID_ARG, "gc_prefix_prefill_attn_q8: unknown flags 0x%x", flags);
  if (n_image_blocks < 0)
    return fail(GC_ERR_INVALID_ARG, "gc_prefix_prefill_attn_q8: negative n_image_blocks");
  if (noop) return GC_OK;
  if (!q8_table || (n_image_blocks > 0 && !q8_image))
    return fail(GC_ERR_INVALID_ARG, "gc_prefix_prefill_attn_q8: NULL q8_image / q8_table");
  if (reinterpret_cast<uintptr_t>(q8_image) % 16)
    return fail(GC_ERR_INVALID_ARG, "gc_prefix_prefill_attn_q8: q8_image not 16-byte aligned");
  const gc::Q8Pages q8{static_cast<const uint8_t*>(q8_image), q8_table, n_image_blocks,
                       (flags & GC_RESTORE_LAYER_MAJOR) != 0};
  return gc::launch_attn_tc_q8(pool, a, q8, stream);
}

gc_status gc_prefix_prefill_attn_simt(const void* q, const gc_kv_pool* pool,
                                      const int32_t* block_table, const int32_t* prefix_lens,
                                      const int32_t* new_lens, void* out, cudaStream_t stream,
                                      int32_t layer, const int32_t* cu_new_lens, int32_t batch,
                                      int32_t max_blocks_per_seq, int32_t num_q_heads,
                                      float softmax_scale, int32_t total_new_tokens) {
  Range range_("gc_prefix_prefill_attn_simt");
  g_msg[0] = 0;
  gc::AttnArgs a;
  bool noop;
  gc_status s = attn_common("gc_prefix_prefill_attn_simt", q, pool, block_table, prefix_lens,
                            new_lens, out, layer, cu_new_lens, batch, max_blocks_per_seq,
                            num_q_heads, softmax_scale, total_new_tokens, &a, &noop);
  if (s != GC_OK || noop) return s;
  return gc::launch_attn_simt(pool, a, stream);
}

size_t gc_paged_decode_workspace_bytes(const gc_kv_pool* pool, int32_t batch,
                                       int32_t max_blocks_per_seq, int32_t num_q_heads) {
  if (!pool || batch <= 0 || max_blocks_per_seq <= 0 || num_q_heads <= 0) return 0;
  return gc::decode_workspace_bytes(pool, batch, max_blocks_per_seq, num_q_heads);
}

gc_status gc_paged_decode_attn(const void* q, const gc_kv_pool* pool, const int32_t* block_table,
                               const int32_t* seq_lens, void* out, cudaStream_t stream,
                               int32_t layer, int32_t batch, int32_t max_blocks_per_seq,
                               int32_t num_q_heads, float softmax_scale, void* workspace,
                               size_t workspace_bytes) {
  Range range_("gc_paged_decode_attn");
  g_msg[0] = 0;
  const char* who = "gc_paged_decode_attn";
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (batch < 0 || max_blocks_per_seq < 0) return fail(GC_ERR_INVALID_ARG, "%s: negative size", who);
  if (layer < 0 || layer >= pool->cfg.num_layers)
    return fail(GC_ERR_OUT_OF_RANGE, "%s: layer %d outside [0, %d)", who, layer,
                pool->cfg.num_layers);
  const int hkv = pool->cfg.num_kv_heads;
  if (num_q_heads <= 0 || num_q_heads % hkv)
    return fail(GC_ERR_INVALID_ARG, "%s: num_q_heads %d not a multiple of num_kv_heads %d", who,
                num_q_heads, hkv);
  const int G = num_q_heads / hkv;
  if (G != 1 && G != 2 && G != 4 && G != 8 && G != 16)
    return fail(GC_ERR_UNSUPPORTED, "%s: q heads per kv head %d not in {1,2,4,8,16}", who, G);
  if (!(softmax_scale > 0.0f) || softmax_scale == __builtin_inff())
    return fail(GC_ERR_INVALID_ARG, "%s: softmax_scale must be positive and finite", who);
  if (batch == 0) return GC_OK;
  if (!q || !out || !block_table || !seq_lens)
    return fail(GC_ERR_INVALID_ARG, "%s: NULL array argument", who);
  if (max_blocks_per_seq == 0) return fail(GC_ERR_INVALID_ARG, "%s: max_blocks_per_seq is 0", who);
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out) |
       reinterpret_cast<uintptr_t>(workspace)) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: q / out / workspace not 16-byte aligned", who);
  const gc::DecodeArgs a{q, out, block_table, seq_lens, batch, max_blocks_per_seq, layer,
                         num_q_heads, softmax_scale, workspace, workspace_bytes};
  return gc::launch_decode(pool, a, stream);
}

gc_status gc_paged_decode_attn_q8(const void* q, const gc_kv_pool* pool,
                                  const int32_t* block_table, const int32_t* seq_lens, void* out,
                                  cudaStream_t stream, int32_t layer, int32_t batch,
                                  int32_t max_blocks_per_seq, int32_t num_q_heads,
                                  float softmax_scale, void* workspace, size_t workspace_bytes,
                                  const void* q8_image, const int32_t* q8_table,
                                  int32_t n_image_blocks, uint32_t flags) {
  Range range_("gc_paged_decode_attn_q8");
  g_msg[0] = 0;
  const char* who = "gc_paged_decode_attn_q8";
  if (!pool) return fail(GC_ERR_INVALID_ARG, "%s: pool is NULL", who);
  if (batch < 0 || max_blocks_per_seq < 0 || n_image_blocks < 0)
    return fail(GC_ERR_INVALID_ARG, "%s: negative size", who);
  if (flags & ~GC_RESTORE_LAYER_MAJOR)
    return fail(GC_ERR_INVALID_ARG, "%s: unknown flags 0x%x", who, flags);
  if (layer < 0 || layer >= pool->cfg.num_layers)
    return fail(GC_ERR_OUT_OF_RANGE, "%s: layer %d outside [0, %d)", who, layer,
                pool->cfg.num_layers);
  const int hkv = pool->cfg.num_kv_heads;
  if (num_q_heads <= 0 || num_q_heads % hkv)
    return fail(GC_ERR_INVALID_ARG, "%s: num_q_heads %d not a multiple of num_kv_heads %d", who,
                num_q_heads, hkv);
  const int G = num_q_heads / hkv;
  if (G != 1 && G != 2 && G != 4 && G != 8 && G != 16)
    return fail(GC_ERR_UNSUPPORTED, "%s: q heads per kv head %d not in {1,2,4,8,16}", who, G);
  if (!(softmax_scale > 0.0f) || softmax_scale == __builtin_inff())
    return fail(GC_ERR_INVALID_ARG, "%s: softmax_scale must be positive and finite", who);
  if (batch == 0) return GC_OK;
  if (!q || !out || !block_table || !seq_lens || !q8_table || (n_image_blocks > 0 && !q8_image))
    return fail(GC_ERR_INVALID_ARG, "%s: NULL array argument", who);
  if (max_blocks_per_seq == 0) return fail(GC_ERR_INVALID_ARG, "%s: max_blocks_per_seq is 0", who);
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out) |
       reinterpret_cast<uintptr_t>(workspace) | reinterpret_cast<uintptr_t>(q8_image)) % 16)
    return fail(GC_ERR_INVALID_ARG, "%s: q / out / workspace / q8_image not 16-byte aligned", who);
  const gc::DecodeArgs a{q, out, block_table, seq_lens, batch, max_blocks_per_seq, layer,
                         num_q_heads, softmax_scale, workspace, workspace_bytes};
  const gc::Q8Pages q8{static_cast<const uint8_t*>(q8_image), q8_table, n_image_blocks,
                       (flags & GC_RESTORE_LAYER_MAJOR) != 0};
  return gc::launch_decode(pool, a, stream, &q8);
}

gc_status gc_selftest_wait_timeout(gc_kv_pool* pool, cudaStream_t stream) {
  g_msg[0] = 0;
  if (!pool) return fail(GC_ERR_INVALID_ARG, "gc_selftest_wait_timeout: pool is NULL");
  return gc::launch_selftest_timeout(pool, stream);
}

}  // extern "C"
