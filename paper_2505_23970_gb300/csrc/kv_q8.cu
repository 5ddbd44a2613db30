// 8-bit cache tier: pool pages <-> an INT8 image with one scale per
// (block, layer, plane, kv head) group of ps*d values.  The 70B runs of
// Sec. 6.1 use INT8; keeping the cached KV in 8 bits halves what the cache
// tier stores (its embodied carbon, Sec. 3.2) and what the host link moves
// on a restore.  The pool itself stays bf16, so attention is unchanged.
//
//   save:    amax = max |x| over the group's finite values
//            s = amax / 127, c = clamp(rne(x * (127 / amax)), -127, 127)
//            (NaN -> 0; all codes 0 when amax is 0)
//   restore: x' = bf16_rne(c * s)
//
// Both directions are bandwidth-bound element maps.  Save gives one warp a
// group: a first pass of 16-byte loads finds amax (warp max-reduction over
// the float bit patterns, which order like the values for |x|), a second
// pass quantises it from registers (or re-reads it from L1/L2 when it is too
// large to hold) and writes 8 codes per 16-byte word.  Restore gives each
// thread 16 codes (one 16-byte load) and writes 16 bf16 values (two 16-byte
// stores).  Both grids are exactly the resident blocks, so the grid-stride
// loops split the work evenly.
#include "gc_internal.cuh"

namespace gc {
namespace {

struct Q8Geom {
  uint64_t chunk_bytes;  // image bytes of one (block, layer, plane)
  uint32_t hdr_bytes;    // scales + zero padding to a multiple of 16 bytes
  uint32_t group;        // ps*d values per kv head
  int32_t L, num_pages, Hkv, n_blocks, layer0, layers, layer_major;
};

__device__ __forceinline__ uint64_t q8_chunk(const Q8Geom& g, int64_t i, int l, int kv) {
  const uint64_t il = g.layer_major ? static_cast<uint64_t>(l) * g.n_blocks + i
                                    : static_cast<uint64_t>(i) * g.L + l;
  return il * 2 + kv;
}

__device__ __forceinline__ uint64_t pool_group_offset(const Q8Geom& g, int l, int kv, int page,
                                                      int h) {
  return ((((static_cast<uint64_t>(l) * 2 + kv) * g.num_pages + page) * g.Hkv + h) * g.group) * 2;
}

// |x| of a bf16 bit pattern as float bits, or 0 for NaN / infinity.
__device__ __forceinline__ uint32_t finite_abs_bits(uint32_t u16) {
  return ((u16 & 0x7f80u) == 0x7f80u) ? 0u : (u16 & 0x7fffu) << 16;
}

__device__ __forceinline__ int q8_code(uint32_t u16, float inv) {
  const float x = __uint_as_float(u16 << 16);
  float v = x * inv;
  if (v != v) return 0;  // NaN input, or infinity * 0 when amax is 0
  v = fminf(fmaxf(v, -127.0f), 127.0f);
  return __float2int_rn(v);
}

__device__ __forceinline__ uint32_t pack4(int a, int b, int c, int d) {
  return (static_cast<uint32_t>(a) & 0xffu) | ((static_cast<uint32_t>(b) & 0xffu) << 8) |
         ((static_cast<uint32_t>(c) & 0xffu) << 16) | (static_cast<uint32_t>(d) << 24);
}

__device__ __forceinline__ uint2 quant8(const uint4& v, float inv) {
  uint2 o;
  o.x = pack4(q8_code(v.x & 0xffffu, inv), q8_code(v.x >> 16, inv), q8_code(v.y & 0xffffu, inv),
              q8_code(v.y >> 16, inv));
  o.y = pack4(q8_code(v.z & 0xffffu, inv), q8_code(v.z >> 16, inv), q8_code(v.w & 0xffffu, inv),
              q8_code(v.w >> 16, inv));
  return o;
}

// Codes of four finite values (two bf16 pairs): |x * inv| <= 127 up to one
// rounding of the product, so round-to-nearest-even alone lands in
// [-127, 127] and no clamp is needed.
__device__ __forceinline__ uint32_t quant4_finite(uint32_t w0, uint32_t w1, float inv) {
  const int a = __float2int_rn(__uint_as_float(w0 << 16) * inv);
  const int b = __float2int_rn(__uint_as_float(w0 & 0xffff0000u) * inv);
  const int c = __float2int_rn(__uint_as_float(w1 << 16) * inv);
  const int d = __float2int_rn(__uint_as_float(w1 & 0xffff0000u) * inv);
  return __byte_perm(__byte_perm(a, b, 0x0040), __byte_perm(c, d, 0x0040), 0x5410);
}

__device__ __forceinline__ uint2 quant8_finite(const uint4& v, float inv) {
  return make_uint2(quant4_finite(v.x, v.y, inv), quant4_finite(v.z, v.w, inv));
}

// Finite-only |x| maximum of 8 bf16 values, as float bits.
__device__ __forceinline__ uint32_t amax8(const uint4& v, uint32_t m) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    m = max(m, finite_abs_bits(w[k] & 0xffffu));
    m = max(m, finite_abs_bits(w[k] >> 16));
  }
  return m;
}

// Maximum of |x| over 8 bf16 values including non-finite ones, per 16-bit
// half (|x| patterns order like the magnitudes; NaN and infinity sort above
// every finite value).
__device__ __forceinline__ uint32_t umax16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.u16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

__device__ __forceinline__ uint32_t absmax8_any(const uint4& v, uint32_t m) {
  m = umax16x2(m, v.x & 0x7fff7fffu);
  m = umax16x2(m, v.y & 0x7fff7fffu);
  m = umax16x2(m, v.z & 0x7fff7fffu);
  return umax16x2(m, v.w & 0x7fff7fffu);
}

// A group of up to 32*kRegWords 16-byte words is held in registers between
// the amax pass and the quantise pass (ps*d <= 2048 bf16 values, e.g. ps 16
// at d 128); larger groups re-read the group, which is then in L1/L2.  The
// common all-finite group takes a short path (packed 16-bit magnitude max,
// no clamps); a group holding NaN or infinity (e.g. stale slots past the end
// of a sequence) takes the general path with the finite-only maximum.
constexpr int kRegWords = 8;

__global__ void __launch_bounds__(256) save_q8_kernel(uint8_t* __restrict__ image,
                                                      const uint8_t* __restrict__ pool,
                                                      const int32_t* __restrict__ block_ids,
                                                      Q8Geom g, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const uint64_t nwarps = (static_cast<uint64_t>(gridDim.x) * blockDim.x) >> 5;
  const uint64_t groups = static_cast<uint64_t>(g.n_blocks) * g.layers * 2 * g.Hkv;
  const uint32_t words = g.group / 8;  // 16-byte words of bf16 per group
  const bool in_regs = words <= 32u * kRegWords;
  for (uint64_t gi = (static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
       gi < groups; gi += nwarps) {
    const int h = static_cast<int>(gi % g.Hkv);
    const uint64_t c = gi / g.Hkv;
    const int kv = static_cast<int>(c % 2);
    const int lr = static_cast<int>((c / 2) % g.layers);
    const int64_t i = static_cast<int64_t>(c / (2 * g.layers));
    const int l = g.layer0 + lr;
    const int32_t id = __ldg(block_ids + i);
    if (id < 0 || id >= g.num_pages) {
      if (lane == 0 && h == 0 && kv == 0 && lr == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
      continue;
    }
    const uint4* src = reinterpret_cast<const uint4*>(pool + pool_group_offset(g, l, kv, id, h));
    uint4 held[kRegWords];
    uint32_t m2 = 0;
    if (in_regs) {
#pragma unroll
      for (int k = 0; k < kRegWords; ++k) {
        const uint32_t j = lane + 32u * k;
        if (j < words) {
          held[k] = __ldg(src + j);
          m2 = absmax8_any(held[k], m2);
        }
      }
    } else {
#pragma unroll 4
      for (uint32_t j = lane; j < words; j += 32) m2 = absmax8_any(__ldg(src + j), m2);
    }
    uint32_t amax_bits = __reduce_max_sync(0xffffffffu, max(m2 & 0xffffu, m2 >> 16)) << 16;
    const bool all_finite = amax_bits < 0x7f800000u;
    if (!all_finite) {  // rare: recompute the maximum over finite values only
      amax_bits = 0;
      if (in_regs) {
#pragma unroll
        for (int k = 0; k < kRegWords; ++k)
          if (lane + 32u * k < words) amax_bits = amax8(held[k], amax_bits);
      } else {
        for (uint32_t j = lane; j < words; j += 32) amax_bits = amax8(__ldg(src + j), amax_bits);
      }
      amax_bits = __reduce_max_sync(0xffffffffu, amax_bits);
    }
    const float amax = __uint_as_float(amax_bits);
    const float scale = amax / 127.0f;
    const float inv = amax > 0.0f ? 127.0f / amax : 0.0f;
    // the short path needs finite values and a finite 127/amax (a group of
    // tiny subnormal values can overflow it)
    const bool finite = all_finite && inv < INFINITY;
    uint8_t* chunk = image + q8_chunk(g, i, l, kv) * g.chunk_bytes;
    if (lane == 0) {
      reinterpret_cast<float*>(chunk)[h] = scale;
      if (h == 0)
        for (uint32_t b = 4u * g.Hkv; b < g.hdr_bytes; ++b) chunk[b] = 0;
    }
    uint2* dst = reinterpret_cast<uint2*>(chunk + g.hdr_bytes + static_cast<uint64_t>(h) * g.group);
    if (in_regs) {
#pragma unroll
      for (int k = 0; k < kRegWords; ++k) {
        const uint32_t j = lane + 32u * k;
        if (j < words) dst[j] = finite ? quant8_finite(held[k], inv) : quant8(held[k], inv);
      }
    } else {
#pragma unroll 4
      for (uint32_t j = lane; j < words; j += 32) {
        const uint4 v = __ldg(src + j);
        dst[j] = finite ? quant8_finite(v, inv) : quant8(v, inv);
      }
    }
  }
}

// Each thread dequantises 16 codes (one 16-byte load) into 16 bf16 values
// (two 16-byte stores; a warp's pair of stores covers 1 KB contiguously).
__global__ void __launch_bounds__(256) restore_q8_kernel(const uint8_t* __restrict__ image,
                                                         uint8_t* __restrict__ pool,
                                                         const int32_t* __restrict__ block_ids,
                                                         Q8Geom g, int32_t* status) {
  const uint32_t words_per_group = g.group / 16;  // 16-byte words of codes
  const uint64_t words_per_chunk = static_cast<uint64_t>(words_per_group) * g.Hkv;
  const uint64_t total = static_cast<uint64_t>(g.n_blocks) * g.layers * 2 * words_per_chunk;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  constexpr int U = 4;
  for (uint64_t base = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; base < total;
       base += stride * U) {
    uint4 v[U];
    float s[U];
    uint4* dst[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const uint64_t w = base + k * stride;
      dst[k] = nullptr;
      if (w >= total) continue;
      const uint64_t c = w / words_per_chunk;
      const uint32_t r = static_cast<uint32_t>(w - c * words_per_chunk);
      const int h = static_cast<int>(r / words_per_group);
      const uint32_t e16 = r - static_cast<uint32_t>(h) * words_per_group;
      const int kv = static_cast<int>(c % 2);
      const int lr = static_cast<int>((c / 2) % g.layers);
      const int64_t i = static_cast<int64_t>(c / (2 * g.layers));
      const int l = g.layer0 + lr;
      const int32_t id = __ldg(block_ids + i);
      if (id < 0 || id >= g.num_pages) {
        if (r == 0 && kv == 0 && lr == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
        continue;
      }
      const uint8_t* chunk = image + q8_chunk(g, i, l, kv) * g.chunk_bytes;
      s[k] = reinterpret_cast<const float*>(chunk)[h];
      v[k] = reinterpret_cast<const uint4*>(chunk + g.hdr_bytes +
                                            static_cast<uint64_t>(h) * g.group)[e16];
      dst[k] = reinterpret_cast<uint4*>(pool + pool_group_offset(g, l, kv, id, h)) + 2 * e16;
    }
#pragma unroll
    for (int k = 0; k < U; ++k) {
      if (!dst[k]) continue;
      uint4 lo, hi;
      q8_dequant16(v[k], s[k], lo, hi);
      dst[k][0] = lo;
      dst[k][1] = hi;
    }
  }
}

// Blocks of `kernel` (256 threads) that fit on one SM, queried once.
template <typename K>
int resident_blocks(K kernel) {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, 256, 0) != cudaSuccess || n < 1) {
    cudaGetLastError();
    n = 1;
  }
  return n;
}

Q8Geom make_geom(const gc_kv_pool* pool, int32_t n_blocks, int32_t layer0, int32_t layers,
                 bool layer_major) {
  Q8Geom g;
  const gc_pool_config& c = pool->cfg;
  g.group = static_cast<uint32_t>(c.page_size) * c.head_dim;
  g.hdr_bytes = static_cast<uint32_t>(q8_header_bytes(c));
  g.chunk_bytes = q8_chunk_bytes(c);
  g.L = c.num_layers;
  g.num_pages = c.num_pages;
  g.Hkv = c.num_kv_heads;
  g.n_blocks = n_blocks;
  g.layer0 = layer0;
  g.layers = layers;
  g.layer_major = layer_major ? 1 : 0;
  return g;
}

}  // namespace

size_t q8_header_bytes(const gc_pool_config& c) {
  return (static_cast<size_t>(c.num_kv_heads) * 4 + 15) / 16 * 16;
}

size_t q8_chunk_bytes(const gc_pool_config& c) {
  return q8_header_bytes(c) + static_cast<size_t>(c.num_kv_heads) * c.page_size * c.head_dim;
}

gc_status launch_save_q8(const gc_kv_pool* pool, uint8_t* image, const int32_t* block_ids,
                         int32_t n_blocks, int32_t layer0, int32_t layers, bool layer_major,
                         cudaStream_t stream) {
  const Q8Geom g = make_geom(pool, n_blocks, layer0, layers, layer_major);
  const uint64_t groups = static_cast<uint64_t>(n_blocks) * layers * 2 * g.Hkv;
  uint64_t grid = (groups + 7) / 8;  // 8 warps per block, a warp per group
  static const int per_sm = resident_blocks(save_q8_kernel);
  const uint64_t cap = static_cast<uint64_t>(pool->num_sms) * per_sm;
  if (grid > cap) grid = cap;
  save_q8_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(image, pool->data, block_ids, g,
                                                                  pool->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_kv_save_q8: kernel launch");
  return GC_OK;
}

gc_status launch_restore_q8(const gc_kv_pool* pool, const uint8_t* image,
                            const int32_t* block_ids, int32_t n_blocks, int32_t layer0,
                            int32_t layers, bool layer_major, cudaStream_t stream) {
  const Q8Geom g = make_geom(pool, n_blocks, layer0, layers, layer_major);
  const uint64_t words = static_cast<uint64_t>(n_blocks) * layers * 2 * g.Hkv * (g.group / 16);
  uint64_t grid = (words + 256 * 4 - 1) / (256 * 4);
  static const int per_sm = resident_blocks(restore_q8_kernel);
  const uint64_t cap = static_cast<uint64_t>(pool->num_sms) * per_sm;
  if (grid > cap) grid = cap;
  restore_q8_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(image, pool->data, block_ids,
                                                                     g, pool->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_kv_restore_q8: kernel launch");
  return GC_OK;
}

}  // namespace gc
