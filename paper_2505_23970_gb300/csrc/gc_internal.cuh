// Internal declarations shared by the libgc translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "gc.h"

struct gc_kv_pool {
  gc_pool_config cfg;
  uint8_t* data;          // KV planes [L][2][num_pages][Hkv][ps][d] bf16
  size_t data_bytes;
  int32_t* status;        // device status word (first error recorded by a kernel)
  int32_t* work_counter;  // attention work-item counter (control block, zeroed per launch)
  int32_t* merge_counters;  // [kMergeCounters] decode merge counters (control block, kept at 0)
  void* owned;            // cudaMalloc'd block, or nullptr if caller-owned
  int device;
  int num_sms;
};

namespace gc {

constexpr int kMergeCounters = 448;  // ints after the first 256 bytes of the control block

// Thread-local error message; returns `s` for convenient `return fail(...)`.
gc_status fail(gc_status s, const char* fmt, ...);
gc_status cuda_fail(cudaError_t e, const char* what);

inline size_t page_bytes(const gc_pool_config& c) {
  return static_cast<size_t>(c.num_kv_heads) * c.page_size * c.head_dim * 2;
}

// Record the first device-side error in the pool's status word.
__device__ __forceinline__ void record_error(int32_t* status, int32_t code) {
  atomicCAS(status, 0, code);
}

// 16 8-bit codes (one 16-byte word, byte i = code i) -> 16 bf16 values
// (lo: codes 0-7, hi: codes 8-15, in order), each c * s in binary32 rounded
// to bf16 (nearest even).  The 8-bit restore and the attention over 8-bit
// pages both dequantise with it, so they produce the same bf16 values.
// float(c) is formed without a conversion instruction: the byte c + 128
// (c xor 0x80) placed in the low mantissa bits of 2^23 is the float
// 2^23 + 128 + c, from which subtracting 2^23 + 128 is exact; the
// subtraction and the product (one rounding, as c * s) run as paired fp32
// operations, two codes at a time.
__device__ __forceinline__ uint32_t q8_pair(uint32_t biased, uint32_t sel, uint64_t s2) {
  const uint32_t a = __byte_perm(biased, 0x4B000000u, 0x7540u + sel);
  const uint32_t b = __byte_perm(biased, 0x4B000000u, 0x7540u + sel + 1);
  uint32_t r;
  asm("{\n\t.reg .b64 t;\n\t.reg .f32 x, y;\n\t"
      "mov.b64 t, {%1, %2};\n\t"
      "add.rn.f32x2 t, t, %3;\n\t"
      "mul.rn.f32x2 t, t, %4;\n\t"
      "mov.b64 {x, y}, t;\n\t"
      "cvt.rn.bf16x2.f32 %0, y, x;\n\t}"
      : "=r"(r)
      : "r"(a), "r"(b), "l"(0xCB000080CB000080ull), "l"(s2));  // -(2^23 + 128), twice
  return r;
}

__device__ __forceinline__ void q8_dequant16(const uint4& v, float s, uint4& lo, uint4& hi) {
  const uint64_t s2 = (static_cast<uint64_t>(__float_as_uint(s)) << 32) | __float_as_uint(s);
  const uint32_t x = v.x ^ 0x80808080u, y = v.y ^ 0x80808080u;
  const uint32_t z = v.z ^ 0x80808080u, w = v.w ^ 0x80808080u;
  lo.x = q8_pair(x, 0, s2);
  lo.y = q8_pair(x, 2, s2);
  lo.z = q8_pair(y, 0, s2);
  lo.w = q8_pair(y, 2, s2);
  hi.x = q8_pair(z, 0, s2);
  hi.y = q8_pair(z, 2, s2);
  hi.z = q8_pair(w, 0, s2);
  hi.w = q8_pair(w, 2, s2);
}

// ---------------------------------------------------------------- launchers
// Each returns GC_OK or a status with the message already set.
// Page copies between a staging image [n_blocks][L][2][chunk] (or, with
// layer_major, [L][n_blocks][2][chunk]) and the pool, layers
// [layer0, layer0 + layers) only; gather = false restores
// (staging -> pool), gather = true saves.
gc_status launch_restore_bulk(const gc_kv_pool* pool, uint8_t* staging, const int32_t* block_ids,
                              int32_t n_blocks, int32_t layer0, int32_t layers, bool layer_major,
                              bool gather, cudaStream_t stream);
gc_status launch_restore_vector(const gc_kv_pool* pool, uint8_t* staging,
                                const int32_t* block_ids, int32_t n_blocks, int32_t layer0,
                                int32_t layers, bool layer_major, bool gather,
                                cudaStream_t stream);
// 8-bit cache tier (INT8 codes + one binary32 scale per (block, layer, plane,
// kv head)); image chunk = scales padded to 16 bytes, then [Hkv][ps][d] int8.
size_t q8_header_bytes(const gc_pool_config& c);
size_t q8_chunk_bytes(const gc_pool_config& c);
gc_status launch_save_q8(const gc_kv_pool* pool, uint8_t* image, const int32_t* block_ids,
                         int32_t n_blocks, int32_t layer0, int32_t layers, bool layer_major,
                         cudaStream_t stream);
gc_status launch_restore_q8(const gc_kv_pool* pool, const uint8_t* image,
                            const int32_t* block_ids, int32_t n_blocks, int32_t layer0,
                            int32_t layers, bool layer_major, cudaStream_t stream);
gc_status launch_selftest_timeout(const gc_kv_pool* pool, cudaStream_t stream);
gc_status launch_append(const gc_kv_pool* pool, const void* k_new, const void* v_new,
                        const int32_t* block_table, const int32_t* prefix_lens,
                        const int32_t* cu_new_lens, int32_t batch, int32_t max_blocks,
                        int32_t layer, int32_t total_new_tokens, cudaStream_t stream);

struct AttnArgs {
  const void* q;
  void* out;
  const int32_t* block_table;
  const int32_t* prefix_lens;
  const int32_t* new_lens;
  const int32_t* cu_new_lens;
  int32_t batch, max_blocks, layer, num_q_heads, total_new_tokens;
  float softmax_scale;
};

gc_status launch_attn_simt(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream);
gc_status launch_attn_tc(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream);
gc_status launch_attn_tc_noalloc(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream);
// Prefill attention with some pages read from a device 8-bit image (the
// cache tier's layout) instead of the pool: q8_table [batch][max_blocks]
// gives, per page of a request, an image block (>= 0) or -1 (pool page).
struct Q8Pages {
  const uint8_t* image;
  const int32_t* table;
  int32_t n_blocks;   // blocks in the image
  bool layer_major;   // image [L][n][2][chunk] instead of [n][L][2][chunk]
};
gc_status launch_attn_tc_q8(const gc_kv_pool* pool, const AttnArgs& a, const Q8Pages& q8,
                            cudaStream_t stream);
// head_dim 128 prefill on CTA pairs (attn_tc2.cu), work items claimed from
// `work_counter` (zeroed by the launch).
gc_status launch_attn_tc2(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream,
                          int* work_counter);
// The same kernel in decode mode: one new token per request (AttnArgs'
// prefix_lens / new_lens / cu_new_lens unused), keys cut into ranges.
struct DecodeMode {
  int32_t split_tiles, max_splits;
  const int32_t* seq_lens;
  float* ws;
};
gc_status launch_attn_tc_decode(const gc_kv_pool* pool, const AttnArgs& a, const DecodeMode& dm,
                                cudaStream_t stream, const Q8Pages* q8 = nullptr);
// Host-side bound of the attention kernels' 32-bit work numbering (items and
// q rows of one call, with a margin of two claims per CTA of `grid`):
// GC_ERR_UNSUPPORTED before anything is launched when a call could pass it.
gc_status check_item_bound(const gc_kv_pool* pool, const AttnArgs& a, const DecodeMode* dm,
                           int grid);

// Paged decode attention (one new token per request), split-KV.
struct DecodeArgs {
  const void* q;
  void* out;
  const int32_t* block_table;
  const int32_t* seq_lens;
  int32_t batch, max_blocks, layer, num_q_heads;
  float softmax_scale;
  void* workspace;
  size_t workspace_bytes;
};
struct DecodeSplit {
  int32_t splits, split_tiles, split_len;  // key ranges per request (at most), their length
  size_t workspace_bytes;     // 0 when requests are not split
};
DecodeSplit decode_split(const gc_kv_pool* pool, int32_t batch, int32_t max_blocks,
                         int32_t num_q_heads);
// With q8, the pages that q8->table maps (>= 0) are read from the 8-bit
// image instead of the pool.
gc_status launch_decode(const gc_kv_pool* pool, const DecodeArgs& a, cudaStream_t stream,
                        const Q8Pages* q8 = nullptr);
// The transposed tensor-core decode kernel (decode_tc.cu): head_dim 128 and
// at most 16 q heads per kv head.
bool decode_tc_supported(const gc_kv_pool* pool, int32_t num_q_heads);
size_t decode_tc_workspace_bytes(const gc_kv_pool* pool, int32_t batch);
// With q8, the pages that q8->table maps (>= 0) are read from the 8-bit
// image instead of the pool.
gc_status launch_decode_tc(const gc_kv_pool* pool, const DecodeArgs& a, cudaStream_t stream,
                           const Q8Pages* q8 = nullptr);
// Workspace bytes of a decode call on either path.
size_t decode_workspace_bytes(const gc_kv_pool* pool, int32_t batch, int32_t max_blocks,
                              int32_t num_q_heads);

}  // namespace gc
