// Paged decode attention: one new token per request (Sec. 2.1: the decode
// phase generates tokens one at a time; with the KV cache it is bound by
// memory, not arithmetic).  For request b with context length T_b (the new
// token's own K/V already appended at position T_b - 1), q head h and kv
// head g = h / G:
//     out[b][h] = sum_{j < T_b} softmax_j(scale * q[b][h] . k_j) v_j
// with k_j, v_j read from the paged pool through block_table[b].
//
// Decode streams every cached K/V row once (2*Hkv*d*2 bytes per key) for
// 4*G*d FLOP per key and kv head, so the bound is HBM.  Two kernels do it:
//  - head_dim 128 with G <= 16 (the 70B-shaped layer): decode_tc.cu, the
//    transposed tensor-core kernel (keys on the TMEM lanes), each CTA an equal
//    share of all K/V tiles;
//  - otherwise: the prefill kernel in decode mode (attn_tc.cu).  Its
//    persistent CTAs stream the pages through a TMA ring, and the tensor cores
//    do the G-row products (a Q tile of G real rows: the padding rows cost
//    tensor time that the memory bound leaves idle).  To fill every SM, each
//    request is cut into key ranges of 4 to 16 K/V tiles, chosen per call
//    from the batch and the block table's capacity (work items = requests x
//    kv heads x ranges); a request with several ranges writes fp32 partials
//    (O unnormalised, reference max in log2 units, sum) and the merge kernel
//    below combines them:
//     out = sum_s O_s 2^(m_s - M) / sum_s l_s 2^(m_s - M),  M = max_s m_s.
#include "gc_internal.cuh"
#include "sm103_ptx.cuh"

namespace gc {
namespace {

constexpr int kTileKeys = 128;     // keys per K/V tile of the attention kernel
constexpr int kMinSplitTiles = 4;  // key ranges of 4..16 K/V tiles (512..2048 keys)
constexpr int kMaxSplitTiles = 16;

__device__ __forceinline__ int request_splits(int T, int cap, int split_tiles) {
  if (T < 1 || T > cap) return 0;  // recorded as an error by the attention kernel
  const int tiles = (T + kTileKeys - 1) / kTileKeys;
  return (tiles + split_tiles - 1) / split_tiles;
}

template <int D>
__global__ void __launch_bounds__(D) decode_merge_kernel(const float* __restrict__ ws,
                                                         const int32_t* __restrict__ seq_lens,
                                                         int32_t batch, int32_t Hq,
                                                         int32_t max_splits, int32_t cap,
                                                         int32_t split_tiles,
                                                         __nv_bfloat16* __restrict__ out) {
  // launched as a programmatic dependent of the attention kernel: the
  // blocks may be resident before it ends, so wait for its results here
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int64_t head = blockIdx.x;
  const int b = static_cast<int>(head / Hq);
  const int nsplit = request_splits(__ldg(seq_lens + b), cap, split_tiles);
  if (nsplit <= 1) return;  // written by the attention kernel itself (or invalid)
  const int d = threadIdx.x;
  const float2* ml = reinterpret_cast<const float2*>(
      ws + static_cast<int64_t>(batch) * Hq * max_splits * D + head * max_splits * 2);
  const float* o = ws + head * max_splits * D + d;
  // independent loads, 8 ranges at a time
  float M = -INFINITY;
  for (int s0 = 0; s0 < nsplit; s0 += 8) {
#pragma unroll
    for (int t = 0; t < 8; ++t)
      if (s0 + t < nsplit) M = fmaxf(M, __ldg(ml + s0 + t).x);
  }
  float acc = 0.f, L = 0.f;
  for (int s0 = 0; s0 < nsplit; s0 += 8) {
    float2 mls[8];
    float os[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const bool in = s0 + t < nsplit;
      mls[t] = in ? __ldg(ml + s0 + t) : make_float2(-INFINITY, 0.f);
      os[t] = in ? __ldg(o + static_cast<int64_t>(s0 + t) * D) : 0.f;
    }
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const float f = ptx::ex2_approx(mls[t].x - M);
      acc = fmaf(os[t], f, acc);
      L = fmaf(mls[t].y, f, L);
    }
  }
  out[head * D + d] = __float2bfloat16_rn(acc / L);
}

}  // namespace

DecodeSplit decode_split(const gc_kv_pool* pool, int32_t batch, int32_t max_blocks,
                         int32_t num_q_heads) {
  DecodeSplit d;
  const int64_t cap = static_cast<int64_t>(max_blocks) * pool->cfg.page_size;
  const int64_t tiles = (cap + kTileKeys - 1) / kTileKeys;
  // Longer ranges cost less per tile (each work item has a fixed start-up and
  // epilogue); shorter ones spread a small batch over more SMs.  Aim for about
  // two items per CTA when every request had the longest context.
  const int64_t tile_units = static_cast<int64_t>(batch) * pool->cfg.num_kv_heads * tiles;
  int split_tiles = kMinSplitTiles;
  while (split_tiles < kMaxSplitTiles &&
         tile_units > static_cast<int64_t>(split_tiles) * 2 * pool->num_sms)
    split_tiles *= 2;
  const int64_t splits = tiles > 0 ? (tiles + split_tiles - 1) / split_tiles : 1;
  d.splits = static_cast<int32_t>(splits);
  d.split_tiles = split_tiles;
  d.split_len = split_tiles * kTileKeys;
  d.workspace_bytes = splits > 1 ? static_cast<size_t>(batch) * num_q_heads * splits *
                                       (pool->cfg.head_dim + 2) * sizeof(float)
                                 : 0;
  return d;
}

size_t decode_workspace_bytes(const gc_kv_pool* pool, int32_t batch, int32_t max_blocks,
                              int32_t num_q_heads) {
  if (decode_tc_supported(pool, num_q_heads)) return decode_tc_workspace_bytes(pool, batch);
  return decode_split(pool, batch, max_blocks, num_q_heads).workspace_bytes;
}

gc_status launch_decode(const gc_kv_pool* pool, const DecodeArgs& a, cudaStream_t stream,
                        const Q8Pages* q8) {
  if (a.batch > 8192) return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: batch %d > 8192", a.batch);
  if (static_cast<int64_t>(a.max_blocks) * pool->cfg.page_size > 2147483647LL)
    return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: %lld-token block table",
                static_cast<long long>(a.max_blocks) * pool->cfg.page_size);
  if (decode_tc_supported(pool, a.num_q_heads)) return launch_decode_tc(pool, a, stream, q8);
  const DecodeSplit sp = decode_split(pool, a.batch, a.max_blocks, a.num_q_heads);
  if (sp.workspace_bytes > 0 && (a.workspace == nullptr || a.workspace_bytes < sp.workspace_bytes))
    return fail(GC_ERR_INVALID_ARG,
                "gc_paged_decode_attn: workspace of %zu bytes needed "
                "(gc_paged_decode_workspace_bytes), got %zu",
                sp.workspace_bytes, a.workspace_bytes);
  const long long items = static_cast<long long>(a.batch) * pool->cfg.num_kv_heads * sp.splits;
  if (items > 2147483647LL)
    return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: %lld work items", items);
  const int64_t cap = static_cast<int64_t>(a.max_blocks) * pool->cfg.page_size;
  AttnArgs args{a.q, a.out, a.block_table, nullptr, nullptr, nullptr, a.batch, a.max_blocks,
                a.layer, a.num_q_heads, a.batch, a.softmax_scale};
  const DecodeMode dm{sp.split_tiles, sp.splits, a.seq_lens, static_cast<float*>(a.workspace)};
  gc_status st = launch_attn_tc_decode(pool, args, dm, stream, q8);
  if (st != GC_OK || sp.splits <= 1) return st;
  const unsigned heads = static_cast<unsigned>(a.batch) * static_cast<unsigned>(a.num_q_heads);
  // programmatic dependent launch: the merge grid is set up while the
  // attention kernel drains, and waits for it with griddepcontrol.wait
  cudaLaunchConfig_t lc = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  lc.gridDim = dim3(heads);
  lc.blockDim = dim3(pool->cfg.head_dim);
  lc.dynamicSmemBytes = 0;
  lc.stream = stream;
  lc.attrs = attr;
  lc.numAttrs = 1;
  const float* wsp = static_cast<const float*>(a.workspace);
  __nv_bfloat16* outp = static_cast<__nv_bfloat16*>(a.out);
  const int32_t cap32 = static_cast<int32_t>(cap);
  const cudaError_t e =
      pool->cfg.head_dim == 128
          ? cudaLaunchKernelEx(&lc, decode_merge_kernel<128>, wsp, a.seq_lens, a.batch,
                               a.num_q_heads, sp.splits, cap32, sp.split_tiles, outp)
          : cudaLaunchKernelEx(&lc, decode_merge_kernel<64>, wsp, a.seq_lens, a.batch,
                               a.num_q_heads, sp.splits, cap32, sp.split_tiles, outp);
  if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: merge kernel launch");
  return GC_OK;
}

}  // namespace gc
