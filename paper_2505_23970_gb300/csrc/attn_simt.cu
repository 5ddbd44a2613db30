// Prefix-reuse causal GQA attention on CUDA cores (no tensor cores): one
// warp per (new token, q head), fp32 throughout, online softmax over the
// keys 0..P_b+i read through the block table (Sec. 2.2: the cached prefix
// KV and the new tokens' KV are processed together).  Slow by design; it is
// the GPU cross-check of the tensor-core kernel's indexing.
#include "gc_internal.cuh"

namespace gc {
namespace {

struct SimtGeom {
  int32_t Hq, Hkv, G, ps_shift, num_pages, batch, max_blocks, layer, total_new;
  float scale_log2;
};

template <int D>
__global__ void __launch_bounds__(128) attn_simt_kernel(
    const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ pool,
    const int32_t* __restrict__ block_table, const int32_t* __restrict__ prefix_lens,
    const int32_t* __restrict__ cu_new_lens, __nv_bfloat16* __restrict__ out, SimtGeom g,
    int32_t* status) {
  constexpr int E = D / 32;  // elements per lane
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int h = blockIdx.y;
  if (t >= g.total_new) return;
  int lo = 0, hi = g.batch;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(cu_new_lens + mid) <= t) lo = mid; else hi = mid;
  }
  const int b = lo;
  const int start = __ldg(cu_new_lens + b), end = __ldg(cu_new_lens + b + 1);
  if (t < start || t >= end || end > g.total_new) {
    if (lane == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
    return;
  }
  const int P = __ldg(prefix_lens + b);
  const int nk = P + (t - start) + 1;
  const int kvh = h / g.G;
  const int ps = 1 << g.ps_shift;
  float qv[E], acc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    qv[e] = __bfloat162float(q[(static_cast<int64_t>(t) * g.Hq + h) * D + lane * E + e]) *
            g.scale_log2;
    acc[e] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  const int64_t plane = static_cast<int64_t>(g.num_pages) * g.Hkv * ps * D;
  const __nv_bfloat16* kplane = pool + (static_cast<int64_t>(g.layer) * 2 + 0) * plane;
  const __nv_bfloat16* vplane = pool + (static_cast<int64_t>(g.layer) * 2 + 1) * plane;
  bool bad = false;
  for (int j = 0; j < nk; ++j) {
    const int blk = j >> g.ps_shift;
    const int page = blk < g.max_blocks
                         ? __ldg(block_table + static_cast<int64_t>(b) * g.max_blocks + blk)
                         : -1;
    if (page < 0 || page >= g.num_pages) {
      bad = true;
      continue;
    }
    const int64_t row = ((static_cast<int64_t>(page) * g.Hkv + kvh) * ps + (j & (ps - 1))) * D;
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < E; ++e) s += qv[e] * __bfloat162float(kplane[row + lane * E + e]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mn = fmaxf(m, s);
    const float alpha = exp2f(m - mn);
    const float p = exp2f(s - mn);
    l = l * alpha + p;
#pragma unroll
    for (int e = 0; e < E; ++e)
      acc[e] = acc[e] * alpha + p * __bfloat162float(vplane[row + lane * E + e]);
    m = mn;
  }
  if (bad && lane == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
  const float inv = 1.f / l;
#pragma unroll
  for (int e = 0; e < E; ++e)
    out[(static_cast<int64_t>(t) * g.Hq + h) * D + lane * E + e] = __float2bfloat16_rn(acc[e] * inv);
}

}  // namespace

gc_status launch_attn_simt(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream) {
  SimtGeom g;
  g.Hq = a.num_q_heads;
  g.Hkv = pool->cfg.num_kv_heads;
  g.G = g.Hq / g.Hkv;
  int s = 0;
  while ((1 << s) < pool->cfg.page_size) ++s;
  g.ps_shift = s;
  g.num_pages = pool->cfg.num_pages;
  g.batch = a.batch;
  g.max_blocks = a.max_blocks;
  g.layer = a.layer;
  g.total_new = a.total_new_tokens;
  g.scale_log2 = a.softmax_scale * 1.4426950408889634f;
  dim3 grid((a.total_new_tokens + 3) / 4, g.Hq);
  auto* q = static_cast<const __nv_bfloat16*>(a.q);
  auto* kv = reinterpret_cast<const __nv_bfloat16*>(pool->data);
  auto* o = static_cast<__nv_bfloat16*>(a.out);
  if (pool->cfg.head_dim == 128)
    attn_simt_kernel<128><<<grid, 128, 0, stream>>>(q, kv, a.block_table, a.prefix_lens,
                                                     a.cu_new_lens, o, g, pool->status);
  else
    attn_simt_kernel<64><<<grid, 128, 0, stream>>>(q, kv, a.block_table, a.prefix_lens,
                                                    a.cu_new_lens, o, g, pool->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn_simt: launch");
  return GC_OK;
}

}  // namespace gc
