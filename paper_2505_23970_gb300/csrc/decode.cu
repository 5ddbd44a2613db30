// Paged decode attention: one new token per request (Sec. 2.1: the decode
// phase generates tokens one at a time; with the KV cache it is bound by
// memory, not arithmetic).  For request b with context length T_b (the new
// token's own K/V already appended at position T_b - 1), q head h and kv
// head g = h / G:
//     out[b][h] = sum_{j < T_b} softmax_j(scale * q[b][h] . k_j) v_j
// with k_j, v_j read from the paged pool through block_table[b].
//
// The work is streaming every cached K/V row once (2*Hkv*d*2 bytes per key)
// with 4*G*d FLOP per key per kv head: about 8 FLOP per byte at G = 8, so it
// runs on the CUDA cores and is shaped for HBM: split-KV work units of
// (request, kv head, 512-key range), claimed by a persistent grid (resident
// blocks on every SM) from a counter, each unit done by one 4-warp CTA.
// A warp takes 64 keys at a time:
//   QK   lane = 2 keys; q of the G heads (fp32) is read from shared memory,
//        16-byte K loads, fp32 dot products for all G heads;
//   max  per head over the 64 keys (warp reduction), online softmax in the
//        log2 domain (running max per warp, O and l rescaled when it grows);
//   PV   lane = d/32 output columns: each key's V row is one coalesced
//        warp-wide load, p of the G heads from shared memory, fp32 FMA.
// The 4 warps of a unit then merge their (max, sum, O) partials, and a
// second kernel merges the units of a request-head when a request is split.
// Everything is fp32 after the bf16 loads; out is rounded to bf16.
#include "gc_internal.cuh"
#include "sm103_ptx.cuh"

namespace gc {
namespace {

constexpr int kWarps = 4;
constexpr int kChunk = 64;      // keys per warp iteration (2 per lane)
constexpr int kSplitLen = 512;  // keys per work unit

struct DecGeom {
  int32_t batch, Hq, Hkv, ps_shift, num_pages, max_blocks, layer, max_splits;
  float scale_log2;
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// 2^x with 2^-inf = 0 (ex2.approx.ftz maps -inf to +0).
__device__ __forceinline__ float exp2f_fast(float x) { return ptx::ex2_approx(x); }

// Work units of a request: kv heads x key ranges of kSplitLen (one range for
// a request whose length is invalid: it writes zeros).
__device__ __forceinline__ int request_splits(int T, int cap) {
  return (T < 1 || T > cap) ? 1 : (T + kSplitLen - 1) / kSplitLen;
}

template <int D, int G>
struct DecSmem {
  struct Loop {
    float q[G][D];                  // q of the G heads, fp32
    float p[kWarps][kChunk][G];     // this chunk's probabilities
    int64_t row[kWarps][kChunk];    // K row of each key (-1: no key)
  };
  struct Merge {
    float o[kWarps][G][D];
  };
  union {
    Loop loop;
    Merge merge;
  };
  float m[kWarps][G];
  float l[kWarps][G];
  int unit;
  // followed by unit_start[batch + 1]
};

template <int G>
struct MinBlocks {
  static constexpr int value = G >= 16 ? 2 : 4;
};

template <int D, int G>
__global__ void __launch_bounds__(kWarps * 32, MinBlocks<G>::value) decode_kernel(
    const __nv_bfloat16* __restrict__ q, const uint8_t* __restrict__ pool,
    const int32_t* __restrict__ block_table, const int32_t* __restrict__ seq_lens, DecGeom geo,
    __nv_bfloat16* __restrict__ out, float* __restrict__ ws, int* __restrict__ counter,
    int32_t* status) {
  constexpr int E = D / 32;  // output columns per lane
  extern __shared__ __align__(16) uint8_t smem_raw[];
  DecSmem<D, G>& sm = *reinterpret_cast<DecSmem<D, G>*>(smem_raw);
  int* unit_start = reinterpret_cast<int*>(smem_raw + sizeof(DecSmem<D, G>));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ps = 1 << geo.ps_shift;
  const int cap = geo.max_blocks << geo.ps_shift;

  // work units per request (kv heads x key ranges), exclusive scan
  if (warp == 0) {
    int running = 0;
    for (int b0 = 0; b0 < geo.batch; b0 += 32) {
      const int b = b0 + lane;
      const int cnt = b < geo.batch ? geo.Hkv * request_splits(__ldg(seq_lens + b), cap) : 0;
      int incl = cnt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (b < geo.batch) unit_start[b] = running + incl - cnt;
      running += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) unit_start[geo.batch] = running;
  }
  __syncthreads();
  const int total_units = unit_start[geo.batch];
  const int64_t plane = static_cast<int64_t>(geo.num_pages) * geo.Hkv * ps;  // rows per plane
  const int64_t k_plane0 = static_cast<int64_t>(geo.layer) * 2 * plane;
  const uint4* pool4 = reinterpret_cast<const uint4*>(pool);
  const uint32_t* pool32 = reinterpret_cast<const uint32_t*>(pool);

  while (true) {
    if (threadIdx.x == 0) sm.unit = atomicAdd(counter, 1);
    __syncthreads();
    const int u = sm.unit;
    if (u >= total_units) break;
    int lo = 0, hi = geo.batch;  // last b with unit_start[b] <= u
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (unit_start[mid] <= u) lo = mid; else hi = mid;
    }
    const int b = lo;
    const int local = u - unit_start[b];
    const int g = local % geo.Hkv, s = local / geo.Hkv;
    const int nsplit = (unit_start[b + 1] - unit_start[b]) / geo.Hkv;
    int T = __ldg(seq_lens + b);
    if (T < 1 || T > cap) {
      if (threadIdx.x == 0 && g == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
      T = 0;  // no keys: the output of this request is zero
    }
    const int k0 = s * kSplitLen;
    const int k1 = min(k0 + kSplitLen, T);

    const __nv_bfloat16* qg = q + (static_cast<int64_t>(b) * geo.Hq + g * G) * D;
    for (int i = threadIdx.x; i < G * D; i += kWarps * 32)
      (&sm.loop.q[0][0])[i] = __bfloat162float(qg[i]);
    __syncthreads();

    const int32_t* bt = block_table + static_cast<int64_t>(b) * geo.max_blocks;
    auto row_of = [&](int key) -> int64_t {
      if (key >= k1) return -1;
      const int page = __ldg(bt + (key >> geo.ps_shift));
      if (page < 0 || page >= geo.num_pages) {
        record_error(status, GC_ERR_OUT_OF_RANGE);
        return -1;
      }
      return k_plane0 + (static_cast<int64_t>(page) * geo.Hkv + g) * ps + (key & (ps - 1));
    };

    float m_w[G], l_ln[G], o[G][E];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      m_w[h] = -INFINITY;
      l_ln[h] = 0.f;
#pragma unroll
      for (int e = 0; e < E; ++e) o[h][e] = 0.f;
    }

    for (int base = k0 + warp * kChunk; base < k1; base += kWarps * kChunk) {
      // ---- QK: this lane's keys base + lane and base + 32 + lane
      const int64_t rA = row_of(base + lane), rB = row_of(base + 32 + lane);
      float aA[G], aB[G];
#pragma unroll
      for (int h = 0; h < G; ++h) aA[h] = aB[h] = 0.f;
      const uint4* kA = pool4 + (rA < 0 ? 0 : rA) * (D / 8);
      const uint4* kB = pool4 + (rB < 0 ? 0 : rB) * (D / 8);
#pragma unroll 4
      for (int c = 0; c < D / 8; ++c) {
        const uint4 va = rA >= 0 ? __ldg(kA + c) : make_uint4(0, 0, 0, 0);
        const uint4 vb = rB >= 0 ? __ldg(kB + c) : make_uint4(0, 0, 0, 0);
        const float ka[8] = {bf_lo(va.x), bf_hi(va.x), bf_lo(va.y), bf_hi(va.y),
                             bf_lo(va.z), bf_hi(va.z), bf_lo(va.w), bf_hi(va.w)};
        const float kb[8] = {bf_lo(vb.x), bf_hi(vb.x), bf_lo(vb.y), bf_hi(vb.y),
                             bf_lo(vb.z), bf_hi(vb.z), bf_lo(vb.w), bf_hi(vb.w)};
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float4 q0 = *reinterpret_cast<const float4*>(&sm.loop.q[h][c * 8]);
          const float4 q1 = *reinterpret_cast<const float4*>(&sm.loop.q[h][c * 8 + 4]);
          aA[h] = fmaf(q0.x, ka[0], aA[h]); aA[h] = fmaf(q0.y, ka[1], aA[h]);
          aA[h] = fmaf(q0.z, ka[2], aA[h]); aA[h] = fmaf(q0.w, ka[3], aA[h]);
          aA[h] = fmaf(q1.x, ka[4], aA[h]); aA[h] = fmaf(q1.y, ka[5], aA[h]);
          aA[h] = fmaf(q1.z, ka[6], aA[h]); aA[h] = fmaf(q1.w, ka[7], aA[h]);
          aB[h] = fmaf(q0.x, kb[0], aB[h]); aB[h] = fmaf(q0.y, kb[1], aB[h]);
          aB[h] = fmaf(q0.z, kb[2], aB[h]); aB[h] = fmaf(q0.w, kb[3], aB[h]);
          aB[h] = fmaf(q1.x, kb[4], aB[h]); aB[h] = fmaf(q1.y, kb[5], aB[h]);
          aB[h] = fmaf(q1.z, kb[6], aB[h]); aB[h] = fmaf(q1.w, kb[7], aB[h]);
        }
      }
      // ---- online softmax over the chunk (log2 domain)
#pragma unroll
      for (int h = 0; h < G; ++h) {
        const float sA = rA >= 0 ? aA[h] * geo.scale_log2 : -INFINITY;
        const float sB = rB >= 0 ? aB[h] * geo.scale_log2 : -INFINITY;
        const float m_new = fmaxf(m_w[h], warp_max(fmaxf(sA, sB)));
        // m_new is -inf only if no key has been seen yet: nothing to rescale
        const float alpha = m_new == -INFINITY ? 1.f : exp2f_fast(m_w[h] - m_new);
        const float pA = m_new == -INFINITY ? 0.f : exp2f_fast(sA - m_new);
        const float pB = m_new == -INFINITY ? 0.f : exp2f_fast(sB - m_new);
        l_ln[h] = l_ln[h] * alpha + (pA + pB);
#pragma unroll
        for (int e = 0; e < E; ++e) o[h][e] *= alpha;
        m_w[h] = m_new;
        sm.loop.p[warp][lane][h] = pA;
        sm.loop.p[warp][32 + lane][h] = pB;
      }
      sm.loop.row[warp][lane] = rA;
      sm.loop.row[warp][32 + lane] = rB;
      __syncwarp();
      // ---- PV: lane owns output columns lane*E .. lane*E + E - 1; the V rows
      // of 8 keys are loaded before they are used
      const int nk = min(kChunk, k1 - base);
      for (int k8 = 0; k8 < nk; k8 += 8) {
        float v[8][E];
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          const int64_t r = sm.loop.row[warp][k8 + t];
          if (r >= 0) {
            const int64_t vrow = r + plane;
            if constexpr (E == 4) {
              const uint2 w2 = __ldg(reinterpret_cast<const uint2*>(pool32 + vrow * (D / 2)) + lane);
              v[t][0] = bf_lo(w2.x); v[t][1] = bf_hi(w2.x);
              v[t][2] = bf_lo(w2.y); v[t][3] = bf_hi(w2.y);
            } else {
              const uint32_t w1 = __ldg(pool32 + vrow * (D / 2) + lane);
              v[t][0] = bf_lo(w1); v[t][1] = bf_hi(w1);
            }
          } else {
#pragma unroll
            for (int e = 0; e < E; ++e) v[t][e] = 0.f;  // no key: p is 0 too
          }
        }
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float p = sm.loop.p[warp][k8 + t][h];
#pragma unroll
            for (int e = 0; e < E; ++e) o[h][e] = fmaf(p, v[t][e], o[h][e]);
          }
      }
      __syncwarp();
    }

    // ---- merge the warps' partials
    float l_w[G];
#pragma unroll
    for (int h = 0; h < G; ++h) l_w[h] = warp_sum(l_ln[h]);
    __syncthreads();  // every warp is done with the loop buffers
#pragma unroll
    for (int h = 0; h < G; ++h) {
#pragma unroll
      for (int e = 0; e < E; ++e) sm.merge.o[warp][h][lane * E + e] = o[h][e];
      if (lane == 0) {
        sm.m[warp][h] = m_w[h];
        sm.l[warp][h] = l_w[h];
      }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < G * D; i += kWarps * 32) {
      const int h = i / D, d = i - h * D;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm.m[w][h]);
      float acc = 0.f, L = 0.f;
      if (M != -INFINITY) {
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
          const float f = exp2f_fast(sm.m[w][h] - M);
          acc = fmaf(sm.merge.o[w][h][d], f, acc);
          L = fmaf(sm.l[w][h], f, L);
        }
      }
      const int64_t head = static_cast<int64_t>(b) * geo.Hq + g * G + h;
      if (nsplit == 1) {
        out[head * D + d] = __float2bfloat16_rn(L > 0.f ? acc / L : 0.f);
      } else {
        ws[(head * geo.max_splits + s) * D + d] = acc;
        if (d == 0) {
          float* ml = ws + static_cast<int64_t>(geo.batch) * geo.Hq * geo.max_splits * D;
          ml[(head * geo.max_splits + s) * 2 + 0] = M;
          ml[(head * geo.max_splits + s) * 2 + 1] = L;
        }
      }
    }
    __syncthreads();  // the loop buffers and sm.unit are reused by the next unit
  }
}

// For requests split over several key ranges:
// out[b][h] = sum_s O_s 2^(m_s - M) / sum_s l_s 2^(m_s - M), M = max_s m_s.
template <int D>
__global__ void __launch_bounds__(D) decode_merge_kernel(const float* __restrict__ ws,
                                                         const int32_t* __restrict__ seq_lens,
                                                         DecGeom geo,
                                                         __nv_bfloat16* __restrict__ out) {
  const int64_t head = blockIdx.x;
  const int b = static_cast<int>(head / geo.Hq);
  const int nsplit = request_splits(__ldg(seq_lens + b), geo.max_blocks << geo.ps_shift);
  if (nsplit <= 1) return;  // written by the unit itself
  const int d = threadIdx.x;
  const float* ml = ws + static_cast<int64_t>(geo.batch) * geo.Hq * geo.max_splits * D +
                    head * geo.max_splits * 2;
  float M = -INFINITY;
  for (int s = 0; s < nsplit; ++s) M = fmaxf(M, ml[2 * s]);
  float acc = 0.f, L = 0.f;
  if (M != -INFINITY) {
    for (int s = 0; s < nsplit; ++s) {
      const float f = exp2f_fast(ml[2 * s] - M);
      acc = fmaf(ws[(head * geo.max_splits + s) * D + d], f, acc);
      L = fmaf(ml[2 * s + 1], f, L);
    }
  }
  out[head * D + d] = __float2bfloat16_rn(L > 0.f ? acc / L : 0.f);
}

template <int D, int G>
gc_status launch_g(const gc_kv_pool* pool, const DecodeArgs& a, const DecGeom& geo,
                   cudaStream_t stream) {
  const size_t smem = sizeof(DecSmem<D, G>) + (static_cast<size_t>(a.batch) + 1) * sizeof(int);
  cudaError_t e = cudaFuncSetAttribute(decode_kernel<D, G>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: smem attribute");
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_kernel<D, G>, kWarps * 32,
                                                    smem);
  if (e != cudaSuccess || per_sm < 1) return cuda_fail(e, "gc_paged_decode_attn: occupancy");
  // units are claimed from a counter in the pool's control block
  e = cudaMemsetAsync(pool->decode_counter, 0, sizeof(int), stream);
  if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: clearing the work counter");
  decode_kernel<D, G><<<pool->num_sms * per_sm, kWarps * 32, smem, stream>>>(
      static_cast<const __nv_bfloat16*>(a.q), pool->data, a.block_table, a.seq_lens, geo,
      static_cast<__nv_bfloat16*>(a.out), static_cast<float*>(a.workspace), pool->decode_counter,
      pool->status);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: kernel launch");
  if (geo.max_splits > 1) {
    decode_merge_kernel<D><<<static_cast<unsigned>(a.batch * geo.Hq), D, 0, stream>>>(
        static_cast<const float*>(a.workspace), a.seq_lens, geo,
        static_cast<__nv_bfloat16*>(a.out));
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: merge kernel launch");
  }
  return GC_OK;
}

template <int D>
gc_status launch_d(const gc_kv_pool* pool, const DecodeArgs& a, const DecGeom& geo, int G,
                   cudaStream_t stream) {
  switch (G) {
    case 1: return launch_g<D, 1>(pool, a, geo, stream);
    case 2: return launch_g<D, 2>(pool, a, geo, stream);
    case 4: return launch_g<D, 4>(pool, a, geo, stream);
    case 8: return launch_g<D, 8>(pool, a, geo, stream);
    default: return launch_g<D, 16>(pool, a, geo, stream);
  }
}

}  // namespace

DecodeSplit decode_split(const gc_kv_pool* pool, int32_t batch, int32_t max_blocks,
                         int32_t num_q_heads) {
  DecodeSplit d;
  const int64_t max_ctx = static_cast<int64_t>(max_blocks) * pool->cfg.page_size;
  const int64_t splits = max_ctx > 0 ? (max_ctx + kSplitLen - 1) / kSplitLen : 1;
  d.splits = static_cast<int32_t>(splits);
  d.split_len = kSplitLen;
  d.workspace_bytes = splits > 1 ? static_cast<size_t>(batch) * num_q_heads * splits *
                                       (pool->cfg.head_dim + 2) * sizeof(float)
                                 : 0;
  return d;
}

gc_status launch_decode(const gc_kv_pool* pool, const DecodeArgs& a, cudaStream_t stream) {
  const DecodeSplit sp = decode_split(pool, a.batch, a.max_blocks, a.num_q_heads);
  if (sp.workspace_bytes > 0 && (a.workspace == nullptr || a.workspace_bytes < sp.workspace_bytes))
    return fail(GC_ERR_INVALID_ARG,
                "gc_paged_decode_attn: workspace of %zu bytes needed "
                "(gc_paged_decode_workspace_bytes), got %zu",
                sp.workspace_bytes, a.workspace_bytes);
  const long long units = static_cast<long long>(a.batch) * pool->cfg.num_kv_heads * sp.splits;
  if (units > 2147483647LL)
    return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: %lld work units", units);
  if (a.batch > 8192) return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: batch %d > 8192", a.batch);
  DecGeom geo;
  geo.batch = a.batch;
  geo.Hq = a.num_q_heads;
  geo.Hkv = pool->cfg.num_kv_heads;
  int sh = 0;
  while ((1 << sh) < pool->cfg.page_size) ++sh;
  geo.ps_shift = sh;
  geo.num_pages = pool->cfg.num_pages;
  geo.max_blocks = a.max_blocks;
  geo.layer = a.layer;
  geo.max_splits = sp.splits;
  geo.scale_log2 = a.softmax_scale * 1.4426950408889634f;
  const int G = a.num_q_heads / pool->cfg.num_kv_heads;
  if (pool->cfg.head_dim == 128) return launch_d<128>(pool, a, geo, G, stream);
  return launch_d<64>(pool, a, geo, G, stream);
}

}  // namespace gc
