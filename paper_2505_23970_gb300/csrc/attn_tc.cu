// Prefix-reuse causal GQA attention on the sm_103a tensor cores.
//
// Operation (Sec. 2.2: the cached context KV and the new tokens' KV are
// processed together; Sec. 2.1: prefill): for request b, q head h, new row
// i < n_b and kv head g = h / G,
//     O[b,i,h] = sum_{j <= P_b + i} softmax_j(scale * q . k_j) v_j
// with keys read from the paged pool through block_table[b].
//
// Design
//  * Work item = (request b, kv head g, pair of 128-row Q tiles), handed out
//    dynamically (an atomic counter in the pool's control block; requests are
//    numbered longest first and a request's items later rows first, so long
//    items start early).  A Q tile packs 128/G new tokens x the G q heads of
//    one kv group (row = token*G + head), so every K/V tile fetched from the
//    pool feeds all G heads, and the two Q tiles of a CTA share each K/V tile.
//  * One persistent CTA per SM, 12 warps:
//      warp 0        TMA producer: Q tiles (3-D map over [T_new][Hq][d]) and
//                    K/V tiles page by page (2-D map over the pool rows) into
//                    a 4-slot ring; the page copies of a tile are issued by
//                    16 lanes, the next tile's pages looked up one tile
//                    ahead; zeroes V rows past the end of the sequence.
//      warp 1        TMEM owner; lane 0 issues Q tile 0's MMAs, lane 0 of
//      warp 2        issues Q tile 1's:
//                      S_i = Q_i K^T   (SS, both operands K-major, fp32 in TMEM)
//                      O_i += P_i V    (TS: P_i read from TMEM, V MN-major)
//                    Each issuer waits for its tile's inputs in chain order,
//                    and tile 1's S(j) also waits until tile 0 has published
//                    P(j), so the two softmax phases alternate and each
//                    tile's MMAs fill the other's softmax time.
//      warps 4-7     softmax of Q tile 0; warps 8-11 softmax of Q tile 1.
//                    One thread per row: S row from TMEM, causal mask, online
//                    softmax in the log2 domain against a running reference
//                    max (the exact max of the row's first tile; recomputed,
//                    with O and l rescaled, only if a later tile's terms
//                    would approach fp32 overflow), P as bf16 written back
//                    over S in TMEM (one arrival per warp), final 1/l
//                    normalisation and the bf16 store of O.  They also
//                    release the ring slots and Q tiles once they have seen
//                    the MMAs that read them complete.
//    Warps 0-3 give registers to the softmax warpgroups (setmaxnreg).
//  * TMEM (512 columns): S0 [0,128) S1 [128,256) O0 [256,256+d) O1 [.., +d).
//    P_i overwrites the first 64 columns of S_i.  Because P_i aliases S_i,
//    S_i(j+1) is issued only after PV_i(j) has completed; the other Q
//    tile's MMAs keep the tensor pipe fed meanwhile.
//  * Decode mode (one new token per request): items are (request, kv head,
//    range of K/V tiles); a request cut into several ranges writes fp32
//    partials that a separate kernel merges.
//  * Pages in the 8-bit cache tier (gc_prefix_prefill_attn_q8): a 16-warp
//    variant whose producer loads an image page's codes (TMA) into the
//    page's rows of the ring slot and whose fourth warpgroup dequantises
//    them there (see "pages of the 8-bit image" below).
//  * Every mbarrier wait and spin is bounded; a timeout raises the CTA's
//    abort flag, all roles leave their loops, in-flight copies and MMAs are
//    drained, TMEM is freed and GC_ERR_TIMEOUT is recorded in the pool
//    status word.
#include <cmath>
#include <mutex>

#include "gc_internal.cuh"
#include "sm103_ptx.cuh"

namespace gc {
namespace {

using namespace ptx;

constexpr int kThreads = 384;
// With pages read from an 8-bit image a fourth warpgroup converts them.
constexpr int kThreadsQ8 = 512;
// Batches up to this size are numbered longest request first (ranked in
// shared memory by every CTA); larger batches keep the given order.
constexpr int kSortMax = 512;
constexpr int kRegsProducer = 88;   // warps 0-3 after setmaxnreg.dec
constexpr int kRegsSoftmax = 208;   // warps 4-11 after setmaxnreg.inc
static_assert(128 * kRegsProducer + 256 * kRegsSoftmax <= kThreads * 168,
              "register split exceeds the launch allocation");
constexpr int kRegsProducerQ8 = 72;  // warps 0-3 of the 8-bit variant
constexpr int kRegsConverter = 56;   // warps 12-15 of the 8-bit variant
constexpr int kRegsSoftmaxQ8 = 192;  // warps 4-11 of the 8-bit variant
static_assert(128 * (kRegsProducerQ8 + kRegsConverter) + 256 * kRegsSoftmaxQ8 <=
                  kThreadsQ8 * 128,
              "register split of the 8-bit variant exceeds the launch allocation");
constexpr int kTileM = 128;     // rows per Q tile
constexpr int kTileN = 128;     // keys per K/V tile
// The running row max is only recomputed when a tile's probabilities, taken
// against the stale max, sum to 2^63 or more (a score grew by more than ~56
// in log2 units).  Any reference value gives the same O = sum p v / sum p;
// this bound only keeps p, l and O far from fp32 overflow.
constexpr float kSpecLimit = 9.223372036854775808e18f;  // 2^63


template <int D>
struct Cfg {
  static constexpr int kHalves = D / 64;               // 128-byte column blocks
  static constexpr int kHalfBytes = kTileM * 128;      // one 64-column block of a tile
  static constexpr int kTileBytes = kHalves * kHalfBytes;
  static constexpr int kStages = D == 128 ? 4 : 8;
  static constexpr uint32_t kColS0 = 0, kColS1 = 128, kColO0 = 256, kColO1 = 256 + D;
  static constexpr uint32_t kIdescQK = idesc_bf16_f32(kTileM, kTileN, false, false);
  static constexpr uint32_t kIdescPV = idesc_bf16_f32(kTileM, D, false, true);
};

struct Geom {
  int32_t batch, Hq, Hkv, G, ps, ps_shift, num_pages, max_blocks, layer, total_new;
  float scale_log2;
  // decode mode: one new token per request, context lengths in seq_lens,
  // each request's keys cut into ranges of split_tiles K/V tiles; a request
  // with several ranges writes fp32 partials (O, max, sum) to ws
  int32_t decode, split_tiles, max_splits;
  const int32_t* seq_lens;
  float* ws;
  // pages read from an 8-bit image (the cache tier's layout): q8_table[b][j]
  // >= 0 names the image block holding page j of request b
  const uint8_t* q8_image;
  const int32_t* q8_table;
  int32_t q8_n_blocks, q8_layer_major, L;
  uint32_t q8_hdr, q8_chunk;  // scale header and whole chunk (one block, layer, plane), bytes
};

struct Barriers {
  uint64_t q_full, q_empty, vfix, drain;
  uint64_t kv_full[8], kv_empty[8];
  uint64_t s_full[2], p_full[2], pv_done[2];
  uint64_t item_full[2], item_empty[2];  // work-item ring, producer -> other roles
  int item_slot[2];
  uint32_t tmem_base;
  int abort_flag;
  int p0_steps;  // P tiles tile 0's softmax has published so far (pacing hint)
};

// Consumers of the work-item ring: the two MMA issuer threads and one
// elected thread per softmax warp.
constexpr int kItemConsumers = 2 + 2 * kTileM / 32;

// A work item and the quantities every role derives from it.
struct Item {
  int b, g, P, n, cu, T;
  int tok0[2], nt_i[2], nt;
  bool valid[2];
  int j0;             // first K/V tile (key range start / kTileN)
  int split, nsplit;  // key range of the item and ranges of its request
};

// item_start[p] = first item of the p-th request in work order; the request
// itself is order[p] when the batch was sorted (order != nullptr), else p.
__device__ __forceinline__ bool decode_item(int it, const int* item_start, const Geom& geo,
                                            const int32_t* __restrict__ prefix_lens,
                                            const int32_t* __restrict__ new_lens,
                                            const int32_t* __restrict__ cu_new_lens, Item& w) {
  int lo = 0, hi = geo.batch;  // last b with item_start[b] <= it
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (item_start[mid] <= it) lo = mid; else hi = mid;
  }
  const int b = geo.batch <= kSortMax ? static_cast<int>(
                    reinterpret_cast<const int16_t*>(item_start + geo.batch + 1)[lo])
                                       : lo;
  w.b = b;
  const int local = it - item_start[lo];
  if (geo.decode) {
    // (request, kv head, key range): one Q tile of G rows, tiles [j0, end)
    w.g = local % geo.Hkv;
    w.split = local / geo.Hkv;
    w.T = __ldg(geo.seq_lens + b);
    w.P = w.T - 1;
    w.n = 1;
    w.cu = b;
    const int nt_full = (w.T + kTileN - 1) / kTileN;
    w.nsplit = (nt_full + geo.split_tiles - 1) / geo.split_tiles;
    w.j0 = w.split * geo.split_tiles;
    w.valid[0] = true;
    w.valid[1] = false;
    w.tok0[0] = w.tok0[1] = 0;
    w.nt_i[0] = min(w.j0 + geo.split_tiles, nt_full);
    w.nt_i[1] = 0;
    w.nt = w.nt_i[0];
    return true;
  }
  w.j0 = 0;
  w.split = 0;
  w.nsplit = 1;
  const int pairs = (item_start[lo + 1] - item_start[lo]) / geo.Hkv;
  const int pair = pairs - 1 - local / geo.Hkv;  // later rows (more keys) first
  w.g = local % geo.Hkv;
  w.P = __ldg(prefix_lens + b);
  w.n = __ldg(new_lens + b);
  w.cu = __ldg(cu_new_lens + b);
  w.T = w.P + w.n;
  const int rows = w.n * geo.G;
  w.nt = 0;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int r0 = pair * 2 * kTileM + i * kTileM;
    w.valid[i] = r0 < rows;
    w.tok0[i] = r0 / geo.G;
    const int r1 = min(r0 + kTileM - 1, rows - 1);
    const int kend = w.P + r1 / geo.G + 1;  // keys [0, kend) reach some row
    w.nt_i[i] = w.valid[i] ? (kend + kTileN - 1) / kTileN : 0;
    w.nt = max(w.nt, w.nt_i[i]);
  }
  return true;
}

// Work items are handed out dynamically: the producer warp claims the next
// one from the launch's counter and publishes it to the other roles through a
// 2-slot ring in shared memory; -1 ends the CTA's work.
__device__ __forceinline__ int claim_item(Barriers& bar, uint32_t k, int* work_counter,
                                          int total_items, volatile int* abortp, bool& ok) {
  const int s = k & 1;
  ok = mbar_wait(&bar.item_empty[s], ((k >> 1) & 1) ^ 1, abortp);
  int it = -1;
  if ((threadIdx.x & 31) == 0 && ok) {
    it = atomicAdd(work_counter, 1);
    if (it >= total_items) it = -1;
    bar.item_slot[s] = it;
    mbar_arrive(&bar.item_full[s]);
  }
  return __shfl_sync(0xffffffffu, it, 0);
}

// Read item k of the ring (all consumer threads); the caller releases the
// slot with one arrival per consumer (see kItemConsumers).
__device__ __forceinline__ int read_item(Barriers& bar, uint32_t k, volatile int* abortp,
                                         bool& ok) {
  ok = mbar_wait(&bar.item_full[k & 1], (k >> 1) & 1, abortp);
  return ok ? *reinterpret_cast<volatile int*>(&bar.item_slot[k & 1]) : -1;
}

// ------------------------------------------------- pages of the 8-bit image
// With an 8-bit image (the cache tier's layout, one fp32 scale per (block,
// layer, plane, kv head)), pages that the q8 table maps to the image reach
// the ring in two stages.  The producer loads a page's ps*d codes (one box of
// a 3-D tensor map over the image's d-byte code rows) into
// the page's own rows of the ring slot (d = 128: code row r in the first
// 128 bytes of tile row r; d = 64: code row k at byte ps*64 + 64k of the
// page's rows) and looks the page's scale up one tile ahead; the converter
// warpgroup (warps 12-15) then turns the codes into bf16 in place, with
// the rounding of the 8-bit restore (bf16_rne(c * s)), at the positions the
// tensor map's 128-byte swizzle gives pool pages, and adds its arrivals to
// the slot's full barrier.  The pool is never written.
constexpr int kConvWarps = 4;
constexpr int kMaxPages = kTileN / 16;  // pages per K/V tile (ps >= 16)

struct Q8State {
  uint64_t codes_full[8];    // per ring slot: the codes have landed (tx bytes)
  uint32_t mask[8];          // per slot: bit p = page p of the tile is an image page
  int32_t rows_end[8];       // per slot: rows below this are keys; -1 ends the work
  float scale[8][kMaxPages];  // per slot and page
};

__device__ __forceinline__ uint64_t q8_chunk_index(const Geom& geo, int blk, int kv) {
  const uint64_t il = geo.q8_layer_major
                          ? static_cast<uint64_t>(geo.layer) * geo.q8_n_blocks + blk
                          : static_cast<uint64_t>(blk) * geo.L + geo.layer;
  return il * 2 + kv;
}

// Converter warp c of the warpgroup.  d = 128: tile rows [32c, 32c+32), in
// batches of 16 rows (a batch lies in one page).  Each batch is read whole
// (code row r sits under output row r's first 128 bytes) before any of it
// is written.  d = 64: pages p = c, c+4, ..., each in ascending batches of
// 16 rows; a batch's output rows only cover code rows of this or earlier
// batches of the same page, which are already in registers or converted.
// Rows at or past rows_end (V rows past the sequence end) are written as
// zeros: their probabilities are zero, and 0 * NaN would poison the product.
template <int D>
__device__ __forceinline__ void convert_batch(uint8_t* tile, const uint8_t* codes, int r0,
                                              int code_row0, float sc, int rows_end, int lane) {
  using C = Cfg<D>;
  constexpr int kWords = D / 16;        // 16-byte words of codes per row
  constexpr int kLanesPerRow = kWords;  // one word per lane and row
  constexpr int kRowsPerPass = 32 / kLanesPerRow;
  constexpr int kPasses = 16 / kRowsPerPass;  // 16 rows per batch
  const int u = lane % kLanesPerRow;
  uint4 v[kPasses];
#pragma unroll
  for (int q = 0; q < kPasses; ++q) {
    const int k = q * kRowsPerPass + lane / kLanesPerRow;  // row of the batch
    v[q] = r0 + k < rows_end
               ? *reinterpret_cast<const uint4*>(codes + (code_row0 + k) * D + u * 16)
               : make_uint4(0, 0, 0, 0);
  }
  __syncwarp();
#pragma unroll
  for (int q = 0; q < kPasses; ++q) {
    const int r = r0 + q * kRowsPerPass + lane / kLanesPerRow;
    uint4 lo = make_uint4(0, 0, 0, 0), hi = lo;
    if (r < rows_end) q8_dequant16(v[q], sc, lo, hi);
    const int h = u >> 2, q0 = (u & 3) * 2, sw = r & 7;
    uint8_t* row = tile + h * C::kHalfBytes + r * 128;
    // at d = 128 the two halves store their chunk pairs in opposite order, so
    // the 8 lanes of a row hit 8 distinct bank groups in each store
    if (h == 0) {
      *reinterpret_cast<uint4*>(row + ((q0 ^ sw) << 4)) = lo;
      *reinterpret_cast<uint4*>(row + (((q0 + 1) ^ sw) << 4)) = hi;
    } else {
      *reinterpret_cast<uint4*>(row + (((q0 + 1) ^ sw) << 4)) = hi;
      *reinterpret_cast<uint4*>(row + ((q0 ^ sw) << 4)) = lo;
    }
  }
  __syncwarp();
}

template <int D>
__device__ void converter(uint8_t* smem_kv, Barriers& bar, Q8State& q8, const Geom& geo) {
  using C = Cfg<D>;
  const int lane = threadIdx.x & 31;
  const int c = (threadIdx.x >> 5) - kThreads / 32;
  volatile int* abortp = &bar.abort_flag;
  for (uint32_t step = 0;; ++step) {
    const int slot = step % C::kStages;
    bool ok = mbar_wait(&q8.codes_full[slot], (step / C::kStages) & 1, abortp);
    if (!__all_sync(0xffffffffu, ok)) break;
    const int rows_end = *reinterpret_cast<volatile int32_t*>(&q8.rows_end[slot]);
    if (rows_end < 0) break;
    const uint32_t mask = *reinterpret_cast<volatile uint32_t*>(&q8.mask[slot]);
    uint8_t* tile = smem_kv + slot * C::kTileBytes;
    if (D == 128) {
#pragma unroll 1
      for (int a = 32 * c; a < 32 * c + 32; a += 16) {
        const int p = a >> geo.ps_shift;
        if ((mask >> p) & 1u) convert_batch<D>(tile, tile, a, a, q8.scale[slot][p], rows_end, lane);
      }
    } else {
#pragma unroll 1
      for (int p = c; p < (kTileN >> geo.ps_shift); p += kConvWarps) {
        if (!((mask >> p) & 1u)) continue;
        const int r0 = p << geo.ps_shift;
        const uint8_t* codes = tile + r0 * 128 + geo.ps * 64;
#pragma unroll 1
        for (int a = 0; a < geo.ps; a += 16)
          convert_batch<D>(tile, codes, r0 + a, a, q8.scale[slot][p], rows_end, lane);
      }
    }
    // the tensor core reads the slot through the async proxy
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(&bar.kv_full[slot]);
  }
}

// ------------------------------------------------------------------ roles
template <int D, bool kQ8>
__device__ void producer(uint8_t* smem_q, uint8_t* smem_kv, Barriers& bar, Q8State* q8,
                         const int* item_start, int total_items, const Geom& geo,
                         const CUtensorMap* map_q, const CUtensorMap* map_kv,
                         const CUtensorMap* map_q8,
                         const int32_t* __restrict__ block_table,
                         const int32_t* __restrict__ prefix_lens,
                         const int32_t* __restrict__ new_lens,
                         const int32_t* __restrict__ cu_new_lens, int32_t* status,
                         int* work_counter) {
  using C = Cfg<D>;
  const int lane = threadIdx.x & 31;
  volatile int* abortp = &bar.abort_flag;
  uint32_t q_count = 0, kv_count = 0, vfix_count = 0;
  uint32_t armed = 0, armed_par = 0;  // per slot: a load in flight, and its phase parity
  uint32_t armed8 = 0, armed8_par = 0;  // the same for the code copies of image pages
  int armed_q = -1, armed_vfix = -1;
  bool ok = true;
  const uint32_t box_bytes = static_cast<uint32_t>(geo.ps) * 128;  // one page, one column block
  const uint32_t page_codes = static_cast<uint32_t>(geo.ps) * D;   // one page of 8-bit codes

  for (uint32_t k = 0; ok; ++k) {
    const int it = claim_item(bar, k, work_counter, total_items, abortp, ok);
    if (!ok || it < 0) break;
    Item w;
    decode_item(it, item_start, geo, prefix_lens, new_lens, cu_new_lens, w);
    // ---- Q tiles
    ok = mbar_wait(&bar.q_empty, (q_count & 1) ^ 1, abortp);
    if (!ok) break;
    if (lane == 0) {
      uint32_t bytes = 0;
#pragma unroll
      for (int i = 0; i < 2; ++i)
        if (w.valid[i]) bytes += C::kTileBytes;
      mbar_arrive_expect_tx(&bar.q_full, bytes);
#pragma unroll
      for (int i = 0; i < 2; ++i)
        if (w.valid[i])
#pragma unroll
          for (int h = 0; h < C::kHalves; ++h)
            tma_load_3d(smem_q + i * C::kTileBytes + h * C::kHalfBytes, map_q, &bar.q_full, h * 64,
                        w.g * geo.G, w.cu + w.tok0[i]);
    }
    armed_q = q_count & 1;
    ++q_count;
    // ---- K/V tiles, page by page.  The copies of a tile are issued by
    // several lanes at once (lane = page * halves + half): one thread issuing
    // every box of a 16-row-page tile could not keep up with the MMAs.
    const int64_t bt_row = static_cast<int64_t>(w.b) * geo.max_blocks;
    const int pg = lane / C::kHalves, hh = lane % C::kHalves;
    // lane p (< pages of the tile) looks up page p of a tile in two stages:
    // its block-table (and q8-table) entries are loaded two tiles ahead, an
    // image page's K and V scales one tile ahead, so no load is waited for
    // while the current tile's copies are issued
    struct Raw {
      int page;  // block-table entry, -1 past max_blocks, -2 no page in this lane
      int ib;    // q8-table entry, or -1
    };
    struct Lookup {
      int page;        // pool page, -1 none (or bad), -2 no page in this lane
      int blk;         // image block, -1 none, -2 out of range
      float sk, sv;    // the image page's scales
    };
    auto load_raw = [&](int j) -> Raw {
      Raw r{-2, -1};
      const int key0 = j * kTileN;
      const int nkeys = min(kTileN, w.T - key0);
      const int npages = (nkeys + geo.ps - 1) >> geo.ps_shift;
      const int blk0 = key0 >> geo.ps_shift;
      if (j < w.nt && lane < npages) {
        const bool in = blk0 + lane < geo.max_blocks;
        r.page = in ? __ldg(block_table + bt_row + blk0 + lane) : -1;
        if (kQ8 && in) r.ib = __ldg(geo.q8_table + bt_row + blk0 + lane);
      }
      return r;
    };
    auto resolve = [&](const Raw& r) -> Lookup {
      Lookup l{r.page, -1, 0.f, 0.f};
      if (kQ8 && r.ib >= 0) {
        l.page = -2;
        if (r.ib >= geo.q8_n_blocks) {
          l.page = -1;
          l.blk = -2;  // reported when the tile is issued
        } else {
          l.blk = r.ib;
          const uint8_t* ck = geo.q8_image + q8_chunk_index(geo, r.ib, 0) * geo.q8_chunk;
          l.sk = __ldg(reinterpret_cast<const float*>(ck) + w.g);
          l.sv = __ldg(reinterpret_cast<const float*>(ck + geo.q8_chunk) + w.g);
        }
      }
      return l;
    };
    Lookup next = resolve(load_raw(w.j0));
    Raw raw2 = load_raw(w.j0 + 1);
    for (int j = w.j0; ok && j < w.nt; ++j) {
      const int key0 = j * kTileN;
      const int nkeys = min(kTileN, w.T - key0);
      Lookup cur = next;
      next = resolve(raw2);
      raw2 = load_raw(j + 2);
      int page = cur.page;
      if (cur.blk == -2 || (page != -2 && cur.blk < 0 && (page < 0 || page >= geo.num_pages))) {
        record_error(status, GC_ERR_OUT_OF_RANGE);
        page = -1;
        cur.blk = -1;
      }
      if (page == -2) page = -1;
      const int good = __popc(__ballot_sync(0xffffffffu, page >= 0));
      const uint32_t img_mask = kQ8 ? __ballot_sync(0xffffffffu, cur.blk >= 0) : 0u;
      const int my_page = __shfl_sync(0xffffffffu, page, pg < 32 ? pg : 0);
      const bool issues = pg < kTileN / 16 && my_page >= 0;
#pragma unroll 1
      for (int kv = 0; kv < 2; ++kv) {
        const int slot = kv_count % C::kStages;
        ok = mbar_wait(&bar.kv_empty[slot], ((kv_count / C::kStages) & 1) ^ 1, abortp);
        if (!ok) break;
        uint8_t* dst = smem_kv + slot * C::kTileBytes;
        const bool fix = kv == 1 && nkeys < kTileN;
        uint64_t* full = fix ? &bar.vfix : &bar.kv_full[slot];
        if (kQ8) {
          // codes of the image pages, converted by the converter warpgroup
          if (cur.blk >= 0) q8->scale[slot][lane] = kv ? cur.sv : cur.sk;
          __syncwarp();
          if (lane == 0) {
            q8->mask[slot] = img_mask;
            q8->rows_end[slot] = fix ? nkeys : kTileN;
            mbar_arrive_expect_tx(&q8->codes_full[slot], __popc(img_mask) * page_codes);
          }
          __syncwarp();
          if (cur.blk >= 0) {
            // rows [g*ps, (g+1)*ps) of the chunk's code rows (d bytes each)
            uint8_t* cdst = dst + lane * box_bytes + (D == 128 ? 0 : geo.ps * 64);
            tma_load_3d(cdst, map_q8, &q8->codes_full[slot], 0, w.g * geo.ps,
                        static_cast<int32_t>(q8_chunk_index(geo, cur.blk, kv)));
          }
          armed8 |= 1u << slot;
          armed8_par = (armed8_par & ~(1u << slot)) | (((kv_count / C::kStages) & 1u) << slot);
        }
        if (lane == 0)
          mbar_arrive_expect_tx(full, static_cast<uint32_t>(good) * box_bytes * C::kHalves);
        __syncwarp();
        if (issues) {
          const int plane_row = (geo.layer * 2 + kv) * geo.num_pages;
          const int row = (((plane_row + my_page) * geo.Hkv + w.g) << geo.ps_shift);
          tma_load_2d(dst + hh * C::kHalfBytes + pg * box_bytes, map_kv, full, hh * 64, row);
        }
        if (fix) {
          // V rows past the end of the sequence must be zero, not stale or NaN:
          // their P is zero but 0 * NaN would poison the PV product.  Rows of
          // image pages are zeroed by the converters (they hold codes here).
          ok = mbar_wait(&bar.vfix, vfix_count & 1, abortp);
          if (!ok) {
            armed &= ~(1u << slot);
            armed_vfix = vfix_count & 1;
            break;
          }
          ++vfix_count;
          const int zrows = kTileN - nkeys;
          for (int h = 0; h < C::kHalves; ++h) {
            uint4* z = reinterpret_cast<uint4*>(dst + h * C::kHalfBytes + nkeys * 128);
            for (int k = lane; k < zrows * 8; k += 32)
              if (!kQ8 || !((img_mask >> ((nkeys + (k >> 3)) >> geo.ps_shift)) & 1u))
                z[k] = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar.kv_full[slot]);
        } else {
          armed |= 1u << slot;
          armed_par = (armed_par & ~(1u << slot)) | (((kv_count / C::kStages) & 1u) << slot);
        }
        ++kv_count;
      }
    }
  }
  if (kQ8 && ok) {
    // tell the converters that the work is done (the slot's previous
    // conversion has been consumed once the slot is free again)
    const int slot = kv_count % C::kStages;
    ok = mbar_wait(&bar.kv_empty[slot], ((kv_count / C::kStages) & 1) ^ 1, abortp);
    if (ok && lane == 0) {
      q8->rows_end[slot] = -1;
      mbar_arrive(&q8->codes_full[slot]);
    }
  }
  if (!ok && lane == 0) {
    // drain copies still in flight before the CTA exits (bounded, ignores abort)
    int no_abort = 0;
    if (armed_q >= 0) mbar_wait(&bar.q_full, armed_q, &no_abort);
    if (armed_vfix >= 0) mbar_wait(&bar.vfix, armed_vfix, &no_abort);
    for (int s = 0; s < C::kStages; ++s) {
      if (armed & (1u << s)) mbar_wait(&bar.kv_full[s], (armed_par >> s) & 1u, &no_abort);
      if (kQ8 && (armed8 & (1u << s)))
        mbar_wait(&q8->codes_full[s], (armed8_par >> s) & 1u, &no_abort);
    }
  }
}

// The MMA issuer of Q tile i (one thread).  Each tile's products are a
// strict chain (P_i aliases S_i, so S_i(j+1) waits for PV_i(j) to complete),
// so the issuer waits for each input in order; the two tiles have separate
// issuer threads, so one tile's waits never delay the other tile's MMAs and
// the tensor pipe interleaves the two chains.
template <int D>
__device__ void mma_issuer(int i, uint8_t* smem_q, uint8_t* smem_kv, Barriers& bar, uint32_t tmem,
                           const int* item_start, int total_items, const Geom& geo,
                           const int32_t* __restrict__ prefix_lens,
                           const int32_t* __restrict__ new_lens,
                           const int32_t* __restrict__ cu_new_lens) {
  using C = Cfg<D>;
  volatile int* abortp = &bar.abort_flag;
  uint32_t q_count = 0, kv_count = 0, s_issued = 0, pv_issued = 0;
  bool ok = true;
  const uint32_t q_addr = smem_addr(smem_q) + i * C::kTileBytes, kv_smem = smem_addr(smem_kv);
  const uint32_t col_s = i ? C::kColS1 : C::kColS0;
  const uint32_t col_o = i ? C::kColO1 : C::kColO0;

  int p0_base = 0;  // tile-0 steps of earlier items
  for (uint32_t k = 0; ok; ++k) {
    const int it = read_item(bar, k, abortp, ok);
    if (!ok) break;
    mbar_arrive(&bar.item_empty[k & 1]);
    if (it < 0) break;
    Item w;
    decode_item(it, item_start, geo, prefix_lens, new_lens, cu_new_lens, w);
    // K_j sits in ring use kv_base + 2j, V_j in use kv_base + 2j + 1
    const uint32_t kv_base = kv_count;
    kv_count += 2 * (w.nt - w.j0);
    const int p0_item = p0_base;
    p0_base += w.nt_i[0] - w.j0;
    const uint32_t q_par = q_count & 1;
    ++q_count;
    if (!w.valid[i]) continue;
    ok = mbar_wait(&bar.q_full, q_par, abortp);
    if (!ok) break;
    tc_fence_after();
    for (int j = w.j0; j < w.nt_i[i]; ++j) {
      // S_i = Q_i K_j^T once K_j is in and PV_i(j-1) has finished reading P_i
      const uint32_t ku = kv_base + 2 * (j - w.j0);
      ok = mbar_wait(&bar.kv_full[ku % C::kStages], (ku / C::kStages) & 1, abortp);
      if (ok && pv_issued > 0) ok = mbar_wait(&bar.pv_done[i], (pv_issued - 1) & 1, abortp);
      if (ok && i == 1 && j < w.nt_i[0]) {
        // pacing: tile 1's S(j) follows tile 0's softmax of step j, so the two
        // tiles' softmax phases alternate instead of sharing the MUFU and
        // their MMAs fill each other's softmax time
        const volatile int* p0 = &bar.p0_steps;
        const long long t0 = clock64();
        while (*p0 < p0_item + (j - w.j0) + 1) {
          if (*abortp || clock64() - t0 > kWaitCycles) {
            *abortp = 1;
            ok = false;
            break;
          }
        }
      }
      if (!ok) break;
      tc_fence_after();
      const uint32_t k_addr = kv_smem + (ku % C::kStages) * C::kTileBytes;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = (kk >> 2) * C::kHalfBytes + (kk & 3) * 32;
        mma_ss(tmem + col_s, sdesc_sw128(q_addr + off, 16, 1024),
               sdesc_sw128(k_addr + off, 16, 1024), C::kIdescQK, kk > 0);
      }
      mma_commit(&bar.s_full[i]);
      ++s_issued;
      // O_i += P_i V_j once the softmax has written P_i(j) and V_j is in
      const uint32_t vu = ku + 1;
      ok = mbar_wait(&bar.p_full[i], (s_issued - 1) & 1, abortp);
      if (ok) ok = mbar_wait(&bar.kv_full[vu % C::kStages], (vu / C::kStages) & 1, abortp);
      if (!ok) break;
      tc_fence_after();
      const uint32_t v_addr = kv_smem + (vu % C::kStages) * C::kTileBytes;
#pragma unroll
      for (int kk = 0; kk < kTileN / 16; ++kk)
        mma_ts(tmem + col_o, tmem + col_s + kk * 8,
               sdesc_sw128(v_addr + kk * 16 * 128, C::kHalfBytes, 1024), C::kIdescPV,
               (j > w.j0 || kk > 0) ? 1u : 0u);
      mma_commit(&bar.pv_done[i]);
      ++pv_issued;
    }
  }
  // wait for every MMA this thread issued before TMEM is released
  mma_commit(&bar.drain);
  int no_abort = 0;
  mbar_wait(&bar.drain, 0, &no_abort);
}

// Row max of a 128-column score tile (raw scores, masked columns -inf).
__device__ __forceinline__ float tile_max(const uint32_t (&sr)[4][32]) {
  float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int c = 0; c < 4; ++c)
#pragma unroll
    for (int e = 0; e < 32; e += 8) {
      mx[0] = fmax3(mx[0], __uint_as_float(sr[c][e + 0]), __uint_as_float(sr[c][e + 1]));
      mx[1] = fmax3(mx[1], __uint_as_float(sr[c][e + 2]), __uint_as_float(sr[c][e + 3]));
      mx[2] = fmax3(mx[2], __uint_as_float(sr[c][e + 4]), __uint_as_float(sr[c][e + 5]));
      mx[3] = fmax3(mx[3], __uint_as_float(sr[c][e + 6]), __uint_as_float(sr[c][e + 7]));
    }
  return fmax3(mx[0], mx[1], fmaxf(mx[2], mx[3]));
}

// p = 2^(s * scale*log2(e) - m) for one row of the tile, written to TMEM at
// tS as bf16 pairs (the A operand of the PV product); returns sum p (fp32).
__device__ __forceinline__ float tile_exp(const uint32_t (&sr)[4][32], uint32_t tS,
                                          float scale_log2, float m) {
  const uint64_t sc2 = f2_pack(scale_log2, scale_log2);
  const uint64_t nm2 = f2_pack(-m, -m);
  uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    uint32_t pk[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      const uint64_t t = f2_fma(f2_pack(__uint_as_float(sr[c][2 * e]),
                                        __uint_as_float(sr[c][2 * e + 1])), sc2, nm2);
      float t0, t1;
      f2_unpack(t, t0, t1);
      const float p0 = ex2_approx(t0), p1 = ex2_approx(t1);
      acc[e & 3] = f2_add(acc[e & 3], f2_pack(p0, p1));
      pk[e] = pack_bf16x2(p0, p1);
    }
    tmem_st16(tS + c * 16, pk);
  }
  float s0, s1, s2, s3;
  f2_unpack(f2_add(acc[0], acc[1]), s0, s1);
  f2_unpack(f2_add(acc[2], acc[3]), s2, s3);
  return (s0 + s2) + (s1 + s3);
}

// O row *= alpha in TMEM (D fp32 columns at tO).
template <int D>
__device__ __forceinline__ void rescale_o(uint32_t tO, float alpha) {
#pragma unroll 1
  for (int c = 0; c < D / 32; ++c) {
    uint32_t o[32];
    tmem_ld32(tO + c * 32, o);
    tmem_wait_ld();
#pragma unroll
    for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
    tmem_st32(tO + c * 32, o);
  }
}

// Make this warp's P writes visible to the MMA issuer: every thread waits
// for its TMEM stores and fences, then one elected thread arrives for the
// warp (one arrival per warp: per-thread arrivals on a single barrier are
// serialised and cost more than the softmax itself).
__device__ __forceinline__ void publish_p(uint64_t* bar) {
  tmem_wait_st();
  tc_fence_before();
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

template <int D, int i>
__device__ void softmax_wg(Barriers& bar, uint32_t tmem, const int* item_start,
                           int total_items, const Geom& geo,
                           const int32_t* __restrict__ prefix_lens,
                           const int32_t* __restrict__ new_lens,
                           const int32_t* __restrict__ cu_new_lens,
                           __nv_bfloat16* __restrict__ out) {
  using C = Cfg<D>;
  volatile int* abortp = &bar.abort_flag;
  const int warp = threadIdx.x >> 5;
  const int r = threadIdx.x - kTileM * (1 + i);               // row of the Q tile (= TMEM lane)
  const uint32_t lane_addr = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
  const uint32_t tS = lane_addr + (i ? C::kColS1 : C::kColS0);
  const uint32_t tO = lane_addr + (i ? C::kColO1 : C::kColO0);
  uint32_t s_count = 0, pv_total = 0, kv_count = 0;
  int p0_published = 0;
  bool ok = true;

  for (uint32_t k = 0; ok; ++k) {
    const int it = read_item(bar, k, abortp, ok);
    if (!ok) break;
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(&bar.item_empty[k & 1]);
    if (it < 0) break;
    Item w;
    decode_item(it, item_start, geo, prefix_lens, new_lens, cu_new_lens, w);
    // K_j sits in ring use kv_base + 2j, V_j in use kv_base + 2j + 1
    const uint32_t kv_base = kv_count;
    kv_count += 2 * (w.nt - w.j0);
    if (!w.valid[i]) continue;
    // This tile releases the ring slots (and the Q tiles) once the MMAs that
    // read them are known complete; for K/V tiles (or Q) the other tile does
    // not use, it arrives on that tile's behalf too.
    const bool rel = threadIdx.x == kTileM * (1 + i);
    const int nt_o = w.valid[1 - i] ? w.nt_i[1 - i] : 0;
    auto release = [&](int j, int kv) {
      const uint32_t use = kv_base + 2 * (j - w.j0) + kv;
      mbar_arrive_cnt(&bar.kv_empty[use % C::kStages], j < nt_o ? 1u : 2u);
    };
    const int tok = w.tok0[i] + r / geo.G;
    const bool row_valid = tok < w.n;
    const int kmax = row_valid ? w.P + tok : w.T - 1;  // last visible key
    float m_run = -INFINITY, l = 0.f;
    for (int j = w.j0; j < w.nt_i[i]; ++j) {
      ok = mbar_wait(&bar.s_full[i], s_count & 1, abortp);
      ++s_count;
      if (!ok) break;
      if (rel) {
        // S_i(j) is complete: K_j is done with for this tile; and S_i(j) was
        // issued after PV_i(j-1) completed, so V_{j-1} is too
        release(j, 0);
        if (j > w.j0) release(j - 1, 1);
        if (j == w.nt_i[i] - 1) mbar_arrive_cnt(&bar.q_empty, w.valid[1 - i] ? 1u : 2u);
      }
      tc_fence_after();
      uint32_t sr[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(tS + c * 32, sr[c]);
      tmem_wait_ld();
      const int key0 = j * kTileN;
      if (key0 + kTileN - 1 > kmax) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (key0 + c * 32 + e > kmax) sr[c][e] = __float_as_uint(-INFINITY);
      }
      const float sl2 = geo.scale_log2;
      float lt;
      if (m_run == -INFINITY) {
        // first tile of the row: exact max (key 0 is always visible)
        m_run = tile_max(sr) * sl2;
        lt = tile_exp(sr, tS, sl2, m_run);
      } else {
        // later tiles keep the running max unless the tile would overflow
        lt = tile_exp(sr, tS, sl2, m_run);
        if (__any_sync(0xffffffffu, !(lt < kSpecLimit))) {
          // O is complete up to tile j-1: S_i(j) was issued after PV_i(j-1)
          tmem_wait_st();
          const float m_new = fmaxf(m_run, tile_max(sr) * sl2);
          const float alpha = m_new > m_run ? ex2_approx(m_run - m_new) : 1.f;
          rescale_o<D>(tO, alpha);
          l *= alpha;
          m_run = m_new;
          lt = tile_exp(sr, tS, sl2, m_run);
        }
      }
      l += lt;
      publish_p(&bar.p_full[i]);
      if (i == 0 && rel) *reinterpret_cast<volatile int*>(&bar.p0_steps) = ++p0_published;
    }
    if (!ok) break;
    // ---- epilogue: O / l -> bf16
    pv_total += w.nt_i[i] - w.j0;
    ok = mbar_wait(&bar.pv_done[i], (pv_total - 1) & 1, abortp);
    if (!ok) break;
    if (rel) release(w.nt_i[i] - 1, 1);
    tc_fence_after();
    const int h = w.g * geo.G + r % geo.G;
    if (w.nsplit > 1) {
      // one key range of a split request: fp32 partials O (unnormalised),
      // reference max (log2 units) and sum, merged by a second kernel
      const int64_t head = static_cast<int64_t>(w.b) * geo.Hq + h;
      float* o_ws = geo.ws + (head * geo.max_splits + w.split) * D;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_wait_ld();
        if (row_valid) {
#pragma unroll
          for (int v = 0; v < 8; ++v)
            reinterpret_cast<uint4*>(o_ws + c * 32)[v] =
                make_uint4(o[4 * v], o[4 * v + 1], o[4 * v + 2], o[4 * v + 3]);
        }
      }
      if (row_valid) {
        float* ml = geo.ws + static_cast<int64_t>(geo.batch) * geo.Hq * geo.max_splits * D +
                    (head * geo.max_splits + w.split) * 2;
        ml[0] = m_run;
        ml[1] = l;
      }
      tc_fence_before();
      continue;
    }
    const float inv_l = 1.f / l;
    uint4* orow = reinterpret_cast<uint4*>(
        out + (static_cast<int64_t>(w.cu + tok) * geo.Hq + h) * D);
#pragma unroll 1
    for (int c = 0; c < D / 32; ++c) {
      uint32_t o[32];
      tmem_ld32(tO + c * 32, o);
      tmem_wait_ld();
      if (row_valid) {
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          uint4 pk;
          pk.x = pack_bf16x2(__uint_as_float(o[8 * v + 0]) * inv_l, __uint_as_float(o[8 * v + 1]) * inv_l);
          pk.y = pack_bf16x2(__uint_as_float(o[8 * v + 2]) * inv_l, __uint_as_float(o[8 * v + 3]) * inv_l);
          pk.z = pack_bf16x2(__uint_as_float(o[8 * v + 4]) * inv_l, __uint_as_float(o[8 * v + 5]) * inv_l);
          pk.w = pack_bf16x2(__uint_as_float(o[8 * v + 6]) * inv_l, __uint_as_float(o[8 * v + 7]) * inv_l);
          orow[c * 4 + v] = pk;
        }
      }
    }
    tc_fence_before();
  }
}

template <int D, bool kQ8>
__global__ void __launch_bounds__(kQ8 ? kThreadsQ8 : kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                   const __grid_constant__ CUtensorMap map_kv,
                   const __grid_constant__ CUtensorMap map_q8,
                   const int32_t* __restrict__ block_table, const int32_t* __restrict__ prefix_lens,
                   const int32_t* __restrict__ new_lens, const int32_t* __restrict__ cu_new_lens,
                   __nv_bfloat16* __restrict__ out, Geom geo, int32_t* status,
                   int* work_counter) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* smem_q = base;
  uint8_t* smem_kv = base + 2 * C::kTileBytes;
  Barriers& bar = *reinterpret_cast<Barriers*>(smem_kv + C::kStages * C::kTileBytes);
  int* item_start = reinterpret_cast<int*>(&bar + 1);  // [batch + 1]
  int16_t* order = reinterpret_cast<int16_t*>(item_start + geo.batch + 1);  // [min(batch, kSortMax)]
  Q8State* q8 = kQ8 ? reinterpret_cast<Q8State*>(
                          (reinterpret_cast<uintptr_t>(order + kSortMax) + 7) & ~uintptr_t(7))
                    : nullptr;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&bar.q_full, 1);
    mbar_init(&bar.q_empty, 2);
    mbar_init(&bar.vfix, 1);
    mbar_init(&bar.drain, 2);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bar.kv_full[s], kQ8 ? 1 + kConvWarps : 1);  // + one arrival per converter warp
      mbar_init(&bar.kv_empty[s], 2);
      if (kQ8) mbar_init(&q8->codes_full[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bar.s_full[i], 1);
      mbar_init(&bar.p_full[i], kTileM / 32);
      mbar_init(&bar.pv_done[i], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bar.item_full[s], 1);
      mbar_init(&bar.item_empty[s], kItemConsumers);
    }
    bar.abort_flag = 0;
    bar.p0_steps = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&map_q);
    prefetch_tensormap(&map_kv);
    if (kQ8) prefetch_tensormap(&map_q8);
  }
  if (warp == 1) {
    tmem_alloc(&bar.tmem_base, 512);
    tmem_relinquish();
  }
  if (geo.batch <= kSortMax) {
    // rank requests by total length, longest first (ties by index)
    auto total_len = [&](int b) {
      return geo.decode ? __ldg(geo.seq_lens + b) : __ldg(prefix_lens + b) + __ldg(new_lens + b);
    };
    for (int b = threadIdx.x; b < geo.batch; b += blockDim.x) {
      const int tb = total_len(b);
      int rank = 0;
      for (int o = 0; o < geo.batch; ++o) {
        const int to = total_len(o);
        rank += (to > tb) || (to == tb && o < b);
      }
      order[rank] = static_cast<int16_t>(b);
    }
  }
  __syncthreads();
  if (warp == 2) {
    // work items per request: Hkv * ceil(n_b * G / 256); exclusive scan in work order
    int running = 0;
    for (int b0 = 0; b0 < geo.batch; b0 += 32) {
      const int p = b0 + lane;
      const int b = p < geo.batch ? (geo.batch <= kSortMax ? order[p] : p) : p;
      int cnt = 0;
      if (p < geo.batch && geo.decode) {
        // a context of T keys, cut into ranges of split_tiles K/V tiles
        const int T = __ldg(geo.seq_lens + b);
        if (T < 1 || T > (geo.max_blocks << geo.ps_shift)) {
          record_error(status, GC_ERR_OUT_OF_RANGE);
        } else {
          const int nt_full = (T + kTileN - 1) / kTileN;
          cnt = geo.Hkv * ((nt_full + geo.split_tiles - 1) / geo.split_tiles);
        }
      } else if (p < geo.batch) {
        const int n = __ldg(new_lens + b), P = __ldg(prefix_lens + b);
        const int cu = __ldg(cu_new_lens + b);
        const bool sane = n >= 0 && P >= 0 && cu >= 0 && cu + n <= geo.total_new;
        if (!sane && n != 0) record_error(status, GC_ERR_OUT_OF_RANGE);
        if (sane && n > 0) cnt = geo.Hkv * ((n * geo.G + 2 * kTileM - 1) / (2 * kTileM));
      }
      int incl = cnt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (p < geo.batch) item_start[p] = running + incl - cnt;
      running += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) item_start[geo.batch] = running;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar.tmem_base;
  const int total_items = item_start[geo.batch];

  if (warp < 4) {
    regs_dec<kQ8 ? kRegsProducerQ8 : kRegsProducer>();
    if (warp == 0) {
      producer<D, kQ8>(smem_q, smem_kv, bar, q8, item_start, total_items, geo, &map_q, &map_kv,
                       &map_q8, block_table, prefix_lens, new_lens, cu_new_lens, status, work_counter);
    } else if (warp == 1 || warp == 2) {
      if (lane == 0)
        mma_issuer<D>(warp - 1, smem_q, smem_kv, bar, tmem, item_start, total_items, geo,
                      prefix_lens, new_lens, cu_new_lens);
      __syncwarp();
    }
  } else if (kQ8 && warp >= kThreads / 32) {
    regs_dec<kRegsConverter>();
    converter<D>(smem_kv, bar, *q8, geo);
  } else {
    regs_inc<kQ8 ? kRegsSoftmaxQ8 : kRegsSoftmax>();
    if (warp < 8)
      softmax_wg<D, 0>(bar, tmem, item_start, total_items, geo, prefix_lens, new_lens,
                       cu_new_lens, out);
    else
      softmax_wg<D, 1>(bar, tmem, item_start, total_items, geo, prefix_lens, new_lens,
                       cu_new_lens, out);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if (threadIdx.x == 0 && bar.abort_flag) record_error(status, GC_ERR_TIMEOUT);
}

}  // namespace

// The work items of one call are numbered with 32-bit ints and handed out by
// a 32-bit counter that every CTA (or CTA pair) raises once more after the
// last item: the items, plus two claims per CTA of margin, must stay below
// 2^31, and so must the q rows of the batch (T_new * G), from which the
// kernel derives each request's item count.  Host-side bound, checked
// before anything is launched.
gc_status check_item_bound(const gc_kv_pool* pool, const AttnArgs& a, const DecodeMode* dm,
                           int grid) {
  const long long hkv = pool->cfg.num_kv_heads;
  const long long G = a.num_q_heads / hkv;
  const long long rows = static_cast<long long>(a.total_new_tokens) * G;
  long long items;
  if (dm) {
    // a request's keys (at most max_blocks * ps) cut into ranges of split_tiles tiles
    const long long tiles =
        (static_cast<long long>(a.max_blocks) * pool->cfg.page_size + kTileN - 1) / kTileN;
    const long long per_req = (tiles + dm->split_tiles - 1) / dm->split_tiles;
    items = hkv * a.batch * per_req;
  } else {
    // sum_b ceil(n_b * G / 256) <= T_new * G / 256 + batch
    items = hkv * (rows / (2 * kTileM) + a.batch);
  }
  const long long limit = 2147483647LL - 2LL * grid;
  if (rows + 2 * kTileM > 2147483647LL || items > limit)
    return fail(GC_ERR_UNSUPPORTED,
                "attention: up to %lld work items (%lld q rows) exceed what the 32-bit work "
                "counter can hand out (%lld)",
                items, rows, limit);
  return GC_OK;
}

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

template <int D>
gc_status launch(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream,
                 int* work_counter, const DecodeMode* dm = nullptr,
                 const Q8Pages* q8 = nullptr) {
  using C = Cfg<D>;
  gc_status bound = check_item_bound(pool, a, dm, pool->num_sms);
  if (bound != GC_OK) return bound;
  auto enc = encode_fn();
  if (!enc) return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: cuTensorMapEncodeTiled unavailable");
  const auto& cfg = pool->cfg;
  Geom geo;
  geo.batch = a.batch;
  geo.Hq = a.num_q_heads;
  geo.Hkv = cfg.num_kv_heads;
  geo.G = geo.Hq / geo.Hkv;
  geo.ps = cfg.page_size;
  int s = 0;
  while ((1 << s) < geo.ps) ++s;
  geo.ps_shift = s;
  geo.num_pages = cfg.num_pages;
  geo.max_blocks = a.max_blocks;
  geo.layer = a.layer;
  geo.total_new = a.total_new_tokens;
  geo.scale_log2 = a.softmax_scale * 1.4426950408889634f;
  geo.decode = dm != nullptr;
  geo.split_tiles = dm ? dm->split_tiles : 0;
  geo.max_splits = dm ? dm->max_splits : 0;
  geo.seq_lens = dm ? dm->seq_lens : nullptr;
  geo.ws = dm ? dm->ws : nullptr;
  geo.L = cfg.num_layers;
  geo.q8_image = q8 ? q8->image : nullptr;
  geo.q8_table = q8 ? q8->table : nullptr;
  geo.q8_n_blocks = q8 ? q8->n_blocks : 0;
  geo.q8_layer_major = q8 && q8->layer_major ? 1 : 0;
  // image chunk of one (block, layer, plane): Hkv fp32 scales padded to 16
  // bytes, then Hkv groups of ps*d codes
  geo.q8_hdr = static_cast<uint32_t>(q8_header_bytes(cfg));
  geo.q8_chunk = static_cast<uint32_t>(q8_chunk_bytes(cfg));

  const uint64_t pool_rows = static_cast<uint64_t>(cfg.num_layers) * 2 * cfg.num_pages *
                             cfg.num_kv_heads * cfg.page_size;
  if (pool_rows >= (1ull << 31))
    return fail(GC_ERR_UNSUPPORTED, "gc_prefix_prefill_attn: pool has %llu rows (limit 2^31)",
                static_cast<unsigned long long>(pool_rows));
  CUtensorMap map_q, map_kv;
  {
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(geo.Hq),
                          static_cast<cuuint64_t>(geo.total_new)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2,
                             static_cast<cuuint64_t>(geo.Hq) * D * 2};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(geo.G), static_cast<cuuint32_t>(kTileM / geo.G)};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = enc(&map_q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: q tensor map (CUresult %d)", (int)r);
  }
  {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(D), pool_rows};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(D) * 2};
    cuuint32_t box[2] = {64, static_cast<cuuint32_t>(geo.ps)};
    cuuint32_t es[2] = {1, 1};
    CUresult r = enc(&map_kv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pool->data, dims, strides, box,
                     es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: pool tensor map (CUresult %d)", (int)r);
  }
  // 8-bit image: its code rows (d bytes each; Hkv*ps rows per chunk after the
  // scale header) as a 3-D map, box = one page of one kv head
  CUtensorMap map_q8 = map_kv;  // unused by the bf16 kernel
  if (q8) {
    const uint64_t chunks = static_cast<uint64_t>(q8->n_blocks) * cfg.num_layers * 2;
    if (chunks >= (1ull << 31))
      return fail(GC_ERR_UNSUPPORTED, "gc_prefix_prefill_attn_q8: image of %llu chunks (limit 2^31)",
                  static_cast<unsigned long long>(chunks));
    // an empty image is never read; the map then points at the pool
    const void* base = chunks ? static_cast<const void*>(q8->image + geo.q8_hdr) : pool->data;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(D),
                          static_cast<cuuint64_t>(cfg.num_kv_heads) * cfg.page_size,
                          chunks ? chunks : 1};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(geo.q8_chunk)};
    cuuint32_t box[3] = {static_cast<cuuint32_t>(D), static_cast<cuuint32_t>(cfg.page_size), 1};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = enc(&map_q8, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void*>(base), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn_q8: image tensor map (CUresult %d)", (int)r);
  }
  const size_t smem = 1024 + 2 * C::kTileBytes + C::kStages * C::kTileBytes + sizeof(Barriers) +
                      (static_cast<size_t>(a.batch) + 1) * sizeof(int) +
                      kSortMax * sizeof(int16_t) + (q8 ? sizeof(Q8State) + 8 : 0);
  auto kernel = q8 ? attn_tc_kernel<D, true> : attn_tc_kernel<D, false>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn: smem attribute");
  // the work items are claimed from a counter in the pool's control block
  e = cudaMemsetAsync(work_counter, 0, sizeof(int), stream);
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn: clearing the work counter");
  kernel<<<pool->num_sms, q8 ? kThreadsQ8 : kThreads, smem, stream>>>(
      map_q, map_kv, map_q8, a.block_table, a.prefix_lens, a.new_lens, a.cu_new_lens,
      static_cast<__nv_bfloat16*>(a.out), geo, pool->status, work_counter);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn: launch");
  return GC_OK;
}

// head_dim 128 prefill runs on the CTA-pair kernel (attn_tc2.cu): measured
// faster than the single-SM kernel above on every layer shape (70B layer 1.50
// against 1.95 ms, Llama-3-8B layer 0.173 against 0.205 ms, the conversation
// mix and the long document alike).  The single-SM kernel serves head_dim
// 64, pages read from the 8-bit image and decode at head_dim 64.
gc_status launch_d128(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream,
                      int* work_counter) {
  return launch_attn_tc2(pool, a, stream, work_counter);
}

}  // namespace

gc_status launch_attn_tc(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream) {
  if (pool->cfg.head_dim == 128) return launch_d128(pool, a, stream, pool->work_counter);
  return launch<64>(pool, a, stream, pool->work_counter);
}

// Pages read from the 8-bit image run on the 16-warp variant of the
// single-SM kernel at either head size: its converter warpgroup dequantises
// them into the same shared-memory tiles the tensor map fills for pool pages.
gc_status launch_attn_tc_q8(const gc_kv_pool* pool, const AttnArgs& a, const Q8Pages& q8,
                            cudaStream_t stream) {
  if (pool->cfg.head_dim == 128) return launch<128>(pool, a, stream, pool->work_counter, nullptr, &q8);
  return launch<64>(pool, a, stream, pool->work_counter, nullptr, &q8);
}

gc_status launch_attn_tc_decode(const gc_kv_pool* pool, const AttnArgs& a, const DecodeMode& dm,
                                cudaStream_t stream, const Q8Pages* q8) {
  if (pool->cfg.head_dim == 128) return launch<128>(pool, a, stream, pool->work_counter, &dm, q8);
  return launch<64>(pool, a, stream, pool->work_counter, &dm, q8);
}

}  // namespace gc

// ------------------------------------------------------- allocation-free variant
// Scratch of gc_prefix_prefill_attn_noalloc: element 0 is the work-item
// counter the kernel's CTAs claim items from.  It lives in the library's own
// device memory, so that entry point needs no buffer from anyone; every GPU
// that loads the library keeps these 256 bytes until the process exits, and
// all calls share them.
static __device__ __align__(256) int32_t g_attn_noalloc_scratch[64];

namespace gc {
namespace {

constexpr int kMaxDevices = 64;

// Unique id of the calling thread's current CUDA context, 0 if there is none
// or the driver cannot say (the lookup below is then repeated on every call).
unsigned long long current_context_id() {
  static PFN_cuCtxGetCurrent_v4000 get_cur = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_cur = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_cur || !get_id || get_cur(&ctx) != CUDA_SUCCESS || !ctx) return 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of the static scratch on `device`, with that device
// current.  Host code cannot use the symbol itself (it only names a
// host-side stand-in), so the address is looked up with
// cudaGetSymbolAddress: once per device and context.  A device reset
// (cudaDeviceReset) makes a new context with the library's module loaded
// again, so the next call looks the address up again instead of using a
// stale one.
gc_status noalloc_scratch(int device, int** out) {
  static std::mutex mu;
  static int* addr[kMaxDevices] = {};
  static unsigned long long ctx_of[kMaxDevices] = {};
  if (device < 0 || device >= kMaxDevices)
    return fail(GC_ERR_UNSUPPORTED, "gc_prefix_prefill_attn_noalloc: device %d >= %d", device,
                kMaxDevices);
  std::lock_guard<std::mutex> lock(mu);
  const unsigned long long ctx = current_context_id();
  if (!addr[device] || ctx == 0 || ctx != ctx_of[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_attn_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn_noalloc: cudaGetSymbolAddress");
    addr[device] = static_cast<int*>(p);
    // the lookup made the context current if it was not yet
    ctx_of[device] = ctx ? ctx : current_context_id();
  }
  *out = addr[device];
  return GC_OK;
}

}  // namespace

gc_status launch_attn_tc_noalloc(const gc_kv_pool* pool, const AttnArgs& a,
                                 cudaStream_t stream) {
  int device = -1;
  cudaError_t e = cudaGetDevice(&device);
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn_noalloc: cudaGetDevice");
  if (device != pool->device)
    return fail(GC_ERR_INVALID_ARG,
                "gc_prefix_prefill_attn_noalloc: current device %d is not the pool's device %d",
                device, pool->device);
  // the item bound is checked again by the launch; checking it first keeps a
  // refused call from touching the device at all
  gc_status st = check_item_bound(pool, a, nullptr, pool->num_sms);
  if (st != GC_OK) return st;
  int* counter = nullptr;
  st = noalloc_scratch(device, &counter);
  if (st != GC_OK) return st;
  if (pool->cfg.head_dim == 128) return launch_d128(pool, a, stream, counter);
  return launch<64>(pool, a, stream, counter);
}

}  // namespace gc
