// Decode attention with the keys on the tensor-memory lanes (d = 128, G <= 16).
//
// One new token per request (Sec. 2.1: the decode phase; with the KV cache it
// is bound by memory): for request b with context length T, kv head g and its
// G q heads h,
//     out[b][h] = sum_{j < T} softmax_j(scale * q[b][h] . k_j) v_j.
// A query has only G rows, so the products are taken transposed, with the
// keys on the 128-row side of the tensor-core tile:
//     S^T (128 keys x 16 heads) = K_tile (128 x d) . Q^T (d x 16)
//     O^T (d x 16 heads)       += V_tile^T (d x 128) . P^T (128 x 16)
// S^T lands in TMEM with one key per lane; the softmax thread of that lane
// turns its key's 16 scores into probabilities and writes them as a column of
// P^T in shared memory; O^T accumulates in TMEM with one output column d per
// lane.  A softmax thread does 16 exponentials per tile, so the kernel keeps
// up with the memory; S^T and P^T are double-buffered, so the next tile's S^T
// product runs while this tile's softmax does.
//
// All 128 keys of a tile share one reference max per head (the operands of
// one P^T V product must): the exact max of the piece's first tile (a 4-warp
// exchange), raised together with O^T's column and the partial sums only when
// a later tile's max exceeds it by more than 2^56.  Any reference gives the
// same softmax; this one keeps every probability below 2^56.
//
// Work split: the K/V tiles of all (request, kv head) pairs, numbered in
// order, are cut into one equal share per CTA, so every SM streams the same
// number of bytes whatever the mix of context lengths.  A pair that a share
// boundary cuts is done in pieces: each writes fp32 partials (O^T unscaled,
// its reference max, its sum) and the last CTA to finish one of the pair's
// pieces combines them (a counter per cut pair in the pool's control block).
//
// Roles: warp 0 TMA producer (Q^T rows, K/V pages into the ring), warp 1 TMEM
// owner and MMA issuer (its commits also free the ring slots and Q^T), warp 2
// the unit scan, warps 4-7 softmax, epilogue and the zeroing of V rows past a
// context.  Every wait is bounded; a timeout raises the abort flag, drains
// copies and MMAs, frees TMEM and records GC_ERR_TIMEOUT.
#include "gc_internal.cuh"
#include "sm103_ptx.cuh"

namespace gc {
namespace {

using namespace ptx;

constexpr int kThreads = 256;
constexpr int kKeys = 128;                  // keys per K/V tile
constexpr int kD = 128;                     // head dim
constexpr int kN = 16;                      // q-head columns of S^T, O^T (G padded)
constexpr int kTileBytes = kKeys * kD * 2;  // 32 KB
// A K/V tile in shared memory: groups of 8 keys (2 KB), each the 8 rows of
// columns 0-63 then the 8 rows of columns 64-127 (1 KB each, 128-byte
// swizzled): key n, column half h at (n / 8) * 2048 + h * 1024 + (n % 8) * 128.
// One 4-D TMA box per page lays a page's rows out this way.
constexpr int kGroupBytes = 2048;
constexpr int kAtomBytes = 1024;
constexpr int kSmallHalf = kN * 128;        // one 64-element block of Q^T or P^T
constexpr int kSmallBytes = 2 * kSmallHalf;
constexpr uint32_t kIdescS = idesc_bf16_f32(128, kN, false, false);
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, kN, true, false);
constexpr uint32_t kColS = 0, kColO = 2 * kN;  // S^T buffers [0,16) [16,32); O^T [32,48)
constexpr uint32_t kTmemCols = 64;
constexpr float kRescaleLog2 = 56.0f;
constexpr int kSoftmaxWarp0 = 4;
constexpr int kMaxStages = 6;

struct DGeom {
  int32_t batch, Hq, Hkv, G, ps, ps_shift, num_pages, max_blocks, layer;
  float scale_log2;
  // pages read from an 8-bit image (the cache tier's layout): q8_table[b][j]
  // >= 0 names the image block holding page j of request b
  const uint8_t* q8_image;
  const int32_t* q8_table;
  int32_t q8_n_blocks, q8_layer_major, L;
  uint32_t q8_chunk;  // bytes of one (block, layer, plane) chunk
};

// ---------------------------------------------------- the 8-bit variant
// Pages of an 8-bit image reach the K/V ring in two stages: the producer
// loads a page's ps x 128 codes (one box of a 3-D tensor map over the
// image's 128-byte code rows) into a ring of 16 KB code slots, code row n of
// the tile at byte 128 n, and its K and V scales (plain loads, a tile
// ahead); two converter warpgroups (warps 8-15) turn them into bf16, with the
// rounding of the 8-bit restore, at the grouped, swizzled positions the
// pool's 4-D boxes give pool pages, once the MMA has freed the tile's slot,
// and add their eight arrivals to the slot's full barrier.  The pool is
// never written.
constexpr int kConvWarpsD = 8;
constexpr int kConvWarp0 = 8;
constexpr int kThreadsQ8 = kThreads + 32 * kConvWarpsD;
constexpr int kCodeStages = 4;
constexpr int kCodeSlotBytes = kKeys * kD;  // 16 KB
constexpr int kMaxPagesD = kKeys / 16;
constexpr int kRegsRolesQ8 = 112;    // warps 0-3 of the 8-bit variant
constexpr int kRegsSoftmaxQ8 = 192;  // warps 4-7
constexpr int kRegsConvQ8 = 104;     // warps 8-15
static_assert(128 * (kRegsRolesQ8 + kRegsSoftmaxQ8) + 32 * kConvWarpsD * kRegsConvQ8 <=
                  kThreadsQ8 * 128,
              "register split of the 8-bit variant exceeds the launch allocation");

struct D8State {
  uint64_t code_full[kCodeStages], code_empty[kCodeStages];
  uint32_t mask[kCodeStages];  // bit p: page p of the step's tile is an image page
  int32_t end[kCodeStages];    // 1: no more steps
  float scale[kCodeStages][kMaxPagesD];
};

__device__ __forceinline__ uint64_t d_chunk_index(const DGeom& geo, int blk, int kv) {
  const uint64_t il = geo.q8_layer_major
                          ? static_cast<uint64_t>(geo.layer) * geo.q8_n_blocks + blk
                          : static_cast<uint64_t>(blk) * geo.L + geo.layer;
  return il * 2 + kv;
}

struct DBar {
  uint64_t q_full[2], q_empty[2], drain;
  uint64_t kv_full[kMaxStages], kv_empty[kMaxStages];
  uint64_t s_full[2], p_full[2], pv_done[2];
  uint64_t xchg;
  uint32_t tmem_base;
  int abort_flag;
  int merge_flag;  // this CTA finished a cut pair last: it merges the pieces
};

// Workspace: each CTA's first and last pieces, when they cover part of a
// (request, kv head) pair only, as fp32 partials.
struct Workspace {
  float* part_o;    // [grid][2][kN][kD]  O^T columns, unnormalised
  float2* part_ml;  // [grid][2][kN]      (reference max in log2 units, sum)
};

__host__ __device__ inline Workspace carve(void* ws, int grid) {
  Workspace w;
  w.part_o = static_cast<float*>(ws);
  w.part_ml = reinterpret_cast<float2*>(w.part_o + static_cast<size_t>(grid) * 2 * kN * kD);
  return w;
}

// A piece: K/V tiles [j0, j1) of kv head g of request b, the part of the
// pair's units that falls in this CTA's range.  slot 0 = the range's first
// piece, 1 = a later one (only the last can be partial).
struct Piece {
  int b, g, T, nt, j0, j1;
  int pair0;  // the pair's first unit
  bool whole;
  int slot;
};

// Units are K/V tiles numbered request by request, kv head by kv head:
// unit_start[b] is request b's first unit (each valid request has Hkv x
// ceil(T/128) units, an invalid one none).  Takes the piece starting at unit
// u (< end) and advances u past it.
__device__ __forceinline__ void next_piece(int& u, int end, int range_start, const int* unit_start,
                                           const DGeom& geo, const int32_t* __restrict__ seq_lens,
                                           Piece& w) {
  int lo = 0, hi = geo.batch;  // the last request whose first unit is <= u
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (unit_start[mid] <= u) lo = mid; else hi = mid;
  }
  w.b = lo;
  w.nt = (unit_start[lo + 1] - unit_start[lo]) / geo.Hkv;
  const int local = u - unit_start[lo];
  w.g = local / w.nt;
  w.j0 = local - w.g * w.nt;
  w.j1 = min(w.nt, w.j0 + (end - u));
  w.T = __ldg(seq_lens + lo);
  w.pair0 = unit_start[lo] + w.g * w.nt;
  w.whole = w.j0 == 0 && w.j1 == w.nt;
  w.slot = u == range_start ? 0 : 1;
  u += w.j1 - w.j0;
}

// ------------------------------------------------------------------ producer
template <int kStages>
__device__ void d_producer(uint8_t* smem_q, uint8_t* smem_kv, DBar& bar, const int* unit_start,
                           int u0, int u1, const DGeom& geo, const CUtensorMap* map_q,
                           const CUtensorMap* map_kv, const int32_t* __restrict__ block_table,
                           const int32_t* __restrict__ seq_lens, int32_t* status) {
  const int lane = threadIdx.x & 31;
  volatile int* abortp = &bar.abort_flag;
  uint32_t q_count = 0, kv_count = 0;
  uint32_t armed = 0, armed_par = 0, armed_q = 0, armed_q_par = 0;
  bool ok = true;
  const uint32_t box_bytes = static_cast<uint32_t>(geo.ps) * kD * 2;  // one page

  // lane p looks up page p of tile jt of piece pc (-2: no such page).  The
  // next tile's lookup (the next piece's first, at a piece's end) is issued
  // before this tile's copies, so its latency is hidden.
  auto lookup = [&](const Piece& pc, int jt) -> int {
    int pid = -2;
    const int key0 = jt * kKeys;
    const int np = (min(kKeys, pc.T - key0) + geo.ps - 1) >> geo.ps_shift;
    const int blk = (key0 >> geo.ps_shift) + lane;
    if (lane < np)
      pid = blk < geo.max_blocks
                ? __ldg(block_table + static_cast<int64_t>(pc.b) * geo.max_blocks + blk)
                : -1;
    return pid;
  };
  int u = u0;
  Piece w, wn;
  bool have = u < u1;
  if (have) next_piece(u, u1, u0, unit_start, geo, seq_lens, w);
  int page_next = have ? lookup(w, w.j0) : -2;
  while (ok && have) {
    // ---- Q^T: the 16 q rows from head g*G of token b (rows past the end read 0)
    const int qs = q_count & 1;
    ok = mbar_wait(&bar.q_empty[qs], ((q_count >> 1) & 1) ^ 1, abortp);
    if (!ok) break;
    if (lane == 0) {
      mbar_arrive_expect_tx(&bar.q_full[qs], kSmallBytes);
      const int row = w.b * geo.Hq + w.g * geo.G;
      uint8_t* dst = smem_q + qs * kSmallBytes;
      tma_load_2d(dst, map_q, &bar.q_full[qs], 0, row);
      tma_load_2d(dst + kSmallHalf, map_q, &bar.q_full[qs], 64, row);
    }
    armed_q |= 1u << qs;
    armed_q_par = (armed_q_par & ~(1u << qs)) | (((q_count >> 1) & 1u) << qs);
    ++q_count;
    // ---- K/V tiles of the piece, page by page (lane = page * 2 + half)
    have = false;
    for (int j = w.j0; ok && j < w.j1; ++j) {
      int page = page_next;
      if (j + 1 < w.j1) {
        page_next = lookup(w, j + 1);
      } else if (u < u1) {
        next_piece(u, u1, u0, unit_start, geo, seq_lens, wn);
        page_next = lookup(wn, wn.j0);
        have = true;
      }
      if (page != -2 && (page < 0 || page >= geo.num_pages)) {
        record_error(status, GC_ERR_OUT_OF_RANGE);
        page = -1;
      }
      if (page == -2) page = -1;
      const int good = __popc(__ballot_sync(0xffffffffu, page >= 0));
      const bool issues = page >= 0;  // lane p copies page p of the tile
#pragma unroll 1
      for (int kv = 0; kv < 2; ++kv) {
        const int slot = kv_count % kStages;
        ok = mbar_wait(&bar.kv_empty[slot], ((kv_count / kStages) & 1) ^ 1, abortp);
        if (!ok) break;
        uint8_t* dst = smem_kv + slot * kTileBytes;
        if (lane == 0)
          mbar_arrive_expect_tx(&bar.kv_full[slot], static_cast<uint32_t>(good) * box_bytes);
        __syncwarp();
        if (issues) {
          const int plane_row = (geo.layer * 2 + kv) * geo.num_pages;
          const int row = (((plane_row + page) * geo.Hkv + w.g) << geo.ps_shift);
          tma_load_4d(dst + lane * box_bytes, map_kv, &bar.kv_full[slot], 0, 0, 0, row >> 3);
        }
        armed |= 1u << slot;
        armed_par = (armed_par & ~(1u << slot)) | (((kv_count / kStages) & 1u) << slot);
        ++kv_count;
      }
    }
    if (have) w = wn;
  }
  if (!ok && lane == 0) {
    // abort: wait (bounded, ignoring the flag) for the copies this warp armed
    int no_abort = 0;
    for (int s = 0; s < 2; ++s)
      if (armed_q & (1u << s)) mbar_wait(&bar.q_full[s], (armed_q_par >> s) & 1u, &no_abort);
    for (int s = 0; s < kStages; ++s)
      if (armed & (1u << s)) mbar_wait(&bar.kv_full[s], (armed_par >> s) & 1u, &no_abort);
  }
}

// The producer of the 8-bit variant: Q^T as above; per K/V step the codes
// of the tile's image pages into the next code slot, then the pool pages
// into the ring slot.  Lane p handles page p; a tile's table entries are
// loaded two tiles ahead and an image page's scales one tile ahead (within a
// piece; the first tile of a piece waits for its lookups).
template <int kStages>
__device__ void d_producer_q8(uint8_t* smem_q, uint8_t* smem_kv, uint8_t* smem_code, DBar& bar,
                              D8State& q8, const int* unit_start, int u0, int u1,
                              const DGeom& geo, const CUtensorMap* map_q,
                              const CUtensorMap* map_kv, const CUtensorMap* map_q8,
                              const int32_t* __restrict__ block_table,
                              const int32_t* __restrict__ seq_lens, int32_t* status) {
  const int lane = threadIdx.x & 31;
  volatile int* abortp = &bar.abort_flag;
  uint32_t q_count = 0, step = 0;
  uint32_t armed = 0, armed_par = 0, armed_q = 0, armed_q_par = 0, armed8 = 0, armed8_par = 0;
  bool ok = true;
  const uint32_t box_bytes = static_cast<uint32_t>(geo.ps) * kD * 2;  // one pool page
  const uint32_t code_bytes = static_cast<uint32_t>(geo.ps) * kD;    // one image page

  struct Raw {
    int page, ib;  // block-table and q8-table entries (-2: no page in this lane)
  };
  struct Look {
    int page;      // pool page, -1 none or bad, -2 no page in this lane
    int blk;       // image block, -1 none, -2 out of range
    float sk, sv;  // the image page's scales
  };
  auto raw_load = [&](const Piece& pc, int jt) -> Raw {
    Raw r{-2, -1};
    const int key0 = jt * kKeys;
    const int np = (min(kKeys, pc.T - key0) + geo.ps - 1) >> geo.ps_shift;
    const int blk = (key0 >> geo.ps_shift) + lane;
    if (lane < np) {
      if (blk < geo.max_blocks) {
        const int64_t e = static_cast<int64_t>(pc.b) * geo.max_blocks + blk;
        r.page = __ldg(block_table + e);
        r.ib = __ldg(geo.q8_table + e);
      } else {
        r.page = -1;
      }
    }
    return r;
  };
  auto resolve = [&](const Piece& pc, const Raw& r) -> Look {
    Look l{r.page, -1, 0.f, 0.f};
    if (r.ib >= 0) {
      l.page = -2;
      if (r.ib >= geo.q8_n_blocks) {
        l.page = -1;
        l.blk = -2;
      } else {
        l.blk = r.ib;
        const uint8_t* ck = geo.q8_image + d_chunk_index(geo, r.ib, 0) * geo.q8_chunk;
        l.sk = __ldg(reinterpret_cast<const float*>(ck) + pc.g);
        l.sv = __ldg(reinterpret_cast<const float*>(ck + geo.q8_chunk) + pc.g);
      }
    }
    return l;
  };
  int u = u0;
  Piece w, wn;
  bool have = u < u1;
  Look next{-2, -1, 0.f, 0.f};
  Raw raw2{-2, -1};
  if (have) {
    next_piece(u, u1, u0, unit_start, geo, seq_lens, w);
    next = resolve(w, raw_load(w, w.j0));
    if (w.j0 + 1 < w.j1) raw2 = raw_load(w, w.j0 + 1);
  }
  while (ok && have) {
    // ---- Q^T: the 16 q rows from head g*G of token b (rows past the end read 0)
    const int qs = q_count & 1;
    ok = mbar_wait(&bar.q_empty[qs], ((q_count >> 1) & 1) ^ 1, abortp);
    if (!ok) break;
    if (lane == 0) {
      mbar_arrive_expect_tx(&bar.q_full[qs], kSmallBytes);
      const int row = w.b * geo.Hq + w.g * geo.G;
      uint8_t* dst = smem_q + qs * kSmallBytes;
      tma_load_2d(dst, map_q, &bar.q_full[qs], 0, row);
      tma_load_2d(dst + kSmallHalf, map_q, &bar.q_full[qs], 64, row);
    }
    armed_q |= 1u << qs;
    armed_q_par = (armed_q_par & ~(1u << qs)) | (((q_count >> 1) & 1u) << qs);
    ++q_count;
    have = false;
    for (int j = w.j0; ok && j < w.j1; ++j) {
      Look cur = next;
      if (j + 1 < w.j1) {
        next = resolve(w, raw2);
        raw2 = j + 2 < w.j1 ? raw_load(w, j + 2) : Raw{-2, -1};
      } else if (u < u1) {
        next_piece(u, u1, u0, unit_start, geo, seq_lens, wn);
        next = resolve(wn, raw_load(wn, wn.j0));
        raw2 = wn.j0 + 1 < wn.j1 ? raw_load(wn, wn.j0 + 1) : Raw{-2, -1};
        have = true;
      }
      int page = cur.page;
      if (cur.blk == -2 || (cur.blk < 0 && page != -2 && (page < 0 || page >= geo.num_pages))) {
        record_error(status, GC_ERR_OUT_OF_RANGE);
        page = -1;
        cur.blk = -1;
      }
      if (page == -2) page = -1;
      const int good = __popc(__ballot_sync(0xffffffffu, page >= 0));
      const uint32_t img = __ballot_sync(0xffffffffu, cur.blk >= 0);
#pragma unroll 1
      for (int kv = 0; kv < 2; ++kv) {
        // codes of the image pages into the next code slot
        const int cs = step % kCodeStages;
        ok = mbar_wait(&q8.code_empty[cs], ((step / kCodeStages) & 1) ^ 1, abortp);
        if (!ok) break;
        if (cur.blk >= 0) q8.scale[cs][lane] = kv ? cur.sv : cur.sk;
        __syncwarp();
        if (lane == 0) {
          q8.mask[cs] = img;
          q8.end[cs] = 0;
          mbar_arrive_expect_tx(&q8.code_full[cs], __popc(img) * code_bytes);
        }
        __syncwarp();
        if (cur.blk >= 0)
          tma_load_3d(smem_code + cs * kCodeSlotBytes + lane * code_bytes, map_q8,
                      &q8.code_full[cs], 0, w.g * geo.ps,
                      static_cast<int32_t>(d_chunk_index(geo, cur.blk, kv)));
        armed8 |= 1u << cs;
        armed8_par = (armed8_par & ~(1u << cs)) | (((step / kCodeStages) & 1u) << cs);
        // pool pages into the ring slot
        const int slot = step % kStages;
        ok = mbar_wait(&bar.kv_empty[slot], ((step / kStages) & 1) ^ 1, abortp);
        if (!ok) break;
        uint8_t* dst = smem_kv + slot * kTileBytes;
        if (lane == 0)
          mbar_arrive_expect_tx(&bar.kv_full[slot], static_cast<uint32_t>(good) * box_bytes);
        __syncwarp();
        if (page >= 0) {
          const int plane_row = (geo.layer * 2 + kv) * geo.num_pages;
          const int row = (((plane_row + page) * geo.Hkv + w.g) << geo.ps_shift);
          tma_load_4d(dst + lane * box_bytes, map_kv, &bar.kv_full[slot], 0, 0, 0, row >> 3);
        }
        armed |= 1u << slot;
        armed_par = (armed_par & ~(1u << slot)) | (((step / kStages) & 1u) << slot);
        ++step;
      }
    }
    if (have) w = wn;
  }
  if (ok) {
    // no more steps: tell the converters through the next code slot
    const int cs = step % kCodeStages;
    ok = mbar_wait(&q8.code_empty[cs], ((step / kCodeStages) & 1) ^ 1, abortp);
    if (ok && lane == 0) {
      q8.end[cs] = 1;
      mbar_arrive(&q8.code_full[cs]);
    }
  }
  if (!ok && lane == 0) {
    // abort: wait (bounded, ignoring the flag) for the copies this warp armed
    int no_abort = 0;
    for (int s = 0; s < 2; ++s)
      if (armed_q & (1u << s)) mbar_wait(&bar.q_full[s], (armed_q_par >> s) & 1u, &no_abort);
    for (int s = 0; s < kCodeStages; ++s)
      if (armed8 & (1u << s)) mbar_wait(&q8.code_full[s], (armed8_par >> s) & 1u, &no_abort);
    for (int s = 0; s < kStages; ++s)
      if (armed & (1u << s)) mbar_wait(&bar.kv_full[s], (armed_par >> s) & 1u, &no_abort);
  }
}

// Converter warp c (warps 8-15) of the 8-bit variant: keys [16c, 16c+16) of
// every step's tile, in batches of 8 keys (a batch lies in one page), for
// the pages the step's mask marks.  Code row n sits at byte 128 n of the code
// slot; key n, column half h lands at (n / 8) * 2048 + h * 1024 + (n % 8) * 128
// with 16-byte chunk q at q ^ (n % 8), as the pool's boxes lay out pool pages.
template <int kStages>
__device__ void d_converter(uint8_t* smem_kv, const uint8_t* smem_code, DBar& bar, D8State& q8,
                            const DGeom& geo) {
  const int lane = threadIdx.x & 31;
  const int c = (threadIdx.x >> 5) - kConvWarp0;
  const int u = lane & 7;                  // 16-code word of a key's row
  const int h = u >> 2, q0 = (u & 3) * 2;  // column half and first chunk it lands in
  volatile int* abortp = &bar.abort_flag;
  for (uint32_t step = 0;; ++step) {
    const int cs = step % kCodeStages;
    bool ok = mbar_wait(&q8.code_full[cs], (step / kCodeStages) & 1, abortp);
    if (!__all_sync(0xffffffffu, ok)) break;
    if (*reinterpret_cast<volatile int32_t*>(&q8.end[cs])) break;
    const uint32_t mask = *reinterpret_cast<volatile uint32_t*>(&q8.mask[cs]);
    const int slot = step % kStages;
    // the ring slot is free once the MMAs of its previous use have completed
    ok = mbar_wait(&bar.kv_empty[slot], ((step / kStages) & 1) ^ 1, abortp);
    if (!__all_sync(0xffffffffu, ok)) break;
    uint8_t* tile = smem_kv + slot * kTileBytes;
    const uint8_t* codes = smem_code + cs * kCodeSlotBytes;
#pragma unroll 1
    for (int a = 16 * c; a < 16 * c + 16; a += 8) {
      const int p = a >> geo.ps_shift;
      if (!((mask >> p) & 1u)) continue;
      const float sc = q8.scale[cs][p];
      uint4 v[2];
#pragma unroll
      for (int q = 0; q < 2; ++q)
        v[q] = *reinterpret_cast<const uint4*>(codes + (a + q * 4 + (lane >> 3)) * 128 + u * 16);
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const int n = a + q * 4 + (lane >> 3);
        uint4 lo, hi;
        q8_dequant16(v[q], sc, lo, hi);
        const int sw = n & 7;
        uint8_t* row = tile + (n >> 3) * kGroupBytes + h * kAtomBytes + sw * 128;
        // the two halves store their chunk pairs in opposite order, so the 8
        // lanes of a key hit 8 distinct bank groups in each store
        if (h == 0) {
          *reinterpret_cast<uint4*>(row + ((q0 ^ sw) << 4)) = lo;
          *reinterpret_cast<uint4*>(row + (((q0 + 1) ^ sw) << 4)) = hi;
        } else {
          *reinterpret_cast<uint4*>(row + (((q0 + 1) ^ sw) << 4)) = hi;
          *reinterpret_cast<uint4*>(row + ((q0 ^ sw) << 4)) = lo;
        }
      }
    }
    // the tensor core reads the slot through the async proxy
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      mbar_arrive(&bar.kv_full[slot]);
      mbar_arrive(&q8.code_empty[cs]);
    }
  }
}

// ------------------------------------------------------------------ issuer
template <int kStages>
__device__ void d_issuer(uint8_t* smem_q, uint8_t* smem_p, uint8_t* smem_kv, DBar& bar,
                         uint32_t tmem, const int* unit_start, int u0, int u1,
                         const DGeom& geo, const int32_t* __restrict__ seq_lens) {
  volatile int* abortp = &bar.abort_flag;
  uint32_t q_count = 0, kv_count = 0, p_bits = 0;
  bool ok = true;
  const uint32_t p_addr = smem_addr(smem_p);
  const uint32_t kv_smem = smem_addr(smem_kv);

  for (int u = u0; ok && u < u1;) {
    Piece w;
    next_piece(u, u1, u0, unit_start, geo, seq_lens, w);
    const uint32_t kv_base = kv_count;
    const int nt = w.j1 - w.j0;
    kv_count += 2 * nt;
    const int qs = q_count & 1;
    ok = mbar_wait(&bar.q_full[qs], (q_count >> 1) & 1, abortp);
    ++q_count;
    if (!ok) break;
    tc_fence_after();
    const uint32_t q_addr = smem_addr(smem_q + qs * kSmallBytes);
    // S^T(t) = K_t Q^T into S buffer t & 1 (free once P^T(t - 2) is written)
    auto issue_s = [&](int t) -> bool {
      const uint32_t ku = kv_base + 2 * t;
      if (!mbar_wait(&bar.kv_full[ku % kStages], (ku / kStages) & 1, abortp)) return false;
      tc_fence_after();
      const uint32_t k_addr = kv_smem + (ku % kStages) * kTileBytes;
#pragma unroll
      for (int kk = 0; kk < kD / 16; ++kk) {
        const uint32_t ka = k_addr + (kk >> 2) * kAtomBytes + (kk & 3) * 32;
        const uint32_t qa = q_addr + (kk >> 2) * kSmallHalf + (kk & 3) * 32;
        mma_ss(tmem + kColS + (t & 1) * kN, sdesc_sw128(ka, 16, kGroupBytes), sdesc_sw128(qa, 16, 1024),
               kIdescS, kk > 0 ? 1u : 0u);
      }
      mma_commit(&bar.s_full[t & 1]);
      mma_commit(&bar.kv_empty[ku % kStages]);        // K_t is free once S^T(t) is done
      if (t == nt - 1) mma_commit(&bar.q_empty[qs]);   // and Q^T after the piece's last S^T
      return true;
    };
    ok = issue_s(0);
    if (ok && nt > 1) ok = issue_s(1);
    for (int t = 0; ok && t < nt; ++t) {
      // O^T += V_t^T P^T(t) once the softmax has written P^T(t) and V_t is in
      const uint32_t vu = kv_base + 2 * t + 1;
      const int pb = t & 1;
      ok = mbar_wait(&bar.p_full[pb], (p_bits >> pb) & 1u, abortp);
      p_bits ^= 1u << pb;
      if (ok) ok = mbar_wait(&bar.kv_full[vu % kStages], (vu / kStages) & 1, abortp);
      if (!ok) break;
      tc_fence_after();
      const uint32_t v_addr = kv_smem + (vu % kStages) * kTileBytes;
      const uint32_t pt = p_addr + pb * kSmallBytes;
#pragma unroll
      for (int kk = 0; kk < kKeys / 16; ++kk) {
        const uint32_t pa = pt + (kk >> 2) * kSmallHalf + (kk & 3) * 32;
        mma_ss(tmem + kColO, sdesc_sw128(v_addr + kk * 2 * kGroupBytes, kAtomBytes, kGroupBytes),
               sdesc_sw128(pa, 16, 1024), kIdescPV, (t > 0 || kk > 0) ? 1u : 0u);
      }
      mma_commit(&bar.pv_done[pb]);
      mma_commit(&bar.kv_empty[vu % kStages]);  // V_t is free once PV(t) is done
      if (t + 2 < nt) ok = issue_s(t + 2);
    }
  }
  // every MMA this thread issued completes before TMEM is freed
  mma_commit(&bar.drain);
  int no_abort = 0;
  mbar_wait(&bar.drain, 0, &no_abort);
}

// Byte offset of P^T element (head n, key) in a 128-byte-swizzled K-major
// tile of kN rows: 64-key blocks; in a row, 16-byte chunk c sits at c ^ (n % 8).
__device__ __forceinline__ uint32_t pt_offset(int n, int key) {
  const int blk = key >> 6, kin = key & 63;
  const int chunk = (kin >> 3) ^ (n & 7);
  return blk * kSmallHalf + n * 128 + (chunk << 4) + ((kin & 7) << 1);
}

// 4-warp exchange through shared memory: r[h] = max (or sum) over the softmax
// warps of v[h].  Two buffers alternate, so one barrier phase per exchange.
__device__ __forceinline__ bool exchange(DBar& bar, float* xbuf, uint32_t& x_count, int warp,
                                         const float (&v)[kN], float (&r)[kN], bool is_max,
                                         volatile int* abortp) {
  float* xb = xbuf + (x_count & 1) * 4 * kN;
  const int lane = threadIdx.x & 31;
  float mine = v[0];
#pragma unroll
  for (int h = 1; h < kN; ++h) mine = lane == h ? v[h] : mine;
  if (lane < kN) xb[warp * kN + lane] = mine;
  __syncwarp();
  if (lane == 0) mbar_arrive(&bar.xchg);
  const bool good = mbar_wait(&bar.xchg, x_count & 1, abortp);
  ++x_count;
  if (!good) return false;
#pragma unroll
  for (int h = 0; h < kN; ++h) {
    const float a = xb[h], b = xb[kN + h], c = xb[2 * kN + h], d = xb[3 * kN + h];
    r[h] = is_max ? fmaxf(fmaxf(a, b), fmaxf(c, d)) : (a + b) + (c + d);
  }
  return true;
}

// The four softmax warps meet (bounded wait); one barrier phase, like exchange().
__device__ __forceinline__ bool sync4(DBar& bar, uint32_t& x_count, volatile int* abortp) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&bar.xchg);
  const bool good = mbar_wait(&bar.xchg, x_count & 1, abortp);
  ++x_count;
  return good;
}

// Combines the pieces of pair w held by CTAs c0..c1 (slot 1 of c0 unless the
// pair starts c0's share, slot 0 of the others):
//     out = sum_s O_s 2^(m_s - M) / sum_s l_s 2^(m_s - M),  M = max_s m_s,
// thread d for column d of each q head.  The partials come from other SMs,
// so they are read through L2.
__device__ void merge_pieces(const Workspace& ws, const Piece& w, int c0, int c1, int per,
                             const DGeom& geo, __nv_bfloat16* __restrict__ out_g) {
  const int d = threadIdx.x - kSoftmaxWarp0 * 32;
  const int first_slot = w.pair0 == c0 * per ? 0 : 1;
  for (int h0 = 0; h0 < geo.G; h0 += 4) {
    float M[4], acc[4], L[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      M[i] = -INFINITY;
      acc[i] = 0.f;
      L[i] = 0.f;
    }
    for (int c = c0; c <= c1; c += 4) {
      float2 ml[4][4];
      float o[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const bool in = h0 + i < geo.G && c + k <= c1;
          const int slot = c + k == c0 ? first_slot : 0;
          const int64_t part = (static_cast<int64_t>(c + k) * 2 + slot) * kN + h0 + i;
          ml[i][k] = in ? __ldcg(ws.part_ml + part) : make_float2(-INFINITY, 0.f);
          o[i][k] = in ? __ldcg(ws.part_o + part * kD + d) : 0.f;
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float Mn = M[i];
#pragma unroll
        for (int k = 0; k < 4; ++k) Mn = fmaxf(Mn, ml[i][k].x);
        const float r = ex2_approx(M[i] - Mn);  // 0 while M is -inf
        acc[i] *= r;
        L[i] *= r;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float f = ex2_approx(ml[i][k].x - Mn);
          acc[i] = fmaf(o[i][k], f, acc[i]);
          L[i] = fmaf(ml[i][k].y, f, L[i]);
        }
        M[i] = Mn;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (h0 + i < geo.G) out_g[(h0 + i) * kD + d] = __float2bfloat16_rn(acc[i] / L[i]);
  }
}

// ------------------------------------------------------------------ softmax
template <int kStages>
__device__ void d_softmax(uint8_t* smem_p, uint8_t* smem_kv, DBar& bar, float* xbuf, uint32_t tmem,
                          const int* unit_start, int u0, int u1, const DGeom& geo,
                          const int32_t* __restrict__ seq_lens, __nv_bfloat16* __restrict__ out,
                          const Workspace& ws, int per, int* merge_counters) {
  volatile int* abortp = &bar.abort_flag;
  const int warp = (threadIdx.x >> 5) - kSoftmaxWarp0;  // 0..3 = TMEM lane quarter
  const int lane = threadIdx.x & 31;
  const int t_id = warp * 32 + lane;                     // key of the tile, column d of O^T
  const uint32_t lane_addr = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  uint32_t s_bits = 0, pv_bits = 0, x_count = 0, kv_count = 0;
  bool ok = true;

  for (int u = u0; ok && u < u1;) {
    Piece w;
    next_piece(u, u1, u0, unit_start, geo, seq_lens, w);
    const int nt = w.j1 - w.j0;
    const uint32_t kv_base = kv_count;
    kv_count += 2 * nt;
    // PV products complete in issue order; wait for each once, in order
    int pv_seen = 0;
    auto wait_pv = [&](int upto) -> bool {
      while (pv_seen <= upto) {
        const int b = pv_seen & 1;
        if (!mbar_wait(&bar.pv_done[b], (pv_bits >> b) & 1u, abortp)) return false;
        pv_bits ^= 1u << b;
        ++pv_seen;
      }
      return true;
    };
    float m_ref[kN], lsum[kN];
#pragma unroll
    for (int h = 0; h < kN; ++h) {
      m_ref[h] = -INFINITY;
      lsum[h] = 0.f;
    }
    const float sl2 = geo.scale_log2;
    for (int t = 0; t < nt; ++t) {
      const int buf = t & 1;
      ok = mbar_wait(&bar.s_full[buf], (s_bits >> buf) & 1u, abortp);
      s_bits ^= 1u << buf;
      if (!ok) break;
      tc_fence_after();
      uint32_t sr[kN];
      tmem_ld16(lane_addr + kColS + buf * kN, sr);
      tmem_wait_ld();
      const bool key_valid = (w.j0 + t) * kKeys + t_id < w.T;
      float s[kN], wmax[kN];
#pragma unroll
      for (int h = 0; h < kN; ++h) {
        s[h] = key_valid && h < geo.G ? __uint_as_float(sr[h]) * sl2 : -INFINITY;
        float m = s[h];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        wmax[h] = m;
      }
      // P^T buffer `buf` is free once PV(t - 2) has completed
      if (t >= 2) {
        ok = wait_pv(t - 2);
        if (!ok) break;
      }
      float tmax[kN];
      ok = exchange(bar, xbuf, x_count, warp, wmax, tmax, true, abortp);
      if (!ok) break;
      if (t == 0) {
#pragma unroll
        for (int h = 0; h < kN; ++h) m_ref[h] = tmax[h];
      } else {
        bool grow = false;
#pragma unroll
        for (int h = 0; h < kN; ++h) grow |= tmax[h] > m_ref[h] + kRescaleLog2;
        if (grow) {
          // rare: raise the reference of the heads that outgrew it.  O^T
          // holds tiles < t, so PV(t - 1) must be complete first.
          ok = wait_pv(t - 1);
          if (!ok) break;
          tc_fence_after();
          uint32_t o[kN];
          tmem_ld16(lane_addr + kColO, o);
          tmem_wait_ld();
#pragma unroll
          for (int h = 0; h < kN; ++h) {
            if (tmax[h] > m_ref[h] + kRescaleLog2) {
              const float alpha = ex2_approx(m_ref[h] - tmax[h]);
              o[h] = __float_as_uint(__uint_as_float(o[h]) * alpha);
              lsum[h] *= alpha;
              m_ref[h] = tmax[h];
            }
          }
          tmem_st16(lane_addr + kColO, o);
          tmem_wait_st();
        }
      }
      if ((w.j0 + t + 1) * kKeys > w.T) {
        // the pair's last, ragged tile: V rows past the context must be zero
        // (their P is 0, and 0 * NaN is NaN); each thread clears its own row
        // once the V tile has landed, before P^T(t) releases PV(t)
        const uint32_t vu = kv_base + 2 * t + 1;
        ok = mbar_wait(&bar.kv_full[vu % kStages], (vu / kStages) & 1, abortp);
        if (!ok) break;
        if (!key_valid) {
          uint8_t* vrow = smem_kv + (vu % kStages) * kTileBytes + (t_id >> 3) * kGroupBytes +
                          (t_id & 7) * 128;
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int c = 0; c < 8; ++c)
              reinterpret_cast<uint4*>(vrow + h * kAtomBytes)[c] = make_uint4(0, 0, 0, 0);
        }
      }
      // this key's probabilities for the 16 head columns: column t_id of P^T
      uint8_t* pt = smem_p + buf * kSmallBytes;
#pragma unroll
      for (int h = 0; h < kN; ++h) {
        const float p = s[h] == -INFINITY ? 0.f : ex2_approx(s[h] - m_ref[h]);
        lsum[h] += p;
        *reinterpret_cast<__nv_bfloat16*>(pt + pt_offset(h, t_id)) = __float2bfloat16_rn(p);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar.p_full[buf]);
    }
    if (!ok) break;
    // ---- epilogue: the last PVs, then O^T / l (or the range's partials)
    ok = wait_pv(nt - 1);
    if (!ok) break;
    tc_fence_after();
    float wsum[kN], L[kN];
#pragma unroll
    for (int h = 0; h < kN; ++h) {
      float v = lsum[h];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      wsum[h] = v;
    }
    ok = exchange(bar, xbuf, x_count, warp, wsum, L, false, abortp);
    if (!ok) break;
    uint32_t o[kN];
    tmem_ld16(lane_addr + kColO, o);
    tmem_wait_ld();
    tc_fence_before();
    const int d = t_id;
    const int64_t head0 = static_cast<int64_t>(w.b) * geo.Hq + w.g * geo.G;
    if (w.whole) {
#pragma unroll
      for (int h = 0; h < kN; ++h)
        if (h < geo.G) out[(head0 + h) * kD + d] = __float2bfloat16_rn(__uint_as_float(o[h]) / L[h]);
    } else {
      const int64_t part = (static_cast<int64_t>(blockIdx.x) * 2 + w.slot) * kN;
#pragma unroll
      for (int h = 0; h < kN; ++h) {
        if (h < geo.G) {
          ws.part_o[(part + h) * kD + d] = __uint_as_float(o[h]);
          if (d == 0) ws.part_ml[part + h] = make_float2(m_ref[h], L[h]);
        }
      }
      // The pair's pieces are the shares of CTAs c0..c1; the last to finish
      // combines them.  Its counter (in the pool's control block, indexed by
      // c0) is back at 0 afterwards.
      const int c0 = w.pair0 / per, c1 = (w.pair0 + w.nt - 1) / per;
      __threadfence();
      ok = sync4(bar, x_count, abortp);
      if (!ok) break;
      int* flag = &bar.merge_flag;
      if (t_id == 0) {
        const int prev = atomicAdd(merge_counters + c0, 1);
        const int last = prev == c1 - c0;
        if (last) {
          merge_counters[c0] = 0;
          __threadfence();
        }
        *flag = last;
      }
      ok = sync4(bar, x_count, abortp);
      if (!ok) break;
      if (*reinterpret_cast<volatile int*>(flag))
        merge_pieces(ws, w, c0, c1, per, geo, out + head0 * kD);
    }
  }
}

template <int kStages, bool kQ8>
__global__ void __launch_bounds__(kQ8 ? kThreadsQ8 : kThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                     const __grid_constant__ CUtensorMap map_kv,
                     const __grid_constant__ CUtensorMap map_q8,
                     const int32_t* __restrict__ block_table, const int32_t* __restrict__ seq_lens,
                     __nv_bfloat16* __restrict__ out, void* ws_raw, DGeom geo,
                     int32_t* status, int* merge_counters) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* smem_q = base;                      // Q^T x 2, 8 KB
  uint8_t* smem_p = base + 2 * kSmallBytes;    // P^T x 2, 8 KB
  uint8_t* smem_kv = base + 4 * kSmallBytes;   // ring, 1024-aligned
  uint8_t* smem_code = smem_kv + kStages * kTileBytes;  // 8-bit variant: code slots
  DBar& bar = *reinterpret_cast<DBar*>(smem_code + (kQ8 ? kCodeStages * kCodeSlotBytes : 0));
  float* xbuf = reinterpret_cast<float*>(&bar + 1);             // [2][4][kN]
  int* unit_start = reinterpret_cast<int*>(xbuf + 2 * 4 * kN);  // [batch + 1]
  D8State* q8 = reinterpret_cast<D8State*>(
      (reinterpret_cast<uintptr_t>(unit_start + geo.batch + 1) + 7) & ~uintptr_t(7));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&bar.drain, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bar.kv_full[s], kQ8 ? 1 + kConvWarpsD : 1);  // + one arrival per converter
      mbar_init(&bar.kv_empty[s], 1);
    }
    if (kQ8) {
      for (int s = 0; s < kCodeStages; ++s) {
        mbar_init(&q8->code_full[s], 1);
        mbar_init(&q8->code_empty[s], kConvWarpsD);
      }
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar.q_full[b], 1);
      mbar_init(&bar.q_empty[b], 1);
      mbar_init(&bar.s_full[b], 1);
      mbar_init(&bar.p_full[b], 4);
      mbar_init(&bar.pv_done[b], 1);
    }
    mbar_init(&bar.xchg, 4);
    bar.abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&map_q);
    prefetch_tensormap(&map_kv);
    if (kQ8) prefetch_tensormap(&map_q8);
  }
  if (warp == 1) {
    tmem_alloc(&bar.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  // Launched as a programmatic dependent of the previous kernel on the
  // stream: the set-up above touches only this CTA's shared memory and TMEM;
  // inputs are read, and outputs written, once the previous grid is complete.
  // The next kernel may in turn be set up on the SMs this grid frees.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (warp == 2) {
    // units per request (kv heads x K/V tiles), exclusive scan; a context
    // length outside [1, block table capacity] gets none and is recorded
    const int cap = geo.max_blocks << geo.ps_shift;
    int running = 0;
    for (int b0 = 0; b0 < geo.batch; b0 += 32) {
      const int b = b0 + lane;
      int cnt = 0;
      if (b < geo.batch) {
        const int T = __ldg(seq_lens + b);
        if (T < 1 || T > cap) {
          record_error(status, GC_ERR_OUT_OF_RANGE);
        } else {
          const int nt = (T + kKeys - 1) / kKeys;
          cnt = geo.Hkv * nt;
        }
      }
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
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bar.tmem_base;
  // this CTA's units: an equal share of all of them, in order
  const int total = unit_start[geo.batch];
  const int per = max(1, (total + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x));
  const int u0 = min(total, static_cast<int>(blockIdx.x) * per);
  const int u1 = min(total, u0 + per);
  const Workspace ws = carve(ws_raw, gridDim.x);

  if (kQ8) {
    // warpgroups: roles, softmax, converters
    if (warp < 4) regs_dec<kRegsRolesQ8>();  // (no change at a 128-register launch)
    else if (warp < 8) regs_inc<kRegsSoftmaxQ8>();
    else regs_dec<kRegsConvQ8>();
  }
  if (warp == 0) {
    if (kQ8)
      d_producer_q8<kStages>(smem_q, smem_kv, smem_code, bar, *q8, unit_start, u0, u1, geo,
                             &map_q, &map_kv, &map_q8, block_table, seq_lens, status);
    else
      d_producer<kStages>(smem_q, smem_kv, bar, unit_start, u0, u1, geo, &map_q, &map_kv,
                          block_table, seq_lens, status);
  } else if (warp == 1) {
    if (lane == 0)
      d_issuer<kStages>(smem_q, smem_p, smem_kv, bar, tmem, unit_start, u0, u1, geo, seq_lens);
    __syncwarp();
  } else if (warp >= kSoftmaxWarp0 && warp < kSoftmaxWarp0 + 4) {
    d_softmax<kStages>(smem_p, smem_kv, bar, xbuf, tmem, unit_start, u0, u1, geo, seq_lens, out, ws, per,
                       merge_counters);
  } else if (kQ8 && warp >= kConvWarp0) {
    d_converter<kStages>(smem_kv, smem_code, bar, *q8, geo);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && bar.abort_flag) record_error(status, GC_ERR_TIMEOUT);
}

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

// One CTA per SM, at most one per merge counter of the pool's control block.
int decode_grid(const gc_kv_pool* pool) { return min(pool->num_sms, kMergeCounters); }

size_t smem_bytes(int stages, int batch, bool q8 = false) {
  return 1024 + 4 * kSmallBytes + static_cast<size_t>(stages) * kTileBytes + sizeof(DBar) +
         2 * 4 * kN * sizeof(float) + (static_cast<size_t>(batch) + 1) * sizeof(int) +
         (q8 ? kCodeStages * static_cast<size_t>(kCodeSlotBytes) + sizeof(D8State) + 8 : 0);
}

template <int kStages, bool kQ8>
gc_status launch_stages(const gc_kv_pool* pool, const DecodeArgs& a, const DGeom& geo,
                        const CUtensorMap& map_q, const CUtensorMap& map_kv,
                        const CUtensorMap& map_q8, cudaStream_t stream) {
  const size_t smem = smem_bytes(kStages, a.batch, kQ8);
  cudaError_t e = cudaFuncSetAttribute(decode_tc_kernel<kStages, kQ8>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: smem attribute");
  cudaLaunchConfig_t lc = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  lc.gridDim = dim3(decode_grid(pool));
  lc.blockDim = dim3(kQ8 ? kThreadsQ8 : kThreads);
  lc.dynamicSmemBytes = smem;
  lc.stream = stream;
  lc.attrs = attr;
  lc.numAttrs = 1;
  e = cudaLaunchKernelEx(&lc, decode_tc_kernel<kStages, kQ8>, map_q, map_kv, map_q8, a.block_table,
                         a.seq_lens,
                         static_cast<__nv_bfloat16*>(a.out), a.workspace, geo, pool->status,
                         pool->merge_counters);
  if (e != cudaSuccess) return cuda_fail(e, "gc_paged_decode_attn: launch");
  return GC_OK;
}

}  // namespace

bool decode_tc_supported(const gc_kv_pool* pool, int32_t num_q_heads) {
  const int G = num_q_heads / pool->cfg.num_kv_heads;
  return pool->cfg.head_dim == kD && G >= 1 && G <= kN;
}

size_t decode_tc_workspace_bytes(const gc_kv_pool* pool, int32_t) {
  const size_t grid = static_cast<size_t>(decode_grid(pool));
  return grid * 2 * kN * kD * sizeof(float) + grid * 2 * kN * sizeof(float2);
}

gc_status launch_decode_tc(const gc_kv_pool* pool, const DecodeArgs& a, cudaStream_t stream,
                           const Q8Pages* q8) {
  const size_t need = decode_tc_workspace_bytes(pool, a.batch);
  if (a.workspace == nullptr || a.workspace_bytes < need)
    return fail(GC_ERR_INVALID_ARG,
                "gc_paged_decode_attn: workspace of %zu bytes needed "
                "(gc_paged_decode_workspace_bytes), got %zu",
                need, a.workspace_bytes);
  const auto& cfg = pool->cfg;
  const long long cap_tiles =
      (static_cast<long long>(a.max_blocks) * cfg.page_size + kKeys - 1) / kKeys;
  if (static_cast<long long>(a.batch) * cfg.num_kv_heads * cap_tiles + 2LL * pool->num_sms >
      2147483647LL)
    return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: %lld K/V tiles per call",
                static_cast<long long>(a.batch) * cfg.num_kv_heads * cap_tiles);
  auto enc = encode_fn();
  if (!enc) return fail(GC_ERR_CUDA, "gc_paged_decode_attn: cuTensorMapEncodeTiled unavailable");
  DGeom geo;
  geo.batch = a.batch;
  geo.Hq = a.num_q_heads;
  geo.Hkv = cfg.num_kv_heads;
  geo.G = geo.Hq / geo.Hkv;
  geo.ps = cfg.page_size;
  int sh = 0;
  while ((1 << sh) < geo.ps) ++sh;
  geo.ps_shift = sh;
  geo.num_pages = cfg.num_pages;
  geo.max_blocks = a.max_blocks;
  geo.layer = a.layer;
  geo.scale_log2 = a.softmax_scale * 1.4426950408889634f;
  geo.q8_image = q8 ? q8->image : nullptr;
  geo.q8_table = q8 ? q8->table : nullptr;
  geo.q8_n_blocks = q8 ? q8->n_blocks : 0;
  geo.q8_layer_major = q8 && q8->layer_major ? 1 : 0;
  geo.L = cfg.num_layers;
  geo.q8_chunk = static_cast<uint32_t>(q8_chunk_bytes(cfg));
  const uint64_t pool_rows = static_cast<uint64_t>(cfg.num_layers) * 2 * cfg.num_pages *
                             cfg.num_kv_heads * cfg.page_size;
  if (pool_rows >= (1ull << 31))
    return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn: pool has %llu rows (limit 2^31)",
                static_cast<unsigned long long>(pool_rows));
  CUtensorMap map_q, map_kv;
  {
    // q as rows of d: [batch * Hq][128]; boxes of 16 rows x 64 columns, rows
    // past the end read as zero
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(kD),
                          static_cast<cuuint64_t>(a.batch) * static_cast<cuuint64_t>(geo.Hq)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(kD) * 2};
    cuuint32_t box[2] = {64, kN};
    cuuint32_t es[2] = {1, 1};
    CUresult r = enc(&map_q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(a.q), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_paged_decode_attn: q tensor map (CUresult %d)", (int)r);
  }
  {
    // pool rows of 128 columns seen as (column in half, row in group of 8,
    // half, group): one box of (64, 8, 2, ps/8) is a page, laid out in
    // shared memory group by group, half by half
    cuuint64_t dims[4] = {64, 8, 2, pool_rows / 8};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(kD) * 2, 128, 8 * static_cast<cuuint64_t>(kD) * 2};
    cuuint32_t box[4] = {64, 8, 2, static_cast<cuuint32_t>(geo.ps / 8)};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = enc(&map_kv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, pool->data, dims, strides, box,
                     es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_paged_decode_attn: pool tensor map (CUresult %d)", (int)r);
  }
  constexpr size_t kSmemLimit = 232448;
  if (q8) {
    // the image's code rows (128 bytes each; Hkv*ps rows per chunk after the
    // scale header) as a 3-D map, box = one page of one kv head
    const uint64_t chunks = static_cast<uint64_t>(q8->n_blocks) * cfg.num_layers * 2;
    if (chunks >= (1ull << 31))
      return fail(GC_ERR_UNSUPPORTED, "gc_paged_decode_attn_q8: image of %llu chunks (limit 2^31)",
                  static_cast<unsigned long long>(chunks));
    const void* base = chunks ? static_cast<const void*>(q8->image + q8_header_bytes(cfg))
                              : pool->data;  // an empty image is never read
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD),
                          static_cast<cuuint64_t>(cfg.num_kv_heads) * cfg.page_size,
                          chunks ? chunks : 1};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(geo.q8_chunk)};
    cuuint32_t box[3] = {static_cast<cuuint32_t>(kD), static_cast<cuuint32_t>(cfg.page_size), 1};
    cuuint32_t es[3] = {1, 1, 1};
    CUtensorMap map_q8;
    CUresult r = enc(&map_q8, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void*>(base), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_paged_decode_attn_q8: image tensor map (CUresult %d)", (int)r);
    // four ring slots and four code slots unless a large batch's unit table
    // needs the room
    return smem_bytes(4, a.batch, true) <= kSmemLimit
               ? launch_stages<4, true>(pool, a, geo, map_q, map_kv, map_q8, stream)
               : launch_stages<3, true>(pool, a, geo, map_q, map_kv, map_q8, stream);
  }
  // six ring slots unless the unit table of a large batch needs the room
  const gc_status st = smem_bytes(6, a.batch) <= kSmemLimit
                           ? launch_stages<6, false>(pool, a, geo, map_q, map_kv, map_kv, stream)
                           : launch_stages<5, false>(pool, a, geo, map_q, map_kv, map_kv, stream);
  return st;
}

}  // namespace gc
