// Prefix-reuse causal GQA attention, head_dim 128, on pairs of SMs
// (tcgen05 cta_group::2).
//
// Operation (Sec. 2.2: the cached context KV and the new tokens' KV are
// processed together; Sec. 2.1: prefill): for request b, q head h, new row
// i < n_b and kv head g = h / G,
//     O[b,i,h] = sum_{j <= P_b + i} softmax_j(scale * q . k_j) v_j
// with keys read from the paged pool through block_table[b].
//
// Design
//  * A work item is (request b, kv head g, 256 q rows); a q row is
//    (token, head) with row = token*G + head, so one item covers 256/G new
//    tokens x the G q heads of kv group g and every K/V tile fetched from
//    the pool feeds all of them.  Items are handed out by a counter, longest
//    request first, later rows first within a request.
//  * Each item runs on a CTA pair (a cluster of two, one CTA per SM).  The
//    MMAs are M = 256 products issued by one thread of the even CTA: each
//    SM holds 128 of the q rows (its half of A and of every product) and
//    half of every K/V tile (B is split by columns between the two SMs), so
//    each SM fetches 32 KB of K/V per 128-key step for 128 rows x 128 keys
//    of work.
//      S = Q K^T    M 256, N 128 keys, K 128 (both operands K-major, smem)
//      O += P V     M 256, N 128 (d), K 128 keys (P from tensor memory,
//                   V MN-major in smem)
//  * Tensor memory per SM: S double-buffered [0,128) [128,256), O [256,384),
//    P double-buffered [384,448) [448,512) (bf16 pairs).  P has its own
//    columns, so S(t+1) and S(t+2) are computed while the softmax works on
//    S(t), and PV(t) overlaps the softmax of step t+1.
//  * Warps per CTA:
//      0     K producer: this SM's Q half of each item, then per 128-key step
//            its K half (64 keys x 128 d, one 4-D box per page) into a ring
//            of 16 KB slots.
//      3     V producer: per step its V half (128 keys x 64 d, one box per
//            page) into a second ring.  Each producer reports its own copies
//            to the even CTA once they have landed, zeroing V rows past the
//            end of the sequence first (their P is 0 but 0 * NaN is NaN).
//      1     tensor-memory owner (both CTAs allocate together); in the even
//            CTA lane 0 issues the pair's S products.
//      2     item table at start-up; in the even CTA lane 0 then issues the
//            pair's PV products.
//      4-11  softmax in two warpgroups, key columns [0, 64) and [64, 128) of
//            every q row (= tensor-memory lane): S from tensor memory, causal
//            mask, p = 2^(s*scale*log2 e - m) against a reference max (the
//            row's first-tile max; raised, with O and l rescaled, only if a
//            later tile would approach fp32 overflow), P as bf16 into tensor
//            memory, final 1/l and the bf16 store of O.
//  * Every wait and spin is bounded; a CTA that gives up raises its own and
//    its peer's abort flag, every role leaves its loop, copies and MMAs in
//    flight are drained, both CTAs meet at a cluster barrier, tensor memory
//    is freed and GC_ERR_TIMEOUT is recorded.
#include <cmath>

#include "gc_internal.cuh"
#include "sm103_ptx.cuh"

namespace gc {
namespace {

using namespace ptx;

constexpr int kD = 128;
// softmax by two warpgroups, half a row each
constexpr int kSoftmaxWarps = 8;
constexpr int kThreads = 128 + 32 * kSoftmaxWarps;
constexpr int kRows = 128;            // q rows per SM
constexpr int kKeys = 128;            // keys per K/V step
constexpr int kRing = 4;              // slots of 16 KB in each of the K and V rings
constexpr int kSlotBytes = 16384;
constexpr int kQBytes = kRows * kD * 2;  // 32 KB: two 64-column blocks of 128 rows
constexpr int kSortMax = 512;
// tensor memory: three S buffers of 128 columns (each half-row's P is written
// over the first 32 of its own 64 S columns), O after them
constexpr int kSBufs = 3;
constexpr uint32_t kColS = 0, kColO = kSBufs * 128;
constexpr uint32_t kIdescQK = idesc_bf16_f32(256, kKeys, false, false);
constexpr uint32_t kIdescPV = idesc_bf16_f32(256, kD, false, true);
// consumers of the work-item ring: in each CTA the V producer and the
// softmax warps, plus the two MMA issuers of the even CTA and the odd CTA's
// K producer
constexpr int kItemConsumers = 2 * (1 + kSoftmaxWarps) + 3;

struct Geom2 {
  int32_t batch, Hq, Hkv, G, ps, ps_shift, num_pages, max_blocks, layer, total_new;
  int32_t box_rows, box_shift;  // TMA box height min(ps, 64) and its log2
  float scale_log2;
};

struct Bars2 {
  uint64_t q_full[2];         // even CTA: both Q halves landed (2 arrivals + both copies' bytes)
  uint64_t q_empty[2];        // the item's last S product done (commit, both CTAs)
  uint64_t k_landed[kRing];   // (unused: K copies always complete on k_full)
  uint64_t k_full[kRing];     // even CTA: both K halves of the slot landed (2 arrivals + bytes)
  uint64_t k_empty[kRing];    // the S product reading the slot done (softmax thread 0)
  uint64_t v_landed[kRing];   // this CTA's V half of an item's last, partial step (tx)
  uint64_t v_full[kRing];     // even CTA: both V halves of the slot ready (2 arrivals + bytes)
  uint64_t v_empty[kRing];    // the PV product reading the slot done (commit, both CTAs)
  uint64_t s_full[kSBufs];    // S buffer computed (commit, both CTAs)
  uint64_t p_full[kSBufs];    // even CTA: P written into the buffer by all softmax warps
  uint64_t pv_done[kSBufs];   // PV product reading the buffer's P done (commit, both CTAs)
  uint64_t o_free;            // even CTA: O read by the epilogue
  uint64_t item_full[2];      // work-item ring, written by the even CTA's K producer
  uint64_t item_empty[2];     // even CTA: item slot read by every consumer of both CTAs
  uint64_t drain;             // even CTA: both issuers' last commits
  int item_msg[2][8];         // a claimed item, decoded: it, b, tile, g, P, n, cu (it < 0: end)
  uint32_t tmem_base;
  int abort_flag;
};

// Shared::cluster addresses of the barriers that live in the even CTA, and
// of the peer's abort flag and item messages.
struct Remote {
  uint32_t q_full, k_full, v_full, p_full, o_free, item_empty, item_full, item_msg,
      abort_peer;
};

struct Item2 {
  int b, g, P, n, cu, T;
  int tok0;      // first token of this CTA's 128 rows
  int nt;        // K/V steps of the item (both CTAs)
  bool rows_ok;  // this CTA has at least one valid row
};

// Which request, kv head and 256-row tile item `it` is (item_start: first
// item of each request in work order, then the order itself when the batch
// was ranked), with the request's lengths: the message the even CTA's
// producer sends to every role of both CTAs.
__device__ __forceinline__ void item_message(int it, const int* item_start, const Geom2& geo,
                                             const int32_t* __restrict__ prefix_lens,
                                             const int32_t* __restrict__ new_lens,
                                             const int32_t* __restrict__ cu_new_lens, int* m) {
  int lo = 0, hi = geo.batch;  // last p with item_start[p] <= it
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (item_start[mid] <= it) lo = mid; else hi = mid;
  }
  const int b = geo.batch <= kSortMax ? static_cast<int>(
                    reinterpret_cast<const int16_t*>(item_start + geo.batch + 1)[lo])
                                       : lo;
  const int local = it - item_start[lo];
  const int tiles = (item_start[lo + 1] - item_start[lo]) / geo.Hkv;
  m[0] = it;
  m[1] = b;
  m[2] = tiles - 1 - local / geo.Hkv;  // later rows (more keys) first
  m[3] = local % geo.Hkv;
  m[4] = __ldg(prefix_lens + b);
  m[5] = __ldg(new_lens + b);
  m[6] = __ldg(cu_new_lens + b);
}

// The quantities a role of CTA `rank` derives from an item message.
__device__ __forceinline__ void item_from_message(const int* m, const Geom2& geo, uint32_t rank,
                                                  Item2& w) {
  w.b = m[1];
  w.g = m[3];
  w.P = m[4];
  w.n = m[5];
  w.cu = m[6];
  w.T = w.P + w.n;
  const int rows = w.n * geo.G;
  const int r0 = m[2] * 2 * kRows;
  w.tok0 = (r0 + static_cast<int>(rank) * kRows) / geo.G;
  w.rows_ok = r0 + static_cast<int>(rank) * kRows < rows;
  const int r_last = min(r0 + 2 * kRows - 1, rows - 1);  // last valid row of the item
  const int kend = w.P + r_last / geo.G + 1;              // keys [0, kend) reach some row
  w.nt = (kend + kKeys - 1) / kKeys;
}

// Read item k of the ring (every consumer thread); the caller releases the
// slot with one arrival per consumer warp on the even CTA's item_empty.
// Returns the item number, -1 at the end.
__device__ __forceinline__ int read_item2(Bars2& bar, uint32_t k, const Geom2& geo,
                                          uint32_t rank, Item2& w, volatile int* abortp,
                                          bool& ok) {
  // the message was written by the even CTA's producer: acquire at cluster scope
  ok = mbar_wait_cluster(&bar.item_full[k & 1], (k >> 1) & 1, abortp);
  if (!ok) return -1;
  const volatile int* m = bar.item_msg[k & 1];
  int mm[7];
#pragma unroll
  for (int i = 0; i < 7; ++i) mm[i] = m[i];
  if (mm[0] >= 0) item_from_message(mm, geo, rank, w);
  return mm[0];
}

// The same for a whole warp (every lane reads the item; the lanes agree).
__device__ __forceinline__ int read_item2_warp(Bars2& bar, uint32_t k, const Geom2& geo,
                                               uint32_t rank, Item2& w, volatile int* abortp,
                                               bool& ok) {
  const int it = read_item2(bar, k, geo, rank, w, abortp, ok);
  ok = __all_sync(0xffffffffu, ok);
  return it;
}

// A wait done by every lane of a warp: the lanes agree on the outcome, so a
// timeout seen by one lane alone cannot split the warp before a warp-wide
// (.sync.aligned) instruction.
__device__ __forceinline__ bool wait_warp(uint64_t* bar, uint32_t parity, volatile int* abortp) {
  const bool ok = mbar_wait(bar, parity, abortp);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void raise_abort(Bars2& bar, const Remote& rm) {
  *reinterpret_cast<volatile int*>(&bar.abort_flag) = 1;
  st_cluster_u32(rm.abort_peer, 1u);
}

// ----------------------------------------------------------------- producers
// Two producer warps per CTA: the K producer (this SM's Q half of each item
// and its 64-key half of every K tile, one 4-D box per page bringing both
// 64-column blocks) and the V producer (its 64-column half of every V tile,
// one 2-D box per page).  Each fills its own ring of 16 KB slots, so that
// neither waits behind the other's slot releases, and the two issue their
// copies in parallel (a copy instruction costs its warp tens of cycles per
// box, and 16-token pages need many boxes).
//
// Both CTAs' copies for a ring slot (or a Q buffer) complete on the even
// CTA's full barrier: each producer arrives there once per use with the bytes
// of its own copies (arrive.expect_tx) and issues them with pair completion,
// so the phase ends once both halves have landed and no copy has to be
// watched and reported (watching and reporting every landed copy made the V
// producer the slowest stage of the pipeline).  The exception is a V step
// that ends before 128 keys (an item's last): its rows past the end must be
// zeroed once they have landed (their P is 0, but 0 * NaN is NaN), so that
// copy completes on this CTA's own landed barrier, the producer waits for it,
// zeroes the rows and then arrives on the full barrier.
template <bool kIsK>
struct Producer {
  uint8_t* ring;         // kRing slots of 16 KB
  uint64_t* landed;      // this CTA's landed barriers of the ring (partial V steps)
  uint64_t* empty;
  uint32_t full_cl;      // shared::cluster address of the even CTA's full barrier 0
  volatile int* abortp;
  int lane;
  uint32_t issued = 0;   // ring uses issued
  uint32_t lphase = 0;   // per slot: parity of the slot's next landed phase

  // bounded wait of the whole warp (the lanes agree on the outcome)
  __device__ __forceinline__ bool wait(uint64_t* b, uint32_t parity) {
    return wait_warp(b, parity, abortp);
  }

  // Copies still in flight when the kernel gives up land before the CTA exits:
  // their completion goes to the even CTA's barriers, so wait out a time far
  // above a copy's latency (about 60 us).
  __device__ void drain() {
    const long long t0 = clock64();
    while (clock64() - t0 < (1ll << 17)) {
    }
  }
};

template <bool kIsK>
__device__ void producer2(uint32_t rank, uint8_t* smem_q, uint8_t* smem_ring, Bars2& bar,
                          const Remote& rm, const int* item_start, int total_items,
                          const Geom2& geo, const CUtensorMap* map_q, const CUtensorMap* map_kv,
                          const int32_t* __restrict__ block_table,
                          const int32_t* __restrict__ prefix_lens,
                          const int32_t* __restrict__ new_lens,
                          const int32_t* __restrict__ cu_new_lens, int32_t* status,
                          int* work_counter) {
  const int lane = threadIdx.x & 31;
  Producer<kIsK> pr{smem_ring, kIsK ? bar.k_landed : bar.v_landed,
                    kIsK ? bar.k_empty : bar.v_empty, kIsK ? rm.k_full : rm.v_full,
                    &bar.abort_flag, lane};
  bool ok = true;
  // K: 64 keys of this CTA, one box (both column blocks) per box_rows keys;
  // V: 128 keys of column block `rank`, one box per box_rows keys
  const int nbox = kIsK ? (64 >> geo.box_shift) : (kKeys >> geo.box_shift);
  const uint32_t box_bytes = static_cast<uint32_t>(geo.box_rows) * (kIsK ? 256 : 128);
  const int pages_per_step = kKeys >> geo.ps_shift;
  const bool claims = kIsK && rank == 0;  // the even CTA's K producer claims the items

  for (uint32_t k = 0; ok; ++k) {
    const int s = k & 1;
    int it = -1;
    Item2 w;
    if (claims) {
      // claim the next item and send it, decoded, to every role of both CTAs
      ok = pr.wait(&bar.item_empty[s], ((k >> 1) & 1) ^ 1);
      if (!ok) break;
      int m[7];
      if (lane == 0) {
        it = atomicAdd(work_counter, 1);
        if (it >= total_items) it = -1;
        m[0] = it;
        if (it >= 0) item_message(it, item_start, geo, prefix_lens, new_lens, cu_new_lens, m);
#pragma unroll
        for (int i = 0; i < 7; ++i) {
          bar.item_msg[s][i] = m[i];
          st_cluster_u32(rm.item_msg + 32 * s + 4 * i, static_cast<uint32_t>(m[i]));
          if (it < 0) break;
        }
        mbar_arrive(&bar.item_full[s]);
        mbar_arrive_cluster(rm.item_full + 8 * s);
      }
      __syncwarp();
    } else {
      ok = pr.wait(&bar.item_full[s], (k >> 1) & 1);
      if (!ok) break;
    }
    {
      // read the message (the even CTA's producer wrote it: acquire at cluster scope)
      ok = mbar_wait_cluster(&bar.item_full[s], (k >> 1) & 1, &bar.abort_flag);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      const volatile int* mv = bar.item_msg[s];
      int mm[7];
#pragma unroll
      for (int i = 0; i < 7; ++i) mm[i] = mv[i];
      it = mm[0];
      if (it >= 0) item_from_message(mm, geo, rank, w);
      __syncwarp();
      if (!claims && lane == 0) mbar_arrive_cluster(rm.item_empty + 8 * s);
    }
    if (it < 0) break;
    if (kIsK) {
      // this CTA's Q half: 128 rows = 128/G tokens x G heads, two column blocks
      const int qb = k & 1;
      ok = pr.wait(&bar.q_empty[qb], ((k >> 1) & 1) ^ 1);
      if (!ok) break;
      if (lane == 0) {
        const uint32_t qf = rm.q_full + 8 * qb;
        mbar_arrive_expect_tx_remote(qf, kQBytes);
#pragma unroll
        for (int h = 0; h < 2; ++h)
          tma_load_3d_pair(smem_q + qb * kQBytes + h * (kRows * 128), map_q, qf, h * 64,
                           w.g * geo.G, w.cu + w.tok0);
      }
      __syncwarp();
    }
    // K/V steps.  Lane i holds the block-table entry of page i of a step
    // (-2: no such page before the end of the sequence); the next step's
    // entries are loaded while this step's copies are issued.
    const int64_t bt_row = static_cast<int64_t>(w.b) * geo.max_blocks;
    auto lookup = [&](int j) -> int {
      const int key = j * kKeys + lane * geo.ps;  // first key of page `lane` of step j
      if (lane >= pages_per_step || key >= w.T) return -2;
      const int blk = key >> geo.ps_shift;
      return blk < geo.max_blocks ? __ldg(block_table + bt_row + blk) : -1;
    };
    const int plane_row = (geo.layer * 2 + (kIsK ? 0 : 1)) * geo.num_pages;
    int pages = lookup(0);
    for (int j = 0; ok && j < w.nt; ++j) {
      const int key0 = j * kKeys;
      const int pages_next = j + 1 < w.nt ? lookup(j + 1) : -2;
      // box `lane`: first key ko of the box within the step
      const int ko = kIsK ? static_cast<int>(rank) * 64 + lane * geo.box_rows : lane * geo.box_rows;
      const int page = __shfl_sync(0xffffffffu, pages, min(ko >> geo.ps_shift, 31));
      int row = -1;
      if (lane < nbox && page != -2 && key0 + ko < w.T) {
        if (page < 0 || page >= geo.num_pages) {
          record_error(status, GC_ERR_OUT_OF_RANGE);
        } else {
          row = (((plane_row + page) * geo.Hkv + w.g) << geo.ps_shift) +
                ((key0 + ko) & (geo.ps - 1));
        }
      }
      const int good = __popc(__ballot_sync(0xffffffffu, row >= 0));
      const uint32_t x = pr.issued, slot = x % kRing;
      ok = pr.wait(&pr.empty[slot], ((x / kRing) & 1) ^ 1);
      if (!ok) break;
      const uint32_t full = pr.full_cl + 8 * slot;
      const uint32_t bytes = static_cast<uint32_t>(good) * box_bytes;
      uint8_t* dst = smem_ring + slot * kSlotBytes + lane * box_bytes;
      const int nkeys = min(kKeys, w.T - key0);
      if (kIsK || nkeys == kKeys) {
        if (lane == 0) mbar_arrive_expect_tx_remote(full, bytes);
        __syncwarp();
        if (row >= 0) {
          if (kIsK)
            tma_load_4d_pair(dst, map_kv, full, 0, 0, 0, row >> 3);
          else
            tma_load_2d_pair(dst, map_kv, full, static_cast<int>(rank) * 64, row);
        }
      } else {
        // an item's last V step: land here, zero the rows past the end, report
        const uint32_t par = (pr.lphase >> slot) & 1u;
        pr.lphase ^= 1u << slot;
        if (lane == 0) mbar_arrive_expect_tx(&pr.landed[slot], bytes);
        __syncwarp();
        if (row >= 0) tma_load_2d(dst, map_kv, &pr.landed[slot], static_cast<int>(rank) * 64, row);
        ok = pr.wait(&pr.landed[slot], par);
        if (!ok) break;
        uint4* z = reinterpret_cast<uint4*>(smem_ring + slot * kSlotBytes + nkeys * 128);
        for (int e = lane; e < (kKeys - nkeys) * 8; e += 32) z[e] = make_uint4(0, 0, 0, 0);
        fence_proxy_async_smem();
        __syncwarp();
        // the zeroed rows are generic-proxy writes the other SM's tensor core
        // reads: publish them at cluster scope
        if (lane == 0) mbar_arrive_cluster(full);
      }
      ++pr.issued;
      pages = pages_next;
    }
  }
  if (!ok) pr.drain();
}

// -------------------------------------------------------------- MMA issuers
// Two threads of the even CTA, in different warps, issue the pair's MMAs:
// one the S products, one the PV products.  Step t uses S buffer t mod 3:
// S(t) writes it, the softmax reads it and writes P(t) over it, PV(t) reads
// P(t) from it.  Operand descriptors are built once per tile and advanced by
// constant offsets.
//
// S issuer: S(t) once K(t) is in and PV(t-3) is done (the buffer's last
// reader), so S runs up to two steps ahead of the softmax and the softmax
// never waits for a P buffer.  Frees the Q buffer by a commit after the
// item's last S product (the softmax frees the K slots).
__device__ void s_issuer2(uint8_t* smem_q, uint8_t* smem_k, Bars2& bar, const Remote& rm,
                          uint32_t tmem, const Geom2& geo) {
  volatile int* abortp = &bar.abort_flag;
  const uint32_t q_smem = smem_addr(smem_q), k_smem = smem_addr(smem_k);
  uint32_t u = 0;  // global step counter
  bool ok = true;
  for (uint32_t k = 0; ok; ++k) {
    Item2 w;
    const int it = read_item2(bar, k, geo, 0, w, abortp, ok);
    if (!ok) break;
    mbar_arrive_cluster(rm.item_empty + 8 * (k & 1));
    if (it < 0) break;
    const int qb = k & 1;
    ok = mbar_wait(&bar.q_full[qb], (k >> 1) & 1, abortp);
    if (!ok) break;
    const uint64_t dq = sdesc_sw128(q_smem + qb * kQBytes, 16, 1024);
    const uint32_t u_last = u + w.nt - 1;
    for (; ok && u <= u_last; ++u) {
      const uint32_t sb = u % kSBufs;
      const uint32_t slot = u % kRing;
      ok = mbar_wait(&bar.k_full[slot], (u / kRing) & 1, abortp);
      if (ok && u >= kSBufs)
        ok = mbar_wait(&bar.pv_done[sb], ((u - kSBufs) / kSBufs) & 1, abortp);
      if (!ok) break;
      tc_fence_after();
      // K half: 8-key groups of 2 KB (the group's 8 rows of columns 0-63,
      // then of columns 64-127), so 8-row groups are 2048 bytes apart
      const uint64_t dk = sdesc_sw128(k_smem + slot * kSlotBytes, 16, 2048);
      const uint32_t d = tmem + kColS + sb * 128;
#pragma unroll
      for (int kk = 0; kk < kD / 16; ++kk) {
        // 16-column steps: 32 bytes within a 128-byte row, then the next
        // 64-column block (Q: 16 KB further, K: 1 KB further)
        constexpr uint32_t kQBlk = kRows * 128 >> 4, kKBlk = 1024 >> 4;
        mma2_ss(d, dq + ((kk >> 2) * kQBlk + (kk & 3) * 2), dk + ((kk >> 2) * kKBlk + (kk & 3) * 2),
                kIdescQK, kk > 0);
      }
      mma2_commit_mc(&bar.s_full[sb], 0x3);
      if (u == u_last) mma2_commit_mc(&bar.q_empty[qb], 0x3);
    }
  }
  // every MMA this thread issued must be complete before tensor memory is freed
  mma2_commit_mc(&bar.drain, 0x1);
  int no_abort = 0;
  mbar_wait(&bar.drain, 0, &no_abort);
}

// PV issuer: O += P(t) V(t) once the softmax has written P(t) and V(t) is
// in; an item's first product (which overwrites O) also waits until the
// previous item's epilogue has read O.  Its commits tell both CTAs when the
// S buffer and the V slot have been read.
__device__ void pv_issuer2(uint8_t* smem_v, Bars2& bar, const Remote& rm, uint32_t tmem,
                           const Geom2& geo) {
  volatile int* abortp = &bar.abort_flag;
  const uint32_t v_smem = smem_addr(smem_v);
  uint32_t u = 0;  // global step counter
  bool ok = true;
  for (uint32_t k = 0; ok; ++k) {
    Item2 w;
    const int it = read_item2(bar, k, geo, 0, w, abortp, ok);
    if (!ok) break;
    mbar_arrive_cluster(rm.item_empty + 8 * (k & 1));
    if (it < 0) break;
    const uint32_t u_first = u, u_last = u + w.nt - 1;
    for (; ok && u <= u_last; ++u) {
      const uint32_t pb = u % kSBufs;
      const uint32_t slot = u % kRing;
      ok = mbar_wait(&bar.p_full[pb], (u / kSBufs) & 1, abortp);
      if (ok) ok = mbar_wait(&bar.v_full[slot], (u / kRing) & 1, abortp);
      const bool first = u == u_first;
      if (ok && first && k > 0) ok = mbar_wait(&bar.o_free, (k - 1) & 1, abortp);
      if (!ok) break;
      tc_fence_after();
      const uint64_t dv = sdesc_sw128(v_smem + slot * kSlotBytes, kSlotBytes, 1024);
      // P of keys [0, 64) at the buffer's column 0, of keys [64, 128) at column
      // 64 (each half-row's own S columns); 16 keys = 8 packed columns
      const uint32_t a = tmem + kColS + pb * 128;
#pragma unroll
      for (int kk = 0; kk < kKeys / 16; ++kk)  // 16 keys = two 8-row groups of 1 KB
        mma2_ts(tmem + kColO, a + (kk >> 2) * 64 + (kk & 3) * 8, dv + kk * (2048 >> 4),
                kIdescPV, (!first || kk > 0) ? 1u : 0u);
      mma2_commit_mc(&bar.pv_done[pb], 0x3);
      mma2_commit_mc(&bar.v_empty[slot], 0x3);
    }
  }
  mma2_commit_mc(&bar.drain, 0x1);
  int no_abort = 0;
  mbar_wait(&bar.drain, 0, &no_abort);
}

// ------------------------------------------------------------------ softmax
// Half-row softmax: two warpgroups, warps 4-7 taking key columns [0, 64)
// and warps 8-11 columns [64, 128) of every row of this CTA (warps w and
// w + 4 share the tensor-memory lanes of quadrant w & 3).  Each thread
// exponentiates 64 scores per step, so a step's softmax takes about half the
// time; the two halves of a row agree on its reference max through a
// per-step exchange of their half-tile maxima in shared memory (one tagged
// 16-bit word per row and half, polled by the partner thread), and add
// their partial sums at the end.
constexpr float kRescaleLog2 = 56.f;  // a term above 2^56 against the reference max

// fp32 -> bf16 bits rounded toward +inf (finite and infinite inputs)
__device__ __forceinline__ uint16_t bf16_bits_ru(float x) {
  uint16_t r;
  asm("cvt.rp.bf16.f32 %0, %1;" : "=h"(r) : "f"(x));
  return r;
}

// bf16 bits -> 15-bit key, monotone in the value, rounded up: negative
// values map to ~b, the others to b | 0x8000 (an order-preserving 16-bit
// key), then half of it rounded up.  key15_to_f32 returns the value of the
// key, at or above the input.
__device__ __forceinline__ uint32_t bf16_key15_ru(uint16_t b) {
  const uint32_t k = (b & 0x8000u) ? (~static_cast<uint32_t>(b) & 0xffffu) : (b | 0x8000u);
  return min((k + 1) >> 1, 0x7fffu);
}

__device__ __forceinline__ float key15_to_f32(uint32_t k15) {
  const uint32_t k = k15 << 1;
  const uint32_t b = (k & 0x8000u) ? (k & 0x7fffu) : (~k & 0xffffu);
  return __uint_as_float(b << 16);
}


__device__ void softmax2h(uint32_t rank, Bars2& bar, const Remote& rm, uint32_t tmem,
                          uint16_t* xch, const int* item_start, const Geom2& geo,
                          const int32_t* __restrict__ prefix_lens,
                          const int32_t* __restrict__ new_lens,
                          const int32_t* __restrict__ cu_new_lens,
                          __nv_bfloat16* __restrict__ out) {
  volatile int* abortp = &bar.abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hw = (warp - 4) >> 2;          // which 64 key columns
  const int quad = warp & 3;
  const int r = quad * 32 + lane;          // q row of this CTA's half = tensor-memory lane
  const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quad * 32) << 16);
  uint32_t xn = 0;  // exchanges so far
  // The partner thread's 15-bit value (same row, other half).  Exchange n
  // writes one 16-bit word, value << 1 | phase with phase = (n >> 1) & 1,
  // into buffer n & 1 of this half, and polls (bounded) the partner's word
  // in the same buffer until it carries that phase: one store, no fence (an
  // aligned word cannot be seen half-written).  The word it replaces is
  // exchange n - 2's, of the other phase.  The partner cannot overwrite a
  // buffer before it is read: it writes exchange n + 2 only after reading
  // exchange n + 1, which this thread writes only once its poll for
  // exchange n has returned.  The words start with phase 1, which neither
  // buffer's first exchange (n = 0, 1) carries.
  auto exchange = [&](uint32_t v15, bool& good) -> uint32_t {
    const uint32_t xb = xn & 1, phase = (xn >> 1) & 1;
    volatile uint16_t* mine = xch + (xb * 2 + hw) * kRows + r;
    volatile uint16_t* theirs = xch + (xb * 2 + (hw ^ 1)) * kRows + r;
    *mine = static_cast<uint16_t>(v15 << 1 | phase);
    ++xn;
    uint32_t t = *theirs;
    bool ok_ = true;
    if ((t & 1u) != phase) {
      const long long t0 = clock64();
      do {
        if (*abortp || clock64() - t0 > kWaitCycles) {
          *abortp = 1;
          ok_ = false;
          break;
        }
        t = *theirs;
      } while ((t & 1u) != phase);
    }
    good = __all_sync(0xffffffffu, ok_);
    return t >> 1;
  };
  uint32_t u = 0;  // global step counter
  // One thread per CTA frees K slot u once it has seen S(u) complete (V slots
  // are freed by the PV issuer's commits).  When the softmax is at step u,
  // PV(u - 3) is complete (S(u) was issued after it), so waits on
  // pv_done for PV(u - 1) or PV(u - 2) cannot see a stale phase.
  const bool rel = warp == 4 && lane == 0;
  bool ok = true;
  for (uint32_t k = 0; ok; ++k) {
    Item2 w;
    const int it = read_item2_warp(bar, k, geo, rank, w, abortp, ok);
    if (!ok) break;
    __syncwarp();
    if (lane == 0) mbar_arrive_cluster(rm.item_empty + 8 * (k & 1));
    if (it < 0) break;
    const int tok = w.tok0 + r / geo.G;
    const bool row_valid = tok < w.n;
    const int kmax = row_valid ? w.P + tok : w.T - 1;  // last visible key
    float m_run = -INFINITY, l = 0.f;
    const float sl2 = geo.scale_log2;
    for (int j = 0; j < w.nt; ++j, ++u) {
      const uint32_t sb = u % kSBufs;
      const uint32_t tS = lane_addr + kColS + sb * 128 + hw * 64;
      const uint32_t tP = tS;  // P over this half's scores, once they are in registers
      ok = wait_warp(&bar.s_full[sb], (u / kSBufs) & 1, abortp);
      if (!ok) break;
      if (rel) mbar_arrive(&bar.k_empty[u % kRing]);
      tc_fence_after();
      uint32_t sr[2][32];
      tmem_ld32(tS, sr[0]);
      tmem_ld32(tS + 32, sr[1]);
      tmem_wait_ld();
      const int key0 = j * kKeys + hw * 64;
      if (key0 + 63 > kmax) {
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (key0 + c * 32 + e > kmax) sr[c][e] = __float_as_uint(-INFINITY);
      }
      float mh[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};  // four short chains
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int e = 0; e < 32; e += 8)
#pragma unroll
          for (int x = 0; x < 4; ++x)
            mh[x] = fmax3(mh[x], __uint_as_float(sr[c][e + 2 * x]),
                          __uint_as_float(sr[c][e + 2 * x + 1]));
      // this half's max, rounded up to bf16 and then to a 15-bit key; both
      // halves of the row then take the max of the same two rounded values,
      // a reference at or above the row's true tile max
      const uint32_t mh_key =
          bf16_key15_ru(bf16_bits_ru(fmaxf(fmaxf(mh[0], mh[1]), fmaxf(mh[2], mh[3]))));
      const uint32_t mo = exchange(mh_key, ok);
      if (!ok) break;
      const float mt = fmaxf(key15_to_f32(mh_key), key15_to_f32(mo)) * sl2;
      if (j == 0) {
        m_run = mt;  // first tile of the row: exact max (key 0 is always visible)
      } else if (__any_sync(0xffffffffu, mt - m_run > kRescaleLog2)) {
        // O must hold every earlier step before it is rescaled; both halves of
        // each row take the same decision from the same two maxima
        ok = wait_warp(&bar.pv_done[(u - 1) % kSBufs], ((u - 1) / kSBufs) & 1, abortp);
        if (!ok) break;
        tc_fence_after();
        const float m_new = fmaxf(m_run, mt);
        const float alpha = m_new > m_run ? ex2_approx(m_run - m_new) : 1.f;
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          uint32_t o[32];
          const uint32_t tO = lane_addr + kColO + hw * 64 + c * 32;
          tmem_ld32(tO, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(tO, o);
        }
        l *= alpha;
        m_run = m_new;
      }
      {
        const uint64_t sc2 = f2_pack(sl2, sl2);
        const uint64_t nm2 = f2_pack(-m_run, -m_run);
        uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
        for (int c = 0; c < 2; ++c) {
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
          tmem_st16(tP + c * 16, pk);
        }
        float s0, s1, s2, s3;
        f2_unpack(f2_add(acc[0], acc[1]), s0, s1);
        f2_unpack(f2_add(acc[2], acc[3]), s2, s3);
        l += (s0 + s2) + (s1 + s3);
      }
      // publish this half of P(u)
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(rm.p_full + 8 * sb);
    }
    if (!ok) break;
    // ---- epilogue: O / l -> bf16 (this half's 64 columns), once the item's last PV is done
    // the partner's partial sum, 15 + 15 + 2 bits
    const uint32_t lb = __float_as_uint(l);
    const uint32_t l0 = exchange(lb >> 17, ok);
    if (!ok) break;
    const uint32_t l1 = exchange((lb >> 2) & 0x7fffu, ok);
    if (!ok) break;
    const uint32_t l2 = exchange(lb & 3u, ok);
    if (!ok) break;
    const float l_row = l + __uint_as_float(l0 << 17 | l1 << 2 | l2);
    const uint32_t ul = u - 1;
    ok = wait_warp(&bar.pv_done[ul % kSBufs], (ul / kSBufs) & 1, abortp);
    if (!ok) break;
    tc_fence_after();
    const int h = w.g * geo.G + r % geo.G;
    const float inv_l = 1.f / l_row;
    uint4* orow = reinterpret_cast<uint4*>(
        out + (static_cast<int64_t>(w.cu + tok) * geo.Hq + h) * kD + hw * 64);
#pragma unroll 1
    for (int c = 0; c < 2; ++c) {
      uint32_t o[32];
      tmem_ld32(lane_addr + kColO + hw * 64 + c * 32, o);
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
    // O may now be overwritten by the next item's first PV
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive_remote(rm.o_free);
  }
}

// ------------------------------------------------------------------- kernel
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc2_kernel(const __grid_constant__ CUtensorMap map_q,
                    const __grid_constant__ CUtensorMap map_k,
                    const __grid_constant__ CUtensorMap map_v,
                    const int32_t* __restrict__ block_table,
                    const int32_t* __restrict__ prefix_lens,
                    const int32_t* __restrict__ new_lens,
                    const int32_t* __restrict__ cu_new_lens, __nv_bfloat16* __restrict__ out,
                    Geom2 geo, int32_t* status, int* work_counter) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* smem_q = base;                     // 2 x 32 KB
  uint8_t* smem_k = base + 2 * kQBytes;       // K ring, kRing x 16 KB
  uint8_t* smem_v = smem_k + kRing * kSlotBytes;  // V ring
  Bars2& bar = *reinterpret_cast<Bars2*>(smem_v + kRing * kSlotBytes);
  int* item_start = reinterpret_cast<int*>(&bar + 1);  // [batch + 1]
  int16_t* order = reinterpret_cast<int16_t*>(item_start + geo.batch + 1);
  // half-row softmax exchange words [2 buffers][2 halves][128 rows]
  uint16_t* xch = reinterpret_cast<uint16_t*>(order + (geo.batch <= kSortMax ? kSortMax : 0));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bar.q_full[i], 2);
      mbar_init(&bar.q_empty[i], 1);
      mbar_init(&bar.item_full[i], 1);
      mbar_init(&bar.item_empty[i], kItemConsumers);
    }
    for (int i = 0; i < kSBufs; ++i) {
      mbar_init(&bar.s_full[i], 1);
      mbar_init(&bar.p_full[i], 2 * kSoftmaxWarps);
      mbar_init(&bar.pv_done[i], 1);
    }
    for (int s = 0; s < kRing; ++s) {
      mbar_init(&bar.k_landed[s], 1);
      mbar_init(&bar.k_full[s], 2);
      mbar_init(&bar.k_empty[s], 1);
      mbar_init(&bar.v_landed[s], 1);
      mbar_init(&bar.v_full[s], 2);
      mbar_init(&bar.v_empty[s], 1);
    }
    mbar_init(&bar.o_free, 2 * kSoftmaxWarps);
    mbar_init(&bar.drain, 2);
    bar.abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&map_q);
    prefetch_tensormap(&map_k);
    prefetch_tensormap(&map_v);
  }
  if (warp == 1) {
    tmem_alloc2(&bar.tmem_base, 512);
    tmem_relinquish2();
  }
  // exchange words start with phase 1 (no exchange has been written)
  for (int i = threadIdx.x; i < 2 * 2 * kRows; i += kThreads) xch[i] = 1;
  if (geo.batch <= kSortMax) {
    // rank requests by total length, longest first (ties by index)
    for (int b = threadIdx.x; b < geo.batch; b += kThreads) {
      const int tb = __ldg(prefix_lens + b) + __ldg(new_lens + b);
      int rk = 0;
      for (int o = 0; o < geo.batch; ++o) {
        const int to = __ldg(prefix_lens + o) + __ldg(new_lens + o);
        rk += (to > tb) || (to == tb && o < b);
      }
      order[rk] = static_cast<int16_t>(b);
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
      if (p < geo.batch) {
        const int n = __ldg(new_lens + b), P = __ldg(prefix_lens + b);
        const int cu = __ldg(cu_new_lens + b);
        const bool sane = n >= 0 && P >= 0 && cu >= 0 && cu + n <= geo.total_new;
        if (!sane && n != 0 && rank == 0) record_error(status, GC_ERR_OUT_OF_RANGE);
        if (sane && n > 0) cnt = geo.Hkv * ((n * geo.G + 2 * kRows - 1) / (2 * kRows));
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
  Remote rm;
  {
    const uint32_t lead = 0, peer = rank ^ 1u;
    rm.q_full = mapa(smem_addr(&bar.q_full[0]), lead);
    rm.k_full = mapa(smem_addr(&bar.k_full[0]), lead);
    rm.v_full = mapa(smem_addr(&bar.v_full[0]), lead);
    rm.p_full = mapa(smem_addr(&bar.p_full[0]), lead);
    rm.o_free = mapa(smem_addr(&bar.o_free), lead);
    rm.item_empty = mapa(smem_addr(&bar.item_empty[0]), lead);
    rm.item_full = mapa(smem_addr(&bar.item_full[0]), peer);
    rm.item_msg = mapa(smem_addr(&bar.item_msg[0][0]), peer);
    rm.abort_peer = mapa(smem_addr(&bar.abort_flag), peer);
  }
  tc_fence_before();
  // both CTAs' barriers are initialised before either CTA touches the other's
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem = bar.tmem_base;
  const int total_items = item_start[geo.batch];

  if (warp == 0) {
    producer2<true>(rank, smem_q, smem_k, bar, rm, item_start, total_items, geo, &map_q,
                    &map_k, block_table, prefix_lens, new_lens, cu_new_lens, status,
                    work_counter);
  } else if (warp == 1) {
    if (rank == 0 && lane == 0) s_issuer2(smem_q, smem_k, bar, rm, tmem, geo);
    __syncwarp();
  } else if (warp == 2) {
    if (rank == 0 && lane == 0) pv_issuer2(smem_v, bar, rm, tmem, geo);
    __syncwarp();
  } else if (warp == 3) {
    producer2<false>(rank, smem_q, smem_v, bar, rm, item_start, total_items, geo, &map_q,
                     &map_v, block_table, prefix_lens, new_lens, cu_new_lens, status,
                     work_counter);
  } else if (warp >= 4) {
    softmax2h(rank, bar, rm, tmem, xch, item_start, geo, prefix_lens, new_lens, cu_new_lens,
              out);
  }
  // a CTA that gave up tells its peer, so that the peer's roles leave their
  // loops instead of waiting for arrivals that will not come
  if (*reinterpret_cast<volatile int*>(&bar.abort_flag) && lane == 0) raise_abort(bar, rm);
  tc_fence_before();
  __syncthreads();
  // neither CTA leaves (or frees tensor memory) while the other may still
  // read its shared memory or arrive on its barriers
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc2(tmem, 512);
  }
  if (threadIdx.x == 0 && bar.abort_flag) record_error(status, GC_ERR_TIMEOUT);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn2() {
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

size_t smem_bytes2(int batch) {
  return 1024 + 2 * kQBytes + static_cast<size_t>(2 * kRing) * kSlotBytes + sizeof(Bars2) +
         (static_cast<size_t>(batch) + 1) * sizeof(int) +
         (batch <= kSortMax ? kSortMax * sizeof(int16_t) : 0) + 2 * 2 * kRows * sizeof(uint16_t);
}

}  // namespace

// Clusters of two that fit on the device at once with this kernel's shared
// memory (the persistent grid), 0 if the query fails.
int attn_tc2_pairs(const gc_kv_pool* pool, int batch) {
  const size_t smem = smem_bytes2(batch);
  if (cudaFuncSetAttribute(attn_tc2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(2 * (pool->num_sms / 2));
  lc.blockDim = dim3(kThreads);
  lc.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  lc.attrs = attr;
  lc.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, attn_tc2_kernel, &lc) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return clusters;
}

gc_status launch_attn_tc2(const gc_kv_pool* pool, const AttnArgs& a, cudaStream_t stream,
                          int* work_counter) {
  const auto& cfg = pool->cfg;
  if (cfg.head_dim != kD)
    return fail(GC_ERR_UNSUPPORTED, "gc_prefix_prefill_attn: pair kernel needs head_dim 128");
  const int pairs = attn_tc2_pairs(pool, a.batch);
  if (pairs <= 0)
    return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: no CTA pair fits on the device");
  gc_status bound = check_item_bound(pool, a, nullptr, 2 * pairs);
  if (bound != GC_OK) return bound;
  auto enc = encode_fn2();
  if (!enc) return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: cuTensorMapEncodeTiled unavailable");
  Geom2 geo;
  geo.batch = a.batch;
  geo.Hq = a.num_q_heads;
  geo.Hkv = cfg.num_kv_heads;
  geo.G = geo.Hq / geo.Hkv;
  geo.ps = cfg.page_size;
  int s = 0;
  while ((1 << s) < geo.ps) ++s;
  geo.ps_shift = s;
  geo.box_rows = geo.ps < 64 ? geo.ps : 64;
  s = 0;
  while ((1 << s) < geo.box_rows) ++s;
  geo.box_shift = s;
  geo.num_pages = cfg.num_pages;
  geo.max_blocks = a.max_blocks;
  geo.layer = a.layer;
  geo.total_new = a.total_new_tokens;
  geo.scale_log2 = a.softmax_scale * 1.4426950408889634f;

  const uint64_t pool_rows = static_cast<uint64_t>(cfg.num_layers) * 2 * cfg.num_pages *
                             cfg.num_kv_heads * cfg.page_size;
  if (pool_rows >= (1ull << 31))
    return fail(GC_ERR_UNSUPPORTED, "gc_prefix_prefill_attn: pool has %llu rows (limit 2^31)",
                static_cast<unsigned long long>(pool_rows));
  CUtensorMap map_q, map_k, map_v;
  {
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(geo.Hq),
                          static_cast<cuuint64_t>(geo.total_new)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(kD) * 2,
                             static_cast<cuuint64_t>(geo.Hq) * kD * 2};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(geo.G),
                         static_cast<cuuint32_t>(kRows / geo.G)};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = enc(&map_q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: q tensor map (CUresult %d)", (int)r);
  }
  {
    // K: 4-D view of the pool rows as (64 columns, 8 rows, 2 column blocks,
    // 8-row groups), one box per page (or per 64 keys of a 128-row page):
    // both column blocks of box_rows rows, laid out as 8-row groups of 2 KB
    cuuint64_t dims[4] = {64, 8, 2, pool_rows / 8};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(kD) * 2, 128,
                             8 * static_cast<cuuint64_t>(kD) * 2};
    cuuint32_t box[4] = {64, 8, 2, static_cast<cuuint32_t>(geo.box_rows / 8)};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = enc(&map_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, pool->data, dims, strides, box,
                     es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: pool K tensor map (CUresult %d)", (int)r);
  }
  {
    // V: 2-D view of the pool rows, one box of 64 columns x box_rows rows
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(kD), pool_rows};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(kD) * 2};
    cuuint32_t box[2] = {64, static_cast<cuuint32_t>(geo.box_rows)};
    cuuint32_t es[2] = {1, 1};
    CUresult r = enc(&map_v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pool->data, dims, strides, box,
                     es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(GC_ERR_CUDA, "gc_prefix_prefill_attn: pool V tensor map (CUresult %d)", (int)r);
  }
  const size_t smem = smem_bytes2(a.batch);
  // the work items are claimed from the given counter (the pool's control
  // block, or the static scratch of the allocation-free entry point)
  cudaError_t e = cudaMemsetAsync(work_counter, 0, sizeof(int), stream);
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn: clearing the work counter");
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(2 * pairs);
  lc.blockDim = dim3(kThreads);
  lc.dynamicSmemBytes = smem;
  lc.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  lc.attrs = attr;
  lc.numAttrs = 1;
  e = cudaLaunchKernelEx(&lc, attn_tc2_kernel, map_q, map_k, map_v, a.block_table, a.prefix_lens,
                         a.new_lens, a.cu_new_lens, static_cast<__nv_bfloat16*>(a.out), geo,
                         pool->status, work_counter);
  if (e != cudaSuccess) return cuda_fail(e, "gc_prefix_prefill_attn: launch");
  return GC_OK;
}

}  // namespace gc
