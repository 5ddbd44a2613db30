"""8-bit cache-tier inputs shared by the 8-bit attention tests."""
import numpy as np

import oracle


class Q8Case:
    """The 8-bit image of a workload's cached pages (made by the oracle's
    quantiser), the q8 table mapping each request's FULL prefix pages to it,
    and the partly cached last pages: those also receive the new tokens
    (gc_kv_append writes into them), so they are dequantised into the pool
    first, as a serving loop does before appending to a page."""

    def __init__(self, w, frac_in_image=1.0, seed=0):
        self.w = w
        self.ids = w.prefix_blocks()
        src_pool = w.empty_pool()
        if self.ids.size:
            oracle.kv_restore(src_pool, w.host_src(), self.ids)
        self.img = oracle.kv_save_q8(src_pool, self.ids)       # [n][L][2][chunk]
        self.table = np.full((w.B, w.max_blocks), -1, dtype=np.int32)
        rng = np.random.default_rng(seed)
        to_pool, off = [], 0
        for b in range(w.B):
            P = int(w.prefix_lens[b])
            nb, full = -(-P // w.ps), P // w.ps
            for j in range(nb):
                if j < full and rng.random() < frac_in_image:
                    self.table[b, j] = off + j
                else:
                    to_pool.append(off + j)   # image index of a page restored to the pool
            off += nb
        self.to_pool = np.asarray(to_pool, dtype=np.int64)

    def oracle_pool(self):
        w = self.w
        pool = w.empty_pool()
        if self.ids.size:
            oracle.kv_restore_q8(pool, self.img, self.ids)
        k, v = w.kv_new()
        for l in range(w.L):
            oracle.kv_append(pool, l, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
        return pool


def all_pages_case(w):
    """Every page of every request (the new tokens' too, the last one partly
    filled) in the 8-bit image, made by the oracle from the pool after the
    append; returns (image, block ids, q8 table, oracle pool)."""
    pool = w.empty_pool()
    if w.prefix_blocks().size:
        oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    table = np.full((w.B, w.max_blocks), -1, dtype=np.int32)
    ids = []
    for b in range(w.B):
        nb = -(-int(w.total_lens[b]) // w.ps)
        table[b, :nb] = np.arange(len(ids), len(ids) + nb)
        ids.extend(w.block_table[b, :nb].tolist())
    ids = np.asarray(ids, dtype=np.int32)
    img = oracle.kv_save_q8(pool, ids)
    ref_pool = w.empty_pool()
    oracle.kv_restore_q8(ref_pool, img, ids)
    return img, ids, table, ref_pool
