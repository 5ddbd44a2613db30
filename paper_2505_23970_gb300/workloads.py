"""Seeded synthetic inputs for prefix-reuse prefill.

This module only draws inputs; it holds none of the method's arithmetic, so
both the float64 oracle and the CUDA path can be fed from it.  Everything is
drawn from numpy's PCG64 (``default_rng([seed, stream])``, one stream per
tensor so that any tensor can be drawn on its own).

The workloads stand in for the paper's serving traffic (Sec. 3.1.1: ShareGPT
multi-turn prompts, 77.2 % with more than 1000 context tokens; TriviaQA
documents with a mean context of 5880 tokens; Sec. 6.1: Llama-3 8B and 70B).
None of those datasets is used: only their shapes and length statistics.

bf16 tensors are numpy ``uint16`` arrays of bit patterns (round to nearest
even from float32).  Layouts:

* q            [T_new][Hq][d]
* k_new, v_new [T_new][Hkv][d]
* host_src     [n_blocks][L][2][Hkv][ps][d]  (cached pages, prefix order)
* pool         [L][2][num_pages][Hkv][ps][d]
* block_table  [B][max_blocks] int32, -1 past a request's last page
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

BF16_NAN = np.uint16(0x7FC0)

# stream ids for default_rng([seed, stream])
_S_LENS, _S_PERM, _S_Q, _S_KP, _S_KN, _S_HIT = 1, 2, 3, 4, 5, 6


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    x = np.asarray(x, dtype=np.float32)
    u = np.ascontiguousarray(x).reshape(-1).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16).reshape(x.shape)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    b = np.asarray(b, dtype=np.uint16)
    u = np.ascontiguousarray(b).reshape(-1).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).reshape(b.shape)


def normal_bf16(seed: int, stream: int, shape) -> np.ndarray:
    rng = np.random.default_rng([seed, stream])
    return f32_to_bf16_bits(rng.standard_normal(size=shape, dtype=np.float32))


@dataclass
class Workload:
    """One batch of requests over one pool.  Lengths are int32 arrays."""
    name: str
    B: int
    Hq: int
    Hkv: int
    d: int
    ps: int
    L: int
    prefix_lens: np.ndarray
    new_lens: np.ndarray
    num_pages: int
    block_table: np.ndarray
    seed: int
    layer: int = 0
    note: str = ""
    _cache: dict = field(default_factory=dict, repr=False)

    # ----------------------------------------------------------- derived sizes
    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.d)

    @property
    def total_lens(self) -> np.ndarray:
        return (self.prefix_lens + self.new_lens).astype(np.int32)

    @property
    def cu_new_lens(self) -> np.ndarray:
        cu = np.zeros(self.B + 1, dtype=np.int32)
        cu[1:] = np.cumsum(self.new_lens)
        return cu

    @property
    def T_new(self) -> int:
        return int(self.new_lens.sum())

    @property
    def max_blocks(self) -> int:
        return int(self.block_table.shape[1])

    @property
    def page_bytes(self) -> int:
        """Bytes of one cached block across all layers and both planes."""
        return self.L * 2 * self.Hkv * self.ps * self.d * 2

    @property
    def pool_shape(self):
        return (self.L, 2, self.num_pages, self.Hkv, self.ps, self.d)

    def prefix_blocks(self) -> np.ndarray:
        """Pool pages that hold cached prefix tokens, request by request."""
        ids = []
        for b in range(self.B):
            nb = -(-int(self.prefix_lens[b]) // self.ps)
            ids.extend(self.block_table[b, :nb].tolist())
        return np.asarray(ids, dtype=np.int32)

    def attn_flops(self) -> float:
        """Causal attention FLOPs of the new rows: 4*d*Hq*sum(n*P + n(n+1)/2)."""
        P = self.prefix_lens.astype(np.float64)
        n = self.new_lens.astype(np.float64)
        return float(4.0 * self.d * self.Hq * np.sum(n * P + n * (n + 1) / 2))

    # --------------------------------------------------------------- tensors
    def q(self) -> np.ndarray:
        if "q" not in self._cache:
            self._cache["q"] = normal_bf16(self.seed, _S_Q, (self.T_new, self.Hq, self.d))
        return self._cache["q"]

    def kv_new(self):
        if "kvn" not in self._cache:
            kv = normal_bf16(self.seed, _S_KN, (2, self.T_new, self.Hkv, self.d))
            self._cache["kvn"] = (kv[0], kv[1])
        return self._cache["kvn"]

    def host_src(self) -> np.ndarray:
        """Cached prefix pages [n_blocks][L][2][Hkv][ps][d].  Slots past a
        request's prefix in its last page hold NaN: a reader that uses them
        instead of masking them shows up in every comparison."""
        if "src" not in self._cache:
            ids = self.prefix_blocks()
            src = normal_bf16(self.seed, _S_KP,
                              (ids.size, self.L, 2, self.Hkv, self.ps, self.d))
            blk = 0
            for b in range(self.B):
                P = int(self.prefix_lens[b])
                nb = -(-P // self.ps)
                if nb and P % self.ps:
                    src[blk + nb - 1, :, :, :, P % self.ps:, :] = BF16_NAN
                blk += nb
            self._cache["src"] = src
        return self._cache["src"]

    def empty_pool(self, fill=BF16_NAN) -> np.ndarray:
        return np.full(self.pool_shape, fill, dtype=np.uint16)

    def drop_tensors(self) -> None:
        self._cache.clear()

    def dense_request(self, pool: np.ndarray, b: int, layer: int = 0):
        """K, V [T_b][Hkv][d] of request b read out of a pool by page (input
        plumbing for the dense second path; no arithmetic)."""
        T = int(self.total_lens[b])
        ids = self.block_table[b, :-(-T // self.ps)]
        k = pool[layer, 0, ids].transpose(0, 2, 1, 3).reshape(-1, self.Hkv, self.d)[:T]
        v = pool[layer, 1, ids].transpose(0, 2, 1, 3).reshape(-1, self.Hkv, self.d)[:T]
        return np.ascontiguousarray(k), np.ascontiguousarray(v)


def make_block_table(seed: int, total_lens: np.ndarray, ps: int, num_pages: int) -> np.ndarray:
    """Each request gets ceil(T_b/ps) pages taken in order from a random
    permutation of the pool; unused entries are -1."""
    need = [-(-int(t) // ps) for t in total_lens]
    if sum(need) > num_pages:
        raise ValueError(f"pool of {num_pages} pages too small for {sum(need)}")
    perm = np.random.default_rng([seed, _S_PERM]).permutation(num_pages).astype(np.int32)
    mb = max(max(need) if need else 1, 1)
    bt = np.full((len(need), mb), -1, dtype=np.int32)
    off = 0
    for b, nb in enumerate(need):
        bt[b, :nb] = perm[off:off + nb]
        off += nb
    return bt


def _mk(name, B, Hq, Hkv, d, ps, P, n, seed, L=1, num_pages=None, pool_factor=1.25, note=""):
    P = np.asarray(P, dtype=np.int32).reshape(B)
    n = np.asarray(n, dtype=np.int32).reshape(B)
    T = P + n
    if num_pages is None:
        num_pages = max(1, math.ceil(pool_factor * int(T.sum()) / ps))
        num_pages = max(num_pages, sum(-(-int(t) // ps) for t in T))
    bt = make_block_table(seed, T, ps, num_pages)
    return Workload(name, B, Hq, Hkv, d, ps, L, P, n, num_pages, bt, seed, note=note)


# ------------------------------------------------------------------ configs
def tiny(seed: int = 0) -> Workload:
    """1 request, GQA 4:1, d 64, cached prefix 256, 64 new tokens, ps 16,
    its 20 pages scattered in a 64-page pool."""
    return _mk("tiny", 1, 4, 1, 64, 16, [256], [64], seed, num_pages=64)


def llama3_8b_layer(seed: int = 0, B: int = 16) -> Workload:
    """Llama-3-8B-shaped layer: 32 q heads / 8 kv heads, d 128, prefix
    lengths uniform in [512, 4096], new lengths uniform in [128, 512]."""
    rng = np.random.default_rng([seed, _S_LENS])
    P = rng.integers(512, 4096, size=B, endpoint=True)
    n = rng.integers(128, 512, size=B, endpoint=True)
    return _mk("llama3-8b-layer", B, 32, 8, 128, 16, P, n, seed)


def llama3_70b_layer(seed: int = 0, B: int = 8, prefix: int = 8192, new: int = 1024) -> Workload:
    """Llama-3-70B-shaped layer: 64 q heads / 8 kv heads, d 128, B requests
    with an 8192-token cached prefix and 1024 new tokens each."""
    return _mk("llama3-70b-layer", B, 64, 8, 128, 16, [prefix] * B, [new] * B, seed)


def llama3_70b_restore_80layer(seed: int = 0, prefix: int = 8192) -> Workload:
    """Full 80-layer KV of one cached 8192-token prefix (restore only)."""
    w = _mk("llama3-70b-80layer-restore", 1, 64, 8, 128, 16, [prefix], [0], seed,
            pool_factor=1.25)
    w.L = 80
    return w


def llama3_70b_80layer_prefill(seed: int = 0, prefix: int = 8192, new: int = 1024,
                               recompute: bool = False, B: int = 1) -> Workload:
    """All 80 layers of the 70B-shaped model for B requests with an
    8192-token cached prefix and 1024 new tokens each (restore of every
    layer's cached pages + append + attention); recompute=True gives the
    same context prefilled from scratch (prefix 0, prefix + new tokens)."""
    if recompute:
        w = _mk("llama3-70b-80layer-recompute", B, 64, 8, 128, 16, [0] * B, [prefix + new] * B,
                seed)
    else:
        w = _mk("llama3-70b-80layer-prefill", B, 64, 8, 128, 16, [prefix] * B, [new] * B, seed)
    w.L = 80
    return w


def llama3_70b_decode(seed: int = 0, B: int = 8, context: int = 9216) -> Workload:
    """Decode step on the 70B-shaped layer: B requests whose context of
    `context` tokens (the 8192 + 1024 of the 70B prefill config) ends with the
    new token: cached prefix context - 1, one new token each."""
    return _mk("llama3-70b-decode", B, 64, 8, 128, 16, [context - 1] * B, [1] * B, seed)


def decode_mix(seed: int = 0, B: int = 64) -> Workload:
    """Decode step after the multi-turn mix: contexts = prefix + suffix of
    the conversation mix (p = 1), one new token each."""
    rng = np.random.default_rng([seed, _S_LENS])
    P = np.clip(np.rint(rng.lognormal(math.log(2048), 1.0, size=B)), 0, 32768).astype(np.int64)
    S = np.clip(np.rint(rng.lognormal(math.log(200), 0.8, size=B)), 16, 4096).astype(np.int64)
    return _mk("decode-mix", B, 64, 8, 128, 16, P + S - 1, [1] * B, seed)


def conversation_mix(seed: int = 0, hit_p: float = 1.0, B: int = 64) -> Workload:
    """Multi-turn mix on the 70B-shaped layer: prefix ~ LogNormal(ln 2048, 1.0)
    clipped to [0, 32768], new ~ LogNormal(ln 200, 0.8) clipped to
    [16, 4096], cache hit ~ Bernoulli(hit_p); a miss prefills the whole
    context as new tokens (prefix 0)."""
    rng = np.random.default_rng([seed, _S_LENS])
    P = np.clip(np.rint(rng.lognormal(math.log(2048), 1.0, size=B)), 0, 32768).astype(np.int64)
    S = np.clip(np.rint(rng.lognormal(math.log(200), 0.8, size=B)), 16, 4096).astype(np.int64)
    hit = np.random.default_rng([seed, _S_HIT]).random(B) < hit_p
    prefix = np.where(hit, P, 0)
    new = np.where(hit, S, P + S)
    return _mk(f"conversation-mix-p{hit_p:g}", B, 64, 8, 128, 16, prefix, new, seed)


def long_document(seed: int = 0, recompute: bool = False, B: int = 2,
                  prefix: int = 131072, new: int = 2048) -> Workload:
    """Long-document reuse on the 70B-shaped layer: 131072-token cached
    prefix + 2048 new tokens, ps 64; recompute=True gives the same context
    prefilled from scratch (prefix 0, 133120 new tokens)."""
    if recompute:
        return _mk("long-document-recompute", B, 64, 8, 128, 64, [0] * B, [prefix + new] * B, seed)
    return _mk("long-document", B, 64, 8, 128, 64, [prefix] * B, [new] * B, seed)


def custom(name, B, Hq, Hkv, d, ps, prefix_lens, new_lens, seed=0, num_pages=None,
           pool_factor=1.25) -> Workload:
    return _mk(name, B, Hq, Hkv, d, ps, prefix_lens, new_lens, seed, num_pages=num_pages,
               pool_factor=pool_factor)


CONFIGS = {
    "tiny": tiny,
    "8b": llama3_8b_layer,
    "70b": llama3_70b_layer,
    "mix": conversation_mix,
    "long": long_document,
    "decode": llama3_70b_decode,
    "decode-mix": decode_mix,
}
