"""Pins of the float64 oracle against what the paper and the mathematics fix.

None of these compares the oracle with a retyped copy of itself: each case is
a closed form, an invariant, a brute-force enumeration, a second independent
code path (dense, unpaged attention) or a number printed in the paper.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2505_23970_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf(x):
    """Exactly representable float values -> bf16 bit patterns."""
    out = wl.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))
    assert np.array_equal(wl.bf16_bits_to_f32(out), np.asarray(x, dtype=np.float32)), x
    return out


# ------------------------------------------------------------------ bf16
@pytest.mark.parametrize("bits,value", [
    (0x3F80, 1.0), (0xC000, -2.0), (0x3FC0, 1.5), (0x4049, 3.140625),
    (0x0001, 2.0 ** -133), (0x8000, -0.0), (0x7F80, math.inf), (0x3C00, 2.0 ** -7),
])
def test_bf16_widening_is_exact(bits, value):
    got = oracle.bf16_to_double(bits)
    assert got == value and math.copysign(1, got) == math.copysign(1, value)


# --------------------------------------------------------------- restore
def _tagged(shape, base=1):
    """Distinct small integers (exact in bf16 up to 256) would run out, so
    tags are written as raw uint16 bit patterns: the copy is bitwise."""
    n = int(np.prod(shape))
    assert n + base < 0x7F80
    return (np.arange(n, dtype=np.uint16) + np.uint16(base)).reshape(shape)


def test_restore_roundtrip_and_untouched_pages():
    L, Hkv, ps, d, NP = 3, 2, 4, 5, 11
    ids = np.array([7, 2, 9, 0], dtype=np.int32)
    src = _tagged((ids.size, L, 2, Hkv, ps, d))
    pool = np.full((L, 2, NP, Hkv, ps, d), 0x7FC0, dtype=np.uint16)
    oracle.kv_restore(pool, src, ids)
    assert np.array_equal(oracle.kv_gather_blocks(pool, ids), src)
    untouched = sorted(set(range(NP)) - set(ids.tolist()))
    assert np.all(pool[:, :, untouched] == 0x7FC0)


@pytest.mark.parametrize("ps", [1, 2, 4])
def test_restore_bruteforce_every_permutation(ps):
    """Every placement of 4 cached blocks into a 4-page pool: each pool
    element decodes back to the (block, layer, plane, head, slot, dim) that
    must land there."""
    L, Hkv, d = 2, 2, 3
    shape = (4, L, 2, Hkv, ps, d)
    src = _tagged(shape)
    for perm in itertools.permutations(range(4)):
        ids = np.asarray(perm, dtype=np.int32)
        pool = np.zeros((L, 2, 4, Hkv, ps, d), dtype=np.uint16)
        oracle.kv_restore(pool, src, ids)
        for (l, kv, page, g, s, c) in np.ndindex(pool.shape):
            i = perm.index(page)
            flat = np.ravel_multi_index((i, l, kv, g, s, c), shape)
            assert pool[l, kv, page, g, s, c] == flat + 1


def test_restore_rejects_out_of_range_block():
    pool = np.zeros((1, 2, 4, 1, 2, 2), dtype=np.uint16)
    src = np.zeros((1, 1, 2, 1, 2, 2), dtype=np.uint16)
    with pytest.raises(oracle.OracleError):
        oracle.kv_restore(pool, src, [4])
    with pytest.raises(oracle.OracleError):
        oracle.kv_restore(pool, src, [-1])


def test_kv_bytes_per_token_matches_paper():
    """Sec. 2.2 prints > 300 TB for a 1000-token context cached for 1 M
    prompts of Llama-3 70B.  The restore image of one page of the
    80-layer 70B-shaped workload must give that size per token (327,680 B)."""
    g = json.load(open(os.path.join(GOLDEN, "kv_bytes_per_token.json")))
    w = wl.llama3_70b_restore_80layer()
    per_token = w.page_bytes // w.ps
    assert per_token == 327_680
    total = per_token * g["context_tokens"] * g["prompts"]
    assert total > g["min_total_bytes"]
    # same order as the printed figure: a doubled byte count would be 655 TB
    assert total < 1.5 * g["min_total_bytes"]


# ---------------------------------------------------------------- append
@pytest.mark.parametrize("prefix", [[0, 5], [8, 3], [7, 0]])
def test_append_places_each_token_after_its_prefix(prefix):
    """Each new value carries a tag; after the append the tag must sit at
    absolute position prefix_len + t of its own request, and nothing else
    in the pool may change."""
    ps, Hkv, d, L, layer = 4, 2, 3, 2, 1
    new = [6, 2]
    w = wl.custom("t", 2, 2, Hkv, d, ps, prefix, new, seed=3, num_pages=12)
    k = _tagged((w.T_new, Hkv, d), base=1)
    v = _tagged((w.T_new, Hkv, d), base=1 + k.size)
    pool = np.zeros((L, 2, w.num_pages, Hkv, ps, d), dtype=np.uint16)
    oracle.kv_append(pool, layer, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    expect = np.zeros_like(pool)
    cu = w.cu_new_lens
    for b in range(2):
        for t in range(new[b]):
            pos = prefix[b] + t
            page = w.block_table[b, pos // ps]
            expect[layer, 0, page, :, pos % ps, :] = k[cu[b] + t]
            expect[layer, 1, page, :, pos % ps, :] = v[cu[b] + t]
    assert np.array_equal(pool, expect)


# ------------------------------------------------------------- attention
def _one_request_pool(K, V, ps, perm_seed=0, extra_pages=3):
    """Lay dense K, V [T][Hkv][d] (bf16 bits) into a permuted pool; slots
    past T hold NaN."""
    T, Hkv, d = K.shape
    nb = -(-T // ps)
    NP = nb + extra_pages
    rng = np.random.default_rng(perm_seed)
    pages = rng.permutation(NP)[:nb].astype(np.int32)
    pool = np.full((1, 2, NP, Hkv, ps, d), 0x7FC0, dtype=np.uint16)
    for j in range(T):
        pool[0, 0, pages[j // ps], :, j % ps, :] = K[j]
        pool[0, 1, pages[j // ps], :, j % ps, :] = V[j]
    return pool, pages.reshape(1, nb)


def test_two_key_closed_form():
    """Scores {0, ln 3} give weights {1/4, 3/4}: out = (v0 + 3 v1) / 4."""
    q = bf([[[1.0, 0.0]]])                      # one new row, one head
    K = bf([[[0.0, 0.0]], [[1.0, 0.0]]])
    V = bf([[[4.0, 0.0]], [[0.0, 8.0]]])
    pool, bt = _one_request_pool(K, V, ps=1)
    w, o = oracle.prefix_attn_row_weights(q, pool, 0, bt, [1], [0, 1], math.log(3.0), 0, 0, 0)
    assert np.allclose(w, [0.25, 0.75], rtol=0, atol=1e-15)
    assert np.allclose(o, [1.0, 6.0], rtol=0, atol=1e-14)
    full = oracle.prefix_attn(q, pool, 0, bt, [1], [0, 1], math.log(3.0))
    assert np.allclose(full[0, 0], [1.0, 6.0], rtol=0, atol=1e-14)


def test_weights_follow_exp_of_scores():
    """Integer scores s_j = j (scale 1): w_j / w_0 = e^j and sum w = 1."""
    T = 6
    q = bf([[[1.0, 0.0, 0.0, 0.0]]])
    K = bf([[[float(j), 0.0, 0.0, 0.0]] for j in range(T)])
    V = bf(np.random.default_rng(1).integers(-4, 5, size=(T, 1, 4)).astype(np.float32))
    pool, bt = _one_request_pool(K, V, ps=4)
    w, _ = oracle.prefix_attn_row_weights(q, pool, 0, bt, [T - 1], [0, 1], 1.0, 0, 0, 0)
    assert abs(w.sum() - 1.0) < 1e-15
    assert np.allclose(w / w[0], np.exp(np.arange(T)), rtol=1e-13, atol=0)


def test_single_key_row_returns_v_exactly():
    w = wl.custom("single", 1, 4, 2, 8, 4, [0], [3], seed=5, num_pages=4)
    pool = w.empty_pool()
    k, v = w.kv_new()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    out = oracle.prefix_attn(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    for h in range(4):
        exact = wl.bf16_bits_to_f32(v[0, h // 2]).astype(np.float64)
        assert np.array_equal(out[0, h], exact)


def test_zero_query_gives_mean_of_visible_values():
    """q = 0 makes every score equal: row i returns the mean of v_0..v_{P+i}."""
    P, n, d = 5, 4, 6
    w = wl.custom("mean", 1, 2, 1, d, 4, [P], [n], seed=2, num_pages=6)
    pool = w.empty_pool()
    oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    q = np.zeros_like(w.q())
    out = oracle.prefix_attn(q, pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    _, V = w.dense_request(pool, 0)
    Vd = wl.bf16_bits_to_f32(V).astype(np.float64)
    for i in range(n):
        for h in range(2):
            assert np.allclose(out[i, h], Vd[:P + i + 1, 0].mean(axis=0), rtol=0, atol=1e-14)


def test_huge_scores_do_not_overflow():
    """Scores near 1e4: without the max shift exp() would overflow; the
    row must return the value of the largest-score key."""
    q = bf([[[64.0, 0.0]]])
    K = bf([[[100.0, 0.0]], [[160.0, 0.0]], [[130.0, 0.0]]])
    V = bf([[[1.0, 2.0]], [[3.0, -5.0]], [[7.0, 11.0]]])
    pool, bt = _one_request_pool(K, V, ps=2)
    out = oracle.prefix_attn(q, pool, 0, bt, [2], [0, 1], 1.0)
    assert np.all(np.isfinite(out))
    assert np.allclose(out[0, 0], [3.0, -5.0], rtol=0, atol=1e-12)


def test_causal_limit_is_prefix_plus_row():
    """Row i sees key P+i and not key P+i+1 (bottom-right aligned mask)."""
    w = wl.custom("causal", 1, 2, 1, 8, 4, [6], [5], seed=7, num_pages=5)
    pool = w.empty_pool()
    oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    args = (0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    base = oracle.prefix_attn(w.q(), pool, *args)
    P, i = 6, 2
    for key, changes in [(P + i, True), (P + i + 1, False)]:
        p2 = pool.copy()
        page = w.block_table[0, key // 4]
        p2[0, 1, page, 0, key % 4, :] = bf(np.full(8, 100.0))
        got = oracle.prefix_attn(w.q(), p2, *args)
        assert (not np.allclose(got[i], base[i])) == changes
        assert np.array_equal(got[:i], base[:i])


def test_gqa_head_to_group_map():
    """Constant V per kv head: q head h must return the constant of kv head
    h // (Hq/Hkv), whatever its scores."""
    Hq, Hkv, d, ps = 8, 2, 4, 4
    w = wl.custom("gqa", 2, Hq, Hkv, d, ps, [5, 3], [3, 4], seed=9, num_pages=8)
    pool = w.empty_pool()
    oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    consts = [3.0, -7.0]
    for g in range(Hkv):
        pool[0, 1, :, g] = np.where(pool[0, 1, :, g] == 0x7FC0, pool[0, 1, :, g], bf(consts[g]))
        v = v.copy()
        v[:, g, :] = bf(consts[g])
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    out = oracle.prefix_attn(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    for h in range(Hq):
        assert np.allclose(out[:, h], consts[h // (Hq // Hkv)], rtol=0, atol=1e-13)


def _fill_pool(w):
    pool = w.empty_pool()
    oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    return pool


@pytest.mark.parametrize("ps", [1, 3, 4, 16])
def test_prefix_reuse_equals_full_recompute(ps):
    """Sec. 2.2: the cached prefix KV stitched with the new tokens' KV and
    processed together must give the same rows as a from-scratch causal
    prefill of the concatenated sequence.  The dense second path reads no
    page table."""
    w = wl.custom("equiv", 3, 6, 2, 16, ps, [0, 13, 37], [9, 1, 20], seed=11)
    pool = _fill_pool(w)
    out = oracle.prefix_attn(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    assert np.all(np.isfinite(out))
    rng = np.random.default_rng(5)
    cu = w.cu_new_lens
    for b in range(w.B):
        P, n = int(w.prefix_lens[b]), int(w.new_lens[b])
        K, V = w.dense_request(pool, b)
        # queries of the cached rows do not affect the new rows: draw any
        q_prefix = wl.f32_to_bf16_bits(rng.standard_normal((P, w.Hq, w.d)).astype(np.float32))
        q_full = np.concatenate([q_prefix, w.q()[cu[b]:cu[b + 1]]], axis=0)
        ref = oracle.full_causal_attn(q_full, K, V, w.scale)
        assert np.max(np.abs(ref[P:] - out[cu[b]:cu[b + 1]])) <= 1e-12


def test_prefix_len_zero_is_textbook_causal_attention():
    """With no cached prefix the path is plain causal self-attention,
    checked here against masked-softmax matrix algebra in numpy."""
    w = wl.custom("p0", 1, 4, 2, 8, 4, [0], [7], seed=13, num_pages=3)
    pool = _fill_pool(w)
    out = oracle.prefix_attn(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    q = wl.bf16_bits_to_f32(w.q()).astype(np.float64)
    k, v = [wl.bf16_bits_to_f32(x).astype(np.float64) for x in w.kv_new()]
    T = w.T_new
    mask = np.tril(np.ones((T, T), dtype=bool))
    for h in range(w.Hq):
        g = h // w.G
        S = (q[:, h] @ k[:, g].T) * w.scale
        S = np.where(mask, S, -np.inf)
        A = np.exp(S - S.max(axis=1, keepdims=True))
        A /= A.sum(axis=1, keepdims=True)
        assert np.max(np.abs(A @ v[:, g] - out[:, h])) <= 1e-13


@pytest.mark.parametrize("ps", [1, 2, 4])
def test_bruteforce_page_permutations_tiny(ps):
    """Every placement of a 6-token sequence's pages in a 6-page pool gives
    the same result as the dense path (d 3, prefix 2, 4 new tokens)."""
    d, P, n = 3, 2, 4
    T = P + n
    rng = np.random.default_rng(17)
    K = wl.f32_to_bf16_bits(rng.standard_normal((T, 1, d)).astype(np.float32))
    V = wl.f32_to_bf16_bits(rng.standard_normal((T, 1, d)).astype(np.float32))
    qf = wl.f32_to_bf16_bits(rng.standard_normal((T, 2, d)).astype(np.float32))
    ref = oracle.full_causal_attn(qf, K, V, 0.7)[P:]
    nb = -(-T // ps)
    for perm in itertools.permutations(range(6), nb):
        pool = np.full((1, 2, 6, 1, ps, d), 0x7FC0, dtype=np.uint16)
        for j in range(T):
            pool[0, 0, perm[j // ps], 0, j % ps] = K[j, 0]
            pool[0, 1, perm[j // ps], 0, j % ps] = V[j, 0]
        bt = np.asarray(perm, dtype=np.int32).reshape(1, nb)
        out = oracle.prefix_attn(qf[P:], pool, 0, bt, [P], [0, n], 0.7, nthreads=1)
        assert np.max(np.abs(out - ref)) <= 1e-13


def test_tiny_config_numpy_crosscheck():
    """Tiny config (GQA 4:1, d 64, prefix 256, 64 new, NaN past the end of
    the last page) against an independent numpy float64 evaluation."""
    w = wl.tiny()
    pool = _fill_pool(w)
    out = oracle.prefix_attn(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    K, V = w.dense_request(pool, 0)
    Kd, Vd = [wl.bf16_bits_to_f32(x).astype(np.float64) for x in (K, V)]
    q = wl.bf16_bits_to_f32(w.q()).astype(np.float64)
    P = 256
    for h in range(w.Hq):
        S = q[:, h] @ Kd[:, 0].T * w.scale            # [64][320]
        lim = P + np.arange(64)[:, None]
        S = np.where(np.arange(P + 64)[None, :] <= lim, S, -np.inf)
        A = np.exp(S - S.max(1, keepdims=True))
        ref = (A @ Vd[:, 0]) / A.sum(1, keepdims=True)
        assert np.max(np.abs(ref - out[:, h])) <= 1e-13


def test_sampled_rows_match_full_output():
    w = wl.custom("rows", 2, 4, 2, 16, 4, [9, 0], [5, 6], seed=23)
    pool = _fill_pool(w)
    full = oracle.prefix_attn(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    rows = np.array([[0, 0, 0], [0, 3, 4], [1, 2, 5], [1, 1, 0]], dtype=np.int32)
    got = oracle.prefix_attn_rows(w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens,
                                  w.scale, rows)
    cu = w.cu_new_lens
    for r, (b, h, i) in enumerate(rows):
        assert np.array_equal(got[r], full[cu[b] + i, h])


def test_thread_count_does_not_change_results():
    w = wl.custom("thr", 3, 4, 2, 16, 4, [3, 8, 1], [4, 2, 7], seed=29)
    pool = _fill_pool(w)
    args = (w.q(), pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale)
    assert np.array_equal(oracle.prefix_attn(*args, nthreads=1), oracle.prefix_attn(*args, nthreads=5))


# ------------------------------------------------------ 8-bit cache tier
def _q8_pool(groups, Hkv=1, ps=1):
    """Pool [1][2][NP][Hkv][ps][d] holding `groups` (one per (plane, page, head))."""
    g = np.asarray(groups, dtype=np.float32)
    d = g.shape[-1] // ps
    n = g.shape[0] // (2 * Hkv)
    pool = wl.f32_to_bf16_bits(g).reshape(2, n, Hkv, ps, d)  # every value here is exact in bf16
    return np.ascontiguousarray(pool.reshape(1, 2, n, Hkv, ps, d))


def test_q8_codes_of_worked_groups():
    """amax = 127/64 makes 127/amax = 64 and s = 1/64 exactly, so each code is
    round_half_even(64 x) by hand, ties included (2.5 -> 2, 3.5 -> 4, -0.5 -> 0,
    1.5 -> 2; half-away-from-zero would give 3, 4, -1, 2).  amax = 2 makes
    127/amax = 63.5, so codes are round_half_even(63.5 x) (63.5 -> 64, -63.5 -> -64)."""
    k = np.array([127, 2.5, 3.5, -0.5, 1.5, 0, -127, 64, -3, 10.5, 11.5, 100, -100.5, 1, -1, 0.5])
    a = k / 64.0
    want_a = [127, 2, 4, 0, 2, 0, -127, 64, -3, 10, 12, 100, -100, 1, -1, 0]
    b = np.array([1.0, -0.5, 0.25, 0.125, 2.0, -2.0, 0.0, 1.5, -1.25, 0.75, 0.0625, -0.0625,
                  0.296875, 0.5, -1.0, 0.109375])
    want_b = [64, -32, 16, 8, 127, -127, 0, 95, -79, 48, 4, -4, 19, 32, -64, 7]
    pool = _q8_pool([a, b])  # K plane: group a, V plane: group b
    img = oracle.kv_save_q8(pool, [0])
    scales, codes = oracle.q8_split(img, 1, 1, 16)
    assert codes[0, 0, 0, 0, 0].tolist() == want_a
    assert codes[0, 0, 1, 0, 0].tolist() == want_b
    assert scales[0, 0, 0, 0] == np.float32(1 / 64)
    assert abs(float(scales[0, 0, 1, 0]) * 127 - 2.0) <= 2.0 * 2.0 ** -23
    out = np.zeros_like(pool)
    oracle.kv_restore_q8(out, img, [0])
    back = wl.bf16_bits_to_f32(out[0, 0, 0, 0, 0])
    assert np.array_equal(back, np.asarray(want_a, np.float32) / 64)  # c/64 is exact in bf16


def _random_q8_pool(seed, L=2, NP=5, Hkv=3, ps=4, d=16, scale=1.0):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((L, 2, NP, Hkv, ps, d)) * scale).astype(np.float32)
    return wl.f32_to_bf16_bits(x)


def test_q8_round_trip_within_half_step():
    """Every restored value is within half a quantisation step of the
    original, plus the final bf16 rounding; each group's largest |x| maps to
    +-127; every code is in [-127, 127]."""
    pool = _random_q8_pool(1)
    ids = np.array([4, 0, 2], np.int32)
    img = oracle.kv_save_q8(pool, ids)
    L, _, NP, Hkv, ps, d = pool.shape
    scales, codes = oracle.q8_split(img, Hkv, ps, d)
    assert codes.min() >= -127 and codes.max() <= 127
    out = np.zeros_like(pool)
    oracle.kv_restore_q8(out, img, ids)
    x = wl.bf16_bits_to_f32(pool[:, :, ids]).astype(np.float64)      # [L][2][n][Hkv][ps][d]
    y = wl.bf16_bits_to_f32(out[:, :, ids]).astype(np.float64)
    s = scales.transpose(1, 2, 0, 3)[..., None, None].astype(np.float64)  # [L][2][n][Hkv]
    assert np.all(np.abs(y - x) <= s / 2 * (1 + 2.0 ** -20) + np.abs(y) * 2.0 ** -8)
    amax = np.abs(x).max(axis=(-1, -2))
    cmax = np.abs(codes.transpose(1, 2, 0, 3, 4, 5).astype(np.int64)).max(axis=(-1, -2))
    assert np.all(cmax == 127) and np.all(amax > 0)
    untouched = np.setdiff1d(np.arange(NP), ids)
    assert np.all(out[:, :, untouched] == 0)


def test_q8_sign_and_power_of_two_scaling():
    """Negating a page negates its codes; multiplying it by 4 (exact in bf16)
    keeps the codes and multiplies the scales by 4."""
    pool = _random_q8_pool(2)
    ids = np.arange(pool.shape[2], dtype=np.int32)
    img = oracle.kv_save_q8(pool, ids)
    neg = pool ^ np.uint16(0x8000)
    x4 = wl.f32_to_bf16_bits(wl.bf16_bits_to_f32(pool) * 4)
    s0, c0 = oracle.q8_split(img, *pool.shape[3:])
    s1, c1 = oracle.q8_split(oracle.kv_save_q8(neg, ids), *pool.shape[3:])
    s4, c4 = oracle.q8_split(oracle.kv_save_q8(x4, ids), *pool.shape[3:])
    assert np.array_equal(c1, -c0) and np.array_equal(s1, s0)
    assert np.array_equal(c4, c0) and np.array_equal(s4, s0 * 4)


def test_q8_zero_nan_and_infinite_values():
    """An all-zero group has scale 0 and restores to +0; NaN codes to 0 and
    infinities saturate, neither counting towards amax."""
    zeros = np.zeros(16)
    special = np.array([np.nan, np.inf, -np.inf, 1.0, -0.5] + [0.25] * 11)
    pool = _q8_pool([zeros, special])
    img = oracle.kv_save_q8(pool, [0])
    scales, codes = oracle.q8_split(img, 1, 1, 16)
    assert scales[0, 0, 0, 0] == 0 and np.all(codes[0, 0, 0] == 0)
    assert scales[0, 0, 1, 0] == np.float32(1.0) / np.float32(127)
    assert codes[0, 0, 1, 0, 0, :5].tolist() == [0, 127, -127, 127, -64]
    out = np.full_like(pool, 0x7FC0)
    oracle.kv_restore_q8(out, img, [0])
    assert np.all(out[0, 0, 0] == 0)


def test_q8_image_layout_and_layer_range():
    """Hkv = 3: 12 scale bytes, 4 zero bytes, then the codes; a layer range
    writes only its chunks and restores only its layers."""
    pool = _random_q8_pool(3, L=4, NP=3, Hkv=3, ps=2, d=8)
    assert oracle.q8_chunk_bytes(3, 2, 8) == 16 + 3 * 2 * 8
    ids = np.array([2, 1], np.int32)
    img = oracle.kv_save_q8(pool, ids, layer_begin=1, layer_count=2)
    assert np.all(img[:, [0, 3]] == 0) and np.all(img[:, 1:3, :, 12:16] == 0)
    full = oracle.kv_save_q8(pool, ids)
    assert np.array_equal(img[:, 1:3], full[:, 1:3])
    out = np.zeros_like(pool)
    oracle.kv_restore_q8(out, full, ids, layer_begin=2, layer_count=1)
    ref = np.zeros_like(pool)
    oracle.kv_restore_q8(ref, full, ids)
    assert np.array_equal(out[2], ref[2]) and np.all(out[[0, 1, 3]] == 0)


def test_q8_attention_on_exact_codes_equals_bf16_attention():
    """Attention over 8-bit pages is defined as the 8-bit restore followed by
    prefix attention.  Pages whose values are integers in [-127, 127] times
    2^-e, with +-127 in every (page, plane, head) group, have scale 2^-e and
    codes equal to those integers exactly, so the 8-bit path must give the
    bf16 path's result bit for bit (stale NaN slots past a prefix included)."""
    w = wl.custom("q8-exact", 3, 8, 2, 16, 4, [13, 8, 0], [5, 6, 3], seed=23)
    src = w.host_src()
    rng = np.random.default_rng(29)
    n = src.shape[0]
    codes = rng.integers(-127, 128, size=src.shape)
    codes[..., 0, 0] = np.where(rng.random(codes.shape[:-2]) < 0.5, 127, -127)
    e = rng.integers(2, 9, size=src.shape[:-2])[..., None, None]
    exact = codes.astype(np.float32) * np.float32(2.0) ** -e.astype(np.float32)
    stale = np.isnan(wl.bf16_bits_to_f32(src))
    w._cache["src"] = np.where(stale, src, wl.f32_to_bf16_bits(exact))
    ids = w.prefix_blocks()
    bf = _fill_pool(w)
    out_bf = oracle.prefix_attn(w.q(), bf, 0, w.block_table, w.prefix_lens, w.cu_new_lens,
                                w.scale)
    cached = w.empty_pool()
    oracle.kv_restore(cached, w.host_src(), ids)                # before the append
    img = oracle.kv_save_q8(cached, ids)
    scales, got = oracle.q8_split(img, w.Hkv, w.ps, w.d)       # [n][L][2][Hkv](...)
    want = np.where(stale, 0, codes)
    assert np.array_equal(got.astype(np.int64), want)
    assert np.array_equal(scales.astype(np.float64), 2.0 ** -e[..., 0, 0].astype(np.float64))
    q8 = w.empty_pool()
    oracle.kv_restore_q8(q8, img, ids)
    k, v = w.kv_new()
    oracle.kv_append(q8, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    out_q8 = oracle.prefix_attn(w.q(), q8, 0, w.block_table, w.prefix_lens, w.cu_new_lens,
                                w.scale)
    assert n == ids.size and np.all(np.isfinite(out_q8))
    assert np.array_equal(out_q8, out_bf)
