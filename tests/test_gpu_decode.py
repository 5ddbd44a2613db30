"""GPU parity of paged decode attention (one new token per request) against
the float64 oracle's prefix attention with one new row, through the C ABI."""
import numpy as np
import pytest

import oracle
from paper_2505_23970_gb300 import binding as gcb
from paper_2505_23970_gb300 import workloads as wl
from paper_2505_23970_gb300.harness import DeviceBatch, _i32

from ._util import assert_attn_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2505_23970_gb300 import build
    build.build()


def oracle_pool(w):
    pool = w.empty_pool()
    if w.prefix_blocks().size:
        oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    return pool


def decode_parity(w):
    db = DeviceBatch(w)
    db.restore()
    db.append()
    db.decode()
    assert db.check() == gcb.GC_OK
    got = db.out_f64()
    splits = gcb.gc_paged_decode_workspace_bytes(db.pool.handle, w.B, w.max_blocks, w.Hq)
    db.close()
    ref = oracle.prefix_attn(w.q(), oracle_pool(w), 0, w.block_table, w.prefix_lens,
                             w.cu_new_lens, w.scale)
    assert_attn_close(got, ref, f"{w.name} decode")
    return splits


def test_llama3_70b_decode_full():
    """8 requests x 9216-token contexts on the 70B-shaped layer (split path)."""
    assert decode_parity(wl.llama3_70b_decode(seed=0)) > 0


def test_decode_mix_full():
    """64 requests with the conversation mix's contexts (lognormal lengths)."""
    decode_parity(wl.decode_mix(seed=1))


def test_wide_batch_of_short_contexts():
    """160 requests of 2..161 keys (d 128): most (request, kv head) pairs lie
    whole inside one CTA's share of the K/V tiles."""
    w = wl.custom("dec-wide", 160, 32, 8, 128, 16, list(range(1, 161)), [1] * 160, seed=3)
    decode_parity(w)


def test_unsplit_path_d64_needs_no_workspace():
    """d 64 runs on the prefill kernel's decode mode: with enough requests x
    kv heads to fill the GPU no request is split and no workspace is needed."""
    w = wl.custom("dec-wide64", 160, 32, 8, 64, 16, list(range(1, 161)), [1] * 160, seed=3)
    assert gcb.gc_paged_decode_workspace_bytes(DeviceBatch(w).pool.handle, w.B, w.max_blocks,
                                               w.Hq) == 0
    assert decode_parity(w) == 0


def test_decode_reference_max_raised_inside_a_piece():
    """Keys aligned with q heads 0 and 1 (k = 12 q: scores ~190 in log2
    units against ~4 elsewhere) in later tiles of a CTA's piece: each head's
    reference max is raised once (O and the sums rescaled).  Without the
    raise the probabilities (2^190) would overflow bf16; with a wrong rescale
    of the sums the output would be off by the old keys' weight."""
    w = wl.custom("dec-rescale", 8, 16, 2, 128, 16, [8999] * 8, [1] * 8, seed=31)
    src = w.host_src()  # cached: the device batch and the oracle see the edit
    q = wl.bf16_bits_to_f32(w.q())
    # 8 x 2 pairs of 71 tiles over 152 CTAs: shares of 8 tiles, so the tiles
    # 13 and 14 of request 0, kv head 0 are the 6th and 7th of one piece
    for tile, h in ((13, 0), (14, 1)):
        for j in range(tile * 128 + 3, tile * 128 + 9):
            blk, row = divmod(j, w.ps)
            src[blk, 0, 0, 0, row] = wl.f32_to_bf16_bits(12.0 * q[0, h])
    decode_parity(w)


def test_decode_batch_with_five_slot_ring():
    """4600 requests: the unit table leaves room for five K/V ring slots
    instead of six."""
    ctx = np.random.default_rng(23).integers(1, 200, size=4600)
    w = wl.custom("dec-5slot", 4600, 16, 2, 128, 16, ctx - 1, np.ones(4600, int), seed=23)
    decode_parity(w)


@pytest.mark.parametrize("G,d,ps", [(1, 128, 16), (2, 64, 32), (4, 64, 16), (8, 128, 64),
                                    (16, 128, 128), (16, 64, 16), (8, 64, 128), (2, 128, 16),
                                    (4, 128, 32)])
def test_decode_head_grouping_dims_and_page_sizes(G, d, ps):
    Hkv = 2
    ctx = [1, 17, 300, 1000, 64, 129]
    w = wl.custom(f"dec-g{G}d{d}p{ps}", len(ctx), Hkv * G, Hkv, d, ps, [c - 1 for c in ctx],
                  [1] * len(ctx), seed=G + d + ps)
    decode_parity(w)


def test_context_of_one_returns_v_bit_exact():
    """A context of one key (the new token only): the output is v exactly."""
    import torch
    w = wl.custom("dec-one", 3, 8, 2, 128, 16, [0, 0, 0], [1, 1, 1], seed=6)
    db = DeviceBatch(w)
    db.append()
    db.decode()
    assert db.check() == gcb.GC_OK
    _, v = w.kv_new()
    got = db.out.view(torch.int16).cpu().numpy().view(np.uint16)
    for b in range(w.B):
        for h in range(w.Hq):
            assert np.array_equal(got[b, h], v[b, h // w.G])
    db.close()


def test_decode_matches_prefill_kernel_with_one_new_token():
    import torch
    w = wl.custom("dec-vs-prefill", 4, 64, 8, 128, 16, [700, 33, 0, 4095], [1] * 4, seed=7)
    a = DeviceBatch(w)
    a.restore()
    a.append()
    a.decode()
    b = DeviceBatch(w)
    b.run()
    assert a.check() == gcb.GC_OK and b.check() == gcb.GC_OK
    assert_attn_close(a.out_f64(), b.out_f64(), "decode vs prefill")
    a.close()
    b.close()


def test_decode_errors():
    import torch
    w = wl.llama3_70b_decode(seed=2, B=2, context=5000)
    db = DeviceBatch(w)
    db.restore()
    db.append()
    need = gcb.gc_paged_decode_workspace_bytes(db.pool.handle, w.B, w.max_blocks, w.Hq)
    assert need > 0
    small = torch.empty(need // 2, dtype=torch.uint8, device="cuda")
    with pytest.raises(gcb.GcError) as e:
        db.decode(workspace=small)
    assert e.value.status == gcb.GC_ERR_INVALID_ARG
    # a context longer than the block table allows, and a bad page
    db.seq_lens = _i32(np.array([w.max_blocks * w.ps + 5, 5000]), "cuda")
    db.decode()
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    bt = w.block_table.copy()
    bt[1, 3] = -7
    db.block_table = _i32(bt, "cuda")
    db.seq_lens = _i32(w.total_lens, "cuda")
    db.decode()
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    # batch 0 is a no-op
    gcb.gc_paged_decode_attn(db.q, db.pool.handle, db.block_table, db.seq_lens, db.out, None, 0,
                             0, w.max_blocks, w.Hq, w.scale)
    assert db.check() == gcb.GC_OK
    db.close()


@pytest.mark.parametrize("B,ctx", [(1, 9216), (2, 700), (40, 3000)])
def test_decode_range_lengths_chosen_per_batch(B, ctx):
    """Small and large batches get different key-range lengths (more ranges
    for few requests); every choice matches the oracle."""
    decode_parity(wl.llama3_70b_decode(seed=B, B=B, context=ctx))


def test_decode_batch_beyond_sorted_ranking():
    """1000 requests (more than the 512 the kernel ranks by length)."""
    ctx = np.random.default_rng(22).integers(1, 600, size=1000)
    w = wl.custom("dec-big-batch", 1000, 16, 4, 64, 16, ctx - 1, np.ones(1000, int), seed=22)
    decode_parity(w)


def test_merge_counters_cleared_after_an_error():
    """A (request, kv head) pair cut between two SMs' shares is merged by the
    last CTA to finish one of its pieces, counted in the pool's control block.
    After any recorded error gc_kv_pool_check clears those counters: raise
    them by hand, record an error (a bad page), check, and the next decode
    matches the oracle again (with raised counters the merges would be
    skipped or early)."""
    import torch
    w = wl.llama3_70b_decode(seed=4, B=2, context=3000)
    db = DeviceBatch(w)
    db.restore()
    db.append()
    control = db.pool.buffer[-2048:]
    control[256:256 + 448 * 4].view(torch.int32).fill_(5)
    bt = w.block_table.copy()
    bt[1, 3] = -7
    db.block_table = _i32(bt, "cuda")
    db.decode()
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    assert int(control[256:256 + 448 * 4].view(torch.int32).abs().sum()) == 0
    db.block_table = _i32(w.block_table, "cuda")
    db.decode()
    assert db.check() == gcb.GC_OK
    got = db.out_f64()
    db.close()
    ref = oracle.prefix_attn(w.q(), oracle_pool(w), 0, w.block_table, w.prefix_lens,
                             w.cu_new_lens, w.scale)
    assert_attn_close(got, ref, "decode after counters were cleared")
