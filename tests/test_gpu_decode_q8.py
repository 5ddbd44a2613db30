"""Paged decode attention over pages kept in the 8-bit cache tier
(gc_paged_decode_attn_q8).

Defined as the 8-bit restore (Sec. 6.1 keeps the 70B KV in INT8) followed by
decode attention (Sec. 2.1), so the oracle is oracle.kv_restore_q8 of every
cached page, oracle.kv_append of the new token and oracle.prefix_attn with one
new row.  The GPU path never writes the 8-bit pages into the pool; it is
checked bit for bit against gc_kv_restore_q8 of every page followed by
gc_paged_decode_attn, and within the attention tolerance against the oracle."""
import numpy as np
import pytest

import oracle
from paper_2505_23970_gb300 import binding as gcb
from paper_2505_23970_gb300 import workloads as wl
from paper_2505_23970_gb300.harness import DeviceBatch, _i32

from ._q8 import Q8Case, all_pages_case
from ._util import assert_attn_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2505_23970_gb300 import build
    build.build()


def _bits_equal(a, b):
    import torch
    return torch.equal(a.view(torch.int16), b.view(torch.int16))


def _workspace(db):
    import torch
    w = db.w
    need = gcb.gc_paged_decode_workspace_bytes(db.pool.handle, w.B, w.max_blocks, w.Hq)
    return torch.empty(max(need, 16), dtype=torch.uint8, device="cuda"), need


def run_decode_q8(case, layer=0, layer_major=False, table=None):
    """Restore the pool-side pages, append the new token, decode over the
    q8 table.  Returns (status, out, pool bits)."""
    import torch
    w = case.w
    db = DeviceBatch(w, with_restore=False)
    if case.to_pool.size:
        part = torch.from_numpy(np.ascontiguousarray(case.img[case.to_pool])).cuda()
        gcb.gc_kv_restore_q8(db.pool.handle, part, _i32(case.ids[case.to_pool], "cuda"),
                             int(case.to_pool.size), 0, w.L, None, None,
                             gcb.GC_RESTORE_SRC_DEVICE)
    for l in range(w.L):
        db.append(layer=l)
    img = case.img
    if layer_major:
        img = np.ascontiguousarray(img.swapaxes(0, 1))
    dimg = torch.from_numpy(img).cuda()
    seq = _i32(w.total_lens, "cuda")
    ws, need = _workspace(db)
    gcb.gc_paged_decode_attn_q8(db.q, db.pool.handle, db.block_table, seq, db.out, None, layer,
                                w.B, w.max_blocks, w.Hq, w.scale, ws, need, dimg,
                                _i32(case.table if table is None else table, "cuda"),
                                int(case.ids.size),
                                gcb.GC_RESTORE_LAYER_MAJOR if layer_major else 0)
    status = db.check()
    out = db.out.clone()
    pool = db.pool_bits()
    db.close()
    return status, out, pool


def run_restore_then_decode(case, layer=0):
    import torch
    w = case.w
    db = DeviceBatch(w, with_restore=False)
    if case.ids.size:
        gcb.gc_kv_restore_q8(db.pool.handle, torch.from_numpy(case.img).cuda(),
                             _i32(case.ids, "cuda"), int(case.ids.size), 0, w.L, None, None,
                             gcb.GC_RESTORE_SRC_DEVICE)
    for l in range(w.L):
        db.append(layer=l)
    db.decode(layer=layer)
    assert db.check() == gcb.GC_OK
    out = db.out.clone()
    db.close()
    return out


def decode_q8_parity(w, layer=0, **kw):
    import torch
    case = Q8Case(w, **kw)
    status, out, _ = run_decode_q8(case, layer=layer)
    assert status == gcb.GC_OK
    assert _bits_equal(out, run_restore_then_decode(case, layer=layer)), \
        f"{w.name}: differs from restore + decode"
    ref = oracle.prefix_attn(w.q(), case.oracle_pool(), layer, w.block_table, w.prefix_lens,
                             w.cu_new_lens, w.scale)
    return assert_attn_close(out.to(torch.float64).cpu().numpy(), ref, f"{w.name} [q8 decode]")


def test_q8_decode_llama3_70b():
    """8 requests x 9216-token contexts on the 70B-shaped layer."""
    decode_q8_parity(wl.llama3_70b_decode(seed=0))


def test_q8_decode_mix():
    """64 requests with the conversation mix's contexts."""
    decode_q8_parity(wl.decode_mix(seed=1))


@pytest.mark.parametrize("G,d,ps", [(1, 128, 16), (4, 128, 32), (16, 128, 64), (8, 128, 128),
                                    (2, 64, 16), (8, 64, 64)])
def test_q8_decode_groupings_and_page_sizes(G, d, ps):
    """Head groupings, both head sizes (d 64 runs the decode mode of the 8-bit
    prefill variant) and page sizes, contexts that end inside a page and on a
    page boundary, one of a single key."""
    Hkv = 2
    ctx = [1, ps, ps + 1, 3 * ps - 1, 700, 129]
    w = wl.custom(f"q8dec-G{G}-d{d}-ps{ps}", len(ctx), G * Hkv, Hkv, d, ps,
                  [c - 1 for c in ctx], [1] * len(ctx), seed=G + ps)
    decode_q8_parity(w)


def test_q8_decode_mixed_pool_and_image_pages():
    w = wl.custom("q8dec-mixed", 4, 32, 4, 128, 16, [3000, 129, 1500, 64], [1] * 4, seed=7)
    decode_q8_parity(w, frac_in_image=0.5, seed=5)


@pytest.mark.parametrize("layer_major", [False, True])
def test_q8_decode_layer_of_a_multilayer_image(layer_major):
    import torch
    w = wl.custom("q8dec-layers", 3, 16, 2, 128, 16, [500, 33, 260], [1] * 3, seed=9)
    w.L = 3
    case = Q8Case(w)
    status, out, _ = run_decode_q8(case, layer=2, layer_major=layer_major)
    assert status == gcb.GC_OK
    assert _bits_equal(out, run_restore_then_decode(case, layer=2))
    ref = oracle.prefix_attn(w.q(), case.oracle_pool(), 2, w.block_table, w.prefix_lens,
                             w.cu_new_lens, w.scale)
    assert_attn_close(out.to(torch.float64).cpu().numpy(), ref, "layer 2 [q8 decode]")


def test_q8_decode_batch_with_three_slot_ring():
    """4500 requests: the unit table takes the room of a ring slot."""
    rng = np.random.default_rng(11)
    ctx = rng.integers(1, 60, size=4500)
    w = wl.custom("q8dec-big", 4500, 8, 1, 128, 16, ctx - 1, [1] * 4500, seed=11)
    decode_q8_parity(w)


def test_q8_decode_pool_untouched_and_bad_entry_reported():
    """The pool pages behind image entries keep their NaN fill; an image block
    >= n_image_blocks is skipped and reported as GC_ERR_OUT_OF_RANGE."""
    import torch
    w = wl.custom("q8dec-bad", 2, 16, 2, 128, 16, [640, 300], [1, 1], seed=12)
    case = Q8Case(w)
    status, out, pool = run_decode_q8(case)
    assert status == gcb.GC_OK and torch.isfinite(out.float()).all()
    for b in range(w.B):
        for j in range(w.max_blocks):
            if case.table[b, j] >= 0:
                assert np.all(pool[0, :, w.block_table[b, j]] == 0x7FC0)
    bad = case.table.copy()
    bad[0, 3] = case.ids.size
    status, _, _ = run_decode_q8(case, table=bad)
    assert status == gcb.GC_ERR_OUT_OF_RANGE


def test_q8_decode_d64_long_contexts_split_and_merged():
    """d 64 with contexts long enough that requests are cut into key ranges
    (fp32 partials merged by the merge kernel)."""
    w = wl.custom("q8dec-d64-split", 3, 16, 4, 64, 16, [8191, 3000, 20], [1] * 3, seed=16)
    decode_q8_parity(w)


def test_q8_decode_host_checks():
    import torch
    img = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    ws = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    w = wl.custom("q8dec-args2", 1, 8, 1, 128, 16, [63], [1], seed=13)
    seq = _i32(w.total_lens, "cuda")
    tab = _i32(np.full((1, w.max_blocks), -1, np.int32), "cuda")
    db = DeviceBatch(w, with_restore=False)
    for image, table, flags in ((img, tab, 0x10), (img, None, 0), (img.data_ptr() + 4, tab, 0)):
        with pytest.raises(gcb.GcError) as e:
            gcb.gc_paged_decode_attn_q8(db.q, db.pool.handle, db.block_table, seq, db.out, None,
                                        0, 1, w.max_blocks, w.Hq, w.scale, ws, ws.numel(), image,
                                        table, 1, flags)
        assert e.value.status == gcb.GC_ERR_INVALID_ARG
    torch.cuda.synchronize()
    db.close()


@pytest.mark.parametrize("d", [128, 64])
def test_q8_decode_every_page_from_the_image(d):
    """The page holding the new token also read from the image: the context
    ends inside an image page (V rows past it zeroed, keys masked)."""
    import torch
    w = wl.custom(f"q8dec-allimg-d{d}", 4, 16, 2, d, 16, [300, 0, 76, 639], [1] * 4,
                  seed=19 + d)
    img, ids, table, ref_pool = all_pages_case(w)
    db = DeviceBatch(w, with_restore=False)
    seq = _i32(w.total_lens, "cuda")
    ws, need = _workspace(db)
    gcb.gc_paged_decode_attn_q8(db.q, db.pool.handle, db.block_table, seq, db.out, None, 0, w.B,
                                w.max_blocks, w.Hq, w.scale, ws, need,
                                torch.from_numpy(img).cuda(), _i32(table, "cuda"),
                                int(ids.size), 0)
    assert db.check() == gcb.GC_OK
    ref = oracle.prefix_attn(w.q(), ref_pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens,
                             w.scale)
    assert_attn_close(db.out.to(torch.float64).cpu().numpy(), ref, f"{w.name} [q8 decode]")
    db.close()


@pytest.mark.parametrize("G", [8, 2])
def test_q8_decode_score_jump_rescales(G):
    """Two pages late in a context whose K scales are 200x the rest: their
    scores exceed the reference max taken from the first tile by far more than
    the lazy-rescale threshold, so O and the sums are rescaled mid-request;
    bit for bit the two-step path, within tolerance of the oracle on the same
    image."""
    import torch
    w = wl.custom(f"q8dec-jump-G{G}", 2, 4 * G, 4, 128, 16, [2000, 700], [1, 1], seed=21 + G)
    case = Q8Case(w)
    for j in (100, 101):  # request 0's pages 100 and 101 (image blocks 100, 101)
        hdr = case.img[j, 0, 0, :4 * w.Hkv].view(np.float32)
        hdr *= 200.0
    status, out, _ = run_decode_q8(case)
    assert status == gcb.GC_OK
    assert _bits_equal(out, run_restore_then_decode(case)), f"{w.name}: differs"
    ref = oracle.prefix_attn(w.q(), case.oracle_pool(), 0, w.block_table, w.prefix_lens,
                             w.cu_new_lens, w.scale)
    assert_attn_close(out.to(torch.float64).cpu().numpy(), ref, f"{w.name} [q8 decode]")


def test_q8_decode_one_long_request_beside_a_short_one():
    """One request of 20000 keys (cut between several CTAs' shares, merged in
    the kernel) next to a request of 3 keys."""
    decode_q8_parity(wl.custom("q8dec-one-long", 2, 64, 8, 128, 16, [19999, 2], [1, 1], seed=23))
