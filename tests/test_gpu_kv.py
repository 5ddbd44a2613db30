"""GPU parity of the paged KV restore and append (bit-exact against the
float64 oracle's index maps), through the C ABI."""
import numpy as np
import pytest

import oracle
from paper_2505_23970_gb300 import binding as gcb
from paper_2505_23970_gb300 import workloads as wl
from paper_2505_23970_gb300.harness import DeviceBatch, _i32, bf16_tensor

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2505_23970_gb300 import build
    build.build()


def oracle_pool(w, restore=True, append=True):
    pool = w.empty_pool()
    if restore and w.prefix_blocks().size:
        oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    if append:
        k, v = w.kv_new()
        oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    return pool


@pytest.mark.parametrize("mode,vector", [("staged", False), ("staged", True), ("device", False),
                                         ("zerocopy", False)])
@pytest.mark.parametrize("make", [wl.tiny, lambda: wl.llama3_8b_layer(seed=1, B=6)])
def test_restore_bit_exact(make, mode, vector):
    w = make()
    db = DeviceBatch(w)
    if mode == "device":
        db.stage()
    db.restore(mode=mode, vector=vector)
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), oracle_pool(w, append=False))
    db.close()


def test_restore_full_80_layer_prefix():
    """Full 80-layer KV of one 8192-token prefix (80 x 2 x 8 x 128 x 8192
    bf16 = 2,684,354,560 bytes) from pinned host into a 640-page pool."""
    w = wl.llama3_70b_restore_80layer()
    assert w.host_src().nbytes == 2_684_354_560
    db = DeviceBatch(w)
    db.restore(mode="staged")
    assert db.check() == gcb.GC_OK
    got = db.pool_bits()
    db.close()
    assert np.array_equal(got, oracle_pool(w, append=False))


def test_restore_skips_out_of_range_block_and_reports_it():
    w = wl.tiny()
    db = DeviceBatch(w)
    ids = w.prefix_blocks().copy()
    ids[3] = w.num_pages          # one bad id; the others must still land
    db.block_ids = _i32(ids, "cuda")
    db.restore(mode="staged")
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    ref = w.empty_pool()
    keep = np.ones(ids.size, bool)
    keep[3] = False
    oracle.kv_restore(ref, w.host_src()[keep], ids[keep])
    assert np.array_equal(db.pool_bits(), ref)
    assert db.check() == gcb.GC_OK  # the status word was cleared
    db.close()


def test_restore_rejects_pageable_host_memory():
    w = wl.tiny()
    db = DeviceBatch(w)
    pageable = np.zeros(w.host_src().size, dtype=np.uint16)
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_kv_restore(db.pool.handle, pageable.ctypes.data, db.block_ids, db.n_blocks, None,
                          db.staging, 0)
    assert e.value.status == gcb.GC_ERR_INVALID_ARG
    db.close()


@pytest.mark.parametrize("make", [
    wl.tiny,
    lambda: wl.llama3_8b_layer(seed=2),
    lambda: wl.conversation_mix(seed=3, hit_p=0.5, B=16),
    lambda: wl.custom("ragged", 5, 8, 2, 64, 32, [0, 31, 32, 33, 100], [1, 0, 64, 5, 31], seed=4),
])
def test_append_bit_exact(make):
    w = make()
    db = DeviceBatch(w)
    db.restore()
    db.append()
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), oracle_pool(w))
    db.close()


def test_append_reports_bad_page():
    w = wl.custom("badpage", 2, 4, 1, 64, 16, [16, 3], [20, 4], seed=5)
    bt = w.block_table.copy()
    bt[0, 2] = w.num_pages + 7    # tokens 32..35 of request 0 have no valid page
    db = DeviceBatch(w)
    db.block_table = _i32(bt, "cuda")
    db.restore()
    db.append()
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    db.close()


def test_zero_sizes_are_noops():
    w = wl.tiny()
    db = DeviceBatch(w)
    before = db.pool_bits()
    gcb.gc_kv_restore(db.pool.handle, db.host_src, db.block_ids, 0, None, db.staging, 0)
    gcb.gc_kv_append(db.pool.handle, db.k_new, db.v_new, db.block_table, db.prefix_lens, None, 0,
                     db.cu_new_lens, 0, w.max_blocks, 0)
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), before)
    db.close()


def test_library_owned_pool_matches_caller_owned():
    """A pool whose memory the library allocates itself gives the same
    attention output, bit for bit, as one in caller-owned memory."""
    import torch
    w = wl.tiny()
    db = DeviceBatch(w)
    db.run()
    ref = db.out.clone()
    cfg = gcb.make_config(w.L, w.Hkv, w.d, w.ps, w.num_pages)
    h = gcb.gc_kv_pool_create(cfg)
    ptr, nbytes = gcb.gc_kv_pool_data(h)
    assert ptr and nbytes == int(np.prod(w.pool_shape)) * 2
    gcb.gc_kv_restore(h, db.host_src, db.block_ids, db.n_blocks, None, db.staging, 0)
    gcb.gc_kv_append(h, db.k_new, db.v_new, db.block_table, db.prefix_lens, None, 0,
                     db.cu_new_lens, w.B, w.max_blocks, w.T_new)
    out = torch.full_like(ref, float("nan"))
    gcb.gc_prefix_prefill_attn(db.q, h, db.block_table, db.prefix_lens, db.new_lens, out, None,
                               0, db.cu_new_lens, w.B, w.max_blocks, w.Hq, w.scale, w.T_new)
    assert gcb.gc_kv_pool_check(h) == gcb.GC_OK
    gcb.gc_kv_pool_destroy(h)
    assert torch.equal(out.view(torch.int16), ref.view(torch.int16))
    db.close()


def _used_pages(w):
    ids = []
    for b in range(w.B):
        ids.extend(w.block_table[b, :-(-int(w.total_lens[b]) // w.ps)].tolist())
    return np.asarray(ids[::-1], dtype=np.int32)  # reversed: not pool order


@pytest.mark.parametrize("mode,vector", [("staged", False), ("staged", True), ("device", False),
                                         ("zerocopy", False)])
@pytest.mark.parametrize("make", [wl.tiny, lambda: wl.llama3_8b_layer(seed=1, B=6)])
def test_save_bit_exact(make, mode, vector):
    """Sec. 2.2 step 1: the pages of processed requests saved to the cache
    tier are byte-for-byte the pool pages (oracle gather of the same ids)."""
    w = make()
    db = DeviceBatch(w)
    db.restore()
    db.append()
    ids = _used_pages(w)
    got = db.save(ids, mode=mode, vector=vector)
    assert db.check() == gcb.GC_OK
    assert np.array_equal(got, oracle.kv_gather_blocks(oracle_pool(w), ids))
    db.close()


def test_save_then_restore_round_trip():
    """Saving pages and restoring them elsewhere reproduces them exactly."""
    w = wl.custom("roundtrip", 3, 8, 2, 128, 32, [70, 0, 300], [10, 40, 3], seed=13)
    a = DeviceBatch(w)
    a.restore()
    a.append()
    ids = _used_pages(w)
    image = a.save(ids, mode="staged")
    b = DeviceBatch(w, with_restore=False)
    new_ids = np.random.default_rng(1).permutation(w.num_pages)[:ids.size].astype(np.int32)
    import torch
    src = torch.from_numpy(image.view(np.int16)).pin_memory()
    staging = torch.empty_like(src, device="cuda")
    gcb.gc_kv_restore(b.pool.handle, src, _i32(new_ids, "cuda"), ids.size, None, staging, 0)
    assert b.check() == gcb.GC_OK and a.check() == gcb.GC_OK
    pa, pb = a.pool_bits(), b.pool_bits()
    assert np.array_equal(pa[:, :, ids], pb[:, :, new_ids])
    a.close()
    b.close()


def test_save_skips_out_of_range_block_and_reports_it():
    w = wl.tiny()
    db = DeviceBatch(w)
    db.restore()
    db.append()
    ids = _used_pages(w)
    ids[2] = -3
    got = db.save(ids, mode="device", fill=0x1234)
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    keep = np.ones(ids.size, bool)
    keep[2] = False
    assert np.array_equal(got[keep], oracle.kv_gather_blocks(oracle_pool(w), ids[keep]))
    assert np.all(got[2] == 0x1234)
    db.close()


def _layered(seed=15):
    w = wl.custom("layered", 3, 8, 2, 64, 16, [90, 0, 257], [7, 3, 20], seed=seed)
    w.L = 5
    return w


@pytest.mark.parametrize("mode,vector", [("staged", False), ("staged", True), ("device", False),
                                         ("zerocopy", False)])
@pytest.mark.parametrize("lb,lc", [(0, 5), (1, 2), (4, 1)])
@pytest.mark.parametrize("layer_major", [False, True])
def test_restore_layers_bit_exact(mode, vector, lb, lc, layer_major):
    """gc_kv_restore_layers writes exactly the chosen layers' pages of the
    cached image (block-major or layer-major) and leaves every other layer
    untouched."""
    w = _layered()
    db = DeviceBatch(w)
    if layer_major:  # the same image with its first two axes swapped (layout only)
        img = np.ascontiguousarray(w.host_src().swapaxes(0, 1))
        db.host_src = bf16_tensor(img, pin=True)
        db.staging = db.staging.view(db.host_src.shape)
    if mode == "device":
        db.stage()
    src = db.staging if mode == "device" else db.host_src
    staging = db.staging if mode == "staged" else None
    flags = (gcb.GC_RESTORE_VECTOR if vector else 0) | (
        gcb.GC_RESTORE_SRC_DEVICE if mode == "device" else 0) | (
        gcb.GC_RESTORE_LAYER_MAJOR if layer_major else 0)
    gcb.gc_kv_restore_layers(db.pool.handle, src, db.block_ids, db.n_blocks, lb, lc, None,
                             staging, flags)
    assert db.check() == gcb.GC_OK
    full = oracle_pool(w, append=False)
    want = w.empty_pool()
    want[lb:lb + lc] = full[lb:lb + lc]
    assert np.array_equal(db.pool_bits(), want)
    db.close()


def test_restore_layers_one_call_per_layer_equals_whole_restore():
    w = _layered(16)
    db = DeviceBatch(w)
    for l in range(w.L):
        gcb.gc_kv_restore_layers(db.pool.handle, db.host_src, db.block_ids, db.n_blocks, l, 1,
                                 None, db.staging, 0)
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), oracle_pool(w, append=False))
    db.close()


@pytest.mark.parametrize("mode", ["staged", "device", "zerocopy"])
@pytest.mark.parametrize("lb,lc", [(0, 5), (2, 3), (3, 1)])
@pytest.mark.parametrize("layer_major", [False, True])
def test_save_layers_bit_exact(mode, lb, lc, layer_major):
    """gc_kv_save_layers writes the chosen layers' slices of the image (the
    oracle's gather; block-major or layer-major) and no other byte of it."""
    import torch
    w = _layered(17)
    db = DeviceBatch(w)
    db.restore()
    db.append()
    ids = _used_pages(w)
    n = ids.size
    shape = (w.L, n, 2, w.Hkv, w.ps, w.d) if layer_major else (n, w.L, 2, w.Hkv, w.ps, w.d)
    fill = int(np.uint16(0x1234).view(np.int16))
    flags = (gcb.GC_SAVE_DST_DEVICE if mode == "device" else 0) | (
        gcb.GC_SAVE_LAYER_MAJOR if layer_major else 0)
    if mode == "device":
        dst = torch.full(shape, fill, dtype=torch.int16, device="cuda")
    else:
        dst = torch.full(shape, fill, dtype=torch.int16).pin_memory()
    staging = torch.empty(shape, dtype=torch.int16, device="cuda") if mode == "staged" else None
    gcb.gc_kv_save_layers(db.pool.handle, dst, _i32(ids, "cuda"), n, lb, lc, None, staging, flags)
    assert db.check() == gcb.GC_OK
    got = dst.cpu().numpy().view(np.uint16)
    if layer_major:
        got = got.swapaxes(0, 1)
    want = np.full((n, w.L, 2, w.Hkv, w.ps, w.d), 0x1234, dtype=np.uint16)
    want[:, lb:lb + lc] = oracle.kv_gather_blocks(oracle_pool(w), ids)[:, lb:lb + lc]
    assert np.array_equal(got, want)
    db.close()


def test_layer_range_checks():
    w = _layered(18)
    db = DeviceBatch(w)
    before = db.pool_bits()
    for lb, lc in [(-1, 1), (0, 6), (5, 1), (2, -1), (4, 2)]:
        for fn, buf in ((gcb.gc_kv_restore_layers, db.host_src),
                        (gcb.gc_kv_save_layers, db.host_src)):
            with pytest.raises(gcb.GcError) as e:
                fn(db.pool.handle, buf, db.block_ids, db.n_blocks, lb, lc, None, db.staging, 0)
            assert e.value.status == gcb.GC_ERR_OUT_OF_RANGE
    gcb.gc_kv_restore_layers(db.pool.handle, db.host_src, db.block_ids, db.n_blocks, 5, 0, None,
                             db.staging, 0)  # empty range at the end: a no-op
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), before)
    db.close()


# ------------------------------------------------------ 8-bit cache tier
def _q8_image_shape(w, n, layer_major):
    import oracle as _o
    chunk = _o.q8_chunk_bytes(w.Hkv, w.ps, w.d)
    return (w.L, n, 2, chunk) if layer_major else (n, w.L, 2, chunk)


@pytest.mark.parametrize("mode", ["staged", "device", "zerocopy"])
@pytest.mark.parametrize("lb,lc", [(0, 5), (1, 3)])
@pytest.mark.parametrize("layer_major", [False, True])
def test_save_q8_bit_exact(mode, lb, lc, layer_major):
    """INT8 codes and scales of the chosen layers equal the oracle's, bit for
    bit (pages carry NaN in their unused tail slots); other chunks untouched."""
    import torch
    w = _layered(19)
    db = DeviceBatch(w)
    db.restore()
    db.append()
    ids = _used_pages(w)
    n = ids.size
    shape = _q8_image_shape(w, n, layer_major)
    flags = (gcb.GC_SAVE_DST_DEVICE if mode == "device" else 0) | (
        gcb.GC_SAVE_LAYER_MAJOR if layer_major else 0)
    if mode == "device":
        dst = torch.full(shape, 0xAB, dtype=torch.uint8, device="cuda")
    else:
        dst = torch.full(shape, 0xAB, dtype=torch.uint8).pin_memory()
    staging = torch.empty(shape, dtype=torch.uint8, device="cuda") if mode == "staged" else None
    gcb.gc_kv_save_q8(db.pool.handle, dst, _i32(ids, "cuda"), n, lb, lc, None, staging, flags)
    assert db.check() == gcb.GC_OK
    got = dst.cpu().numpy()
    if layer_major:
        got = got.swapaxes(0, 1)
    want = np.full((n, w.L, 2, shape[-1]), 0xAB, dtype=np.uint8)
    oracle.kv_save_q8(oracle_pool(w), ids, lb, lc, out=want)
    assert np.array_equal(got, want)
    db.close()


@pytest.mark.parametrize("mode", ["staged", "device", "zerocopy"])
@pytest.mark.parametrize("lb,lc", [(0, 5), (2, 1)])
@pytest.mark.parametrize("layer_major", [False, True])
def test_restore_q8_bit_exact(mode, lb, lc, layer_major):
    """Dequantising an oracle-made INT8 image into the pool gives the
    oracle's pool bit for bit; other layers and pages are untouched."""
    import torch
    w = _layered(20)
    ids = w.prefix_blocks()
    src_pool = w.empty_pool()
    oracle.kv_restore(src_pool, w.host_src(), ids)
    img = oracle.kv_save_q8(src_pool, ids)                    # [n][L][2][chunk]
    want = w.empty_pool()
    oracle.kv_restore_q8(want, img, ids, lb, lc)
    db = DeviceBatch(w)
    if layer_major:
        img = np.ascontiguousarray(img.swapaxes(0, 1))
    host = torch.from_numpy(img).pin_memory()
    flags = gcb.GC_RESTORE_LAYER_MAJOR if layer_major else 0
    if mode == "device":
        src, staging, flags = host.cuda(), None, flags | gcb.GC_RESTORE_SRC_DEVICE
    elif mode == "staged":
        src, staging = host, torch.empty_like(host, device="cuda")
    else:
        src, staging = host, None
    gcb.gc_kv_restore_q8(db.pool.handle, src, db.block_ids, db.n_blocks, lb, lc, None, staging,
                         flags)
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), want)
    db.close()


def test_q8_gpu_round_trip_and_bad_id():
    """GPU save then GPU restore reproduces the oracle's round trip; a bad
    block id is skipped and reported by both calls."""
    import torch
    w = _layered(21)
    db = DeviceBatch(w)
    db.restore()
    db.append()
    ids = _used_pages(w)
    n = ids.size
    img = torch.zeros(_q8_image_shape(w, n, False), dtype=torch.uint8, device="cuda")
    gcb.gc_kv_save_q8(db.pool.handle, img, _i32(ids, "cuda"), n, 0, w.L, None, None,
                      gcb.GC_SAVE_DST_DEVICE)
    b = DeviceBatch(w, with_restore=False)
    gcb.gc_kv_restore_q8(b.pool.handle, img, _i32(ids, "cuda"), n, 0, w.L, None, None,
                         gcb.GC_RESTORE_SRC_DEVICE)
    assert db.check() == gcb.GC_OK and b.check() == gcb.GC_OK
    ref = w.empty_pool()
    oracle.kv_restore_q8(ref, oracle.kv_save_q8(oracle_pool(w), ids), ids)
    assert np.array_equal(b.pool_bits(), ref)
    bad = ids.copy()
    bad[1] = w.num_pages
    gcb.gc_kv_save_q8(db.pool.handle, img, _i32(bad, "cuda"), n, 0, w.L, None, None,
                      gcb.GC_SAVE_DST_DEVICE)
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    gcb.gc_kv_restore_q8(b.pool.handle, img, _i32(bad, "cuda"), n, 0, w.L, None, None,
                         gcb.GC_RESTORE_SRC_DEVICE)
    assert b.check() == gcb.GC_ERR_OUT_OF_RANGE
    db.close()
    b.close()


def test_q8_subnormal_and_large_groups_match_oracle():
    """Groups of tiny (subnormal) values, where 127/amax overflows, and of
    large values take the general path and still match the oracle bit for bit."""
    import torch
    w = _layered(22)
    src = wl.bf16_bits_to_f32(w.host_src())
    src[0::3] *= 2.0 ** -130          # subnormal magnitudes in bf16
    src[1::3] *= 2.0 ** 100
    w._cache["src"] = wl.f32_to_bf16_bits(src)
    db = DeviceBatch(w)
    db.restore()
    ids = w.prefix_blocks()
    n = ids.size
    img = torch.zeros(_q8_image_shape(w, n, False), dtype=torch.uint8, device="cuda")
    gcb.gc_kv_save_q8(db.pool.handle, img, db.block_ids, n, 0, w.L, None, None,
                      gcb.GC_SAVE_DST_DEVICE)
    assert db.check() == gcb.GC_OK
    want = oracle.kv_save_q8(oracle_pool(w, append=False), ids)
    assert np.array_equal(img.cpu().numpy(), want)
    b = DeviceBatch(w, with_restore=False)
    gcb.gc_kv_restore_q8(b.pool.handle, img, db.block_ids, n, 0, w.L, None, None,
                         gcb.GC_RESTORE_SRC_DEVICE)
    assert b.check() == gcb.GC_OK
    ref = w.empty_pool()
    oracle.kv_restore_q8(ref, want, ids)
    assert np.array_equal(b.pool_bits(), ref)
    db.close()
    b.close()


# --------------------------------------------------------- failure handling
def test_bounded_wait_times_out_and_reports():
    """A device wait nobody satisfies gives up after its limit (~1.5 s), is
    reported as GC_ERR_TIMEOUT, and leaves the context usable."""
    import time
    pool = gcb.KVPool.create(1, 1, 64, 16, 4)
    t0 = time.time()
    gcb.gc_selftest_wait_timeout(pool.handle)
    assert pool.check() == gcb.GC_ERR_TIMEOUT
    assert 0.5 < time.time() - t0 < 30
    assert pool.check() == gcb.GC_OK  # read and cleared
    pool.close()
    w = wl.tiny()
    db = DeviceBatch(w)
    db.restore()
    assert db.check() == gcb.GC_OK
    assert np.array_equal(db.pool_bits(), oracle_pool(w, append=False))
    db.close()


def test_pool_create_out_of_memory_is_reported():
    """A library-owned pool larger than the GPU fails with GC_ERR_OOM and
    later allocations still succeed."""
    cfg = gcb.make_config(1, 8, 128, 16, 2**24)  # 1 TiB of pages
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_kv_pool_create(cfg)
    assert e.value.status == gcb.GC_ERR_OOM
    h = gcb.gc_kv_pool_create(gcb.make_config(1, 1, 64, 16, 4))
    gcb.gc_kv_pool_destroy(h)
