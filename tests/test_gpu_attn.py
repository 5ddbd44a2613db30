"""GPU parity of prefix-reuse attention against the float64 oracle, through
the C ABI, plus metamorphic checks that need no oracle (bit-exact)."""
import numpy as np
import pytest

import oracle
from paper_2505_23970_gb300 import binding as gcb
from paper_2505_23970_gb300 import workloads as wl
from paper_2505_23970_gb300.harness import DeviceBatch, _i32, bf16_tensor

from ._util import assert_attn_close, gather_rows, sample_rows

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


def full_parity(w, impl="tc"):
    db = DeviceBatch(w)
    db.run(impl=impl)
    assert db.check() == gcb.GC_OK
    got = db.out_f64()
    db.close()
    ref = oracle.prefix_attn(w.q(), oracle_pool(w), 0, w.block_table, w.prefix_lens,
                             w.cu_new_lens, w.scale)
    return assert_attn_close(got, ref, f"{w.name} [{impl}]")


def sampled_parity(w, n_random=512, impl="tc"):
    db = DeviceBatch(w)
    db.run(impl=impl)
    assert db.check() == gcb.GC_OK
    got = db.out_f64()
    db.close()
    rows = sample_rows(w, n_random)
    ref = oracle.prefix_attn_rows(w.q(), oracle_pool(w), 0, w.block_table, w.prefix_lens,
                                  w.cu_new_lens, w.scale, rows)
    return assert_attn_close(gather_rows(got, w, rows), ref, f"{w.name} sampled [{impl}]")


# ------------------------------------------------------------ the five configs
@pytest.mark.parametrize("impl", ["tc", "simt"])
def test_tiny_config(impl):
    full_parity(wl.tiny(), impl)


@pytest.mark.parametrize("impl", ["tc", "simt"])
def test_llama3_8b_layer(impl):
    full_parity(wl.llama3_8b_layer(seed=0), impl)


def test_llama3_70b_layer_sampled():
    sampled_parity(wl.llama3_70b_layer(seed=0), n_random=768)


@pytest.mark.parametrize("hit_p", [0.0, 0.5, 1.0])
def test_conversation_mix_sampled(hit_p):
    sampled_parity(wl.conversation_mix(seed=1, hit_p=hit_p), n_random=512)


def test_long_document_sampled():
    sampled_parity(wl.long_document(seed=0), n_random=256)


def test_long_document_recompute_sampled():
    sampled_parity(wl.long_document(seed=0, recompute=True), n_random=128)


# --------------------------------------------------------------- edge cases
@pytest.mark.parametrize("G,d,ps", [(1, 128, 16), (2, 64, 32), (4, 64, 16), (8, 128, 64),
                                    (16, 128, 128), (8, 64, 128), (4, 128, 32)])
def test_head_grouping_dims_and_page_sizes(G, d, ps):
    Hkv = 2
    w = wl.custom(f"g{G}d{d}p{ps}", 4, Hkv * G, Hkv, d, ps, [0, 77, 300, 129], [200, 1, 45, 130],
                  seed=G * 7 + d + ps)
    full_parity(w)


def test_ragged_lengths_and_empty_requests():
    """Requests with no new tokens, prefixes ending mid-page, new rows that
    do not fill a Q tile, a prefix of 0 and one-token requests."""
    w = wl.custom("ragged", 7, 16, 2, 128, 16, [0, 5, 17, 128, 255, 0, 1000],
                  [3, 0, 1, 129, 17, 1, 0], seed=3)
    full_parity(w)


def test_batch_with_no_new_tokens_is_noop():
    import torch
    w = wl.custom("none", 2, 8, 1, 64, 16, [10, 20], [0, 0], seed=4)
    db = DeviceBatch(w)
    db.restore()
    gcb.gc_prefix_prefill_attn(db.q, db.pool.handle, db.block_table, db.prefix_lens, db.new_lens,
                               db.out, None, 0, db.cu_new_lens, w.B, w.max_blocks, w.Hq, w.scale,
                               0)
    assert db.check() == gcb.GC_OK
    db.close()


def test_single_key_row_returns_v_bit_exact():
    """prefix 0, row 0: one visible key, so the output is v_0 exactly."""
    import torch
    w = wl.custom("single", 3, 8, 2, 128, 16, [0, 0, 0], [1, 5, 130], seed=6)
    db = DeviceBatch(w)
    db.run()
    assert db.check() == gcb.GC_OK
    cu = w.cu_new_lens
    _, v = w.kv_new()
    for b in range(w.B):
        row = db.out[cu[b]].view(torch.int16).cpu().numpy().view(np.uint16)
        for h in range(w.Hq):
            assert np.array_equal(row[h], v[cu[b], h // w.G])
    db.close()


def test_tc_matches_simt_kernel():
    w = wl.custom("xcheck", 3, 32, 4, 128, 16, [700, 33, 0], [300, 70, 260], seed=8)
    a = DeviceBatch(w)
    a.run(impl="tc")
    b = DeviceBatch(w)
    b.run(impl="simt")
    assert a.check() == gcb.GC_OK and b.check() == gcb.GC_OK
    assert_attn_close(a.out_f64(), b.out_f64(), "tc vs simt")
    a.close()
    b.close()


# -------------------------------------------------------------- metamorphic
def test_deterministic_run_to_run():
    import torch
    w = wl.llama3_8b_layer(seed=5, B=6)
    db = DeviceBatch(w)
    db.run()
    first = db.out.clone()
    for _ in range(2):
        db.out.fill_(0)
        db.attn()
        assert torch.equal(db.out.view(torch.int16), first.view(torch.int16))
    db.close()


def test_page_permutation_invariance():
    """Moving every page elsewhere in the pool (and the block table with it)
    leaves the output bit-identical."""
    import torch
    w = wl.custom("perm", 3, 16, 2, 128, 16, [100, 0, 260], [90, 33, 64], seed=9)
    a = DeviceBatch(w)
    a.run()
    w2 = wl.custom("perm", 3, 16, 2, 128, 16, [100, 0, 260], [90, 33, 64], seed=9)
    perm = np.random.default_rng(0).permutation(w2.num_pages).astype(np.int32)
    bt = np.where(w2.block_table >= 0, perm[np.maximum(w2.block_table, 0)], -1).astype(np.int32)
    w2.block_table = bt
    w2._cache = dict(w._cache)  # same tensors, new placement
    b = DeviceBatch(w2)
    b.run()
    assert a.check() == gcb.GC_OK and b.check() == gcb.GC_OK
    assert torch.equal(a.out.view(torch.int16), b.out.view(torch.int16))
    a.close()
    b.close()


def test_batch_composition_invariance():
    """A request's output does not depend on the other requests in the batch."""
    import torch
    P, n = [300, 17, 1000, 0], [40, 129, 7, 250]
    w = wl.custom("batch", 4, 32, 4, 128, 16, P, n, seed=10)
    full = DeviceBatch(w)
    full.run()
    assert full.check() == gcb.GC_OK
    cu = w.cu_new_lens
    for b in range(4):
        wb = wl.custom("one", 1, 32, 4, 128, 16, [P[b]], [n[b]], seed=10)
        # same tensors as request b of the batch
        pool_src = w.host_src()
        blocks = [-(-p // 16) for p in P]
        start = sum(blocks[:b])
        wb._cache["src"] = pool_src[start:start + blocks[b]]
        k, v = w.kv_new()
        wb._cache["kvn"] = (k[cu[b]:cu[b + 1]], v[cu[b]:cu[b + 1]])
        wb._cache["q"] = w.q()[cu[b]:cu[b + 1]]
        one = DeviceBatch(wb)
        one.run()
        assert one.check() == gcb.GC_OK
        assert torch.equal(one.out.view(torch.int16), full.out[cu[b]:cu[b + 1]].view(torch.int16))
        one.close()
    full.close()


def test_bad_block_table_entry_is_reported_not_faulted():
    w = wl.custom("badbt", 2, 8, 1, 64, 16, [40, 8], [30, 9], seed=11)
    db = DeviceBatch(w)
    db.run()
    assert db.check() == gcb.GC_OK
    bt = w.block_table.copy()
    bt[1, 0] = -5
    db.block_table = _i32(bt, "cuda")
    db.attn()
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    db.close()


def test_large_score_jumps_take_the_exact_path():
    """Keys whose scores jump far above the running row max (by more than
    the overflow guard, in the second half of one tile and the first half of
    a later one) must still give the softmax definition."""
    w = wl.custom("jumps", 1, 8, 1, 128, 16, [512], [64], seed=12)
    src = wl.bf16_bits_to_f32(w.host_src())          # [32 blocks][1][2][1][16][128]
    keys = src[:, 0, 0, 0].reshape(-1, 128)            # prefix keys in order
    keys[192:256] *= 256.0                             # tile 1, second half
    keys[256:320] *= 1024.0                            # tile 2, first half
    src[:, 0, 0, 0] = keys.reshape(-1, 16, 128)
    w._cache["src"] = wl.f32_to_bf16_bits(src)
    full_parity(w)


@pytest.mark.parametrize("schedule", ["copy-stream", "side-restore"])
def test_layer_pipelined_schedule_matches_serial_and_oracle(schedule):
    """Restoring layer l in a pipeline with the layers' compute — each layer's
    copy on a copy stream (gc_kv_stage_layers) and its scatter right before
    its append and attention, or one staged gc_kv_restore_layers call per
    layer on a side stream — leaves the pool and every layer's output
    bit-identical to restoring all layers first; the pool equals the
    oracle's and the outputs match its attention."""
    import torch
    from paper_2505_23970_gb300.harness import LayerStack
    w = wl.custom("layers", 2, 16, 2, 128, 16, [700, 33], [64, 130], seed=14)
    w.L = 4
    serial = LayerStack(w, keep_outputs=True)
    serial.run(pipelined=False)
    piped = LayerStack(w, keep_outputs=True)
    piped.run(pipelined=True, schedule=schedule)
    assert serial.check() == gcb.GC_OK and piped.check() == gcb.GC_OK
    for a, b in zip(serial.outs, piped.outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    pool = w.empty_pool()
    oracle.kv_restore(pool, w.host_src(), w.prefix_blocks())
    k, v = w.kv_new()
    for l in range(w.L):
        oracle.kv_append(pool, l, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    assert np.array_equal(piped.pool_bits(), pool)
    assert np.array_equal(serial.pool_bits(), pool)
    for l in (0, 3):
        ref = oracle.prefix_attn(w.q(), pool, l, w.block_table, w.prefix_lens, w.cu_new_lens,
                                 w.scale)
        assert_attn_close(piped.outs[l].to(torch.float64).cpu().numpy(), ref, f"layer {l}")
    serial.close()
    piped.close()


def test_layer_pipeline_from_the_8bit_tier_matches_whole_restore():
    """With the cache tier holding the 8-bit image, the copy-stream pipeline
    (gc_kv_stage_layers with GC_STAGE_Q8, then gc_kv_restore_q8 of one layer
    from the device image) leaves the same pool and outputs, bit for bit, as
    dequantising every layer at once before the compute."""
    import torch
    from paper_2505_23970_gb300.harness import LayerStack
    w = wl.custom("layers-q8", 2, 16, 2, 128, 16, [520, 47], [40, 129], seed=15)
    w.L = 3
    stacks = []
    for pipelined in (False, True):
        st = LayerStack(w, keep_outputs=True)
        st.restore_all(None)
        st.use_q8()
        st.pool.planes().view(torch.int16).fill_(0x7FC0)
        st.run(pipelined=pipelined)
        assert st.check() == gcb.GC_OK
        stacks.append(st)
    serial, piped = stacks
    assert np.array_equal(serial.pool_bits(), piped.pool_bits())
    for a, b in zip(serial.outs, piped.outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    for st in stacks:
        st.close()


def test_batch_beyond_sorted_ranking():
    """More requests than the kernel ranks by length (512): work items keep
    the given request order; outputs still match the oracle."""
    rng = np.random.default_rng(21)
    B = 700
    P = rng.integers(0, 300, size=B)
    n = rng.integers(0, 40, size=B)
    w = wl.custom("big-batch", B, 16, 4, 64, 16, P, n, seed=21)
    full_parity(w)


def test_output_canaries_untouched():
    """Prefill and decode write exactly their output rows: a canary after the
    end of the output buffer keeps its bytes."""
    import torch
    w = wl.custom("canary", 3, 16, 2, 128, 16, [100, 0, 37], [20, 5, 1], seed=23)
    db = DeviceBatch(w)
    db.restore()
    db.append()
    rows = w.T_new * w.Hq * w.d
    buf = torch.full((rows + 4096,), -7.0, dtype=torch.bfloat16, device="cuda")
    out = buf[:rows].view(w.T_new, w.Hq, w.d)
    db.attn(out=out)
    assert db.check() == gcb.GC_OK
    assert torch.all(buf[rows:] == -7.0)
    wd = wl.custom("canary-dec", 3, 16, 2, 128, 16, [100, 0, 37], [1, 1, 1], seed=24)
    dd = DeviceBatch(wd)
    dd.restore()
    dd.append()
    rows = wd.B * wd.Hq * wd.d
    buf = torch.full((rows + 4096,), -7.0, dtype=torch.bfloat16, device="cuda")
    dd.decode(out=buf[:rows].view(wd.B, wd.Hq, wd.d))
    assert dd.check() == gcb.GC_OK
    assert torch.all(buf[rows:] == -7.0)
    db.close()
    dd.close()


def test_work_item_bound_refused_before_launch():
    """A call whose 32-bit work numbering could overflow (q rows or work items
    near 2^31) is refused on the host with GC_ERR_UNSUPPORTED: the dummy
    arrays below are far too small and are never touched."""
    import torch
    dummy = torch.zeros(1024, dtype=torch.int32, device="cuda")
    # 16 q heads per kv head x 2^27 new tokens = 2^31 q rows
    pool = gcb.KVPool.create(1, 64, 64, 16, 1)
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_prefix_prefill_attn(dummy, pool.handle, dummy, dummy, dummy, dummy, None, 0, dummy,
                                   1, 1, 64 * 16, 0.125, 2**27)
    assert e.value.status == gcb.GC_ERR_UNSUPPORTED
    assert "work items" in gcb.gc_last_error()
    assert pool.check() == gcb.GC_OK
    pool.close()
    # q rows within bounds, but 512 kv heads x (2^31 - 512) / 256 row groups
    # give more work items than the counter can hand out
    pool = gcb.KVPool.create(1, 512, 64, 16, 1)
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_prefix_prefill_attn(dummy, pool.handle, dummy, dummy, dummy, dummy, None, 0, dummy,
                                   1, 1, 512, 0.125, 2**31 - 512)
    assert e.value.status == gcb.GC_ERR_UNSUPPORTED
    assert "work items" in gcb.gc_last_error()
    assert pool.check() == gcb.GC_OK
    pool.close()


# ------------------------------------------------------- the CTA-pair kernel
# head_dim 128 prefill runs on the CTA-pair kernel; these cases also widen
# the block table with unused (-1) columns to a 65536-token capacity, as a
# long-context server's tables are.
PAIR_KEYS = 65536


def on_pair_kernel(w):
    cols = -(-PAIR_KEYS // w.ps)
    if w.max_blocks < cols:
        w.block_table = np.pad(w.block_table, ((0, 0), (0, cols - w.max_blocks)),
                               constant_values=-1).astype(np.int32)
    return w


@pytest.mark.parametrize("make", [
    lambda: wl.llama3_8b_layer(seed=0),
    lambda: wl.custom("pair-g1", 4, 2, 2, 128, 16, [0, 77, 300, 129], [200, 1, 45, 130], seed=31),
    lambda: wl.custom("pair-g8p64", 4, 16, 2, 128, 64, [0, 77, 300, 129], [200, 1, 45, 130], seed=32),
    lambda: wl.custom("pair-g16p128", 4, 32, 2, 128, 128, [0, 77, 300, 129], [200, 1, 45, 130],
                      seed=33),
    lambda: wl.custom("pair-g4p32", 4, 8, 2, 128, 32, [0, 77, 300, 129], [200, 1, 45, 130], seed=34),
    lambda: wl.custom("pair-ragged", 7, 16, 2, 128, 16, [0, 5, 17, 128, 255, 0, 1000],
                      [3, 0, 1, 129, 17, 1, 0], seed=35),
], ids=["8b", "g1p16", "g8p64", "g16p128", "g4p32", "ragged"])
def test_pair_kernel_parity(make):
    full_parity(on_pair_kernel(make()))


def test_pair_kernel_70b_sampled():
    sampled_parity(on_pair_kernel(wl.llama3_70b_layer(seed=2)), n_random=384)


def test_pair_kernel_single_key_row_returns_v_bit_exact():
    import torch
    w = on_pair_kernel(wl.custom("pair-single", 3, 8, 2, 128, 16, [0, 0, 0], [1, 5, 130], seed=36))
    db = DeviceBatch(w)
    db.run()
    assert db.check() == gcb.GC_OK
    cu = w.cu_new_lens
    _, v = w.kv_new()
    for b in range(w.B):
        row = db.out[cu[b]].view(torch.int16).cpu().numpy().view(np.uint16)
        for h in range(w.Hq):
            assert np.array_equal(row[h], v[cu[b], h // w.G])
    db.close()


def test_pair_kernel_large_score_jumps():
    w = on_pair_kernel(wl.custom("pair-jumps", 1, 8, 1, 128, 16, [512], [64], seed=12))
    src = wl.bf16_bits_to_f32(w.host_src())
    keys = src[:, 0, 0, 0].reshape(-1, 128)
    keys[192:256] *= 256.0
    keys[256:320] *= 1024.0
    src[:, 0, 0, 0] = keys.reshape(-1, 16, 128)
    w._cache["src"] = wl.f32_to_bf16_bits(src)
    full_parity(w)


def test_pair_kernel_deterministic_and_page_permutation_invariant():
    import torch
    w = on_pair_kernel(wl.custom("pair-perm", 3, 16, 2, 128, 16, [100, 0, 260], [90, 33, 64],
                                 seed=37))
    a = DeviceBatch(w)
    a.run()
    first = a.out.clone()
    a.out.fill_(0)
    a.attn()
    assert torch.equal(a.out.view(torch.int16), first.view(torch.int16))
    w2 = on_pair_kernel(wl.custom("pair-perm", 3, 16, 2, 128, 16, [100, 0, 260], [90, 33, 64],
                                  seed=37))
    perm = np.random.default_rng(1).permutation(w2.num_pages).astype(np.int32)
    w2.block_table = np.where(w2.block_table >= 0, perm[np.maximum(w2.block_table, 0)],
                              -1).astype(np.int32)
    w2._cache = dict(w._cache)
    b = DeviceBatch(w2)
    b.run()
    assert a.check() == gcb.GC_OK and b.check() == gcb.GC_OK
    assert torch.equal(first.view(torch.int16), b.out.view(torch.int16))
    a.close()
    b.close()


def test_pair_kernel_bad_block_table_entry_is_reported_not_faulted():
    w = on_pair_kernel(wl.custom("pair-badbt", 2, 8, 1, 128, 16, [40, 8], [30, 9], seed=38))
    db = DeviceBatch(w)
    db.run()
    assert db.check() == gcb.GC_OK
    bt = w.block_table.copy()
    bt[1, 0] = -5
    db.block_table = _i32(bt, "cuda")
    db.attn()
    assert db.check() == gcb.GC_ERR_OUT_OF_RANGE
    db.close()


@pytest.mark.parametrize("q8", [False, True])
def test_layer_pipeline_captured_in_a_cuda_graph(q8):
    """The copy-stream layer pipeline recorded into a CUDA graph and replayed
    gives the eager run's pool and outputs bit for bit."""
    import torch
    from paper_2505_23970_gb300.harness import LayerStack
    w = wl.custom("layers-graph", 2, 16, 2, 128, 16, [520, 47], [40, 129], seed=16)
    w.L = 3
    eager = LayerStack(w, keep_outputs=True)
    if q8:
        eager.restore_all(None)
        eager.use_q8()
    eager.run(pipelined=True)
    torch.cuda.synchronize()
    assert eager.check() == gcb.GC_OK
    graphed = LayerStack(w, keep_outputs=True)
    if q8:
        graphed.restore_all(None)
        graphed.use_q8()
    g = graphed.capture(pipelined=True)
    for o in graphed.outs:
        o.fill_(float("nan"))
    graphed.pool.planes().view(torch.int16).fill_(0x7FC0)
    g.replay()
    torch.cuda.synchronize()
    assert graphed.check() == gcb.GC_OK
    assert np.array_equal(eager.pool_bits(), graphed.pool_bits())
    for a, b in zip(eager.outs, graphed.outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    eager.close()
    graphed.close()


# ------------------------------------------------------- the largest batch
def _max_batch_workload(seed, d=128):
    rng = np.random.default_rng(seed)
    B = 8192
    P = rng.integers(0, 40, size=B)
    n = rng.integers(0, 4, size=B)
    return wl.custom(f"batch-8192-{seed}-d{d}", B, 4, 2, d, 16, P, n, seed=seed)


@pytest.mark.parametrize("kernel", ["one-sm", "pairs"])
def test_largest_batch(kernel):
    """8192 requests, the most one call takes (the unit table then fills
    the shared memory both kernels have left), on the one-SM kernel (head_dim
    64) and on SM pairs (head_dim 128); 8193 requests are refused before
    anything is launched."""
    w = _max_batch_workload(41, d=64 if kernel == "one-sm" else 128)
    full_parity(w)
    import torch
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    pool = gcb.KVPool.create(1, 2, 128, 16, 4)
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_prefix_prefill_attn(dummy, pool.handle, dummy, dummy, dummy, dummy, None, 0, dummy,
                                   8193, 1, 4, 0.1, 16)
    assert e.value.status == gcb.GC_ERR_UNSUPPORTED
    pool.close()
