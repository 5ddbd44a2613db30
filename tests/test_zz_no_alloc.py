"""The allocation-free attention entry point.

gc_prefix_prefill_attn_noalloc exists for callers that cannot allocate
device memory, such as code running inside a framework whose caching
allocator owns the GPU's memory: its only scratch is a small static array in
libgc. These tests call it through the C ABI and check it against
gc_prefix_prefill_attn on two calls in a row (the second call must find the
shared scratch usable again). This file sorts last so that a run stopping at
the first failure has already run every other test.
"""
import numpy as np
import pytest

from paper_2505_23970_gb300 import binding as gcb
from paper_2505_23970_gb300 import workloads as wl
from paper_2505_23970_gb300.harness import DeviceBatch

from ._util import assert_attn_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2505_23970_gb300 import build
    build.build()


def _call_noalloc(db, out):
    w = db.w
    gcb.gc_prefix_prefill_attn_noalloc(db.q, db.pool.handle, db.block_table, db.prefix_lens,
                                       db.new_lens, out, None, 0, db.cu_new_lens, w.B,
                                       w.max_blocks, w.Hq, w.scale, w.T_new)


def test_noalloc_matches_regular_entry_point_on_two_calls():
    import torch
    w = wl.custom("noalloc", 5, 16, 2, 128, 16, [300, 0, 77, 1000, 5], [64, 200, 1, 33, 129],
                  seed=21)
    db = DeviceBatch(w)
    db.run()                                   # gc_kv_restore + gc_kv_append + attention
    assert db.check() == gcb.GC_OK
    ref = db.out_f64()
    for _ in range(2):
        out = torch.full_like(db.out, float("nan"))
        _call_noalloc(db, out)
        assert db.check() == gcb.GC_OK
        got = out.to(torch.float64).cpu().numpy()
        assert_attn_close(got, ref, "noalloc vs gc_prefix_prefill_attn")
    db.close()


def test_noalloc_allocates_no_device_memory():
    """The pool here lives in memory the caller owns (KVPool.create passes a
    torch buffer as dev_mem).  After the first call, which looks up the static
    scratch's address once, further calls leave the device's free memory
    unchanged: nothing is allocated, not even by the CUDA runtime."""
    import torch
    w = wl.custom("noalloc-mem", 3, 16, 2, 128, 16, [260, 0, 31], [70, 129, 2], seed=22)
    db = DeviceBatch(w)
    db.run()
    assert db.check() == gcb.GC_OK
    ref = db.out_f64()
    out = torch.full_like(db.out, float("nan"))
    _call_noalloc(db, out)                      # first call: symbol lookup
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        _call_noalloc(db, out)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"free device memory changed by {free0 - free1} bytes"
    assert db.check() == gcb.GC_OK
    assert_attn_close(out.to(torch.float64).cpu().numpy(), ref, "noalloc, caller-owned pool")
    db.close()


def test_noalloc_rejects_calls_beyond_its_limit():
    """Up to 2^31 - 1 work items per call fit the static work counter; a call
    that could need more is refused before anything is launched."""
    import torch
    pool = gcb.KVPool.create(1, 64, 64, 16, 1)
    dummy = torch.zeros(1024, dtype=torch.int32, device="cuda")
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_prefix_prefill_attn_noalloc(dummy, pool.handle, dummy, dummy, dummy, dummy, None, 0,
                                           dummy, 8192, 1, 64 * 16, 0.125, 2**31 - 1)
    assert e.value.status == gcb.GC_ERR_UNSUPPORTED
    assert "work items" in gcb.gc_last_error()
    pool.close()
