"""The C-ABI library loads on a machine without a GPU and exports every
symbol include/gc.h declares; host-side checks answer without touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2505_23970_gb300 import binding as gcb
from paper_2505_23970_gb300 import build as gbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    gbuild.build()
    return gcb.load()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "gc.h")).read()
    return sorted(set(re.findall(r"GC_API\s+[\w\s\*]+?\b(gc_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("gc_kv_pool_create", "gc_kv_restore", "gc_kv_append",
                     "gc_prefix_prefill_attn"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(gcb.EXPORTED) == set(declared_functions())


def test_pool_bytes_arithmetic(lib):
    cfg = gcb.make_config(80, 8, 128, 16, 640)
    planes = 80 * 2 * 640 * 8 * 16 * 128 * 2
    assert gcb.gc_kv_pool_bytes(cfg) == planes + 2048
    assert gcb.gc_kv_pool_bytes(gcb.make_config(0, 8, 128, 16, 10)) == 0


@pytest.mark.parametrize("cfg,status", [
    ((1, 1, 64, 16, 0), gcb.GC_ERR_INVALID_ARG),
    ((1, 0, 64, 16, 4), gcb.GC_ERR_INVALID_ARG),
    ((1, 1, 96, 16, 4), gcb.GC_ERR_UNSUPPORTED),
    ((1, 1, 128, 8, 4), gcb.GC_ERR_UNSUPPORTED),
])
def test_pool_create_rejects_bad_configs(lib, cfg, status):
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_kv_pool_create(gcb.make_config(*cfg))
    assert e.value.status == status
    assert gcb.gc_last_error()


def test_null_pool_is_rejected_before_any_launch(lib):
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_kv_restore(None, 16, 16, 1, None, None, 0)
    assert e.value.status == gcb.GC_ERR_INVALID_ARG
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_kv_append(None, 16, 16, 16, 16, None, 0, 16, 1, 1, 1)
    assert e.value.status == gcb.GC_ERR_INVALID_ARG
    for fn in (gcb.gc_prefix_prefill_attn, gcb.gc_prefix_prefill_attn_simt):
        with pytest.raises(gcb.GcError) as e:
            fn(16, None, 16, 16, 16, 16, None, 0, 16, 1, 1, 8, 0.1, 1)
        assert e.value.status == gcb.GC_ERR_INVALID_ARG
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_prefix_prefill_attn_q8(16, None, 16, 16, 16, 16, None, 0, 16, 1, 1, 8, 0.1, 1,
                                      16, 16, 1, 0)
    assert e.value.status == gcb.GC_ERR_INVALID_ARG
    with pytest.raises(gcb.GcError) as e:
        gcb.gc_paged_decode_attn_q8(16, None, 16, 16, 16, None, 0, 1, 1, 8, 0.1, 16, 1 << 20,
                                    16, 16, 1, 0)
    assert e.value.status == gcb.GC_ERR_INVALID_ARG


def test_status_strings(lib):
    assert gcb.gc_status_string(gcb.GC_OK) == "GC_OK"
    assert gcb.gc_status_string(gcb.GC_ERR_TIMEOUT) == "GC_ERR_TIMEOUT"
    assert gcb.gc_status_string(99) == "GC_ERR_UNKNOWN"


def test_destroy_null_is_noop(lib):
    gcb.gc_kv_pool_destroy(None)
