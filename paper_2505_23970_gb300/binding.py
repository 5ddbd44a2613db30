"""ctypes binding of libgc (include/gc.h), argument marshalling only.

Every function keeps the C name and argument order.  Array arguments accept
a raw address (int), ``None`` or any object with ``data_ptr()`` (a torch
tensor); stream arguments accept an address, ``None`` (legacy default
stream) or an object with ``cuda_stream`` (a ``torch.cuda.Stream``).  A
non-OK status raises :class:`GcError` with the library's message.

There is no fallback: if ``libgc.so`` has not been built, loading raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libgc.so")

GC_OK = 0
GC_ERR_INVALID_ARG = 1
GC_ERR_OUT_OF_RANGE = 2
GC_ERR_OOM = 3
GC_ERR_CUDA = 4
GC_ERR_UNSUPPORTED = 5
GC_ERR_TIMEOUT = 6

GC_RESTORE_SRC_DEVICE = 1
GC_RESTORE_VECTOR = 2
GC_SAVE_DST_DEVICE = 1
GC_SAVE_VECTOR = 2
GC_RESTORE_LAYER_MAJOR = 4
GC_SAVE_LAYER_MAJOR = 4
GC_STAGE_Q8 = 8

EXPORTED = (
    "gc_kv_pool_bytes", "gc_kv_pool_create", "gc_kv_pool_destroy", "gc_kv_pool_data",
    "gc_kv_pool_check", "gc_kv_restore", "gc_kv_save", "gc_kv_restore_layers",
    "gc_kv_save_layers", "gc_kv_stage_layers", "gc_kv_q8_chunk_bytes", "gc_kv_save_q8",
    "gc_kv_restore_q8",
    "gc_kv_append", "gc_prefix_prefill_attn",
    "gc_prefix_prefill_attn_simt", "gc_prefix_prefill_attn_noalloc",
    "gc_prefix_prefill_attn_q8", "gc_paged_decode_attn_q8",
    "gc_paged_decode_workspace_bytes", "gc_paged_decode_attn", "gc_selftest_wait_timeout",
    "gc_last_error",
    "gc_status_string",
)


class gc_pool_config(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("num_pages", ctypes.c_int32)]


class GcError(RuntimeError):
    def __init__(self, status: int, func: str, message: str):
        self.status = status
        super().__init__(f"{func} -> {status_name(status)}: {message}")


_lock = threading.Lock()
_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libgc.so once; raise if it is missing (it is never emulated)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is not built; run __graft_entry__.build() "
                               "(nvcc for sm_103a) first")
        lib = ctypes.CDLL(path)
        vp, i32, u32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint32, ctypes.c_size_t
        cfgp = ctypes.POINTER(gc_pool_config)
        lib.gc_kv_pool_bytes.argtypes = [cfgp]
        lib.gc_kv_pool_bytes.restype = sz
        lib.gc_kv_pool_create.argtypes = [cfgp, vp, sz, ctypes.POINTER(vp)]
        lib.gc_kv_pool_destroy.argtypes = [vp]
        lib.gc_kv_pool_data.argtypes = [vp, ctypes.POINTER(vp), ctypes.POINTER(sz)]
        lib.gc_kv_pool_check.argtypes = [vp, vp, ctypes.POINTER(i32)]
        lib.gc_kv_restore.argtypes = [vp, vp, vp, i32, vp, vp, u32]
        lib.gc_kv_save.argtypes = [vp, vp, vp, i32, vp, vp, u32]
        lib.gc_kv_restore_layers.argtypes = [vp, vp, vp, i32, i32, i32, vp, vp, u32]
        lib.gc_kv_save_layers.argtypes = [vp, vp, vp, i32, i32, i32, vp, vp, u32]
        lib.gc_kv_stage_layers.argtypes = [vp, vp, vp, i32, i32, i32, vp, u32]
        lib.gc_kv_q8_chunk_bytes.argtypes = [ctypes.POINTER(gc_pool_config)]
        lib.gc_kv_q8_chunk_bytes.restype = ctypes.c_size_t
        lib.gc_kv_save_q8.argtypes = [vp, vp, vp, i32, i32, i32, vp, vp, u32]
        lib.gc_kv_restore_q8.argtypes = [vp, vp, vp, i32, i32, i32, vp, vp, u32]
        lib.gc_kv_append.argtypes = [vp, vp, vp, vp, vp, vp, i32, vp, i32, i32, i32]
        attn = [vp, vp, vp, vp, vp, vp, vp, i32, vp, i32, i32, i32, ctypes.c_float, i32]
        lib.gc_prefix_prefill_attn.argtypes = attn
        lib.gc_prefix_prefill_attn_simt.argtypes = attn
        lib.gc_prefix_prefill_attn_noalloc.argtypes = attn
        lib.gc_prefix_prefill_attn_q8.argtypes = attn + [vp, vp, i32, u32]
        lib.gc_selftest_wait_timeout.argtypes = [vp, vp]
        lib.gc_selftest_wait_timeout.restype = ctypes.c_int
        lib.gc_paged_decode_workspace_bytes.argtypes = [vp, i32, i32, i32]
        lib.gc_paged_decode_workspace_bytes.restype = ctypes.c_size_t
        lib.gc_paged_decode_attn.argtypes = [vp, vp, vp, vp, vp, vp, i32, i32, i32, i32,
                                             ctypes.c_float, vp, ctypes.c_size_t]
        lib.gc_paged_decode_attn_q8.argtypes = lib.gc_paged_decode_attn.argtypes + [vp, vp, i32,
                                                                                  u32]
        for f in ("gc_kv_pool_create", "gc_kv_pool_destroy", "gc_kv_pool_data",
                  "gc_kv_pool_check", "gc_kv_restore", "gc_kv_save", "gc_kv_restore_layers",
                  "gc_kv_save_layers", "gc_kv_stage_layers", "gc_kv_save_q8", "gc_kv_restore_q8",
                  "gc_kv_append",
                  "gc_prefix_prefill_attn", "gc_prefix_prefill_attn_simt",
                  "gc_prefix_prefill_attn_noalloc", "gc_prefix_prefill_attn_q8",
                  "gc_paged_decode_attn", "gc_paged_decode_attn_q8"):
            getattr(lib, f).restype = ctypes.c_int
        lib.gc_last_error.argtypes = []
        lib.gc_last_error.restype = ctypes.c_char_p
        lib.gc_status_string.argtypes = [ctypes.c_int]
        lib.gc_status_string.restype = ctypes.c_char_p
        _lib = lib
        return lib


def _addr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "value"):  # ctypes.c_void_p
        return x.value
    raise TypeError(f"cannot take a device/host address of {type(x).__name__}")


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    if hasattr(s, "cuda_stream"):
        return s.cuda_stream
    raise TypeError(f"not a stream: {type(s).__name__}")


def _check(st: int, func: str) -> None:
    if st != GC_OK:
        raise GcError(st, func, gc_last_error())


def status_name(st: int) -> str:
    return load().gc_status_string(st).decode()


def gc_last_error() -> str:
    return load().gc_last_error().decode()


def gc_status_string(st: int) -> str:
    return status_name(st)


def make_config(num_layers, num_kv_heads, head_dim, page_size, num_pages) -> gc_pool_config:
    return gc_pool_config(num_layers, num_kv_heads, head_dim, page_size, num_pages)


def gc_kv_pool_bytes(cfg: gc_pool_config) -> int:
    return load().gc_kv_pool_bytes(ctypes.byref(cfg))


def gc_kv_pool_create(cfg: gc_pool_config, dev_mem=None, dev_bytes: int = 0) -> ctypes.c_void_p:
    h = ctypes.c_void_p()
    _check(load().gc_kv_pool_create(ctypes.byref(cfg), _addr(dev_mem), dev_bytes, ctypes.byref(h)),
           "gc_kv_pool_create")
    return h


def gc_kv_pool_destroy(pool) -> None:
    _check(load().gc_kv_pool_destroy(pool), "gc_kv_pool_destroy")


def gc_kv_pool_data(pool):
    p, n = ctypes.c_void_p(), ctypes.c_size_t()
    _check(load().gc_kv_pool_data(pool, ctypes.byref(p), ctypes.byref(n)), "gc_kv_pool_data")
    return p.value, n.value


def gc_kv_pool_check(pool, stream=None) -> int:
    st = ctypes.c_int32()
    _check(load().gc_kv_pool_check(pool, _stream(stream), ctypes.byref(st)), "gc_kv_pool_check")
    return st.value


def gc_kv_restore(pool, host_src, block_ids, n_blocks: int, stream=None, dev_staging=None,
                  flags: int = 0) -> None:
    _check(load().gc_kv_restore(pool, _addr(host_src), _addr(block_ids), n_blocks,
                                _stream(stream), _addr(dev_staging), flags), "gc_kv_restore")


def gc_kv_save(pool, host_dst, block_ids, n_blocks: int, stream=None, dev_staging=None,
               flags: int = 0) -> None:
    _check(load().gc_kv_save(pool, _addr(host_dst), _addr(block_ids), n_blocks, _stream(stream),
                             _addr(dev_staging), flags), "gc_kv_save")


def gc_kv_restore_layers(pool, host_src, block_ids, n_blocks: int, layer_begin: int,
                         layer_count: int, stream=None, dev_staging=None, flags: int = 0) -> None:
    _check(load().gc_kv_restore_layers(pool, _addr(host_src), _addr(block_ids), n_blocks,
                                       layer_begin, layer_count, _stream(stream),
                                       _addr(dev_staging), flags), "gc_kv_restore_layers")


def gc_kv_save_layers(pool, host_dst, block_ids, n_blocks: int, layer_begin: int,
                      layer_count: int, stream=None, dev_staging=None, flags: int = 0) -> None:
    _check(load().gc_kv_save_layers(pool, _addr(host_dst), _addr(block_ids), n_blocks,
                                    layer_begin, layer_count, _stream(stream), _addr(dev_staging),
                                    flags), "gc_kv_save_layers")


def gc_kv_stage_layers(pool, host_src, dev_image, n_blocks: int, layer_begin: int,
                       layer_count: int, stream=None, flags: int = 0) -> None:
    _check(load().gc_kv_stage_layers(pool, _addr(host_src), _addr(dev_image), n_blocks,
                                     layer_begin, layer_count, _stream(stream), flags),
           "gc_kv_stage_layers")


def gc_kv_q8_chunk_bytes(cfg: gc_pool_config) -> int:
    return int(load().gc_kv_q8_chunk_bytes(ctypes.byref(cfg)))


def gc_kv_save_q8(pool, dst, block_ids, n_blocks: int, layer_begin: int, layer_count: int,
                  stream=None, dev_staging=None, flags: int = 0) -> None:
    _check(load().gc_kv_save_q8(pool, _addr(dst), _addr(block_ids), n_blocks, layer_begin,
                                layer_count, _stream(stream), _addr(dev_staging), flags),
           "gc_kv_save_q8")


def gc_kv_restore_q8(pool, src, block_ids, n_blocks: int, layer_begin: int, layer_count: int,
                     stream=None, dev_staging=None, flags: int = 0) -> None:
    _check(load().gc_kv_restore_q8(pool, _addr(src), _addr(block_ids), n_blocks, layer_begin,
                                   layer_count, _stream(stream), _addr(dev_staging), flags),
           "gc_kv_restore_q8")


def gc_kv_append(pool, k_new, v_new, block_table, seq_lens, stream, layer: int, cu_new_lens,
                 batch: int, max_blocks_per_seq: int, total_new_tokens: int) -> None:
    _check(load().gc_kv_append(pool, _addr(k_new), _addr(v_new), _addr(block_table),
                               _addr(seq_lens), _stream(stream), layer, _addr(cu_new_lens), batch,
                               max_blocks_per_seq, total_new_tokens), "gc_kv_append")


def gc_prefix_prefill_attn(q, pool, block_table, prefix_lens, new_lens, out, stream, layer: int,
                           cu_new_lens, batch: int, max_blocks_per_seq: int, num_q_heads: int,
                           softmax_scale: float, total_new_tokens: int) -> None:
    _check(load().gc_prefix_prefill_attn(_addr(q), pool, _addr(block_table), _addr(prefix_lens),
                                         _addr(new_lens), _addr(out), _stream(stream), layer,
                                         _addr(cu_new_lens), batch, max_blocks_per_seq,
                                         num_q_heads, softmax_scale, total_new_tokens),
           "gc_prefix_prefill_attn")


def gc_prefix_prefill_attn_simt(q, pool, block_table, prefix_lens, new_lens, out, stream,
                                layer: int, cu_new_lens, batch: int, max_blocks_per_seq: int,
                                num_q_heads: int, softmax_scale: float,
                                total_new_tokens: int) -> None:
    _check(load().gc_prefix_prefill_attn_simt(_addr(q), pool, _addr(block_table),
                                              _addr(prefix_lens), _addr(new_lens), _addr(out),
                                              _stream(stream), layer, _addr(cu_new_lens), batch,
                                              max_blocks_per_seq, num_q_heads, softmax_scale,
                                              total_new_tokens), "gc_prefix_prefill_attn_simt")


def gc_prefix_prefill_attn_noalloc(q, pool, block_table, prefix_lens, new_lens, out, stream,
                                   layer: int, cu_new_lens, batch: int, max_blocks_per_seq: int,
                                   num_q_heads: int, softmax_scale: float,
                                   total_new_tokens: int) -> None:
    """gc_prefix_prefill_attn for callers that cannot allocate device memory:
    its only scratch is a static array inside libgc (see include/gc.h)."""
    _check(load().gc_prefix_prefill_attn_noalloc(_addr(q), pool, _addr(block_table),
                                                 _addr(prefix_lens), _addr(new_lens), _addr(out),
                                                 _stream(stream), layer, _addr(cu_new_lens),
                                                 batch, max_blocks_per_seq, num_q_heads,
                                                 softmax_scale, total_new_tokens),
           "gc_prefix_prefill_attn_noalloc")


def gc_prefix_prefill_attn_q8(q, pool, block_table, prefix_lens, new_lens, out, stream,
                              layer: int, cu_new_lens, batch: int, max_blocks_per_seq: int,
                              num_q_heads: int, softmax_scale: float, total_new_tokens: int,
                              q8_image, q8_table, n_image_blocks: int, flags: int = 0) -> None:
    """gc_prefix_prefill_attn with the pages that q8_table maps (>= 0) read
    from the 8-bit image q8_image instead of the pool."""
    _check(load().gc_prefix_prefill_attn_q8(_addr(q), pool, _addr(block_table),
                                            _addr(prefix_lens), _addr(new_lens), _addr(out),
                                            _stream(stream), layer, _addr(cu_new_lens), batch,
                                            max_blocks_per_seq, num_q_heads, softmax_scale,
                                            total_new_tokens, _addr(q8_image), _addr(q8_table),
                                            n_image_blocks, flags),
           "gc_prefix_prefill_attn_q8")


@dataclass
class KVPool:
    """A pool whose device memory is a caller-owned torch buffer (so tests
    and benchmarks can view it), created through gc_kv_pool_create."""
    cfg: gc_pool_config
    buffer: object          # torch.uint8 CUDA tensor of gc_kv_pool_bytes(cfg)
    handle: ctypes.c_void_p

    @classmethod
    def create(cls, num_layers, num_kv_heads, head_dim, page_size, num_pages, device="cuda"):
        import torch
        cfg = make_config(num_layers, num_kv_heads, head_dim, page_size, num_pages)
        nbytes = gc_kv_pool_bytes(cfg)
        if nbytes == 0:
            raise GcError(GC_ERR_INVALID_ARG, "gc_kv_pool_bytes", "invalid configuration")
        buf = torch.empty(nbytes, dtype=torch.uint8, device=device)
        h = gc_kv_pool_create(cfg, buf, nbytes)
        return cls(cfg, buf, h)

    @property
    def shape(self):
        c = self.cfg
        return (c.num_layers, 2, c.num_pages, c.num_kv_heads, c.page_size, c.head_dim)

    def planes(self):
        """The KV planes as a bf16 tensor [L][2][num_pages][Hkv][ps][d] (a view)."""
        import torch
        n = 1
        for s in self.shape:
            n *= s
        return self.buffer[: 2 * n].view(torch.bfloat16).view(self.shape)

    def check(self, stream=None) -> int:
        return gc_kv_pool_check(self.handle, stream)

    def close(self):
        if self.handle:
            gc_kv_pool_destroy(self.handle)
            self.handle = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def gc_paged_decode_workspace_bytes(pool, batch: int, max_blocks_per_seq: int,
                                    num_q_heads: int) -> int:
    return int(load().gc_paged_decode_workspace_bytes(pool, batch, max_blocks_per_seq,
                                                      num_q_heads))


def gc_paged_decode_attn(q, pool, block_table, seq_lens, out, stream, layer: int, batch: int,
                         max_blocks_per_seq: int, num_q_heads: int, softmax_scale: float,
                         workspace=None, workspace_bytes: int = 0) -> None:
    _check(load().gc_paged_decode_attn(_addr(q), pool, _addr(block_table), _addr(seq_lens),
                                       _addr(out), _stream(stream), layer, batch,
                                       max_blocks_per_seq, num_q_heads, softmax_scale,
                                       _addr(workspace), workspace_bytes),
           "gc_paged_decode_attn")


def gc_paged_decode_attn_q8(q, pool, block_table, seq_lens, out, stream, layer: int, batch: int,
                            max_blocks_per_seq: int, num_q_heads: int, softmax_scale: float,
                            workspace, workspace_bytes: int, q8_image, q8_table,
                            n_image_blocks: int, flags: int = 0) -> None:
    """gc_paged_decode_attn with the pages that q8_table maps (>= 0) read from
    the 8-bit image q8_image instead of the pool."""
    _check(load().gc_paged_decode_attn_q8(_addr(q), pool, _addr(block_table), _addr(seq_lens),
                                          _addr(out), _stream(stream), layer, batch,
                                          max_blocks_per_seq, num_q_heads, softmax_scale,
                                          _addr(workspace), workspace_bytes, _addr(q8_image),
                                          _addr(q8_table), n_image_blocks, flags),
           "gc_paged_decode_attn_q8")


def gc_selftest_wait_timeout(pool, stream=None) -> None:
    _check(load().gc_selftest_wait_timeout(pool, _stream(stream)), "gc_selftest_wait_timeout")
