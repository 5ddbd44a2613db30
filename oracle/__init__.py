"""Float64 CPU oracle for prefix-reuse prefill (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
leg of ``bench.py`` may import this package.  The product path (the CUDA
library under ``paper_2505_23970_gb300``) never imports it, and this package
never imports the product.  The arithmetic lives in ``gc_oracle.c`` (plain C,
float64); this module only builds it with gcc and marshals numpy arrays.

bf16 tensors are passed as ``numpy.uint16`` arrays holding the bit patterns.
Results are float64.  Layouts follow the definitions in ``gc_oracle.c``:
pool ``[L][2][num_pages][Hkv][ps][d]``, staging image
``[n_blocks][L][2][Hkv][ps][d]``, queries ``[T_new][Hq][d]``, new keys and
values ``[T_new][Hkv][d]``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gc_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libgc_oracle.so")
_lock = threading.Lock()
_lib = None

# -ffp-contract=off: no fused multiply-add, so x86_64 and aarch64 builds give
# bit-identical float64 results.
CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-pthread", "-ffp-contract=off"]


def build(force: bool = False) -> str:
    """Compile gc_oracle.c into _build/libgc_oracle.so (gcc, no CUDA)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            i32, dbl = ctypes.c_int, ctypes.c_double
            p = ctypes.c_void_p
            lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
            lib.oracle_bf16_to_double.restype = dbl
            lib.oracle_kv_restore.argtypes = [p, i32, i32, i32, i32, i32, p, p, i32]
            lib.oracle_kv_gather_blocks.argtypes = [p, i32, i32, i32, i32, i32, p, i32, p]
            lib.oracle_q8_chunk_bytes.argtypes = [i32, i32, i32]
            lib.oracle_q8_chunk_bytes.restype = ctypes.c_size_t
            lib.oracle_kv_save_q8.argtypes = [p, i32, i32, i32, i32, i32, p, i32, i32, i32, p]
            lib.oracle_kv_restore_q8.argtypes = [p, i32, i32, i32, i32, i32, p, p, i32, i32, i32]
            lib.oracle_kv_append.argtypes = [p, i32, i32, i32, i32, i32, i32, p, p, p, i32, p, p, i32]
            lib.oracle_prefix_attn.argtypes = [p, p, i32, i32, i32, i32, i32, i32, p, i32, p, p,
                                               i32, i32, dbl, p, i32]
            lib.oracle_prefix_attn_rows.argtypes = [p, p, i32, i32, i32, i32, i32, i32, p, i32, p,
                                                    p, i32, i32, dbl, p, i32, p, i32]
            lib.oracle_prefix_attn_row_weights.argtypes = [p, p, i32, i32, i32, i32, i32, i32, p,
                                                           i32, p, p, i32, i32, dbl, i32, i32,
                                                           i32, p, p]
            lib.oracle_full_causal_attn.argtypes = [p, p, p, i32, i32, i32, i32, dbl, p, i32]
            for f in ("oracle_kv_restore", "oracle_kv_gather_blocks", "oracle_kv_append",
                      "oracle_prefix_attn", "oracle_prefix_attn_rows",
                      "oracle_prefix_attn_row_weights", "oracle_full_causal_attn"):
                getattr(lib, f).restype = i32
            _lib = lib
    return _lib


class OracleError(RuntimeError):
    pass


_CODES = {1: "invalid argument", 2: "index out of range", 3: "out of memory"}


def _check(st: int, what: str) -> None:
    if st != 0:
        raise OracleError(f"{what}: {_CODES.get(st, st)}")


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _u16(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError(f"bf16 arrays are passed as uint16 bit patterns, got {a.dtype}")
    return a


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def default_threads() -> int:
    return os.cpu_count() or 1


def bf16_to_double(bits: int) -> float:
    return _load().oracle_bf16_to_double(int(bits) & 0xFFFF)


def kv_restore(pool: np.ndarray, host_src: np.ndarray, block_ids) -> None:
    """In place: pool[l][kv][block_ids[i]] = host_src[i][l][kv]."""
    L, two, NP, Hkv, ps, d = pool.shape
    assert two == 2 and pool.flags.c_contiguous and pool.dtype == np.uint16
    ids = _i32(block_ids)
    src = _u16(host_src)
    assert src.shape == (ids.size, L, 2, Hkv, ps, d)
    _check(_load().oracle_kv_restore(_ptr(pool), L, Hkv, ps, d, NP, _ptr(src), _ptr(ids), ids.size),
           "kv_restore")


def kv_gather_blocks(pool: np.ndarray, block_ids) -> np.ndarray:
    """Inverse of kv_restore: the staging image of pages block_ids."""
    L, _, NP, Hkv, ps, d = pool.shape
    ids = _i32(block_ids)
    out = np.empty((ids.size, L, 2, Hkv, ps, d), dtype=np.uint16)
    _check(_load().oracle_kv_gather_blocks(_ptr(_u16(pool)), L, Hkv, ps, d, NP, _ptr(ids),
                                           ids.size, _ptr(out)), "kv_gather_blocks")
    return out


def q8_chunk_bytes(Hkv: int, ps: int, d: int) -> int:
    """Bytes of one (block, layer, plane) chunk of the 8-bit image."""
    return int(_load().oracle_q8_chunk_bytes(Hkv, ps, d))


def kv_save_q8(pool: np.ndarray, block_ids, layer_begin: int = 0, layer_count=None,
               out: np.ndarray | None = None) -> np.ndarray:
    """8-bit image [n_blocks][L][2][chunk] (uint8) of pages block_ids, layers
    [layer_begin, layer_begin + layer_count) written (into `out` if given,
    else into a zero image)."""
    L, _, NP, Hkv, ps, d = pool.shape
    if layer_count is None:
        layer_count = L - layer_begin
    ids = _i32(block_ids)
    chunk = q8_chunk_bytes(Hkv, ps, d)
    if out is None:
        out = np.zeros((ids.size, L, 2, chunk), dtype=np.uint8)
    assert out.dtype == np.uint8 and out.flags.c_contiguous and out.shape == (ids.size, L, 2, chunk)
    _check(_load().oracle_kv_save_q8(_ptr(_u16(pool)), L, Hkv, ps, d, NP, _ptr(ids), ids.size,
                                     layer_begin, layer_count, _ptr(out)), "kv_save_q8")
    return out


def kv_restore_q8(pool: np.ndarray, image: np.ndarray, block_ids, layer_begin: int = 0,
                  layer_count=None) -> None:
    """In place: dequantise the 8-bit image's chunks into the pool pages."""
    assert pool.dtype == np.uint16 and pool.flags.c_contiguous
    L, _, NP, Hkv, ps, d = pool.shape
    if layer_count is None:
        layer_count = L - layer_begin
    ids = _i32(block_ids)
    img = np.ascontiguousarray(image, dtype=np.uint8)
    assert img.size == ids.size * L * 2 * q8_chunk_bytes(Hkv, ps, d)
    _check(_load().oracle_kv_restore_q8(_ptr(pool), L, Hkv, ps, d, NP, _ptr(img), _ptr(ids),
                                        ids.size, layer_begin, layer_count), "kv_restore_q8")


def q8_split(image: np.ndarray, Hkv: int, ps: int, d: int):
    """(scales [n][L][2][Hkv] float32, codes [n][L][2][Hkv][ps][d] int8) views
    of an 8-bit image (layout plumbing, no arithmetic)."""
    n, L = image.shape[:2]
    chunk = q8_chunk_bytes(Hkv, ps, d)
    hdr = chunk - Hkv * ps * d
    flat = image.reshape(n, L, 2, chunk)
    scales = np.ascontiguousarray(flat[..., :4 * Hkv]).view(np.float32)
    codes = np.ascontiguousarray(flat[..., hdr:]).view(np.int8).reshape(n, L, 2, Hkv, ps, d)
    return scales, codes


def kv_append(pool: np.ndarray, layer: int, k_new, v_new, block_table, prefix_lens,
              cu_new_lens) -> None:
    """In place: write the new tokens' K and V after each request's prefix."""
    L, _, NP, Hkv, ps, d = pool.shape
    assert pool.flags.c_contiguous and pool.dtype == np.uint16
    bt = _i32(block_table)
    pl, cu = _i32(prefix_lens), _i32(cu_new_lens)
    k, v = _u16(k_new), _u16(v_new)
    batch = pl.size
    max_blocks = bt.shape[1] if bt.ndim == 2 else 0
    _check(_load().oracle_kv_append(_ptr(pool), L, Hkv, ps, d, NP, layer, _ptr(k), _ptr(v),
                                    _ptr(bt), max_blocks, _ptr(pl), _ptr(cu), batch),
           "kv_append")


def _attn_common(pool, block_table, prefix_lens, cu_new_lens):
    L, _, NP, Hkv, ps, d = pool.shape
    bt = _i32(block_table)
    max_blocks = bt.shape[1] if bt.ndim == 2 else 0
    return (L, NP, Hkv, ps, d, bt, max_blocks, _i32(prefix_lens), _i32(cu_new_lens))


def prefix_attn(q, pool, layer, block_table, prefix_lens, cu_new_lens, scale,
                nthreads: int | None = None) -> np.ndarray:
    """O[T_new][Hq][d] (float64) of every new-token row."""
    q = _u16(q)
    T_new, Hq, d_q = q.shape
    L, NP, Hkv, ps, d, bt, mb, pl, cu = _attn_common(pool, block_table, prefix_lens, cu_new_lens)
    assert d_q == d
    out = np.zeros((T_new, Hq, d), dtype=np.float64)
    _check(_load().oracle_prefix_attn(_ptr(q), _ptr(_u16(pool)), L, Hkv, ps, d, NP, layer,
                                      _ptr(bt), mb, _ptr(pl), _ptr(cu), pl.size, Hq, float(scale),
                                      _ptr(out), nthreads or default_threads()), "prefix_attn")
    return out


def prefix_attn_rows(q, pool, layer, block_table, prefix_lens, cu_new_lens, scale, rows,
                     nthreads: int | None = None) -> np.ndarray:
    """Rows (b, h, i) only: out[n_rows][d] (float64), each exact over all its keys."""
    q = _u16(q)
    T_new, Hq, _ = q.shape
    L, NP, Hkv, ps, d, bt, mb, pl, cu = _attn_common(pool, block_table, prefix_lens, cu_new_lens)
    rows = _i32(rows).reshape(-1, 3)
    out = np.zeros((rows.shape[0], d), dtype=np.float64)
    _check(_load().oracle_prefix_attn_rows(_ptr(q), _ptr(_u16(pool)), L, Hkv, ps, d, NP, layer,
                                           _ptr(bt), mb, _ptr(pl), _ptr(cu), pl.size, Hq,
                                           float(scale), _ptr(rows), rows.shape[0], _ptr(out),
                                           nthreads or default_threads()), "prefix_attn_rows")
    return out


def prefix_attn_row_weights(q, pool, layer, block_table, prefix_lens, cu_new_lens, scale,
                            b: int, h: int, i: int):
    """(weights[P_b + i + 1], out_row[d]) of one row, both float64."""
    q = _u16(q)
    _, Hq, _ = q.shape
    L, NP, Hkv, ps, d, bt, mb, pl, cu = _attn_common(pool, block_table, prefix_lens, cu_new_lens)
    w = np.zeros(int(pl[b]) + i + 1, dtype=np.float64)
    o = np.zeros(d, dtype=np.float64)
    _check(_load().oracle_prefix_attn_row_weights(_ptr(q), _ptr(_u16(pool)), L, Hkv, ps, d, NP,
                                                  layer, _ptr(bt), mb, _ptr(pl), _ptr(cu),
                                                  pl.size, Hq, float(scale), b, h, i, _ptr(w),
                                                  _ptr(o)), "prefix_attn_row_weights")
    return w, o


def full_causal_attn(q, k, v, scale, nthreads: int | None = None) -> np.ndarray:
    """Dense, unpaged causal attention: q [T][Hq][d], k, v [T][Hkv][d]."""
    q, k, v = _u16(q), _u16(k), _u16(v)
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    assert k.shape == (T, Hkv, d) and v.shape == k.shape
    out = np.zeros((T, Hq, d), dtype=np.float64)
    _check(_load().oracle_full_causal_attn(_ptr(q), _ptr(k), _ptr(v), T, Hq, Hkv, d, float(scale),
                                           _ptr(out), nthreads or default_threads()),
           "full_causal_attn")
    return out
