"""Device-side plumbing around the C ABI for one batch of requests.

``DeviceBatch`` places a :class:`workloads.Workload`'s inputs in device (and
pinned host) memory with torch, then runs the three steps of the path —
restore, append, attention — through :mod:`binding`.  It moves inputs and
allocates buffers only; every result is computed by libgc's kernels.
"""
from __future__ import annotations

import numpy as np

from . import binding as gcb
from .workloads import BF16_NAN, Workload


def _i32(a, device):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(device)


def bf16_tensor(bits: np.ndarray, device="cuda", pin: bool = False):
    """uint16 bit patterns -> torch.bfloat16 tensor (device, or pinned host)."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    if pin:
        return t.pin_memory()
    return t.to(device)


def bf16_bits(t) -> np.ndarray:
    """torch.bfloat16 tensor -> numpy uint16 bit patterns (host copy)."""
    import torch
    return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)


class DeviceBatch:
    def __init__(self, w: Workload, device: str = "cuda", fill=BF16_NAN, with_restore=True,
                 staging: bool = True):
        import torch
        self.w = w
        self.device = device
        self.pool = gcb.KVPool.create(w.L, w.Hkv, w.d, w.ps, w.num_pages, device=device)
        self.pool.planes().view(torch.int16).fill_(int(np.int16(np.uint16(fill).view(np.int16))))
        self.block_table = _i32(w.block_table, device)
        self.prefix_lens = _i32(w.prefix_lens, device)
        self.new_lens = _i32(w.new_lens, device)
        self.cu_new_lens = _i32(w.cu_new_lens, device)
        self.n_blocks = 0
        if with_restore:
            ids = w.prefix_blocks()
            self.n_blocks = int(ids.size)
            self.block_ids = _i32(ids, device)
            self.host_src = bf16_tensor(w.host_src(), pin=True) if self.n_blocks else None
            self.staging = (torch.empty_like(self.host_src, device=device)
                            if staging and self.n_blocks else None)
        k, v = w.kv_new()
        self.k_new = bf16_tensor(k, device)
        self.v_new = bf16_tensor(v, device)
        self.q = bf16_tensor(w.q(), device)
        self.out = torch.full((w.T_new, w.Hq, w.d), float("nan"), dtype=torch.bfloat16,
                              device=device)

    # ---------------------------------------------------------------- steps
    def restore(self, stream=None, mode: str = "staged", vector: bool = False):
        """mode: 'staged' (pinned host -> staging -> pool), 'device' (staging
        already holds the image: scatter only) or 'zerocopy' (kernel reads
        pinned host memory)."""
        if self.n_blocks == 0:
            return
        flags = gcb.GC_RESTORE_VECTOR if vector else 0
        if mode == "staged":
            gcb.gc_kv_restore(self.pool.handle, self.host_src, self.block_ids, self.n_blocks,
                              stream, self.staging, flags)
        elif mode == "device":
            gcb.gc_kv_restore(self.pool.handle, self.staging, self.block_ids, self.n_blocks,
                              stream, None, flags | gcb.GC_RESTORE_SRC_DEVICE)
        elif mode == "zerocopy":
            gcb.gc_kv_restore(self.pool.handle, self.host_src, self.block_ids, self.n_blocks,
                              stream, None, flags)
        else:
            raise ValueError(mode)

    def save(self, block_ids, mode: str = "staged", vector: bool = False, stream=None,
             fill=0x7FC0) -> np.ndarray:
        """gc_kv_save of pages `block_ids` into a fresh image [n][L][2][Hkv][ps][d]
        pre-filled with `fill`; mode 'staged' (device staging, then a copy to
        pinned host), 'device' (device destination) or 'zerocopy' (kernel writes
        pinned host memory). Returns the image's bf16 bit patterns."""
        import torch
        w = self.w
        ids = _i32(block_ids, self.device)
        n = int(ids.numel())
        shape = (n, w.L, 2, w.Hkv, w.ps, w.d)
        flags = gcb.GC_SAVE_VECTOR if vector else 0
        fill_i16 = int(np.uint16(fill).view(np.int16))
        if mode == "device":
            dst = torch.full(shape, fill_i16, dtype=torch.int16, device=self.device)
            flags |= gcb.GC_SAVE_DST_DEVICE
        else:
            dst = torch.full(shape, fill_i16, dtype=torch.int16).pin_memory()
        staging = (torch.empty(shape, dtype=torch.int16, device=self.device)
                   if mode == "staged" else None)
        if mode not in ("staged", "device", "zerocopy"):
            raise ValueError(mode)
        gcb.gc_kv_save(self.pool.handle, dst, ids, n, stream, staging, flags)
        torch.cuda.synchronize()
        return dst.cpu().numpy().view(np.uint16)

    def stage(self, stream=None):
        """Copy the pinned image into the device staging buffer (torch copy)."""
        if self.n_blocks:
            self.staging.copy_(self.host_src, non_blocking=True)

    def append(self, stream=None, layer: int = 0):
        w = self.w
        gcb.gc_kv_append(self.pool.handle, self.k_new, self.v_new, self.block_table,
                         self.prefix_lens, stream, layer, self.cu_new_lens, w.B, w.max_blocks,
                         w.T_new)

    def attn(self, stream=None, impl: str = "tc", layer: int = 0, out=None):
        w = self.w
        fn = gcb.gc_prefix_prefill_attn if impl == "tc" else gcb.gc_prefix_prefill_attn_simt
        fn(self.q, self.pool.handle, self.block_table, self.prefix_lens, self.new_lens,
           self.out if out is None else out, stream, layer, self.cu_new_lens, w.B, w.max_blocks,
           w.Hq, w.scale, w.T_new)

    def decode(self, stream=None, layer: int = 0, out=None, workspace=None):
        """gc_paged_decode_attn of the batch's one new token per request over
        its whole context (seq_lens = prefix + 1); allocates the workspace the
        library asks for unless one is given."""
        import torch
        w = self.w
        assert np.all(w.new_lens == 1), "decode takes one new token per request"
        if not hasattr(self, "seq_lens"):
            self.seq_lens = _i32(w.total_lens, self.device)
        need = gcb.gc_paged_decode_workspace_bytes(self.pool.handle, w.B, w.max_blocks, w.Hq)
        if workspace is None and need:
            if getattr(self, "_dec_ws", None) is None or self._dec_ws.numel() < need:
                self._dec_ws = torch.empty(need, dtype=torch.uint8, device=self.device)
            workspace = self._dec_ws
        gcb.gc_paged_decode_attn(self.q, self.pool.handle, self.block_table, self.seq_lens,
                                 self.out if out is None else out, stream, layer, w.B,
                                 w.max_blocks, w.Hq, w.scale, workspace,
                                 0 if workspace is None else workspace.numel())

    def run(self, stream=None, restore_mode: str = "staged", impl: str = "tc"):
        self.restore(stream, restore_mode)
        self.append(stream)
        self.attn(stream, impl)

    def check(self, stream=None) -> int:
        return self.pool.check(stream)

    def pool_bits(self) -> np.ndarray:
        return bf16_bits(self.pool.planes())

    def out_f64(self) -> np.ndarray:
        import torch
        return self.out.to(torch.float64).cpu().numpy()

    def close(self):
        self.pool.close()


class LayerStack:
    """One batch of requests through all `w.L` layers of one pool, the way a
    serving loop prefills with reused context: per layer, the cached pages
    of that layer are restored, the layer's new K/V appended and its
    attention run.

    ``run(pipelined=True)`` splits each layer's restore into its two legs:
    every layer's host -> device copy (gc_kv_stage_layers) is issued up front
    on a copy stream, back to back, each followed by a CUDA event, so the
    host link never waits for a kernel; the main stream waits for layer l's
    event, then runs layer l's scatter (gc_kv_restore_layers from the device
    image), append and attention.  The copies of later layers overlap the
    compute of earlier ones, and the scatter, which needs the SMs the
    attention of the previous layer holds, sits where it is needed anyway.
    ``run(pipelined=True, schedule="side-restore")`` is the simpler schedule
    it replaced: one staged gc_kv_restore_layers per layer (copy + scatter)
    on a side stream, so each copy waits behind the previous layer's
    scatter, which waits for the attention holding the SMs.
    ``run(pipelined=False)`` restores all layers first (one gc_kv_restore)
    and then computes layer by layer on one stream.  Q and the new tokens' K/V are the same tensors for every layer
    (inputs of the attention step, not produced here); the cached pages
    differ per layer.  Only streams, events and buffers are handled here:
    every byte is moved or computed by libgc."""

    def __init__(self, w: Workload, device: str = "cuda", fill=BF16_NAN, keep_outputs=False,
                 staging: bool = True, layer_major: bool = True):
        import torch
        self.w, self.device = w, device
        self.pool = gcb.KVPool.create(w.L, w.Hkv, w.d, w.ps, w.num_pages, device=device)
        self.pool.planes().view(torch.int16).fill_(int(np.uint16(fill).view(np.int16)))
        self.block_table = _i32(w.block_table, device)
        self.prefix_lens = _i32(w.prefix_lens, device)
        self.new_lens = _i32(w.new_lens, device)
        self.cu_new_lens = _i32(w.cu_new_lens, device)
        ids = w.prefix_blocks()
        self.n_blocks = int(ids.size)
        self.block_ids = _i32(ids, device)
        # the cached image, layer-major [L][n][2][Hkv][ps][d] by default so
        # that each layer's slice is one contiguous host span
        self.flags = gcb.GC_RESTORE_LAYER_MAJOR if layer_major else 0
        img = w.host_src()
        if layer_major and self.n_blocks:
            img = np.ascontiguousarray(img.swapaxes(0, 1))
        self.host_src = bf16_tensor(img, pin=True) if self.n_blocks else None
        del img
        self.staging = (torch.empty_like(self.host_src, device=device)
                        if staging and self.n_blocks else None)
        k, v = w.kv_new()
        self.k_new, self.v_new = bf16_tensor(k, device), bf16_tensor(v, device)
        self.q = bf16_tensor(w.q(), device)
        n_out = w.L if keep_outputs else 1
        self.outs = [torch.empty((w.T_new, w.Hq, w.d), dtype=torch.bfloat16, device=device)
                     for _ in range(n_out)]
        self.side = torch.cuda.Stream(device=device)
        self.copy = torch.cuda.Stream(device=device)
        self.events = [torch.cuda.Event() for _ in range(w.L)]

    def use_q8(self):
        """Switch the cache tier to the 8-bit image: quantise what the pool
        holds now (after a restore) into a pinned layer-major INT8 image with
        gc_kv_save_q8; later restores dequantise it with gc_kv_restore_q8."""
        import torch
        w = self.w
        chunk = gcb.gc_kv_q8_chunk_bytes(self.pool.cfg)
        shape = (w.L, self.n_blocks, 2, chunk)
        self.q8_staging = torch.empty(shape, dtype=torch.uint8, device=self.device)
        self.q8_host = torch.empty(shape, dtype=torch.uint8).pin_memory()
        gcb.gc_kv_save_q8(self.pool.handle, self.q8_host, self.block_ids, self.n_blocks, 0, w.L,
                          None, self.q8_staging, gcb.GC_SAVE_LAYER_MAJOR)
        torch.cuda.synchronize()
        self.q8 = True

    q8 = False

    def restore_layer(self, l, stream):
        if self.n_blocks and self.q8:
            gcb.gc_kv_restore_q8(self.pool.handle, self.q8_host, self.block_ids, self.n_blocks,
                                 l, 1, stream, self.q8_staging, gcb.GC_RESTORE_LAYER_MAJOR)
        elif self.n_blocks:
            gcb.gc_kv_restore_layers(self.pool.handle, self.host_src, self.block_ids,
                                     self.n_blocks, l, 1, stream, self.staging, self.flags)

    def stage_layer(self, l, stream):
        """Host -> device copy of layer l's slice of the cached image."""
        if not self.n_blocks:
            return
        if self.q8:
            gcb.gc_kv_stage_layers(self.pool.handle, self.q8_host, self.q8_staging, self.n_blocks,
                                   l, 1, stream, gcb.GC_RESTORE_LAYER_MAJOR | gcb.GC_STAGE_Q8)
        else:
            gcb.gc_kv_stage_layers(self.pool.handle, self.host_src, self.staging, self.n_blocks,
                                   l, 1, stream, self.flags)

    def scatter_layer(self, l, stream):
        """Layer l's pages from the device image into the pool."""
        if not self.n_blocks:
            return
        if self.q8:
            gcb.gc_kv_restore_q8(self.pool.handle, self.q8_staging, self.block_ids, self.n_blocks,
                                 l, 1, stream, None,
                                 gcb.GC_RESTORE_SRC_DEVICE | gcb.GC_RESTORE_LAYER_MAJOR)
        else:
            gcb.gc_kv_restore_layers(self.pool.handle, self.staging, self.block_ids,
                                     self.n_blocks, l, 1, stream, None,
                                     gcb.GC_RESTORE_SRC_DEVICE | self.flags)

    def restore_all(self, stream):
        if self.n_blocks and self.q8:
            gcb.gc_kv_restore_q8(self.pool.handle, self.q8_host, self.block_ids, self.n_blocks,
                                 0, self.w.L, stream, self.q8_staging, gcb.GC_RESTORE_LAYER_MAJOR)
        elif self.n_blocks:
            gcb.gc_kv_restore(self.pool.handle, self.host_src, self.block_ids, self.n_blocks,
                              stream, self.staging, self.flags)

    def prefill_layer(self, l, stream):
        w = self.w
        h = self.pool.handle
        gcb.gc_kv_append(h, self.k_new, self.v_new, self.block_table, self.prefix_lens, stream, l,
                         self.cu_new_lens, w.B, w.max_blocks, w.T_new)
        gcb.gc_prefix_prefill_attn(self.q, h, self.block_table, self.prefix_lens, self.new_lens,
                                   self.outs[l % len(self.outs)], stream, l, self.cu_new_lens,
                                   w.B, w.max_blocks, w.Hq, w.scale, w.T_new)

    def run(self, pipelined: bool = True, schedule: str = "copy-stream", trace=None):
        """Restore + append + attention of every layer, issued on the current
        stream (and, when pipelined, the copy or side stream).  `trace`, a
        dict, receives per-layer timing events of the copy-stream schedule:
        'copied' (copy stream, after layer l's copy), 'scattered' (main, after
        layer l's scatter) and 'computed' (main, after layer l's attention)."""
        import torch
        main = torch.cuda.current_stream(self.device)
        L = self.w.L
        if not pipelined:
            self.restore_all(main)
            for l in range(L):
                self.prefill_layer(l, main)
            return
        if schedule == "side-restore":
            self.side.wait_stream(main)  # the restores may not pass earlier work on main
            for l in range(L):
                self.restore_layer(l, self.side)
                self.events[l].record(self.side)
            for l in range(L):
                main.wait_event(self.events[l])
                self.prefill_layer(l, main)
            return
        if schedule != "copy-stream":
            raise ValueError(schedule)
        if trace is not None:
            for k in ("copied", "scattered", "computed"):
                trace[k] = [torch.cuda.Event(enable_timing=True) for _ in range(L)]
        self.copy.wait_stream(main)  # the copies may not pass earlier work on main
        for l in range(L):
            self.stage_layer(l, self.copy)
            self.events[l].record(self.copy)
            if trace is not None:
                trace["copied"][l].record(self.copy)
        for l in range(L):
            main.wait_event(self.events[l])
            self.scatter_layer(l, main)
            if trace is not None:
                trace["scattered"][l].record(main)
            self.prefill_layer(l, main)
            if trace is not None:
                trace["computed"][l].record(main)

    def capture(self, pipelined: bool = True, schedule: str = "copy-stream"):
        """Record one run() into a CUDA graph (torch.cuda.CUDAGraph) after one
        eager run on the capture's side stream; replay() then re-issues every
        copy, kernel and event dependency of the whole layer stack with one
        launch, so the host's per-call cost and jitter leave the step.  The
        graph reuses this stack's buffers: its inputs are whatever they hold
        at replay time."""
        import torch
        side = torch.cuda.Stream(device=self.device)
        side.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(side):
            self.run(pipelined=pipelined, schedule=schedule)
        torch.cuda.current_stream(self.device).wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            self.run(pipelined=pipelined, schedule=schedule)
        return graph

    def prefill_only(self):
        """Append + attention of every layer (the compute half alone)."""
        import torch
        main = torch.cuda.current_stream(self.device)
        for l in range(self.w.L):
            self.prefill_layer(l, main)

    def check(self) -> int:
        return self.pool.check(None)

    def pool_bits(self) -> np.ndarray:
        return bf16_bits(self.pool.planes())

    def close(self):
        self.pool.close()
