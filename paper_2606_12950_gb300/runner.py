"""Device-side holders for a pool and a decode batch, driving the C ABI.

PyTorch provides the device memory and the streams; every step of the path
(append, attention, split combine) runs in libkvpool's kernels through
``kvpool``.  Host arrays use uint16 for bf16 bit patterns.
"""
from __future__ import annotations

import numpy as np
import torch

from . import kvpool as K


def _dev_u16(a: np.ndarray, device) -> torch.Tensor:
    """Host uint16 (bf16 bits) -> device bfloat16 tensor with the same bits."""
    t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16))
    return t.to(device).view(torch.bfloat16)


def _host_u16(t: torch.Tensor) -> np.ndarray:
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


class DevicePool:
    """A caller-owned device buffer managed by a kv_pool handle."""

    def __init__(self, n_pages: int, page_bytes: int, block_size: int, layouts, shuffle_seed: int = 0,
                 device: str = "cuda"):
        self.device = torch.device(device)
        self.n_pages = int(n_pages)
        self.page_bytes = int(page_bytes)
        self.buf = torch.empty(self.n_pages * self.page_bytes, dtype=torch.uint8, device=self.device)
        self.err = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.handle = K.kv_pool_create(self.buf, self.buf.numel(), block_size, layouts, self.err,
                                       page_bytes=page_bytes, shuffle_seed=shuffle_seed)

    def upload(self, pool_u16: np.ndarray) -> None:
        src = torch.from_numpy(np.ascontiguousarray(pool_u16).view(np.uint8))
        self.buf.copy_(src.to(self.device))

    def fill_u16(self, value: int) -> None:
        self.buf.view(torch.int16).fill_(np.array(value, np.uint16).view(np.int16).item())

    def download(self) -> np.ndarray:
        return self.buf.cpu().numpy().view(np.uint16)

    def error(self, stream=None) -> int:
        return K.kv_pool_get_error(self.handle, stream)

    def set_variant(self, v: int) -> None:
        K.kv_set_attn_variant(self.handle, v)

    def set_step_overlap(self, on: bool) -> None:
        K.kv_set_attn_step_overlap(self.handle, on)

    def close(self) -> None:
        if self.handle:
            K.kv_pool_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class _RawDevice:
    """A device byte range seen through __cuda_array_interface__ (no ownership)."""

    def __init__(self, ptr: int, nbytes: int):
        self.__cuda_array_interface__ = {"shape": (nbytes,), "typestr": "|u1", "data": (ptr, False),
                                         "version": 3}


class VmmPool:
    """A VMM-backed elastic pool (kv_pool_create_vmm, CUDA backend): the
    library reserves the virtual range and maps physical chunks as blocks are
    allocated.  ``pages`` views the whole range (n_pages x page_bytes); only
    rows of allocated blocks may be touched."""

    def __init__(self, virtual_bytes: int, page_bytes: int, block_size: int, layouts, physical_limit: int = 0,
                 budget=None, shuffle_seed: int = 0, chunk_bytes: int = 0, device: str = "cuda"):
        self.device = torch.device(device)
        dev_index = self.device.index if self.device.index is not None else torch.cuda.current_device()
        self.err = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.handle = K.kv_pool_create_vmm(virtual_bytes, block_size, layouts, self.err, page_bytes=page_bytes,
                                           shuffle_seed=shuffle_seed, chunk_bytes=chunk_bytes,
                                           physical_limit=physical_limit, budget=budget, device=dev_index)
        self.base = K.kv_pool_get_base(self.handle)
        st = K.kv_pool_stats(self.handle)
        self.page_bytes = int(page_bytes)
        self.n_pages = int(st["pages_total"])
        raw = torch.as_tensor(_RawDevice(self.base, self.n_pages * self.page_bytes), device=self.device)
        self.pages = raw.view(self.n_pages, self.page_bytes)

    def write_pages(self, ids, data_u16: np.ndarray) -> None:
        """Rows of the given page ids (allocated blocks' first pages) <- data."""
        idx = torch.as_tensor(np.asarray(ids, np.int64), device=self.device)
        src = torch.from_numpy(np.ascontiguousarray(data_u16).view(np.uint8)).to(self.device)
        self.pages.index_copy_(0, idx, src.view(len(idx), -1))

    def fill_random(self, ids, seed: int) -> None:
        """Finite bf16 values (N(0,1) rounded) in the given pages."""
        g = torch.Generator(device=self.device)
        g.manual_seed(seed)
        idx = torch.as_tensor(np.asarray(ids, np.int64), device=self.device)
        vals = torch.randn((len(idx), self.page_bytes // 2), generator=g, device=self.device).to(torch.bfloat16)
        self.pages.index_copy_(0, idx, vals.view(torch.uint8))

    def read_pages(self, ids) -> np.ndarray:
        idx = torch.as_tensor(np.asarray(ids, np.int64), device=self.device)
        return self.pages.index_select(0, idx).cpu().numpy().view(np.uint16)

    def stats(self) -> dict:
        return K.kv_pool_stats(self.handle)

    def trim(self) -> int:
        return K.kv_pool_trim(self.handle)

    def error(self, stream=None) -> int:
        return K.kv_pool_get_error(self.handle, stream)

    def set_variant(self, v: int) -> None:
        K.kv_set_attn_variant(self.handle, v)

    def set_step_overlap(self, on: bool) -> None:
        K.kv_set_attn_step_overlap(self.handle, on)

    def close(self) -> None:
        if self.handle:
            torch.cuda.synchronize()
            self.pages = None
            K.kv_pool_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class DeviceBatch:
    """One layout's decode batch on the device (q, new K/V rows, table,
    lengths, output, workspace)."""

    def __init__(self, pool: DevicePool, layout: int, b, num_splits: int = 0):
        dev = pool.device
        self.pool = pool
        self.layout = layout
        self.b = b
        self.S, self.Hq, self.d, self.max_blocks = b.S, b.Hq, b.d, b.max_blocks
        self.q = _dev_u16(b.q, dev)
        self.k_new = _dev_u16(b.k_new, dev)
        self.v_new = _dev_u16(b.v_new, dev)
        self.table = torch.empty((b.S, b.max_blocks), dtype=torch.int32, device=dev)
        self.lens = torch.empty(b.S, dtype=torch.int32, device=dev)
        self.out = torch.empty((b.S, b.Hq, b.d), dtype=torch.bfloat16, device=dev)
        self.num_splits = num_splits
        self.ws_bytes = K.kv_workspace_bytes(pool.handle, layout, b.S, b.Hq, b.max_blocks, num_splits)
        self.ws = torch.zeros(max(256, self.ws_bytes), dtype=torch.uint8, device=dev)
        self.upload_table(b.table, b.ctx_lens)

    def upload_table(self, table, lens, stream=None) -> None:
        K.kv_block_table_upload(self.pool.handle, self.layout, table, lens, self.table, self.lens, stream)

    def set_rows(self, q, k_new, v_new) -> None:
        dev = self.pool.device
        self.q.copy_(_dev_u16(q, dev))
        self.k_new.copy_(_dev_u16(k_new, dev))
        self.v_new.copy_(_dev_u16(v_new, dev))

    def append(self, stream=None) -> None:
        K.kv_append(self.pool.handle, self.layout, self.k_new, self.v_new, self.table, self.lens,
                    self.max_blocks, self.S, stream)

    def attend(self, num_splits: int | None = None, stream=None) -> None:
        ns = self.num_splits if num_splits is None else num_splits
        if ns != self.num_splits:
            need = K.kv_workspace_bytes(self.pool.handle, self.layout, self.S, self.Hq, self.max_blocks, ns)
            if need > self.ws.numel():
                self.ws = torch.zeros(need, dtype=torch.uint8, device=self.pool.device)
            self.num_splits = ns
            self.ws_bytes = need
        K.paged_decode_attn(self.pool.handle, self.layout, self.q, self.out, self.table, self.lens,
                            self.max_blocks, self.S, self.Hq, self.b.scale, ns, self.ws,
                            self.ws.numel(), stream)

    def append_attend(self, stream=None) -> None:
        """The fused append + attention pass."""
        K.paged_decode_attn_append(self.pool.handle, self.layout, self.q, self.k_new, self.v_new, self.out,
                                   self.table, self.lens, self.max_blocks, self.S, self.Hq, self.b.scale,
                                   self.num_splits, self.ws, self.ws.numel(), stream)

    def batch(self, fused: bool = True) -> dict:
        """This batch as a paged_decode_attn_multi entry."""
        return {"layout": self.layout, "q": self.q, "k_new": self.k_new if fused else None,
                "v_new": self.v_new if fused else None, "out": self.out, "dev_table": self.table,
                "dev_ctx_lens": self.lens, "max_blocks": self.max_blocks, "S": self.S, "Hq": self.Hq,
                "scale": self.b.scale, "workspace": self.ws, "ws_bytes": self.ws.numel()}

    def cascade(self, plan, fused: bool = True, stream=None) -> None:
        """Shared-prefix attention (with the fused append unless fused=False)."""
        need = K.kv_cascade_workspace_bytes(self.pool.handle, self.layout, self.S, self.Hq, self.max_blocks)
        if need > self.ws.numel():
            self.ws = torch.zeros(need, dtype=torch.uint8, device=self.pool.device)
        K.paged_decode_attn_cascade(self.pool.handle, self.layout, self.q, self.k_new if fused else None,
                                    self.v_new if fused else None, self.out, self.table, self.lens,
                                    self.max_blocks, self.S, self.Hq, self.b.scale, plan, self.ws,
                                    self.ws.numel(), stream)

    def out_f64(self) -> np.ndarray:
        return self.out.float().cpu().numpy().astype(np.float64)

    def out_bits(self) -> np.ndarray:
        return _host_u16(self.out)


class DeviceSteps:
    """Device buffers of a decode batch whose table and lengths come from a
    host sequence table (rows >= S table rows; the first S rows decode)."""

    def __init__(self, pool: DevicePool, layout: int, rows: int, S: int, Hq: int, Hkv: int, d: int,
                 max_blocks: int, scale: float, q, k_new, v_new, num_splits: int = 0):
        dev = pool.device
        self.pool, self.layout = pool, layout
        self.rows, self.S, self.Hq, self.Hkv, self.d = rows, S, Hq, Hkv, d
        self.max_blocks, self.scale, self.num_splits = max_blocks, scale, num_splits
        self.table = torch.full((rows, max_blocks), -1, dtype=torch.int32, device=dev)
        self.lens = torch.zeros(rows, dtype=torch.int32, device=dev)
        # q, k_new and v_new are views of one contiguous buffer, so a step's
        # inputs reach the device with a single copy (each view stays 16-byte
        # aligned: every part is a whole number of d-element rows, d % 8 == 0)
        parts = [np.ascontiguousarray(a).reshape(-1) for a in (q, k_new, v_new)]
        self.inputs = _dev_u16(np.concatenate(parts), dev)
        sizes = [p.size for p in parts]
        q_, k_, v_ = torch.split(self.inputs, sizes)
        self.q = q_.view(np.shape(q))
        self.k_new = k_.view(np.shape(k_new))
        self.v_new = v_.view(np.shape(v_new))
        self.out = torch.empty((S, Hq, d), dtype=torch.bfloat16, device=dev)
        self.ws_bytes = K.kv_workspace_bytes(pool.handle, layout, S, Hq, max_blocks, num_splits)
        self.ws = torch.empty(max(256, self.ws_bytes), dtype=torch.uint8, device=dev)
        self._shapes = (np.shape(q), np.shape(k_new), np.shape(v_new))
        self._device_io = (self.inputs, self.out)

    def io(self, inputs=None, out=None) -> None:
        """Point q / k_new / v_new at `inputs` (bf16, laid out like
        self.inputs: q, then k_new, then v_new) and the output at `out`:
        device tensors, or pinned host tensors that the kernels read and
        write directly over the GPU's coherent link to host memory.  With no
        arguments, back to this batch's device buffers."""
        if inputs is None:
            inputs, out = self._device_io
        if inputs.numel() != self._device_io[0].numel() or out.numel() != self._device_io[1].numel():
            raise ValueError("io buffers must match the batch's input and output sizes")
        if inputs.device.type == "cpu" and not (inputs.is_pinned() and out.is_pinned()):
            raise ValueError("host io buffers must be pinned")
        sizes = [int(np.prod(sh)) for sh in self._shapes]
        q_, k_, v_ = torch.split(inputs.view(torch.bfloat16).reshape(-1), sizes)
        self.inputs = inputs
        self.q, self.k_new, self.v_new = (t.view(sh) for t, sh in zip((q_, k_, v_), self._shapes))
        self.out = out.view(self._device_io[1].shape)

    def sync(self, seqtab, stream=None) -> None:
        seqtab.sync(self.table, self.lens, stream)

    def append_attend(self, stream=None) -> None:
        K.paged_decode_attn_append(self.pool.handle, self.layout, self.q, self.k_new, self.v_new, self.out,
                                   self.table, self.lens, self.max_blocks, self.S, self.Hq, self.scale,
                                   self.num_splits, self.ws, self.ws.numel(), stream)

    def batch(self, fused: bool = True) -> dict:
        """This batch as a paged_decode_attn_multi entry."""
        return {"layout": self.layout, "q": self.q, "k_new": self.k_new if fused else None,
                "v_new": self.v_new if fused else None, "out": self.out, "dev_table": self.table,
                "dev_ctx_lens": self.lens, "max_blocks": self.max_blocks, "S": self.S, "Hq": self.Hq,
                "scale": self.scale, "workspace": self.ws, "ws_bytes": self.ws.numel()}

    def sync_append_attend(self, seqtab, stream=None) -> None:
        """seqtab's table sync, the append and the attention: one launch of
        the decode kernel (plus the combine) when the sync fits in it."""
        K.paged_decode_attn_seqtab(self.pool.handle, seqtab, self.q, self.k_new, self.v_new, self.out, self.table,
                                   self.lens, self.S, self.Hq, self.scale, self.num_splits, self.ws, self.ws.numel(),
                                   stream)

    def append(self, stream=None) -> None:
        K.kv_append(self.pool.handle, self.layout, self.k_new, self.v_new, self.table, self.lens,
                    self.max_blocks, self.S, stream)

    def attend(self, stream=None) -> None:
        K.paged_decode_attn(self.pool.handle, self.layout, self.q, self.out, self.table, self.lens,
                            self.max_blocks, self.S, self.Hq, self.scale, self.num_splits, self.ws,
                            self.ws.numel(), stream)

    def use_cascade(self) -> None:
        """Size the workspace for paged_decode_attn_cascade."""
        need = K.kv_cascade_workspace_bytes(self.pool.handle, self.layout, self.S, self.Hq, self.max_blocks)
        if need > self.ws.numel():
            self.ws = torch.empty(need, dtype=torch.uint8, device=self.pool.device)

    def cascade(self, plan, fused: bool = True, stream=None) -> None:
        K.paged_decode_attn_cascade(self.pool.handle, self.layout, self.q, self.k_new if fused else None,
                                    self.v_new if fused else None, self.out, self.table, self.lens,
                                    self.max_blocks, self.S, self.Hq, self.scale, plan, self.ws,
                                    self.ws.numel(), stream)

    def sync_cascade(self, seqtab, plan, stream=None) -> None:
        """seqtab's table sync, then shared-prefix attention with the fused
        append; the sync rides in the kernel that writes the plan when it fits."""
        K.paged_decode_attn_cascade_seqtab(self.pool.handle, seqtab, self.q, self.k_new, self.v_new, self.out,
                                           self.table, self.lens, self.S, self.Hq, self.scale, plan, self.ws,
                                           self.ws.numel(), stream)
