"""Glue between the synthetic manifests and the loader's Python binding, for tests, the smoke
check and the benchmark: marshals manifest columns, lays destinations out in device memory with
guard bands, and builds generator-backed callback sources.  No loader arithmetic here."""
import ctypes

import numpy as np

from . import gen
from .manifests import DTYPE_SIZE

GUARD_BYTE = 0xA5


def entries_for(m, with_names=False):
    import paper_2607_18957_gb300 as cfa
    return cfa.make_entries(dtype=list(m.e_dtype), shape=(m.e_shape, m.e_ndim),
                            offset=m.e_offset, dst=m.e_dst, row=m.e_row, cast=m.e_cast,
                            cksum=m.e_cksum, layer=m.e_layer,
                            names=m.e_name if with_names else None,
                            src_row_stride=m.e_stride)


class DeviceDsts:
    """All destinations of a manifest in one device buffer.

    Destination j starts at a 256-byte boundary plus `misalign` bytes (a multiple of the
    element size), with `guard` bytes of GUARD_BYTE before the first destination, between
    destinations and after the last, so that stray writes show up."""

    def __init__(self, m, device="cuda", guard=256, misalign=0, fill=GUARD_BYTE):
        import torch
        self.m = m
        offs = []
        pos = guard
        for j in range(m.n_dsts):
            es = DTYPE_SIZE[str(m.d_dtype[j])]
            mis = (misalign // es) * es
            pos = (pos + 255) // 256 * 256 + mis
            offs.append(pos)
            pos += m.d_nbytes(j) + guard
        self.total = pos + 256
        self.offsets = offs
        self.buf = torch.full((self.total,), fill, dtype=torch.uint8, device=device)
        base = self.buf.data_ptr()
        self.base = base
        self.cfa_dsts = [(base + offs[j], str(m.d_dtype[j]), m.d_shape_tuple(j))
                         for j in range(m.n_dsts)]

    def view(self, j):
        o = self.offsets[j]
        return self.buf[o:o + self.m.d_nbytes(j)]

    def host_bytes(self, j):
        return self.view(j).cpu().numpy()

    def host_region(self, j0, j1):
        """Destinations j0 .. j1-1 with one device->host copy: {j: uint8 array}."""
        lo = self.offsets[j0]
        hi = self.offsets[j1 - 1] + self.m.d_nbytes(j1 - 1)
        h = self.buf[lo:hi].cpu().numpy()
        return {j: h[self.offsets[j] - lo:self.offsets[j] - lo + self.m.d_nbytes(j)]
                for j in range(j0, j1)}

    def guards_intact(self):
        """True if every byte outside the destinations still holds GUARD_BYTE."""
        import torch
        mask = torch.ones(self.total, dtype=torch.bool, device=self.buf.device)
        for j in range(self.m.n_dsts):
            o = self.offsets[j]
            mask[o:o + self.m.d_nbytes(j)] = False
        return bool((self.buf[mask] == GUARD_BYTE).all().item())


class CallbackSource:
    """A generator-backed fill callback (wl_fill_cb in blobgen.c) for a manifest's blob."""

    class _C(ctypes.Structure):
        _fields_ = [("kind", ctypes.c_int32), ("reserved", ctypes.c_int32),
                    ("seed", ctypes.c_uint64), ("period", ctypes.c_uint64),
                    ("fail_from", ctypes.c_uint64), ("delay_us", ctypes.c_uint64)]

    def __init__(self, m, fail_from=None, delay_us=0):
        lib = gen._load()
        self.c = self._C()
        self.c.kind = {"bits": 0, "f32mix": 1, "f16fin": 2}[m.blob_kind]
        self.c.seed = m.seed & 0xFFFFFFFFFFFFFFFF
        self.c.period = m.period or 0
        self.c.fail_from = 0xFFFFFFFFFFFFFFFF if fail_from is None else int(fail_from)
        self.c.delay_us = int(delay_us)
        self.fn = ctypes.cast(lib.wl_fill_cb, ctypes.c_void_p).value
        self.user = ctypes.addressof(self.c)

    def source(self):
        import paper_2607_18957_gb300 as cfa
        s = cfa.Source.callback(self.fn, self.user)
        s._keep = self  # the struct must outlive the load
        return s


class _HugePinned:
    """n bytes of page-locked host memory: an anonymous mapping aligned to 512 MiB with
    MADV_HUGEPAGE (transparent huge pages where the kernel allows them), page-locked with
    cudaHostRegister after it has been written.  Unregistered and unmapped when the last tensor
    over it is freed.  torch's pinned allocator instead rounds a request up to a power of two
    (93.6 GB -> 128 GiB) and uses the base pages."""

    ALIGN = 512 << 20

    def __init__(self, n):
        self.libc = ctypes.CDLL(None, use_errno=True)
        self.libc.mmap.restype = ctypes.c_void_p
        self.libc.mmap.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_int,
                                   ctypes.c_int, ctypes.c_long]
        self.libc.munmap.argtypes = [ctypes.c_void_p, ctypes.c_size_t]
        self.libc.madvise.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int]
        self.n = n
        self.size = n + self.ALIGN
        self.p = self.libc.mmap(None, self.size, 0x3, 0x22, -1, 0)  # RW, PRIVATE|ANONYMOUS
        if self.p is None or self.p == ctypes.c_void_p(-1).value:
            raise OSError(ctypes.get_errno(), "mmap of the pinned blob failed")
        self.base = (self.p + self.ALIGN - 1) // self.ALIGN * self.ALIGN
        self.libc.madvise(self.base, n, 14)  # MADV_HUGEPAGE; a refusal only costs speed
        self.registered = False

    def register(self):
        import torch
        rc = torch.cuda.cudart().cudaHostRegister(self.base, self.n, 0)
        if int(getattr(rc, "value", rc)) != 0:
            raise RuntimeError(f"cudaHostRegister failed ({rc})")
        self.registered = True

    def __del__(self):
        try:
            if self.registered:
                import torch
                torch.cuda.cudart().cudaHostUnregister(self.base)
            self.libc.munmap(self.p, self.size)
        except Exception:
            pass


def pinned_blob(m, threads=None):
    """A page-locked torch uint8 tensor holding the source bytes of the manifest's blob (huge
    pages, exact size; torch's pinned allocator if that cannot be had)."""
    import torch
    n = m.source_bytes()
    try:
        h = _HugePinned(max(n, 1))
        m.fill_source_ptr(h.base, threads)  # written first, so that the pages are huge
        h.register()
    except (OSError, RuntimeError, AttributeError):
        t = torch.empty(n, dtype=torch.uint8, pin_memory=True)
        m.fill_source_ptr(t.data_ptr(), threads)
        return t
    arr = (ctypes.c_uint8 * max(n, 1)).from_address(h.base)
    arr._owner = h  # the tensor keeps the array, the array keeps the mapping
    return torch.frombuffer(arr, dtype=torch.uint8)[:n]


def device_blob(m, host=None):
    """A device torch uint8 tensor holding the source bytes (copied from `host` if given)."""
    import torch
    if host is None:
        host = pinned_blob(m)
    d = torch.empty(m.source_bytes(), dtype=torch.uint8, device="cuda")
    d.copy_(host, non_blocking=False)
    return d


def entry_host_bytes(m, i):
    """Blob bytes entry i spans (its source bytes, plus the gaps of a column slice)."""
    return m.blob_range(int(m.e_offset[i]), m.e_extent(i))


__all__ = ["entries_for", "DeviceDsts", "CallbackSource", "pinned_blob", "device_blob",
           "entry_host_bytes", "GUARD_BYTE", "np"]
