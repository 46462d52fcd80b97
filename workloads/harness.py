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

    def __init__(self, m, device="cuda", guard=256, misalign=0, fill=GUARD_BYTE, order="index"):
        """order "index": destinations in index order; "blob": in the order of their first
        blob byte, so that a load writes them front to back."""
        import torch
        self.m = m
        offs = [0] * m.n_dsts
        pos = guard
        seq = range(m.n_dsts)
        if order == "blob":
            first = np.full(m.n_dsts, np.iinfo(np.uint64).max, dtype=np.uint64)
            np.minimum.at(first, m.e_dst, m.e_offset)
            seq = np.argsort(first, kind="stable")
        for j in seq:
            j = int(j)
            es = DTYPE_SIZE[str(m.d_dtype[j])]
            mis = (misalign // es) * es
            pos = (pos + 255) // 256 * 256 + mis
            offs[j] = pos
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

    def host_region(self, j0, j1):  # index order layouts only
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


def pinned_blob(m, threads=None):
    """A page-locked torch uint8 tensor holding the source bytes of the manifest's blob."""
    import torch
    t = torch.empty(m.source_bytes(), dtype=torch.uint8, pin_memory=True)
    m.fill_source_ptr(t.data_ptr(), threads)
    return t


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
