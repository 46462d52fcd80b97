"""GB300 loader of model checkpoints into a serving engine's final parameter layout.

Python face of the C ABI in include/cfa.h (libcfa.so, built in-tree by `build.py`).  Every
step of a load runs in the library (host plan builder in C, staging pipeline on CUDA streams,
unpack kernels for sm_103a); this module only marshals arguments.  PyTorch is used for device
memory and streams only, and is imported lazily.

    entries = make_entries(dtype=[...], shape=[...], offset=[...], dst=[...], row=[...])
    plan = Plan(entries, dsts=[(tensor.data_ptr(), "bf16", tensor.shape), ...],
                blob_bytes=n)
    plan.load_async(Source.pinned(ptr))      # enqueue; returns at once
    plan.wait_layer(3)                       # readiness group 3 Loaded
    plan.wait_layer()                        # whole load
    ck = plan.checksums()
"""
import contextlib
import ctypes
import gc
import itertools

import numpy as np

from . import _lib
from ._lib import ALL, DTYPE, ENTRY_DTYPE, DST_DTYPE, PIECE_DTYPE  # noqa: F401

__all__ = ["Plan", "Source", "FileSource", "Safetensors", "StTensor", "CfaError", "make_entries",
           "make_dsts", "ALL", "library_path", "segment_range", "AllGather"]


class CfaError(RuntimeError):
    def __init__(self, status, detail):
        self.status = status
        self.name = _lib.STATUS.get(status, str(status))
        super().__init__(f"{self.name}: {detail}")


def library_path():
    return _lib.LIB_PATH


def _check(st, plan_handle=None):
    if st != _lib.CFA_OK:
        lib = _lib.load()
        detail = lib.cfa_last_error(plan_handle)
        raise CfaError(st, detail.decode(errors="replace") if detail else "")


def _stream_handle(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _shape_columns(shapes, n):
    """Shapes (sequences of ints) -> ([n, 8] int64 array, [n] int32 ndim), without a Python loop
    per element."""
    if not isinstance(shapes, (list, tuple)):
        shapes = list(shapes)
    if len(shapes) != n:
        raise ValueError(f"{len(shapes)} shapes for {n} entries")
    nd = np.fromiter(map(len, shapes), dtype=np.int32, count=n)
    if n and int(nd.max()) > 8:
        raise ValueError("more than 8 dimensions")
    out = np.zeros((n, 8), dtype=np.int64)
    total = int(nd.sum())
    if total:
        flat = np.fromiter(itertools.chain.from_iterable(shapes), dtype=np.int64, count=total)
        rows = np.repeat(np.arange(n), nd)
        starts = np.repeat(np.cumsum(nd) - nd, nd)
        out[rows, np.arange(total) - starts] = flat
    return out, nd


def make_entries(dtype, shape, offset, dst, row=None, cast=None, cksum=None, layer=None,
                 names=None, src_row_stride=None):
    """Builds the cfa_tensor_entry array from columns.

    dtype   sequence of dtype names ("bf16", "f32", ...), or of CFA_DTYPE_* codes
    shape   sequence of shapes (tuples), or an [N, 8] int array plus `ndim` via a tuple
            (shape_array, ndim_array)
    offset  blob byte offsets;  dst  destination indices;  row  destination row offsets
    cast, cksum  booleans (default: no conversion, checksum on); cast converts the source
            elements to the destination's dtype (CFA_ENTRY_CONVERT);  layer  readiness groups
    names   optional list of str (kept alive by the returned object)
    src_row_stride  source elements between row starts for strided (column-slice) entries;
            0 = contiguous (default)
    """
    n = len(dst)
    e = np.zeros(n, dtype=ENTRY_DTYPE)
    codes = _dtype_codes(dtype)
    e["src_dtype"] = codes if n else 0
    if isinstance(shape, tuple) and len(shape) == 2 and isinstance(shape[0], np.ndarray):
        e["shape"] = shape[0]
        e["ndim"] = shape[1]
    else:
        e["shape"], e["ndim"] = _shape_columns(shape, n)
    e["blob_offset"] = np.asarray(offset, dtype=np.uint64) if n else 0
    e["dst_index"] = np.asarray(dst, dtype=np.int32) if n else 0
    if row is not None:
        e["dst_row_offset"] = np.asarray(row, dtype=np.int64)
    fl = np.zeros(n, dtype=np.uint32)
    if cast is not None:
        fl |= np.asarray(cast, dtype=bool).astype(np.uint32) * _lib.ENTRY_CONVERT
    if cksum is None:
        fl |= _lib.ENTRY_CKSUM
    else:
        fl |= np.asarray(cksum, dtype=bool).astype(np.uint32) * _lib.ENTRY_CKSUM
    e["flags"] = fl
    if layer is not None:
        e["layer"] = np.asarray(layer, dtype=np.int32)
    if src_row_stride is not None:
        e["src_row_stride"] = np.asarray(src_row_stride, dtype=np.uint32)
    keep = None
    if names is not None:
        enc = [s.encode() for s in names]
        blob = b"\0".join(enc) + b"\0"
        keep = ctypes.create_string_buffer(blob, len(blob))
        size = np.fromiter(map(len, enc), dtype=np.uint64, count=n) + np.uint64(1)
        e["name"] = np.uint64(ctypes.addressof(keep)) + np.cumsum(size, dtype=np.uint64) - size
    return _Entries(e, keep)


@contextlib.contextmanager
def _no_cyclic_gc():
    """Pauses the cyclic garbage collector while a large table of tuples is built (they form no
    cycles; with 10^5 of them the collector's repeated scans took half the time)."""
    was = gc.isenabled()
    gc.disable()
    try:
        yield
    finally:
        if was:
            gc.enable()


class _Entries:
    def __init__(self, arr, keep):
        self.arr = arr
        self.keep = keep

    def __len__(self):
        return len(self.arr)


def _dtype_codes(dtypes):
    """dtype names or CFA_DTYPE_* codes -> int32 array of codes."""
    if isinstance(dtypes, np.ndarray) and dtypes.dtype.kind in "iu":
        return dtypes.astype(np.int32)
    if all(isinstance(x, str) for x in dtypes):  # names: one lookup per distinct name
        names, inverse = np.unique(np.asarray(dtypes, dtype=str), return_inverse=True)
        return np.array([DTYPE[k] for k in names.tolist()], dtype=np.int32)[inverse.ravel()]
    memo = {}

    def code(x):
        if isinstance(x, (int, np.integer)):
            return int(x)
        k = str(x)
        if k not in memo:
            memo[k] = DTYPE[k]
        return memo[k]
    return np.fromiter((code(x) for x in dtypes), dtype=np.int32)


def make_dsts(dsts):
    """[(device pointer, dtype name or code, shape), ...] -> cfa_dst array."""
    n = len(dsts)
    d = np.zeros(n, dtype=DST_DTYPE)
    if n:
        ptrs, dts, shapes = zip(*dsts)
        d["dev_ptr"] = np.fromiter((int(x) for x in ptrs), dtype=np.uint64, count=n)
        d["dtype"] = _dtype_codes(dts)
        d["shape"], d["ndim"] = _shape_columns(shapes, n)
    return d


class Source:
    """Where the blob comes from (cfa_source)."""

    def __init__(self, kind, base=0, period=0, fill=None, user=None, size=0):
        self.kind, self.base, self.period, self.fill, self.user = kind, base, period, fill, user
        self.size = size  # bytes readable at base; 0: not stated (a load checks it when stated)

    @classmethod
    def host(cls, ptr, period=0, size=0):
        """Pageable host memory, copied into pinned slots by the plan's threads."""
        return cls(_lib.SRC_HOST, ptr, period, size=size)

    @classmethod
    def pinned(cls, ptr, period=0, size=0):
        """Page-locked host memory, copied straight to the device."""
        return cls(_lib.SRC_PINNED, ptr, period, size=size)

    @classmethod
    def device(cls, ptr, period=0, size=0):
        """Device memory that already holds the blob (no staging, no copies)."""
        return cls(_lib.SRC_DEVICE, ptr, period, size=size)

    @classmethod
    def host_direct(cls, ptr, period=0, size=0):
        """Host memory (pageable or page-locked, 8-byte aligned) that the unpack kernel reads in
        place over the host link; pageable memory needs a device with pageable memory access."""
        return cls(_lib.SRC_HOST_DIRECT, ptr, period, size=size)

    @classmethod
    def callback(cls, fill_fn_ptr, user_ptr=0):
        """A C function int fill(void *user, uint64 off, void *dst, uint64 len), as an address
        (for example from ctypes.cast(ctypes_function, c_void_p).value)."""
        return cls(_lib.SRC_CALLBACK, 0, 0, fill_fn_ptr, user_ptr)

    def to_c(self):
        s = _lib.Source()
        s.kind = self.kind
        s.base = self.base or None
        s.period_bytes = self.period
        s.fill = self.fill or None
        s.user = self.user or None
        s.size_bytes = self.size
        return s


class FileSource(Source):
    """A checkpoint file (cfa_file_source_open): blob byte o is file byte data_offset + o.  By
    default the plan's fill threads read it with pread; direct=True reads with O_DIRECT, past
    the page cache; mapped=True copies from a read-only mapping of the file (faster for page-
    cache-resident files); in_place=True maps the file and lets the unpack kernels read the
    mapping over the host link, with no fill threads, pinned slots or copies (devices with
    pageable memory access; data_offset a multiple of 8).  A mapped file must not shrink while
    mapped.  Close the source after the last load that uses it has completed (the context
    manager does)."""

    def __init__(self, path, data_offset=0, direct=False, mapped=False, in_place=False):
        lib = _lib.load()
        self._lib = lib
        self._c = _lib.Source()
        flags = ((_lib.FILE_DIRECT if direct else 0) | (_lib.FILE_MMAP if mapped else 0) |
                 (_lib.FILE_MMAP_IN_PLACE if in_place else 0))
        st = lib.cfa_file_source_open(str(path).encode(), int(data_offset), flags,
                                      ctypes.byref(self._c))
        _check(st)
        super().__init__(self._c.kind, self._c.base or 0, 0, self._c.fill, self._c.user,
                         size=self._c.size_bytes)
        self.path, self.data_offset, self.direct = str(path), int(data_offset), bool(direct)
        self.in_place = bool(in_place)

    def to_c(self):
        if not self._c.user:
            raise CfaError(-1, "file source is closed")
        return self._c

    def close(self):
        if self._c.user:
            _check(self._lib.cfa_file_source_close(ctypes.byref(self._c)))

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


Source.file = staticmethod(lambda path, data_offset=0, direct=False, mapped=False,
                           in_place=False: FileSource(path, data_offset, direct, mapped,
                                                      in_place))


class StTensor(tuple):
    """(name, dtype, shape, offset, nbytes) of one safetensors tensor; offset is a blob offset
    into the data section."""
    __slots__ = ()
    name = property(lambda s: s[0])
    dtype = property(lambda s: s[1])
    shape = property(lambda s: s[2])
    offset = property(lambda s: s[3])
    nbytes = property(lambda s: s[4])


class Safetensors:
    """A parsed safetensors header (cfa_safetensors).  The file's data section is the loader's
    blob: `tensors[i].offset` is a blob offset, `data_offset` is where the data section starts in
    the file and `data_bytes` its length."""

    def __init__(self, handle):
        lib = _lib.load()
        n, off, nb = ctypes.c_size_t(), ctypes.c_uint64(), ctypes.c_uint64()
        try:
            _check(lib.cfa_safetensors_info(handle, ctypes.byref(n), ctypes.byref(off),
                                            ctypes.byref(nb)))
            # the whole tensor table in one call; names are read before the handle is closed
            rec = np.zeros(n.value, dtype=_lib.ST_TENSOR_DTYPE)
            _check(lib.cfa_safetensors_tensors(handle, 0, n.value,
                                               rec.ctypes.data if n.value else None))
            nbytes = ctypes.c_uint64()
            _check(lib.cfa_safetensors_names(handle, None, 0, ctypes.byref(nbytes)))
            buf = ctypes.create_string_buffer(max(nbytes.value, 1))
            _check(lib.cfa_safetensors_names(handle, buf, nbytes.value, ctypes.byref(nbytes)))
            names = buf.raw[:nbytes.value].decode("utf-8").split("\0")[:n.value]
            dt_name = {v: k for k, v in DTYPE.items()}
            with _no_cyclic_gc():
                out = [StTensor((nm, dt_name[c], tuple(sh[:k]), o, b))
                       for nm, c, sh, k, o, b in zip(names, rec["dtype"].tolist(),
                                                     rec["shape"].tolist(), rec["ndim"].tolist(),
                                                     rec["blob_offset"].tolist(),
                                                     rec["nbytes"].tolist())]
        finally:
            lib.cfa_safetensors_close(handle)
        self.tensors = out
        self.data_offset, self.data_bytes = off.value, nb.value

    @classmethod
    def open(cls, path):
        """Reads and validates the header of a safetensors file."""
        lib = _lib.load()
        h = ctypes.c_void_p()
        _check(lib.cfa_safetensors_open(str(path).encode(), ctypes.byref(h)))
        return cls(h)

    @classmethod
    def parse(cls, header, file_bytes):
        """Parses the JSON header bytes of a file of `file_bytes` bytes."""
        lib = _lib.load()
        h = ctypes.c_void_p()
        buf = ctypes.create_string_buffer(bytes(header), len(header))
        _check(lib.cfa_safetensors_parse(buf, len(header), int(file_bytes), ctypes.byref(h)))
        return cls(h)

    def entries(self, targets, whole_file=False):
        """Manifest entries for the tensors named in `targets`, in the order of `targets` (a
        name the file does not hold raises KeyError).  A target is
        (dst, row) or (dst, row, layer), or a dict with keys dst, row, layer, cast, cksum and at
        most one of rows=(r0, r1) (a range of the tensor's first dimension) or cols=(c0, c1) (a
        range of its last dimension, read with a source row stride: a tensor-parallel column
        shard).  With whole_file the blob is the whole file (offsets shifted by data_offset), so
        that a mapping of the file from its first byte can serve as the source."""
        n = len(targets)
        dtype, shape, names = [None] * n, [None] * n, [None] * n
        offset, dst, row, layer = [0] * n, [0] * n, [0] * n, [0] * n
        cast, cksum, stride = [False] * n, [True] * n, [0] * n
        shift = self.data_offset if whole_file else 0
        by_name = {t[0]: t for t in self.tensors}
        size = _lib.DTYPE_SIZE
        for i, (name, v) in enumerate(targets.items()):
            t = by_name.get(name)
            if t is None:
                raise KeyError(f"the file holds no tensor named {name!r}")
            tname, tdt, tshape, toff = t[0], t[1], t[2], t[3]
            dtype[i], shape[i], names[i], offset[i] = tdt, tshape, tname, toff + shift
            if not isinstance(v, dict):  # (dst, row) or (dst, row, layer)
                dst[i] = v[0]
                if len(v) > 1:
                    row[i] = v[1]
                if len(v) > 2:
                    layer[i] = v[2]
                continue
            dst[i] = v["dst"]
            row[i] = v.get("row", 0)
            layer[i] = v.get("layer", 0)
            cast[i] = bool(v.get("cast", False))
            cksum[i] = bool(v.get("cksum", True))
            if "rows" in v and "cols" in v:
                raise ValueError(f"{tname}: give rows or cols, not both")
            es = size[tdt]
            if "rows" in v:
                r0, r1 = v["rows"]
                if not (len(tshape) >= 1 and 0 <= r0 <= r1 <= tshape[0]):
                    raise ValueError(f"{tname}: rows {r0}:{r1} outside shape {tshape}")
                per_row = int(np.prod(tshape[1:], dtype=np.int64))
                offset[i] += r0 * per_row * es
                shape[i] = (r1 - r0,) + tuple(tshape[1:])
            elif "cols" in v:
                c0, c1 = v["cols"]
                if not (len(tshape) >= 1 and 0 <= c0 <= c1 <= tshape[-1]):
                    raise ValueError(f"{tname}: cols {c0}:{c1} outside shape {tshape}")
                offset[i] += c0 * es
                if int(np.prod(tshape[:-1], dtype=np.int64)) > 1:
                    stride[i] = tshape[-1]
                shape[i] = tuple(tshape[:-1]) + (c1 - c0,)
        return make_entries(dtype=dtype, shape=shape, offset=offset, dst=dst, row=row,
                            cast=cast, cksum=cksum, layer=layer, names=names,
                            src_row_stride=stride)


def segment_range(blob_bytes, chunk_bytes, world, rank, chunk):
    """(blob offset, bytes) of rank `rank`'s segment of chunk `chunk` in a segmented load of
    `world` ranks (cfa_segment_range)."""
    off, n = ctypes.c_uint64(), ctypes.c_uint64()
    _check(_lib.load().cfa_segment_range(int(blob_bytes), int(chunk_bytes), int(world),
                                         int(rank), int(chunk), ctypes.byref(off),
                                         ctypes.byref(n)))
    return off.value, n.value


class _RawBytes:
    """`n` bytes at device address `ptr`, seen by torch through __cuda_array_interface__."""

    def __init__(self, ptr, n):
        self.__cuda_array_interface__ = {"shape": (n,), "typestr": "|u1", "data": (ptr, False),
                                         "version": 3, "strides": None}


class AllGather:
    """The gather step of a segmented load (section 4.2, "Optimization of Distributed
    Loading"; section 5: AllGather over a torch.distributed group, NCCL on GPUs): a callable for
    Plan(gather=...) that gathers every rank's segment into the chunk's slot in place, enqueued
    on the loader's gather stream.  `device` "cuda" (slot in device memory, the library's case)
    or "cpu" (host memory: the same exchange over gloo, for tests without a GPU)."""

    def __init__(self, group=None, device="cuda"):
        self.group = group
        self.device = device

    def slot(self, ptr, n):
        import torch
        if self.device == "cpu":
            buf = (ctypes.c_uint8 * n).from_address(ptr)
            return torch.frombuffer(buf, dtype=torch.uint8, count=n)
        return torch.as_tensor(_RawBytes(ptr, n), device="cuda")

    def __call__(self, chunk_ptr, segment_bytes, world, rank, chunk, stream):
        import torch
        import torch.distributed as dist
        out = self.slot(chunk_ptr, segment_bytes * world)
        mine = out[rank * segment_bytes:(rank + 1) * segment_bytes]
        if self.device == "cpu":
            dist.all_gather_into_tensor(out, mine, group=self.group)
            return
        with torch.cuda.stream(torch.cuda.ExternalStream(stream)):
            dist.all_gather_into_tensor(out, mine, group=self.group)


class Plan:
    """A loading plan (cfa_plan): validated manifest, chunk <-> tensor mapping, descriptor table,
    staging slots, streams and events."""

    def __init__(self, entries, dsts, blob_bytes, chunk_bytes=512 << 20, host_slots=2,
                 dev_slots=3, fill_threads=None, slab_bytes=0, tiny_bytes=8192, strict=True,
                 host_only=False, timing=False, bulk=True, no_merge=False, stage_slices=False,
                 device=-1,
                 workspace=0, workspace_bytes=0, world=1, rank=0, gather=None,
                 pull_percent=None):
        """world > 1 makes a segmented plan (cfa_plan_opts.seg_world): this process loads
        rank `rank`'s segment of every chunk and `gather(chunk_ptr, segment_bytes, world, rank,
        chunk, stream_handle)` assembles each chunk in the device slot (e.g. AllGather(group)).
        An exception raised by `gather` fails the load with CFA_ERR_GATHER."""
        lib = _lib.load()
        self._lib = lib
        self._handle = None
        if not isinstance(entries, _Entries):
            entries = _Entries(np.ascontiguousarray(entries, dtype=ENTRY_DTYPE), None)
        self._entries = entries
        if not isinstance(dsts, np.ndarray):
            dsts = make_dsts(dsts)
        self._dsts = np.ascontiguousarray(dsts, dtype=DST_DTYPE)
        o = _lib.PlanOpts()
        lib.cfa_plan_opts_default(ctypes.byref(o))
        o.chunk_bytes = chunk_bytes
        o.host_slots = host_slots
        o.dev_slots = dev_slots
        if fill_threads is not None:  # None: the library's default (one per usable CPU)
            o.fill_threads = fill_threads
        o.device = device
        o.slab_bytes = slab_bytes
        o.tiny_bytes = tiny_bytes
        o.flags = ((_lib.OPT_STRICT_COVERAGE if strict else 0) |
                   (_lib.OPT_HOST_ONLY if host_only else 0) |
                   (_lib.OPT_TIMING if timing else 0) |
                   (_lib.OPT_BULK if bulk else 0) |
                   (_lib.OPT_NO_MERGE if no_merge else 0) |
                   (_lib.OPT_STAGE_SLICES if stage_slices else 0))
        o.workspace = workspace or None
        o.workspace_bytes = workspace_bytes
        if pull_percent is not None:  # None: the library's default
            o.pull_percent = pull_percent
        o.seg_world = world
        o.seg_rank = rank
        self._gather = None
        if gather is not None:
            def trampoline(_user, chunk_ptr, seg_bytes, w, r, chunk, stream):
                try:
                    gather(chunk_ptr, seg_bytes, w, r, chunk, stream or 0)
                    return 0
                except Exception as e:  # reported as CFA_ERR_GATHER by the library
                    self.gather_error = e
                    return 1
            self._gather = _lib.GATHER_FN(trampoline)  # kept alive with the plan
            o.gather = ctypes.cast(self._gather, ctypes.c_void_p).value
        self.gather_error = None
        h = ctypes.c_void_p()
        ea = entries.arr
        st = lib.cfa_plan_create(ea.ctypes.data if len(ea) else None, len(ea),
                                 self._dsts.ctypes.data if len(self._dsts) else None,
                                 len(self._dsts), int(blob_bytes), ctypes.byref(o),
                                 ctypes.byref(h))
        _check(st, None)
        self._handle = h
        self.n_entries = len(ea)
        self.chunk_bytes = chunk_bytes
        self._sources = []

    # -- loading -------------------------------------------------------------------------------
    def load_async(self, source, stream=None):
        """Enqueues one full load; returns at once.  Keeps `source` alive until the next load."""
        s = source.to_c()
        self._sources = [source, s]
        st = self._lib.cfa_load_async(self._handle, ctypes.byref(s),
                                      ctypes.c_void_p(_stream_handle(stream)))
        _check(st, self._handle)

    def wait_layer(self, layer=ALL, stream=None, timeout_ns=-1, host=None):
        """Waits for readiness group `layer` (ALL = the whole load).  With a stream (or host=False
        and the current stream) the stream waits on the GPU; otherwise the host blocks."""
        if stream is None and host is False:
            stream = _stream_handle(None)
        h = None if stream is None else ctypes.c_void_p(_stream_handle(stream))
        st = self._lib.cfa_wait_layer(self._handle, layer, h, timeout_ns)
        _check(st, self._handle)

    def try_wait_layer(self, layer=ALL, timeout_ns=0):
        """Host wait that returns the status code instead of raising."""
        return self._lib.cfa_wait_layer(self._handle, layer, None, timeout_ns)

    def checksums(self, n=None):
        n = self.n_entries if n is None else n
        out = np.zeros(n, dtype=np.uint64)
        st = self._lib.cfa_get_checksums(self._handle, out.ctypes.data if n else None, n)
        _check(st, self._handle)
        return out

    def stats(self):
        s = _lib.Stats()
        _check(self._lib.cfa_get_stats(self._handle, ctypes.byref(s)), self._handle)
        return {name: getattr(s, name) for name, _ in _lib.Stats._fields_}

    def timeline(self):
        """Per-chunk timeline of the last load (CFA_OPT_TIMING plans): a float32 array [n_chunks,
        4] of h2d begin/end and unpack begin/end in ms from the load's first operation (-1 where
        the step did not run)."""
        n = self.info()["n_chunks"]
        out = np.zeros((n, 4), dtype=np.float32)
        _check(self._lib.cfa_get_timeline(self._handle, out.ctypes.data if n else None, n),
               self._handle)
        return out

    def layer_times(self, n=None):
        if n is None:
            n = self.info()["n_layers"]
        out = np.zeros(n, dtype=np.float32)
        _check(self._lib.cfa_get_layer_times(self._handle, out.ctypes.data if n else None, n),
               self._handle)
        return out

    def info(self):
        a, b, c = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
        _check(self._lib.cfa_plan_info(self._handle, ctypes.byref(a), ctypes.byref(b),
                                       ctypes.byref(c)), self._handle)
        return {"n_layers": a.value, "n_pieces": b.value, "n_chunks": c.value}

    def pieces(self):
        n = self.info()["n_pieces"]
        out = np.zeros(n, dtype=PIECE_DTYPE)
        got = ctypes.c_size_t()
        _check(self._lib.cfa_plan_get_pieces(self._handle, out.ctypes.data if n else None, n,
                                             ctypes.byref(got)), self._handle)
        return out[:got.value]

    def unpack_chunks_async(self, chunk_begin, chunk_end, src_ptr, stream=None):
        st = self._lib.cfa_unpack_chunks_async(self._handle, chunk_begin, chunk_end,
                                               ctypes.c_void_p(src_ptr),
                                               ctypes.c_void_p(_stream_handle(stream)))
        _check(st, self._handle)

    def reset_checksums(self, stream=None):
        _check(self._lib.cfa_reset_checksums(self._handle,
                                             ctypes.c_void_p(_stream_handle(stream))),
               self._handle)

    def close(self):
        if self._handle is not None:
            self._lib.cfa_plan_destroy(self._handle)
            self._handle = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
