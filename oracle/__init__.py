"""ORACLE -- plain CPU unpacker used to check the GPU loader.  Test infrastructure only.

Only the test suite, `__graft_entry__.smoke()` and the benchmark's CPU-baseline / reference leg
may import this package.  It shares no code with the loader library (the library lives in
`paper_2607_18957_gb300/`); both consume the same seeded manifests and blob bytes from
`workloads/`, which hold none of the method's arithmetic.

The arithmetic is in cfa_oracle.c (InstantInfer section 4.2 and Theorem 2: the naive per-tensor
loader, element by element).  This wrapper only marshals numpy arrays.

Functions:
  rne_bf16(u32 array) -> u16 array               the bitwise round-to-nearest-even cast
  unpack(manifest, blob, ...) -> OracleResult     destinations, checksums, coverage
"""
import ctypes
import os
import subprocess
import tempfile
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cfa_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

# The oracle's own dtype codes (cfa_oracle.c); dtype names are the manifest's.
_DTYPE_CODE = {"u8": 1, "bf16": 2, "f16": 3, "f32": 4, "i32": 5, "i64": 6, "f64": 7, "i16": 8}
_ELEM = {"u8": 1, "bf16": 2, "f16": 2, "f32": 4, "i32": 4, "i64": 8, "f64": 8, "i16": 2}
_CONVERT, _CKSUM = 1, 2
# conversion ids of oracle_convert_array
CONV = {("f32", "bf16"): 1, ("f32", "f16"): 2, ("f16", "bf16"): 3, ("bf16", "f32"): 4,
        ("f16", "f32"): 5}

ORC_OK, ORC_E_INVAL, ORC_E_DTYPE, ORC_E_ALIGN, ORC_E_OOB, ORC_E_SHAPE, ORC_E_OVERLAP, \
    ORC_E_COVERAGE = range(8)
STATUS_NAME = {0: "ok", 1: "inval", 2: "dtype", 3: "align", 4: "oob", 5: "shape",
               6: "overlap", 7: "coverage"}


def build(force=False):
    """Compiles cfa_oracle.c into liboracle.so (plain C; no vectorisation flags)."""
    if not force and os.path.exists(_LIB_PATH) and \
            os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    subprocess.run(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"],
                   check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _bind(path):
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    U64 = ctypes.c_uint64
    lib.oracle_rne_bf16.argtypes = [ctypes.c_uint32]
    lib.oracle_rne_bf16.restype = ctypes.c_uint16
    lib.oracle_rne_bf16_array.argtypes = [P, P, U64]
    lib.oracle_rne_bf16_array.restype = None
    lib.oracle_unpack.argtypes = [U64, P, P, P, P, P, P, P, P, U64, P, P, P, P, P, P, U64,
                                  U64, U64, P, P]
    lib.oracle_unpack.restype = ctypes.c_int
    lib.oracle_check_cover.argtypes = [U64, P, P, P]
    lib.oracle_check_cover.restype = ctypes.c_int
    lib.oracle_convert_array.argtypes = [ctypes.c_int, P, P, U64]
    lib.oracle_convert_array.restype = None
    lib.oracle_f32_to_f16.argtypes = [ctypes.c_uint32]
    lib.oracle_f32_to_f16.restype = ctypes.c_uint16
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            _lib = _bind(_LIB_PATH)
    return _lib


def rne_bf16_scalar(u, lib=None):
    return int((lib or _load()).oracle_rne_bf16(int(u) & 0xFFFFFFFF))


def rne_bf16(u32, lib=None):
    """Bitwise fp32 -> bf16 round-to-nearest-even over a uint32 array."""
    a = np.ascontiguousarray(u32, dtype=np.uint32)
    out = np.empty(a.shape, dtype=np.uint16)
    (lib or _load()).oracle_rne_bf16_array(a.ctypes.data, out.ctypes.data, a.size)
    return out


def convert(src_dtype, dst_dtype, bits, lib=None):
    """Converts an array of source bit patterns (uint16 or uint32) to destination bit patterns
    with the oracle's conversion for that dtype pair."""
    conv = CONV[(src_dtype, dst_dtype)]
    a = np.ascontiguousarray(bits, dtype=np.uint16 if src_dtype in ("f16", "bf16") else np.uint32)
    out = np.empty(a.shape, dtype=np.uint16 if dst_dtype in ("f16", "bf16") else np.uint32)
    (lib or _load()).oracle_convert_array(conv, a.ctypes.data, out.ctypes.data, a.size)
    return out


def f32_to_f16_scalar(u, lib=None):
    return int((lib or _load()).oracle_f32_to_f16(int(u) & 0xFFFFFFFF))


class OracleResult:
    def __init__(self, status, bad_entry, dst, cksum, cover):
        self.status = status          # ORC_* code
        self.bad_entry = bad_entry    # first failing entry or -1
        self.dst = dst                # {dst index: uint8 array of the destination's bytes}
        self.cksum = cksum            # uint64 [n_entries]
        self.cover = cover            # {dst index: uint32 per-byte write counts} or None

    @property
    def status_name(self):
        return STATUS_NAME[self.status]


def _ptr_array(arrs):
    out = (ctypes.c_void_p * len(arrs))()
    for i, a in enumerate(arrs):
        out[i] = None if a is None else a.ctypes.data
    return out


def _columns(m):
    """The manifest's columns in the oracle's own codes (marshalling only; cached on m)."""
    c = getattr(m, "_oracle_columns", None)
    if c is None:
        c = (np.array([_DTYPE_CODE[str(x)] for x in m.e_dtype], dtype=np.int32),
             np.array([_DTYPE_CODE[str(x)] for x in m.d_dtype], dtype=np.int32),
             (m.e_cast.astype(np.uint32) * _CONVERT) | (m.e_cksum.astype(np.uint32) * _CKSUM),
             np.ascontiguousarray(m.e_ndim, dtype=np.int32),
             np.ascontiguousarray(m.e_shape, dtype=np.int64),
             np.ascontiguousarray(m.e_offset, dtype=np.uint64),
             np.ascontiguousarray(m.e_dst, dtype=np.int32),
             np.ascontiguousarray(m.e_row, dtype=np.int64),
             np.ascontiguousarray(m.d_ndim, dtype=np.int32),
             np.ascontiguousarray(m.d_shape, dtype=np.int64),
             np.ascontiguousarray(getattr(m, "e_stride", np.zeros(m.n_entries)),
                                  dtype=np.uint32))
        try:
            m._oracle_columns = c
        except AttributeError:
            pass
    return c


def unpack(m, blob, blob_begin=0, dsts=None, cover=False, fill=0, lib=None):
    """Runs the naive loader over manifest `m`.

    blob        uint8 array holding blob bytes [blob_begin, blob_begin + len(blob)).
    dsts        destination indices to materialise (default: all).  Entries into other
                destinations are validated only.
    cover       also return per-byte write counts (and check the strict-coverage rule via
                check_cover).
    fill        initial byte value of the destination buffers.
    lib         a library bound with load_variant (default: the oracle itself).
    """
    lib = lib or _load()
    n, nd = m.n_entries, m.n_dsts
    sel = range(nd) if dsts is None else sorted(set(int(j) for j in dsts))
    (e_dtype, d_dtype, e_flags, e_ndim, e_shape, e_off, e_dst, e_row, d_ndim,
     d_shape, e_stride) = _columns(m)
    bufs = [None] * nd
    covs = [None] * nd
    for j in sel:
        nel = int(np.prod(m.d_shape[j, :m.d_ndim[j]], dtype=np.int64))
        nb = nel * _ELEM[str(m.d_dtype[j])]
        bufs[j] = np.full(nb, fill, dtype=np.uint8)
        if cover:
            covs[j] = np.zeros(nb, dtype=np.uint32)
    blob = np.ascontiguousarray(blob, dtype=np.uint8)
    ck = np.zeros(n, dtype=np.uint64)
    bad = ctypes.c_int64(-1)
    st = lib.oracle_unpack(
        n, e_dtype.ctypes.data, e_ndim.ctypes.data, e_shape.ctypes.data, e_off.ctypes.data,
        e_dst.ctypes.data, e_row.ctypes.data, e_flags.ctypes.data, e_stride.ctypes.data,
        nd, d_dtype.ctypes.data, d_ndim.ctypes.data, d_shape.ctypes.data,
        _ptr_array(bufs), _ptr_array(covs) if cover else None,
        blob.ctypes.data if blob.size else None, blob_begin, blob_begin + blob.size,
        m.blob_bytes, ck.ctypes.data, ctypes.byref(bad))
    return OracleResult(st, bad.value, {j: bufs[j] for j in sel}, ck,
                        {j: covs[j] for j in sel} if cover else None)


def check_cover(res, lib=None):
    """Strict-coverage rule over an unpack(..., cover=True) result: returns (code, dst)."""
    lib = lib or _load()
    keys = sorted(res.cover)
    nbytes = np.array([res.cover[j].size for j in keys], dtype=np.uint64)
    bad = ctypes.c_int64(-1)
    st = lib.oracle_check_cover(len(keys), nbytes.ctypes.data,
                                _ptr_array([res.cover[j] for j in keys]), ctypes.byref(bad))
    return st, (keys[bad.value] if bad.value >= 0 else -1)


def load_variant(path):
    """Binds another build of cfa_oracle.c (the mutation tests compile deliberately broken
    copies to show that the pins catch them); pass the result as `lib=`."""
    return _bind(path)


SOURCE_PATH = _SRC
