"""ctypes bindings of libcfa.so (the C ABI in include/cfa.h).  Argument marshalling only."""
import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcfa.so")

# status codes (cfa.h)
CFA_OK = 0
STATUS = {0: "CFA_OK", -1: "CFA_ERR_INVAL", -2: "CFA_ERR_OVERLAP", -3: "CFA_ERR_OOB",
          -4: "CFA_ERR_COVERAGE", -5: "CFA_ERR_CUDA", -6: "CFA_ERR_SOURCE", -7: "CFA_ERR_TIMEOUT",
          -8: "CFA_ERR_BUSY", -9: "CFA_ERR_NOMEM", -10: "CFA_ERR_DTYPE", -11: "CFA_ERR_ALIGN",
          -12: "CFA_ERR_DEVICE", -13: "CFA_ERR_SHAPE",
          -14: "CFA_ERR_SUSPECT", -15: "CFA_ERR_GATHER"}
DTYPE = {"u8": 1, "bf16": 2, "f16": 3, "f32": 4, "i32": 5, "i64": 6, "f64": 7, "i16": 8}
DTYPE_SIZE = {"u8": 1, "bf16": 2, "f16": 2, "f32": 4, "i32": 4, "i64": 8, "f64": 8, "i16": 2}
ENTRY_CAST_BF16, ENTRY_CKSUM, ENTRY_CONVERT = 0x1, 0x2, 0x4
OPT_STRICT_COVERAGE, OPT_HOST_ONLY, OPT_TIMING, OPT_BULK, OPT_NO_MERGE = 0x1, 0x2, 0x4, 0x8, 0x10
OPT_STAGE_SLICES = 0x20
SRC_HOST, SRC_PINNED, SRC_CALLBACK, SRC_DEVICE, SRC_HOST_DIRECT = 1, 2, 3, 4, 5
FILE_DIRECT, FILE_MMAP, FILE_MMAP_IN_PLACE = 0x1, 0x2, 0x4
ALL = -1

# cfa_tensor_entry and cfa_dst as numpy records (fast for 10^5 entries)
ENTRY_DTYPE = np.dtype([("name", "<u8"), ("src_dtype", "<i4"), ("ndim", "<i4"),
                        ("shape", "<i8", (8,)), ("blob_offset", "<u8"), ("dst_index", "<i4"),
                        ("layer", "<i4"), ("dst_row_offset", "<i8"), ("flags", "<u4"),
                        ("src_row_stride", "<u4")])
DST_DTYPE = np.dtype([("dev_ptr", "<u8"), ("dtype", "<i4"), ("ndim", "<i4"),
                      ("shape", "<i8", (8,))])

FILL_FN = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p,
                           ctypes.c_uint64)
# cfa_gather_fn(user, chunk_dev, segment_bytes, world, rank, chunk, stream)
GATHER_FN = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint64,
                             ctypes.c_int32, ctypes.c_int32, ctypes.c_uint32, ctypes.c_void_p)


class PlanOpts(ctypes.Structure):
    _fields_ = [("chunk_bytes", ctypes.c_uint64), ("host_slots", ctypes.c_int32),
                ("dev_slots", ctypes.c_int32), ("fill_threads", ctypes.c_int32),
                ("device", ctypes.c_int32), ("slab_bytes", ctypes.c_uint32),
                ("tiny_bytes", ctypes.c_uint32), ("flags", ctypes.c_uint32),
                ("pull_percent", ctypes.c_uint32), ("workspace", ctypes.c_void_p),
                ("workspace_bytes", ctypes.c_uint64), ("seg_world", ctypes.c_int32),
                ("seg_rank", ctypes.c_int32), ("gather", ctypes.c_void_p),
                ("gather_user", ctypes.c_void_p)]


class Source(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("base", ctypes.c_void_p), ("period_bytes", ctypes.c_uint64),
                ("fill", ctypes.c_void_p), ("user", ctypes.c_void_p),
                ("size_bytes", ctypes.c_uint64)]


class Stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_uint64) for n in (
        "blob_bytes", "n_entries", "n_dsts", "n_chunks", "n_layers", "n_pieces", "n_slabs",
        "n_bulk", "n_tiny", "n_strided", "bytes_read", "bytes_written", "descriptor_bytes",
        "staged_bytes", "loads",
        "kernel_launches")] + [(n, ctypes.c_double) for n in (
            "plan_ms", "load_ms", "h2d_ms", "unpack_ms")]


class Piece(ctypes.Structure):
    _fields_ = [("chunk", ctypes.c_uint32), ("entry", ctypes.c_uint32),
                ("src_offset", ctypes.c_uint64), ("dst_index", ctypes.c_uint32),
                ("conv", ctypes.c_uint32), ("dst_offset", ctypes.c_uint64),
                ("n_elems", ctypes.c_uint64), ("rows", ctypes.c_uint32),
                ("src_row_stride", ctypes.c_uint32)]


class StTensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("dtype", ctypes.c_int32), ("ndim", ctypes.c_int32),
                ("shape", ctypes.c_int64 * 8), ("blob_offset", ctypes.c_uint64),
                ("nbytes", ctypes.c_uint64)]


# cfa_st_tensor as a numpy record (bulk reads of a header's tensor table)
ST_TENSOR_DTYPE = np.dtype([("name", "<u8"), ("dtype", "<i4"), ("ndim", "<i4"),
                            ("shape", "<i8", (8,)), ("blob_offset", "<u8"), ("nbytes", "<u8")])

assert ST_TENSOR_DTYPE.itemsize == ctypes.sizeof(StTensor)

PIECE_DTYPE = np.dtype([("chunk", "<u4"), ("entry", "<u4"), ("src_offset", "<u8"),
                        ("dst_index", "<u4"), ("conv", "<u4"), ("dst_offset", "<u8"),
                        ("n_elems", "<u8"), ("rows", "<u4"), ("src_row_stride", "<u4")])

# Every function cfa.h declares, with its ctypes signature.
_P, _U64, _I32, _SZ = ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int32, ctypes.c_size_t
SIGNATURES = {
    "cfa_plan_opts_default": (None, [_P]),
    "cfa_plan_create": (ctypes.c_int, [_P, _SZ, _P, _SZ, _U64, _P, _P]),
    "cfa_load_async": (ctypes.c_int, [_P, _P, _P]),
    "cfa_wait_layer": (ctypes.c_int, [_P, _I32, _P, ctypes.c_int64]),
    "cfa_get_checksums": (ctypes.c_int, [_P, _P, _SZ]),
    "cfa_get_stats": (ctypes.c_int, [_P, _P]),
    "cfa_get_layer_times": (ctypes.c_int, [_P, _P, _SZ]),
    "cfa_plan_info": (ctypes.c_int, [_P, _P, _P, _P]),
    "cfa_plan_get_pieces": (ctypes.c_int, [_P, _P, _SZ, _P]),
    "cfa_unpack_chunks_async": (ctypes.c_int, [_P, ctypes.c_uint32, ctypes.c_uint32, _P, _P]),
    "cfa_reset_checksums": (ctypes.c_int, [_P, _P]),
    "cfa_segment_range": (ctypes.c_int, [_U64, _U64, _I32, _I32, ctypes.c_uint32, _P, _P]),
    "cfa_plan_destroy": (ctypes.c_int, [_P]),
    "cfa_last_error": (ctypes.c_char_p, [_P]),
    "cfa_status_name": (ctypes.c_char_p, [ctypes.c_int]),
    "cfa_abi_sizeof": (_SZ, [ctypes.c_char_p]),
    "cfa_unpack_noalloc": (ctypes.c_int, [_P, _SZ, _P, _SZ, _P, _U64, _P, _P, _P,
                                          ctypes.c_char_p, _SZ]),
    "cfa_safetensors_open": (ctypes.c_int, [ctypes.c_char_p, _P]),
    "cfa_safetensors_parse": (ctypes.c_int, [_P, _U64, _U64, _P]),
    "cfa_safetensors_info": (ctypes.c_int, [_P, _P, _P, _P]),
    "cfa_safetensors_tensor": (ctypes.c_int, [_P, _SZ, _P]),
    "cfa_safetensors_tensors": (ctypes.c_int, [_P, _SZ, _SZ, _P]),
    "cfa_safetensors_names": (ctypes.c_int, [_P, _P, _U64, _P]),
    "cfa_safetensors_close": (ctypes.c_int, [_P]),
    "cfa_file_source_open": (ctypes.c_int, [ctypes.c_char_p, _U64, ctypes.c_uint32, _P]),
    "cfa_file_source_close": (ctypes.c_int, [_P]),
    "cfa_selftest_wait_timeout": (ctypes.c_int, [ctypes.c_int, _P]),
    "cfa_get_timeline": (ctypes.c_int, [_P, _P, _SZ]),
}

_lib = None


def load():
    """Loads libcfa.so from the package directory.  There is no fallback: without the compiled
    library nothing here works, and the error says how to build it."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            f"{LIB_PATH} is missing: build it with `python -m paper_2607_18957_gb300.build` "
            "(nvcc for sm_103a)")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in SIGNATURES.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _check_layouts(lib)
    _lib = lib
    return lib


def _check_layouts(lib):
    want = {"cfa_tensor_entry": ENTRY_DTYPE.itemsize, "cfa_dst": DST_DTYPE.itemsize,
            "cfa_plan_opts": ctypes.sizeof(PlanOpts), "cfa_source": ctypes.sizeof(Source),
            "cfa_stats": ctypes.sizeof(Stats), "cfa_piece": ctypes.sizeof(Piece),
            "cfa_st_tensor": ST_TENSOR_DTYPE.itemsize,
            "cfa_chunk_times": 16}
    for name, size in want.items():
        got = lib.cfa_abi_sizeof(name.encode())
        if got != size:
            raise RuntimeError(f"ABI mismatch for {name}: library {got} B, binding {size} B")
