"""Python side of the counter-based blob generator (blobgen.c).

`fill(kind, seed, off, length)` returns blob bytes [off, off + length) as a numpy uint8 array;
`fill_ptr` writes them to a raw host address (pinned torch buffers).  Large ranges are split
over threads; ctypes releases the GIL, and the result does not depend on the split because
every word is a pure function of (seed, word index).
"""
import ctypes
import os
import subprocess
import tempfile
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "blobgen.c")
_LIB_PATH = os.path.join(_HERE, "libwlgen.so")
_lock = threading.Lock()
_lib = None

KINDS = ("bits", "f32mix", "f16fin")


def build(force=False):
    """Compiles blobgen.c into libwlgen.so next to it (plain C, any host architecture)."""
    if not force and os.path.exists(_LIB_PATH) and \
            os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            lib.wl_fill_bits.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                         ctypes.c_void_p]
            lib.wl_fill_bits.restype = None
            lib.wl_fill_f32mix.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                           ctypes.c_void_p]
            lib.wl_fill_f32mix.restype = ctypes.c_int
            lib.wl_fill_f16fin.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                           ctypes.c_void_p]
            lib.wl_fill_f16fin.restype = ctypes.c_int
            lib.wl_splitmix64_word.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
            lib.wl_splitmix64_word.restype = ctypes.c_uint64
            _lib = lib
    return _lib


def splitmix64_word(seed, w):
    return int(_load().wl_splitmix64_word(seed & 0xFFFFFFFFFFFFFFFF, w))


def _fill_one(kind, seed, off, length, ptr):
    lib = _load()
    if kind == "bits":
        lib.wl_fill_bits(seed, off, length, ptr)
    elif kind == "f32mix":
        if lib.wl_fill_f32mix(seed, off, length, ptr) != 0:
            raise ValueError("f32mix ranges must start and end on 4-byte boundaries")
    elif kind == "f16fin":
        if lib.wl_fill_f16fin(seed, off, length, ptr) != 0:
            raise ValueError("f16fin ranges must start and end on 2-byte boundaries")
    else:
        raise ValueError(f"unknown blob kind {kind!r}")


def _default_threads():
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def fill_ptr(kind, seed, off, length, ptr, threads=None):
    """Writes blob bytes [off, off + length) of (kind, seed) to host address `ptr`."""
    seed &= 0xFFFFFFFFFFFFFFFF
    if length <= 0:
        return
    threads = threads or _default_threads()
    piece = 64 << 20
    if threads == 1 or length <= piece:
        _fill_one(kind, seed, off, length, ptr)
        return
    # split on 64 MiB boundaries of the blob so the pieces stay word-aligned
    cuts = [off]
    nxt = (off // piece + 1) * piece
    while nxt < off + length:
        cuts.append(nxt)
        nxt += piece
    cuts.append(off + length)
    with ThreadPoolExecutor(max_workers=threads) as ex:
        futs = [ex.submit(_fill_one, kind, seed, a, b - a, ptr + (a - off))
                for a, b in zip(cuts[:-1], cuts[1:])]
        for f in futs:
            f.result()


def fill(kind, seed, off, length, threads=None):
    """Returns blob bytes [off, off + length) of (kind, seed) as a numpy uint8 array."""
    out = np.empty(int(length), dtype=np.uint8)
    if length:
        fill_ptr(kind, seed, int(off), int(length), out.ctypes.data, threads)
    return out
