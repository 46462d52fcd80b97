"""Writes a manifest's blob as a safetensors checkpoint file (test and benchmark input).

The file holds every checkpoint tensor the manifest's entries read, at full size and at its
blob offset, so the file's data section is byte for byte the manifest's blob.  Gaps left by
alignment or jitter become filler U8 tensors named `__gap_<k>`, which keeps the data section
contiguous as the format asks.  The header is padded with spaces so that the data section
starts on an 8-byte boundary.
"""
import json
import os
import struct

import numpy as np

from .manifests import DTYPE_SIZE

ST_DTYPE = {"u8": "U8", "i16": "I16", "bf16": "BF16", "f16": "F16", "f32": "F32", "i32": "I32",
            "i64": "I64", "f64": "F64"}


def file_tensors(m):
    """[(name, dtype, full shape, offset, nbytes)] of the checkpoint tensors, in blob order,
    with filler tensors over the gaps so the list covers [0, m.blob_bytes) exactly."""
    seen = {}
    for i in range(m.n_entries):
        name, full, off = m.e_name[i], tuple(int(x) for x in m.e_full[i]), int(m.e_full_offset[i])
        dt = str(m.e_dtype[i])
        nb = DTYPE_SIZE[dt] * int(np.prod(full, dtype=np.int64))
        key = (name, dt, full, off, nb)
        if name in seen and seen[name] != key:
            raise ValueError(f"two different tensors named {name}")
        seen[name] = key
    for name, dt, full, off in m.unread:
        nb = DTYPE_SIZE[dt] * int(np.prod(full, dtype=np.int64))
        if name in seen:
            raise ValueError(f"two different tensors named {name}")
        seen[name] = (name, dt, tuple(int(x) for x in full), int(off), nb)
    ts = sorted(seen.values(), key=lambda t: t[3])
    out, pos, k = [], 0, 0
    for t in ts:
        if t[3] < pos:
            raise ValueError(f"tensor {t[0]} overlaps the one before it")
        if t[3] > pos:
            out.append((f"__gap_{k}", "u8", (t[3] - pos,), pos, t[3] - pos))
            k += 1
        out.append(t)
        pos = t[3] + t[4]
    if pos < m.blob_bytes:
        out.append((f"__gap_{k}", "u8", (m.blob_bytes - pos,), pos, m.blob_bytes - pos))
    return out


def header_bytes(tensors, metadata=None, data_align=8):
    """The JSON header, padded with spaces so that the data section (after the 8-byte length
    word and the header) starts at a multiple of data_align bytes."""
    h = {}
    if metadata is not None:
        h["__metadata__"] = metadata
    for name, dt, shape, off, nb in tensors:
        h[name] = {"dtype": ST_DTYPE[dt], "shape": list(shape), "data_offsets": [off, off + nb]}
    raw = json.dumps(h, separators=(",", ":")).encode()
    return raw + b" " * ((-(8 + len(raw))) % data_align)


def write_safetensors(m, path, piece=64 << 20, data_align=8):
    """Writes m's blob as a safetensors file at `path`; returns the data section's file offset."""
    hdr = header_bytes(file_tensors(m), metadata={"format": "pt", "source": m.name},
                       data_align=data_align)
    tmp = str(path) + ".part"
    with open(tmp, "wb") as f:
        f.write(struct.pack("<Q", len(hdr)))
        f.write(hdr)
        for a in range(0, m.blob_bytes, piece):
            f.write(m.blob_range(a, min(piece, m.blob_bytes - a)).tobytes())
    os.replace(tmp, path)
    return 8 + len(hdr)


def targets_for(m):
    """The Safetensors.entries() targets that rebuild m's entries (in m's entry order) from a
    file written by write_safetensors(m, ...)."""
    out = {}
    for i in range(m.n_entries):
        v = {"dst": int(m.e_dst[i]), "row": int(m.e_row[i]), "layer": int(m.e_layer[i]),
             "cast": bool(m.e_cast[i]), "cksum": bool(m.e_cksum[i])}
        sl = m.e_slice[i]
        if sl is not None:
            v[sl[0]] = (int(sl[1]), int(sl[2]))
        if m.e_name[i] in out:
            raise ValueError(f"two entries read {m.e_name[i]}")
        out[m.e_name[i]] = v
    return out
