"""Checkpoint files on the host (no GPU): the safetensors header parser against Python's json
module, the format's corner cases and malformed headers, manifests rebuilt from a file (whole
tensors, row and column shards), and the pread file source's fill function."""
import ctypes
import json
import os
import random
import struct
import subprocess

import numpy as np
import pytest

import paper_2607_18957_gb300 as cfa
from paper_2607_18957_gb300 import _lib
from workloads import dense_config, moe_config
from workloads.harness import entries_for
from workloads.stfile import ST_DTYPE, file_tensors, header_bytes, targets_for, write_safetensors

from test_host_pool import sanitizer_could_not_start

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

ST_NAME = {v: k for k, v in ST_DTYPE.items()}
ST_NAME.update({"BOOL": "u8", "I8": "u8", "F8_E4M3": "u8", "F8_E5M2": "u8", "U16": "i16",
                "U32": "i32", "U64": "i64"})


def configs():
    return [
        dense_config("st_dense", 81, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64, inter=640,
                     vocab=512, align=2, jitter=5),
        dense_config("st_f32_tp4r1", 82, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                     inter=640, vocab=512, src_dtype="f32", align=4, jitter=3, tp=4, rank=1),
        moe_config("st_moe_tp2r1", 83, layers=1, hidden=128, n_q=2, n_kv=2, head_dim=64,
                   inter=256, n_experts=4, vocab=256, n_extra=200, align=2, jitter=3, tp=2,
                   rank=1),
    ]


def write_file(path, header, data=b""):
    with open(path, "wb") as f:
        f.write(struct.pack("<Q", len(header)))
        f.write(header)
        f.write(data)


def expect_from_json(raw, file_bytes):
    """The tensor list by Python's json module (an independent reading of the header)."""
    h = json.loads(raw)
    out = []
    for name, v in h.items():
        if name == "__metadata__":
            continue
        b, e = v["data_offsets"]
        out.append((name, ST_NAME[v["dtype"]], tuple(v["shape"]), b, e - b))
    return out, 8 + len(raw), file_bytes - 8 - len(raw)


@pytest.mark.parametrize("idx", [0, 1, 2])
def test_parse_matches_json_and_the_manifest(tmp_path, idx):
    m = configs()[idx]
    p = tmp_path / "model.safetensors"
    off = write_safetensors(m, p)
    raw = p.read_bytes()
    (n,) = struct.unpack("<Q", raw[:8])
    assert off == 8 + n and off % 8 == 0
    st = cfa.Safetensors.open(p)
    want, data_off, data_bytes = expect_from_json(raw[8:8 + n], len(raw))
    assert [tuple(t) for t in st.tensors] == want
    assert (st.data_offset, st.data_bytes) == (data_off, data_bytes) == (off, m.blob_bytes)
    assert [tuple(t) for t in st.tensors] == file_tensors(m)
    # the same bytes through the in-memory parser
    st2 = cfa.Safetensors.parse(raw[8:8 + n], len(raw))
    assert st2.tensors == st.tensors
    # the data section is the manifest's blob
    assert np.array_equal(np.frombuffer(raw, np.uint8, offset=off), m.blob_range(0, m.blob_bytes))


@pytest.mark.parametrize("idx", [0, 1, 2])
def test_entries_from_a_file_equal_the_manifest(tmp_path, idx):
    """Whole tensors, row shards and column shards (source row stride) rebuilt from the header
    equal the entries the manifest builder made, field by field."""
    m = configs()[idx]
    p = tmp_path / "model.safetensors"
    off = write_safetensors(m, p)
    st = cfa.Safetensors.open(p)
    ref = entries_for(m).arr
    for whole, shift in ((False, 0), (True, off)):
        got = st.entries(targets_for(m), whole_file=whole).arr
        for f in ("src_dtype", "ndim", "shape", "dst_index", "layer", "dst_row_offset", "flags",
                  "src_row_stride"):
            assert np.array_equal(got[f], ref[f]), f
        assert np.array_equal(got["blob_offset"], ref["blob_offset"] + np.uint64(shift))
    if idx:
        assert (ref["src_row_stride"] > 0).any(), "the shard config has no column slices"


def test_entry_slices_are_checked():
    hdr = header_bytes([("w", "bf16", (4, 6), 0, 48)])
    st = cfa.Safetensors.parse(hdr, 8 + len(hdr) + 48)
    e = st.entries({"w": {"dst": 0, "cols": (2, 5)}}).arr
    assert (e["blob_offset"][0], tuple(e["shape"][0, :2]), e["src_row_stride"][0]) == (4, (4, 3), 6)
    e = st.entries({"w": {"dst": 0, "rows": (1, 3)}}).arr
    assert (e["blob_offset"][0], tuple(e["shape"][0, :2]), e["src_row_stride"][0]) == (12, (2, 6), 0)
    with pytest.raises(ValueError):
        st.entries({"w": {"dst": 0, "cols": (5, 7)}})
    with pytest.raises(ValueError):
        st.entries({"w": {"dst": 0, "rows": (0, 1), "cols": (0, 1)}})
    with pytest.raises(KeyError):
        st.entries({"missing": (0, 0)})


def test_format_corner_cases():
    """Keys in any order, unknown keys, nested metadata, escapes and non-ASCII names, scalars,
    zero-size tensors, every dtype name, whitespace around tokens."""
    names = ["café.weight", "emoji\U0001F600", 'quote"d', "back\\slash", "tab\tname", "/"]
    h = {"__metadata__": {"a": [1, 2.5e3, -3, {"b": None}], "c": True, "d": False, "e": "x"}}
    off = 0
    dts = ["BOOL", "U8", "I8", "F8_E4M3", "F8_E5M2", "I16", "U16", "F16", "BF16", "I32", "U32",
           "F32", "I64", "U64", "F64"]
    size = {"BOOL": 1, "U8": 1, "I8": 1, "F8_E4M3": 1, "F8_E5M2": 1, "I16": 2, "U16": 2,
            "F16": 2, "BF16": 2, "I32": 4, "U32": 4, "F32": 4, "I64": 8, "U64": 8, "F64": 8}
    for k, dt in enumerate(dts):
        shape = [[], [0], [3], [2, 3], [1, 1, 1, 1, 1, 1, 1, 5]][k % 5]
        nb = size[dt] * int(np.prod(shape, dtype=np.int64))
        name = names[k] if k < len(names) else f"t{k}"
        v = {"shape": shape, "data_offsets": [off, off + nb], "extra": {"x": [1]}, "dtype": dt}
        if k % 2:
            v = dict(reversed(list(v.items())))
        h[name] = v
        off += nb
    for raw in (json.dumps(h).encode(), json.dumps(h, indent=3).encode(),
                json.dumps(h, ensure_ascii=False).encode()):
        st = cfa.Safetensors.parse(raw, 8 + len(raw) + off)
        want, _, _ = expect_from_json(raw, 8 + len(raw) + off)
        assert [tuple(t) for t in st.tensors] == want
    empty = cfa.Safetensors.parse(b"{}", 10)
    assert empty.tensors == [] and empty.data_bytes == 0
    meta_only = cfa.Safetensors.parse(b' {"__metadata__" : {} }   ', 8 + 26)
    assert meta_only.tensors == []


BAD_HEADERS = [
    b"",
    b"{",
    b"[]",
    b'{"a": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]}} x',
    b'{"a": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]},}',
    b'{"a": {"dtype": "F4", "shape": [2], "data_offsets": [0, 1]}}',
    b'{"a": {"dtype": "F32", "shape": [2], "data_offsets": [0, 12]}}',
    b'{"a": {"dtype": "F32", "shape": [2], "data_offsets": [8, 0]}}',
    b'{"a": {"dtype": "F32", "shape": [2], "data_offsets": [64, 72]}}',
    b'{"a": {"dtype": "F32", "shape": [-2], "data_offsets": [0, 8]}}',
    b'{"a": {"dtype": "F32", "shape": [2.0], "data_offsets": [0, 8]}}',
    b'{"a": {"dtype": "F32", "shape": [1,1,1,1,1,1,1,1,2], "data_offsets": [0, 8]}}',
    b'{"a": {"dtype": "F32", "data_offsets": [0, 8]}}',
    b'{"a": {"dtype": "F32", "shape": [2]}}',
    b'{"a": {"shape": [2], "data_offsets": [0, 8]}}',
    b'{"a": {}}',
    b'{"a": 3}',
    b'{"a\\x": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]}}',
    b'{"\\ud800": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]}}',
    b'{"a": {"dtype": "F32", "shape": [99999999999999999999], "data_offsets": [0, 8]}}',
    b'{"a": {"dtype": "U8", "shape": [4294967296, 4294967296], "data_offsets": [0, 8]}}',
    b'{"__metadata__": ' + b"[" * 100 + b"]" * 100 + b"}",
    b'{"a": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]}',
    b'{"__metadata__": {"x": 1\x002}}',
    b'{"a\x00": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]}}',
    b'{"a\\u0000b": {"dtype": "F32", "shape": [2], "data_offsets": [0, 8]}}',
]


@pytest.mark.parametrize("k", range(len(BAD_HEADERS)))
def test_malformed_headers_are_rejected(k):
    raw = BAD_HEADERS[k]
    with pytest.raises(cfa.CfaError) as e:
        cfa.Safetensors.parse(raw, 8 + len(raw) + 16)
    assert e.value.name == "CFA_ERR_INVAL"


ST_ES = {"BOOL": 1, "U8": 1, "I8": 1, "F8_E4M3": 1, "F8_E5M2": 1, "I16": 2, "U16": 2, "F16": 2,
         "BF16": 2, "I32": 4, "U32": 4, "F32": 4, "I64": 8, "U64": 8, "F64": 8}


def json_reading(raw, file_bytes):
    """The tensor list a strict reading of the header by Python's json module gives, or None
    where the format rejects the header.  The rules: UTF-8 JSON text, no NaN or Infinity; every
    string a sequence of Unicode scalar values other than U+0000 (a lone surrogate escape or a
    \\u0000 is rejected); a top-level
    object whose values other than __metadata__ are objects with a known dtype, a shape of at most
    8 integers in [0, 2^63) whose non-zero product fits in 64 bits, and data_offsets [b, e] with
    b <= e <= the data section's size and e - b the shape's byte size.  Repeated names are kept,
    in order (the parser does not check them)."""
    def reject_constant(name):
        raise ValueError(name)

    def scalar_values_only(x):
        if isinstance(x, str):
            try:
                x.encode("utf-8")
            except UnicodeEncodeError:
                return False
            return "\x00" not in x  # a C string cannot hold U+0000
        if isinstance(x, (list, tuple)):
            return all(scalar_values_only(y) for y in x)
        return True

    try:
        h = json.loads(raw.decode("utf-8"), object_pairs_hook=list,
                       parse_constant=reject_constant)
    except ValueError:  # includes UnicodeDecodeError and json.JSONDecodeError
        return None
    if not isinstance(h, list) or not scalar_values_only(h):
        return None
    data_bytes = file_bytes - 8 - len(raw)
    out = []
    for name, v in h:
        if name == "__metadata__":
            continue
        if not isinstance(v, list):
            return None
        d = dict(v)
        if not {"dtype", "shape", "data_offsets"} <= d.keys():
            return None
        dt, shape, offs = d["dtype"], d["shape"], d["data_offsets"]
        if (not isinstance(dt, str) or dt not in ST_ES or not isinstance(shape, list)
                or len(shape) > 8 or not isinstance(offs, list) or len(offs) != 2):
            return None
        if any(type(x) is not int or not 0 <= x < 1 << 63 for x in shape):
            return None
        if any(type(x) is not int or not 0 <= x < 1 << 64 for x in offs):
            return None
        nz = 1
        for x in shape:
            nz *= x or 1
        if nz >= 1 << 64:
            return None
        nbytes = 0 if 0 in shape else ST_ES[dt] * nz
        b, e = offs
        if not b <= e <= data_bytes or e - b != nbytes:
            return None
        out.append((name, ST_NAME[dt], tuple(shape), b, e - b))
    return out


_FUZZ_TOKENS = [b"{", b"}", b"[", b"]", b",", b":", b'"', b"\\", b"\\u", b"\\u00", b"\\ud800",
                b"\\udc00", b"\\ud800\\udc00", b"\\u0000", b"1e999", b"-1", b"-0", b"01", b"1.5",
                b"2.0", b"1E2",
                b"18446744073709551615", b"18446744073709551616", b"9223372036854775808",
                b"99999999999999999999999", b"null", b"true", b"NaN", b"\x00", b"\t", b"\n",
                b"\xff", b"\xc3\xa9", b"\xe2\x82", b"\xed\xa0\x80", b"\xf4\x90\x80\x80", b"\xc0\xaf",
                b'"dtype"', b'"shape"', b'"data_offsets"', b'"__metadata__"', b"[[", b"]]"]


def mutated_headers(seed, n):
    """n (header, file size) pairs: valid headers (every dtype, 0-3 dimensions, metadata,
    non-ASCII names) with up to three random deletions, token insertions, byte changes or
    truncations each."""
    rng = random.Random(seed)
    for _ in range(n):
        h, off = {}, 0
        if rng.random() < 0.5:
            h["__metadata__"] = {"format": "pt", "k": "v\u00e9\"x\\n", "l": [1, 2.5, None, True]}
        for i in range(rng.randint(0, 5)):
            dt = rng.choice(sorted(ST_ES))
            shape = [rng.randint(0, 5) for _ in range(rng.randint(0, 3))]
            nb = ST_ES[dt] * int(np.prod(shape, dtype=np.int64))
            h[f"layer.{i}.w\u00e9"] = {"dtype": dt, "shape": shape, "data_offsets": [off, off + nb]}
            off += nb
        b = bytearray(json.dumps(h, ensure_ascii=rng.random() < 0.5).encode())
        for _ in range(rng.randint(0, 3)):
            r = rng.random()
            if r < 0.3 and b:
                i = rng.randrange(len(b))
                del b[i:i + rng.randint(1, 6)]
            elif r < 0.7:
                i = rng.randrange(len(b) + 1)
                b[i:i] = rng.choice(_FUZZ_TOKENS)
            elif r < 0.9 and b:
                b[rng.randrange(len(b))] = rng.randrange(256)
            else:
                b = b[:rng.randrange(len(b) + 1)]
        yield bytes(b), 8 + len(b) + off + rng.choice([0, 0, 0, 1, 1 << 40])


@pytest.mark.parametrize("seed", [1, 2])
def test_mutated_headers_parse_as_python_json_reads_them(seed):
    accepted = rejected = 0
    for raw, file_bytes in mutated_headers(seed, 3000):
        want = json_reading(raw, file_bytes)
        try:
            got = [tuple(t) for t in cfa.Safetensors.parse(raw, file_bytes).tensors]
        except cfa.CfaError as e:
            assert e.name == "CFA_ERR_INVAL"
            got = None
        assert got == want, raw
        accepted += got is not None
        rejected += got is None
    assert accepted > 100 and rejected > 100


def test_header_parser_under_address_sanitizer(tmp_path):
    exe = tmp_path / "st_header_fuzz"
    csrc = os.path.join(ROOT, "paper_2607_18957_gb300", "csrc")
    r = subprocess.run(["gcc", "-g", "-O1", "-std=c11", "-fsanitize=address,undefined",
                        "-fno-sanitize-recover=all", "-I", csrc, "-I", os.path.join(ROOT, "include"),
                        os.path.join(ROOT, "tests", "st_header_fuzz.c"),
                        os.path.join(csrc, "cfa_files.c"), "-o", str(exe), "-lpthread"],
                       capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("no AddressSanitizer runtime for gcc here: " + r.stderr[-200:])
    inputs = tmp_path / "headers.bin"
    with open(inputs, "wb") as f:
        for raw, file_bytes in mutated_headers(7, 20000):
            f.write(struct.pack("<IQ", len(raw), file_bytes) + raw)
        for raw in BAD_HEADERS:
            f.write(struct.pack("<IQ", len(raw), 8 + len(raw) + 16) + raw)
    r = subprocess.run([str(exe), str(inputs)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr[-2000:]


def test_malformed_files_are_rejected(tmp_path):
    p = tmp_path / "x.safetensors"
    with pytest.raises(cfa.CfaError) as e:
        cfa.Safetensors.open(tmp_path / "missing.safetensors")
    assert e.value.name == "CFA_ERR_SOURCE"
    p.write_bytes(b"\x05\x00")  # shorter than the length word
    with pytest.raises(cfa.CfaError) as e:
        cfa.Safetensors.open(p)
    assert e.value.name == "CFA_ERR_SOURCE"
    p.write_bytes(struct.pack("<Q", 100) + b"{}")  # length past the end of the file
    with pytest.raises(cfa.CfaError) as e:
        cfa.Safetensors.open(p)
    assert e.value.name == "CFA_ERR_INVAL"
    # a tensor running past the end of a truncated file
    hdr = header_bytes([("w", "f32", (4,), 0, 16)])
    write_file(p, hdr, b"\0" * 12)
    with pytest.raises(cfa.CfaError) as e:
        cfa.Safetensors.open(p)
    assert e.value.name == "CFA_ERR_INVAL" and "data_offsets" in str(e.value)
    write_file(p, hdr, b"\0" * 16)
    assert cfa.Safetensors.open(p).tensors[0] == ("w", "f32", (4,), 0, 16)


FillFn = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p,
                          ctypes.c_uint64)


def _direct_supported(path):
    try:
        fd = os.open(path, os.O_RDONLY | os.O_DIRECT)
    except OSError:
        return False
    os.close(fd)
    return True


@pytest.mark.parametrize("mode,data_align", [("pread", 8), ("direct", 8), ("direct", 4096),
                                             ("mmap", 8), ("mmap", 4096)])
def test_file_source_fill_reads_the_data_section(tmp_path, mode, data_align):
    """Random ranges, destinations at every offset class within a 4 KiB block (for direct
    reads: bounced, and block-congruent with the file so the middle blocks land in place),
    ranges ending at the end of the file, and nothing written outside the range."""
    m = configs()[0]
    p = tmp_path / "model.safetensors"
    off = write_safetensors(m, p, data_align=data_align)
    assert off % data_align == 0
    direct = mode == "direct"
    if direct and not _direct_supported(p):
        pytest.skip("the file system has no O_DIRECT")
    blob = m.blob_range(0, m.blob_bytes)
    rng = np.random.default_rng(5)
    B = 4096
    with cfa.Source.file(p, off, direct=direct, mapped=mode == "mmap") as src:
        c = src.to_c()
        assert c.kind == _lib.SRC_CALLBACK and c.fill and c.user
        fill = FillFn(c.fill)
        cases = []
        for k in range(60):
            a = int(rng.integers(0, m.blob_bytes))
            n = int(rng.integers(0, min(9 << 20, m.blob_bytes - a) + 1))
            cases.append((a, n))
        cases += [(m.blob_bytes - 5, 5), (m.blob_bytes - (3 << 20) - 7, (3 << 20) + 7),
                  (0, m.blob_bytes), (B - off % B, 5 * B), (0, 1)]
        for k, (a, n) in enumerate(cases):
            raw = np.full(n + 3 * B, 0xAB, dtype=np.uint8)
            base = raw.ctypes.data
            if k % 2:  # block-congruent with the file offset
                lead = ((off + a) - (base + 64)) % B + 64
            else:
                lead = 64 + 7 * k % B
            assert fill(c.user, a, base + lead, n) == 0, (a, n)
            assert np.array_equal(raw[lead:lead + n], blob[a:a + n]), (a, n, lead)
            assert (raw[:lead] == 0xAB).all() and (raw[lead + n:] == 0xAB).all()
        buf = np.zeros(16, dtype=np.uint8)
        assert fill(c.user, m.blob_bytes - 8, buf.ctypes.data, 16) != 0  # past the end
        assert fill(c.user, (1 << 64) - 4, buf.ctypes.data, 8) != 0    # offset wraps
    with pytest.raises(cfa.CfaError):
        src.to_c()  # closed
    with pytest.raises(cfa.CfaError) as e:
        cfa.Source.file(tmp_path / "missing")
    assert e.value.name == "CFA_ERR_SOURCE"


def test_host_only_plan_from_a_file_matches_the_manifest_plan(tmp_path):
    """The plan built from the file's entries (pieces, work split, staged bytes) is the plan
    built from the manifest's."""
    m = configs()[1]
    p = tmp_path / "model.safetensors"
    write_safetensors(m, p)
    st = cfa.Safetensors.open(p)
    dsts = [(0x10000 * (j + 1) << 12, str(m.d_dtype[j]), tuple(m.d_shape[j, :m.d_ndim[j]]))
            for j in range(m.n_dsts)]
    kw = dict(chunk_bytes=64 << 10, host_only=True)
    with cfa.Plan(st.entries(targets_for(m)), dsts, st.data_bytes, **kw) as a, \
            cfa.Plan(entries_for(m), dsts, m.blob_bytes, **kw) as b:
        assert np.array_equal(a.pieces(), b.pieces())
        sa, sb = a.stats(), b.stats()
        for f in ("n_pieces", "n_slabs", "n_tiny", "n_strided", "staged_bytes", "bytes_written"):
            assert sa[f] == sb[f], f


def test_file_abi_is_exported():
    lib = _lib.load()
    for name in ("cfa_safetensors_open", "cfa_safetensors_parse", "cfa_safetensors_info",
                 "cfa_safetensors_tensor", "cfa_safetensors_close", "cfa_file_source_open",
                 "cfa_file_source_close"):
        assert hasattr(lib, name)
    assert lib.cfa_abi_sizeof(b"cfa_st_tensor") == ctypes.sizeof(_lib.StTensor) == 96
    assert os.path.basename(cfa.library_path()) == "libcfa.so"


def test_file_source_flags_are_checked(tmp_path):
    p = tmp_path / "f.bin"
    p.write_bytes(b"\0" * 4096)
    with pytest.raises(cfa.CfaError) as e:
        cfa.Source.file(p, 0, direct=True, mapped=True)
    assert e.value.name == "CFA_ERR_INVAL"
    lib = _lib.load()
    c = _lib.Source()
    assert lib.cfa_file_source_open(str(p).encode(), 0, 0x80, ctypes.byref(c)) == -1
    empty = tmp_path / "empty.bin"
    empty.write_bytes(b"")
    with cfa.Source.file(empty, 0, mapped=True) as src:  # nothing to map, nothing to read
        fill = FillFn(src.to_c().fill)
        assert fill(src.to_c().user, 0, None, 0) == 0
        assert fill(src.to_c().user, 0, None, 1) != 0


@pytest.mark.parametrize("data_align", [8, 4096])
def test_in_place_file_source_maps_the_data_section(tmp_path, data_align):
    """CFA_FILE_MMAP_IN_PLACE gives a HOST_DIRECT source whose base is the data section inside
    a read-only mapping of the whole file and whose size is the rest of the file; closing it
    unmaps the file."""
    m = configs()[0]
    p = tmp_path / "model.safetensors"
    off = write_safetensors(m, p, data_align=data_align)
    size = os.path.getsize(p)
    with cfa.Source.file(p, off, in_place=True) as src:
        c = src.to_c()
        assert c.kind == _lib.SRC_HOST_DIRECT and c.base and c.user and c.fill
        assert c.base % 8 == 0 and c.size_bytes == size - off == m.blob_bytes
        assert src.base == c.base and src.size == c.size_bytes
        got = np.frombuffer(ctypes.string_at(c.base, c.size_bytes), dtype=np.uint8)
        assert np.array_equal(got, m.blob_range(0, m.blob_bytes))
    with pytest.raises(cfa.CfaError):
        src.to_c()  # closed


def test_in_place_file_source_rules(tmp_path):
    p = tmp_path / "f.bin"
    p.write_bytes(bytes(range(256)) * 16)
    for kw in (dict(direct=True), dict(mapped=True)):
        with pytest.raises(cfa.CfaError) as e:
            cfa.Source.file(p, 0, in_place=True, **kw)
        assert e.value.name == "CFA_ERR_INVAL"
    with pytest.raises(cfa.CfaError) as e:
        cfa.Source.file(p, 12, in_place=True)  # elements would not be aligned
    assert e.value.name == "CFA_ERR_ALIGN" and "multiple of 8" in str(e.value)
    with pytest.raises(cfa.CfaError) as e:
        cfa.Source.file(p, 4096 + 8, in_place=True)
    assert e.value.name == "CFA_ERR_SOURCE" and "past the end" in str(e.value)
    with cfa.Source.file(p, 4096, in_place=True) as src:  # an empty data section at the end
        assert src.to_c().size_bytes == 0
    with cfa.Source.file(p, 8, in_place=True) as src:
        c = src.to_c()
        assert c.size_bytes == 4088 and ctypes.string_at(c.base, 4) == bytes([8, 9, 10, 11])
    empty = tmp_path / "empty.bin"
    empty.write_bytes(b"")
    with cfa.Source.file(empty, 0, in_place=True) as src:  # nothing to map
        assert not src.to_c().base and src.to_c().size_bytes == 0
    # a HOST_DIRECT source the library did not open is not closed by cfa_file_source_close
    lib = _lib.load()
    c = _lib.Source()
    c.kind, c.user = _lib.SRC_HOST_DIRECT, 1234
    assert lib.cfa_file_source_close(ctypes.byref(c)) == -1


@pytest.mark.parametrize("sanitizer", ["thread", "address,undefined"])
def test_concurrent_fills_under_sanitizers(tmp_path, sanitizer):
    """tests/file_fill_stress.c: eight threads fill random ranges of a 24 MiB file at random
    destination alignments in every read mode, at a block-aligned and an unaligned data offset,
    with requests past the end and wrapping around 64 bits refused; built with ThreadSanitizer
    and with AddressSanitizer + UBSan."""
    exe = tmp_path / "file_fill_stress"
    csrc = os.path.join(ROOT, "paper_2607_18957_gb300", "csrc")
    r = subprocess.run(["gcc", "-g", "-O1", "-std=c11", "-pthread", f"-fsanitize={sanitizer}",
                        "-fno-sanitize-recover=all", "-I", csrc, "-I", os.path.join(ROOT, "include"),
                        os.path.join(ROOT, "tests", "file_fill_stress.c"),
                        os.path.join(csrc, "cfa_files.c"), "-o", str(exe)],
                       capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip(f"no {sanitizer} sanitizer runtime for gcc here: " + r.stderr[-200:])
    path = tmp_path / "file.bin"
    path.write_bytes(np.random.default_rng(5).integers(0, 256, (24 << 20) + 777, np.uint8)
                     .tobytes())
    for data_offset in (4096, 4104):
        r = subprocess.run([str(exe), str(path), str(data_offset)], capture_output=True,
                           text=True, timeout=600,
                           env={**os.environ, "TSAN_OPTIONS": "halt_on_error=1 exitcode=66"})
        if r.returncode != 0 and sanitizer_could_not_start(r.stderr):
            pytest.skip(f"the {sanitizer} sanitizer runtime cannot start here: " + r.stderr[:200])
        assert r.returncode == 0, (data_offset, r.stdout + r.stderr[-3000:])
