"""The loader library on the host (no GPU): it loads, exports every function cfa.h declares,
agrees with the binding's struct layouts, and its plan builder (validation, tensor x chunk
pieces, fused placement) agrees with the oracle.  Plans here are CFA_OPT_HOST_ONLY: no CUDA
call is made."""
import os
import re

import numpy as np
import pytest
import torch

import oracle
import paper_2607_18957_gb300 as cfa
from paper_2607_18957_gb300 import _lib
from paper_2607_18957_gb300 import build as cfa_build
from workloads import DTYPE_SIZE, dense_config, moe_config, tiny_config
from workloads.harness import entries_for

import _pins
from _golden import manifest_case

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_library():
    cfa_build.build()
    return _lib.load()


def header_functions():
    text = open(os.path.join(ROOT, "include", "cfa.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cfa_\w+)\s*\(", text)))


def test_exports_every_declared_function(built_library):
    names = header_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(built_library, n), n
    assert set(names) == set(_lib.SIGNATURES), "binding and header disagree"


def test_struct_layouts_match():
    lib = _lib.load()  # raises on a mismatch
    assert lib.cfa_abi_sizeof(b"cfa_tensor_entry") == 112
    assert lib.cfa_abi_sizeof(b"nonsense") == 0
    assert lib.cfa_status_name(-2) == b"CFA_ERR_OVERLAP"
    # every status code of cfa.h has its name in the library and in the binding
    import re
    with open(os.path.join(ROOT, "include", "cfa.h")) as f:
        codes = dict((int(v), k) for k, v in
                     re.findall(r"#define (CFA_OK|CFA_ERR_\w+)\s+\(?(-?\d+)\)?", f.read()))
    assert codes[-14] == "CFA_ERR_SUSPECT" and codes[-15] == "CFA_ERR_GATHER"
    for v, name in codes.items():
        assert lib.cfa_status_name(v) == name.encode(), name
        assert _lib.STATUS[v] == name


FAKE_BASE = 0x7F00_0000_0000


def fake_dsts(m, misalign=0, guard=256):
    out, pos = [], guard
    for j in range(m.n_dsts):
        es = DTYPE_SIZE[str(m.d_dtype[j])]
        pos = (pos + 255) // 256 * 256 + (misalign // es) * es
        out.append((FAKE_BASE + pos, str(m.d_dtype[j]), m.d_shape_tuple(j)))
        pos += m.d_nbytes(j) + guard
    return out


def host_plan(m, chunk_bytes=512 << 20, misalign=0, **kw):
    return cfa.Plan(entries_for(m, with_names=True), fake_dsts(m, misalign), m.blob_bytes,
                    chunk_bytes=chunk_bytes, host_only=True, **kw)


def execute_pieces_on_cpu(m, pieces, blob):
    """Applies the plan's pieces with numpy/torch: no offsets are recomputed here."""
    out = {j: np.zeros(m.d_nbytes(j), np.uint8) for j in range(m.n_dsts)}
    for pc in pieces:
        i = int(pc["entry"])
        es_s = DTYPE_SIZE[str(m.e_dtype[i])]
        rows = int(pc["rows"])
        cols = int(pc["n_elems"]) // rows
        step = int(pc["src_row_stride"]) * es_s if rows > 1 else cols * es_s
        o = int(pc["dst_offset"])
        for k in range(rows):
            a = int(pc["src_offset"]) + k * step
            src = blob[a:a + cols * es_s]
            if pc["conv"]:
                s_dt, d_dt = str(m.e_dtype[i]), str(m.d_dtype[int(pc["dst_index"])])
                src = _pins.torch_convert_bits(s_dt, d_dt,
                                               src.view(_pins._BITS[s_dt][0])).view(np.uint8)
            out[int(pc["dst_index"])][o:o + src.size] = src
            o += src.size
    return out


def mini_configs():
    return [
        tiny_config(seed=51, n=40, lo=2, hi=20000, align=2, jitter=7),
        dense_config("d", 52, 2, 64, 4, 2, 16, 96, 100, align=2, jitter=3),
        dense_config("d32", 53, 2, 64, 4, 2, 16, 96, 100, src_dtype="f32", align=4, jitter=2),
        moe_config("m", 54, 2, 32, 4, 2, 8, 48, 3, 50, n_extra=30, align=2, jitter=3),
        # tensor-parallel ranks: column slices read with a source row stride
        dense_config("d_tp2r1", 55, 2, 64, 4, 2, 16, 96, 100, align=2, jitter=3, tp=2, rank=1),
        dense_config("d32_tp4r2", 56, 2, 64, 4, 2, 16, 96, 100, src_dtype="f32", align=4,
                     jitter=2, tp=4, rank=2),
        moe_config("m_tp2r0", 57, 2, 32, 4, 2, 8, 48, 3, 52, n_extra=30, align=2, jitter=3,
                   tp=2, rank=0),
        # dtype conversions
        dense_config("f32_f16", 58, 2, 64, 4, 2, 16, 96, 100, src_dtype="f32", dst_dtype="f16",
                     align=4, jitter=2),
        dense_config("f16_bf16", 59, 2, 64, 4, 2, 16, 96, 100, src_dtype="f16",
                     norm_dtype="f32", align=2, jitter=3, tp=2, rank=1),
    ]


@pytest.mark.parametrize("chunk", [256, 4096 + 256, 1 << 20, 512 << 20])
def test_plan_pieces_reproduce_the_oracle(chunk):
    for m in mini_configs():
        blob = m.blob_range(0, m.blob_bytes)
        with host_plan(m, chunk_bytes=chunk) as p:
            pcs = p.pieces()
            info = p.info()
        assert info["n_chunks"] == -(-m.blob_bytes // chunk)
        # every piece lies inside one chunk
        es = np.array([DTYPE_SIZE[str(m.e_dtype[int(i)])] for i in pcs["entry"]])
        start = pcs["src_offset"].astype(np.int64)
        rows = pcs["rows"].astype(np.int64)
        cols = pcs["n_elems"].astype(np.int64) // rows
        step = np.where(rows > 1, pcs["src_row_stride"].astype(np.int64), cols)
        end = start + ((rows - 1) * step + cols) * es
        assert (start // chunk == pcs["chunk"]).all()
        assert ((end - 1) // chunk == pcs["chunk"]).all()
        # chunk-major order
        assert (np.diff(pcs["chunk"].astype(np.int64)) >= 0).all()
        got = execute_pieces_on_cpu(m, pcs, blob)
        ref = oracle.unpack(m, blob)
        assert ref.status == 0
        for j in range(m.n_dsts):
            assert np.array_equal(got[j], ref.dst[j]), (m.name, chunk, m.d_name[j])


def test_golden_manifests_through_the_plan():
    for name in ("fused_tiny.txt", "moe_tiny.txt"):
        m, blob, exp_dst, _ = manifest_case(name)
        with host_plan(m, chunk_bytes=256) as p:
            got = execute_pieces_on_cpu(m, p.pieces(), blob)
        for j, want in exp_dst.items():
            assert np.array_equal(got[j], want), (name, j)


_ORACLE_TO_CFA = {oracle.ORC_E_INVAL: "CFA_ERR_INVAL", oracle.ORC_E_DTYPE: "CFA_ERR_DTYPE",
                  oracle.ORC_E_ALIGN: "CFA_ERR_ALIGN", oracle.ORC_E_OOB: "CFA_ERR_OOB",
                  oracle.ORC_E_SHAPE: "CFA_ERR_SHAPE", oracle.ORC_E_OVERLAP: "CFA_ERR_OVERLAP",
                  oracle.ORC_E_COVERAGE: "CFA_ERR_COVERAGE"}


def _plan_status(m, **kw):
    try:
        host_plan(m, chunk_bytes=256, **kw).close()
        return "CFA_OK"
    except cfa.CfaError as e:
        return e.name


def test_validation_agrees_with_the_oracle():
    m, blob, _, _ = manifest_case("fused_tiny.txt")
    cases = [
        (dict(i=0, offset=32), None), (dict(i=0, offset=5), None), (dict(i=0, row=3), None),
        (dict(i=0, dtype="f16"), None), (dict(i=3, cast=False), None),
        (dict(i=0, shape=(1, 4)), None), (dict(i=5, row=2), None),
        (dict(i=1, row=1), "cover"), (dict(i=4, shape=(0,)), "cover"),
    ]
    for change, how in cases:
        i = change.pop("i")
        mv = _pins._variant(m, i, **change)
        r = oracle.unpack(mv, blob, cover=(how == "cover"))
        code = oracle.check_cover(r)[0] if how == "cover" else r.status
        assert code != 0
        assert _plan_status(mv) == _ORACLE_TO_CFA[code], (change, oracle.STATUS_NAME[code])
    # the valid manifest passes both
    assert oracle.unpack(m, blob).status == 0 and _plan_status(m) == "CFA_OK"
    # non-strict mode accepts the gap
    gap = _pins._variant(m, 4, shape=(0,))
    assert _plan_status(gap, strict=False) == "CFA_OK"


def test_destinations_overlapping_in_memory_are_rejected():
    m, _, _, _ = manifest_case("fused_tiny.txt")
    d = fake_dsts(m)
    d[1] = (d[0][0] + 8, d[1][1], d[1][2])  # norm starts inside qkv
    with pytest.raises(cfa.CfaError) as e:
        cfa.Plan(entries_for(m), d, m.blob_bytes, host_only=True)
    assert e.value.name == "CFA_ERR_OVERLAP"


def test_slab_size_follows_the_load_size():
    """slab_bytes 0 (the default) gives about 4096 block-level items per load, a power of two in
    [32 KiB, 256 KiB]: the same work items as that size given explicitly."""
    def items(p):
        st = p.stats()
        return st["n_slabs"], st["n_bulk"], st["n_tiny"]
    import workloads
    cases = [(workloads.named_config("tiny_1000"), 32 << 10),          # 131 MB of destinations
             (dense_config("mid", 3, layers=2, hidden=2048, n_q=16, n_kv=4, head_dim=128,
                           inter=8192, vocab=32000), 64 << 10),         # 505 MB
             (dense_config("big", 3, layers=4, hidden=2048, n_q=16, n_kv=4, head_dim=128,
                           inter=8192, vocab=32000), 128 << 10),        # 748 MB
             (workloads.named_config("llama3_8b_bf16"), 256 << 10)]    # 16 GB
    for m, want in cases:
        with host_plan(m) as auto, host_plan(m, slab_bytes=want) as fixed, \
                host_plan(m, slab_bytes=want // 2) as half:
            assert items(auto) == items(fixed), (m.name, want)
            assert items(auto) != items(half), (m.name, want)


def test_bad_options_and_misaligned_destination():
    m, _, _, _ = manifest_case("fused_tiny.txt")
    with pytest.raises(cfa.CfaError) as e:
        host_plan(m, chunk_bytes=100)
    assert e.value.name == "CFA_ERR_INVAL"
    with pytest.raises(cfa.CfaError) as e:
        host_plan(m, slab_bytes=1000)
    assert e.value.name == "CFA_ERR_INVAL"
    with pytest.raises(cfa.CfaError) as e:
        host_plan(m, pull_percent=101)
    assert e.value.name == "CFA_ERR_INVAL"
    for pct in (0, 50, 100):
        host_plan(m, pull_percent=pct).close()
    d = fake_dsts(m)
    d[0] = (d[0][0] + 1, d[0][1], d[0][2])
    with pytest.raises(cfa.CfaError) as e:
        cfa.Plan(entries_for(m), d, m.blob_bytes, host_only=True)
    assert e.value.name == "CFA_ERR_ALIGN"


def test_conversion_flags():
    """CFA_ENTRY_CAST_BF16 accepts only fp32 -> bf16; CFA_ENTRY_CONVERT any listed pair."""
    m = dense_config("conv", 60, 1, 64, 4, 2, 16, 96, 100, src_dtype="f32", dst_dtype="f16",
                     align=4)
    ents = entries_for(m)
    ok = cfa.Plan(ents, fake_dsts(m), m.blob_bytes, host_only=True)
    ok.close()
    ents.arr["flags"] = (ents.arr["flags"] & ~np.uint32(_lib.ENTRY_CONVERT)) | _lib.ENTRY_CAST_BF16
    with pytest.raises(cfa.CfaError) as e:
        cfa.Plan(ents, fake_dsts(m), m.blob_bytes, host_only=True)
    assert e.value.name == "CFA_ERR_DTYPE"
    # an unsupported pair (bf16 -> f16) is refused by both sides
    mb = dense_config("conv2", 61, 1, 64, 4, 2, 16, 96, 100, src_dtype="bf16", dst_dtype="f16")
    assert _plan_status(mb) == "CFA_ERR_DTYPE"
    assert oracle.unpack(mb, mb.blob_range(0, mb.blob_bytes)).status == oracle.ORC_E_DTYPE


def test_strided_entries_are_validated_like_the_oracle():
    m, blob, _, _ = manifest_case("tp_shard_tiny.txt")
    assert _plan_status(m) == "CFA_OK" and oracle.unpack(m, blob).status == 0
    # a stride shorter than the row, and a column slice reading past the blob
    for change, name in ((dict(stride=1), "CFA_ERR_INVAL"), (dict(offset=40), "CFA_ERR_OOB")):
        mv = _pins._variant(m, 2, **change)
        assert _plan_status(mv) == name
        assert _ORACLE_TO_CFA[oracle.unpack(mv, blob).status] == name


def test_empty_manifest_and_zero_sized_entries():
    from workloads import Manifest
    with cfa.Plan(cfa.make_entries([], [], [], []), [], 0, host_only=True) as p:
        assert p.info() == {"n_layers": 0, "n_pieces": 0, "n_chunks": 0}
    ents = [{"name": "a", "dtype": "bf16", "shape": (0, 4), "offset": 0, "dst": 0, "row": 0},
            {"name": "b", "dtype": "bf16", "shape": (2,), "offset": 0, "dst": 1, "row": 0,
             "layer": 2}]
    dsts = [{"name": "A", "dtype": "bf16", "shape": (0, 4)},
            {"name": "B", "dtype": "bf16", "shape": (2,)}]
    m = Manifest("zero", ents, dsts, 4, "bits", 0)
    with host_plan(m) as p:
        assert p.info()["n_pieces"] == 1 and p.info()["n_layers"] == 3


def test_host_only_plan_refuses_to_load():
    m, _, _, _ = manifest_case("fused_tiny.txt")
    with host_plan(m) as p:
        with pytest.raises(cfa.CfaError) as e:
            p.load_async(cfa.Source.host(1), stream=0)
        assert e.value.name == "CFA_ERR_INVAL"


def test_staged_bytes_cover_exactly_what_pieces_read():
    """Staged loads copy only the byte ranges pieces read: the whole checkpoint for a 1:1 model,
    about one eighth of it for a tensor-parallel rank of eight."""
    import workloads
    m = workloads.named_config("llama3_8b_bf16")
    with host_plan(m, chunk_bytes=m.chunk_bytes) as p:
        st = p.stats()
    assert m.total_src_bytes() <= st["staged_bytes"] <= m.blob_bytes
    m = workloads.named_config("llama3_70b_bf16_tp8r3")
    with host_plan(m, chunk_bytes=m.chunk_bytes) as p:
        st = p.stats()
    assert st["bytes_read"] <= st["staged_bytes"] < 0.2 * m.blob_bytes


def test_full_size_manifests_plan_on_the_host():
    import workloads
    for name in ("llama3_8b_bf16", "llama3_70b_bf16"):
        m = workloads.named_config(name)
        with host_plan(m, chunk_bytes=m.chunk_bytes) as p:
            st = p.stats()
            assert st["bytes_written"] == m.total_dst_bytes()
            assert st["n_chunks"] == -(-m.blob_bytes // m.chunk_bytes)
            assert st["n_layers"] == m.n_groups()
            pcs = p.pieces()
            assert int(pcs["n_elems"].sum()) == sum(m.e_numel(i) for i in range(m.n_entries))


def test_default_options_take_the_bulk_path():
    """cfa_plan_opts_default turns the TMA bulk path on; the binding's default follows it."""
    import ctypes
    lib = _lib.load()
    o = _lib.PlanOpts()
    lib.cfa_plan_opts_default(ctypes.byref(o))
    assert o.flags & _lib.OPT_BULK and o.flags & _lib.OPT_STRICT_COVERAGE
    import inspect
    assert inspect.signature(cfa.Plan).parameters["bulk"].default is True
    # aligned cast-free slabs become bulk items by default, and never with bulk=False
    m = dense_config("d_aligned", 52, 2, 64, 4, 2, 16, 96, 100, align=256)
    with host_plan(m, chunk_bytes=1 << 20, tiny_bytes=0) as p:
        st = p.stats()
        assert st["n_bulk"] > 0 and st["n_slabs"] == 0
    with host_plan(m, chunk_bytes=1 << 20, tiny_bytes=0, bulk=False) as p:
        st = p.stats()
        assert st["n_bulk"] == 0 and st["n_slabs"] > 0


def test_default_staging_options_match_the_header():
    """The documented staging defaults: 512 MiB chunks, 2 pinned and 3 device slots, the whole
    of each range pulled by the SMs, automatic slab size, 8 KiB tiny threshold; the binding's
    Plan() takes the same device slot count and leaves pull_percent to the library."""
    import ctypes
    import inspect
    import re
    lib = _lib.load()
    o = _lib.PlanOpts()
    lib.cfa_plan_opts_default(ctypes.byref(o))
    assert (o.chunk_bytes, o.host_slots, o.dev_slots) == (512 << 20, 2, 3)
    assert (o.pull_percent, o.slab_bytes, o.tiny_bytes, o.seg_world) == (100, 0, 8192, 1)
    params = inspect.signature(cfa.Plan).parameters
    assert params["dev_slots"].default == o.dev_slots
    assert params["pull_percent"].default is None
    hdr = open(os.path.join(os.path.dirname(__file__), "..", "include", "cfa.h")).read()
    assert re.search(r"dev_slots;.*?default 3", hdr, re.S)
    assert re.search(r"pull_percent;.*?Default 100", hdr, re.S)


def test_log_lines_on_request():
    """CFA_LOG=1 prints one line per plan and per error on stderr (a child process, so the
    variable is read fresh)."""
    import subprocess
    import sys
    code = ("import paper_2607_18957_gb300 as cfa\n"
            "e = cfa.make_entries(dtype=['bf16'], shape=[(1024,)], offset=[0], dst=[0])\n"
            "cfa.Plan(e, [(0x100000, 'bf16', (1024,))], 2048, host_only=True).close()\n"
            "try:\n"
            "    cfa.Plan(e, [(0x100000, 'bf16', (1000,))], 2048, host_only=True)\n"
            "except cfa.CfaError:\n"
            "    pass\n")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, CFA_LOG="1", PYTHONPATH=root)
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=120)
    assert r.returncode == 0, r.stderr
    lines = [x for x in r.stderr.splitlines() if x.startswith("cfa: ")]
    assert any(x.startswith("cfa: plan: 1 entries") for x in lines), r.stderr
    assert any("rows fall outside the destination" in x for x in lines), r.stderr
    env["CFA_LOG"] = "0"
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=120)
    assert "cfa: " not in r.stderr


def _noalloc_status(m, ents=None, blob_ptr=FAKE_BASE, blob_bytes=None):
    """Calls cfa_unpack_noalloc with fake device pointers; only its validation may run."""
    import ctypes
    lib = _lib.load()
    e = ents if ents is not None else entries_for(m)
    d = cfa.make_dsts(fake_dsts(m))
    err = ctypes.create_string_buffer(512)
    st = lib.cfa_unpack_noalloc(e.arr.ctypes.data, len(e.arr), d.ctypes.data, len(d), blob_ptr,
                                m.blob_bytes if blob_bytes is None else blob_bytes, None, None,
                                None, err, len(err))
    return _lib.STATUS.get(st, str(st)), err.value.decode()


@pytest.mark.skipif(torch.cuda.is_available(),
                    reason="fake device pointers: run only where no kernel can be launched")
def test_noalloc_validation_rejects_what_the_planned_path_rejects():
    # every malformed entry is refused before any CUDA call, with the planned path's status
    m, blob, _, _ = manifest_case("fused_tiny.txt")
    cases = [dict(i=0, offset=32), dict(i=0, offset=5), dict(i=0, row=3), dict(i=0, dtype="f16"),
             dict(i=3, cast=False), dict(i=0, shape=(1, 4)), dict(i=5, row=2),
             # sizes that wrap around 64 bits must not slip through the bounds checks
             dict(i=0, shape=(1 << 40, 1 << 40, 2)), dict(i=5, row=(1 << 62) + 1),
             dict(i=5, shape=(1 << 62,))]
    for change in cases:
        i = change.pop("i")
        mv = _pins._variant(m, i, **change)
        planned = _plan_status(mv)
        assert planned != "CFA_OK", change
        st, msg = _noalloc_status(mv)
        assert st == planned, (change, st, msg)
        assert msg.startswith("cfa_unpack_noalloc:"), msg


@pytest.mark.skipif(torch.cuda.is_available(),
                    reason="fake device pointers: run only where no kernel can be launched")
def test_noalloc_argument_checks():
    m, _, _, _ = manifest_case("fused_tiny.txt")
    assert _noalloc_status(m, blob_ptr=FAKE_BASE + 16)[0] == "CFA_ERR_ALIGN"  # blob not 256-aligned
    assert _noalloc_status(m, blob_ptr=0)[0] == "CFA_ERR_INVAL"               # NULL blob
    # column slices need the plan's strided pieces
    mv = _pins._variant(m, 0, stride=3)
    assert _plan_status(mv) == "CFA_OK"
    assert _noalloc_status(mv)[0] == "CFA_ERR_INVAL"
    # more work items than the fixed scratch holds: one per tensor below 8 KiB
    from workloads import Manifest
    n = 16385
    big = Manifest("too_many", [{"name": f"t{k}", "dtype": "bf16", "shape": (4,), "offset": 8 * k,
                                 "dst": k} for k in range(n)],
                   [{"name": f"d{k}", "dtype": "bf16", "shape": (4,)} for k in range(n)],
                   8 * n, "bits", 1)
    st, msg = _noalloc_status(big)
    assert st == "CFA_ERR_INVAL" and "16384" in msg


def test_plain_c_program_through_the_header(tmp_path):
    """tests/c_consumer.c: strict C11 against include/cfa.h, linked to libcfa.so; struct sizes
    agree with the library's, a host-only plan gives hand-computed pieces, errors carry their
    messages, and a safetensors header parses.  Makes no CUDA call."""
    import subprocess
    exe = tmp_path / "c_consumer"
    pkg = os.path.dirname(_lib.LIB_PATH)
    subprocess.run(["gcc", "-std=c11", "-pedantic", "-Wall", "-Wextra", "-Werror",
                    "-I", os.path.join(ROOT, "include"), os.path.join(ROOT, "tests", "c_consumer.c"),
                    "-L", pkg, "-lcfa", "-Wl,-rpath," + pkg, "-o", str(exe)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr
