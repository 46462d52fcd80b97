"""GPU parity for checkpoint files: a safetensors file written from a seeded manifest is loaded
through its header (Safetensors.entries) and compared byte for byte, checksum for checksum,
with the oracle on the manifest.  Sources: the pread file source (data section staged through
the pinned ring, buffered or O_DIRECT, or the mapped file read in place by the kernels), and
the whole file read into page-locked or pageable memory with the blob being the whole file.  Whole tensors, row and column shards, conversions; a file that shrinks
under a load is reported as a source error and the plan recovers."""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_18957_gb300 as cfa
from workloads import dense_config, moe_config
from workloads.harness import DeviceDsts
from workloads.stfile import targets_for, write_safetensors

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def cfg(name):
    if name == "dense":
        return dense_config("file_dense", 91, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                            inter=1536, vocab=1000, align=2, jitter=5)
    if name == "f32_tp":
        return dense_config("file_f32_tp4r2", 92, layers=2, hidden=512, n_q=8, n_kv=2,
                            head_dim=64, inter=1536, vocab=1000, src_dtype="f32", align=4,
                            jitter=3, tp=4, rank=2)
    if name == "moe_tp":
        return moe_config("file_moe_tp2r1", 93, layers=2, hidden=256, n_q=4, n_kv=2,
                          head_dim=64, inter=512, n_experts=4, vocab=500, n_extra=500, align=2,
                          jitter=3, tp=2, rank=1)
    if name == "f32_f16":
        return dense_config("file_f32_f16", 94, layers=2, hidden=512, n_q=8, n_kv=2,
                            head_dim=64, inter=1536, vocab=1000, src_dtype="f32",
                            dst_dtype="f16", align=4, jitter=3)
    raise ValueError(name)


_CACHE = {}


def prepared(name, tmp_path_factory):
    """(manifest, file path, data offset, oracle result) for config `name`."""
    if name not in _CACHE:
        m = cfg(name)
        path = tmp_path_factory.mktemp("ckpt") / f"{m.name}.safetensors"
        off = write_safetensors(m, path)
        r = oracle.unpack(m, m.blob_range(0, m.blob_bytes))
        assert r.status == 0, r.status_name
        _CACHE[name] = (m, str(path), off, r)
    return _CACHE[name]


def aligned_pageable(nbytes, align=256):
    buf = np.empty(nbytes + align, dtype=np.uint8)
    off = (-buf.ctypes.data) % align
    return buf[off:off + nbytes]


def compare(m, d, ck, ref, what):
    for j in range(m.n_dsts):
        got = d.host_bytes(j)
        if not np.array_equal(got, ref.dst[j]):
            bad = np.nonzero(got != ref.dst[j])[0]
            raise AssertionError(f"{what} {m.d_name[j]}: {bad.size} bytes differ, first at "
                                 f"{bad[0]}")
    assert np.array_equal(ck, ref.cksum), f"{what}: checksums differ"
    assert d.guards_intact(), f"{what}: wrote outside a destination"


@pytest.mark.parametrize("chunk", [64 << 10, 1 << 20])
@pytest.mark.parametrize("kind", ["file", "file_mapped", "file_in_place", "whole_pinned",
                                  "whole_direct_pageable"])
@pytest.mark.parametrize("name", ["dense", "f32_tp", "moe_tp", "f32_f16"])
def test_parity_from_a_safetensors_file(tmp_path_factory, name, kind, chunk):
    m, path, off, ref = prepared(name, tmp_path_factory)
    st = cfa.Safetensors.open(path)
    whole = kind.startswith("whole")
    entries = st.entries(targets_for(m), whole_file=whole)
    keep = []
    if not whole:
        src = cfa.Source.file(path, st.data_offset, mapped=kind == "file_mapped",
                              in_place=kind == "file_in_place")
        keep.append(src)
        blob_bytes = st.data_bytes
    else:
        data = np.fromfile(path, dtype=np.uint8)
        blob_bytes = data.size
        if kind == "whole_pinned":
            h = torch.from_numpy(data).pin_memory()
            src = cfa.Source.pinned(h.data_ptr())
        else:
            h = aligned_pageable(data.size)
            h[:] = data
            src = cfa.Source.host_direct(h.ctypes.data)
        keep.append(h)
    d = DeviceDsts(m)
    with cfa.Plan(entries, d.cfa_dsts, blob_bytes, chunk_bytes=chunk) as plan:
        plan.load_async(src)
        plan.wait_layer()
        ck = plan.checksums()
        stats = plan.stats()
    torch.cuda.synchronize()
    if not whole:
        src.close()
    compare(m, d, ck, ref, f"{m.name} [{kind}, chunk {chunk}]")
    if not whole:
        # only the byte ranges the pieces read are read from the file
        assert stats["staged_bytes"] <= st.data_bytes


@pytest.mark.parametrize("phase", [0, 8])
@pytest.mark.parametrize("name", ["dense", "f32_tp", "moe_tp", "f32_f16"])
def test_parity_from_a_file_read_in_place(tmp_path_factory, tmp_path, name, phase):
    """CFA_FILE_MMAP_IN_PLACE: the kernels read the mapped file over the host link, with the
    data section at a 16-byte boundary of the file or 8 bytes past one (header padded with
    spaces), so that every 16-byte phase of the source reaches the vector kernels."""
    from workloads.stfile import file_tensors, header_bytes
    import struct
    m, _, _, ref = prepared(name, tmp_path_factory)
    hdr = header_bytes(file_tensors(m), data_align=16) + b" " * phase
    path = str(tmp_path / "in_place.safetensors")
    with open(path, "wb") as f:
        f.write(struct.pack("<Q", len(hdr)))
        f.write(hdr)
        f.write(m.blob_range(0, m.blob_bytes).tobytes())
    st = cfa.Safetensors.open(path)
    assert st.data_offset % 16 == phase
    d = DeviceDsts(m)
    with cfa.Source.file(path, st.data_offset, in_place=True) as src, \
            cfa.Plan(st.entries(targets_for(m)), d.cfa_dsts, st.data_bytes,
                     chunk_bytes=256 << 10) as plan:
        for _ in range(2):
            plan.load_async(src)
            plan.wait_layer()
            ck = plan.checksums()
            compare(m, d, ck, ref, f"{m.name} [in place, phase {phase}]")
            d.buf.fill_(0xA5)
        assert plan.stats()["staged_bytes"] <= st.data_bytes
    # a plan that reads past the source's stated size is refused before any GPU work
    with cfa.Source.file(path, st.data_offset, in_place=True) as src, \
            cfa.Plan(st.entries(targets_for(m), whole_file=True), d.cfa_dsts,
                     st.data_offset + st.data_bytes, chunk_bytes=256 << 10) as plan:
        with pytest.raises(cfa.CfaError) as e:
            plan.load_async(src)
        assert e.value.name == "CFA_ERR_INVAL" and "holds" in str(e.value)
    torch.cuda.synchronize()
    assert (d.buf == 0xA5).all()


def test_source_size_and_direct_alignment_rules(tmp_path_factory):
    """A stated source size smaller than what the plan reads is refused for every in-place
    kind; a direct host source needs 8-byte alignment only (a pageable copy 8 bytes past a
    16-byte boundary loads exactly)."""
    m, path, off, ref = prepared("dense", tmp_path_factory)
    st = cfa.Safetensors.open(path)
    data = np.fromfile(path, dtype=np.uint8)[st.data_offset:]
    h = aligned_pageable(data.size + 16)
    h8 = h[8:8 + data.size]
    h8[:] = data
    pinned = torch.from_numpy(np.ascontiguousarray(data)).pin_memory()
    d = DeviceDsts(m)
    with cfa.Plan(st.entries(targets_for(m)), d.cfa_dsts, st.data_bytes,
                  chunk_bytes=1 << 20) as plan:
        for src in (cfa.Source.host_direct(h8.ctypes.data, size=st.data_bytes - 1),
                    cfa.Source.host(h8.ctypes.data, size=100),
                    cfa.Source.pinned(pinned.data_ptr(), size=st.data_bytes - 2)):
            with pytest.raises(cfa.CfaError) as e:
                plan.load_async(src)
            assert e.value.name == "CFA_ERR_INVAL"
        with pytest.raises(cfa.CfaError) as e:
            plan.load_async(cfa.Source.host_direct(h8.ctypes.data + 4))
        assert e.value.name == "CFA_ERR_ALIGN"
        plan.load_async(cfa.Source.host_direct(h8.ctypes.data, size=st.data_bytes))
        plan.wait_layer()
        ck = plan.checksums()
    compare(m, d, ck, ref, "direct host source 8 bytes past a 16-byte boundary")


@pytest.mark.parametrize("data_align", [8, 4096])
@pytest.mark.parametrize("name", ["dense", "f32_tp", "moe_tp"])
def test_parity_from_a_file_with_direct_reads(tmp_path_factory, tmp_path, name, data_align):
    """O_DIRECT reads: through bounce buffers (data section at an 8-byte boundary), or for the
    most part straight into the pinned slots (data section at a 4 KiB boundary)."""
    m, _, _, ref = prepared(name, tmp_path_factory)
    path = str(tmp_path / "direct.safetensors")
    off = write_safetensors(m, path, data_align=data_align)
    try:
        src = cfa.Source.file(path, off, direct=True)
    except cfa.CfaError as e:
        pytest.skip(f"no O_DIRECT here: {e}")
    st = cfa.Safetensors.open(path)
    d = DeviceDsts(m)
    with src, cfa.Plan(st.entries(targets_for(m)), d.cfa_dsts, st.data_bytes,
                       chunk_bytes=1 << 20) as plan:
        plan.load_async(src)
        plan.wait_layer()
        ck = plan.checksums()
    compare(m, d, ck, ref, f"{m.name} [direct, data at {data_align}]")


def test_file_that_shrinks_is_reported_and_the_plan_recovers(tmp_path_factory, tmp_path):
    m, path, off, ref = prepared("dense", tmp_path_factory)
    st = cfa.Safetensors.open(path)
    victim = str(tmp_path / "shrinking.safetensors")
    with open(path, "rb") as f:
        whole = f.read()
    with open(victim, "wb") as f:
        f.write(whole)
    entries = st.entries(targets_for(m))
    d = DeviceDsts(m)
    with cfa.Plan(entries, d.cfa_dsts, st.data_bytes, chunk_bytes=256 << 10) as plan:
        with cfa.Source.file(victim, st.data_offset) as src:
            os.truncate(victim, off + st.data_bytes // 2)
            plan.load_async(src)
            with pytest.raises(cfa.CfaError) as e:
                plan.wait_layer()
            assert e.value.name == "CFA_ERR_SOURCE"
        with cfa.Source.file(path, st.data_offset) as src:
            plan.load_async(src)
            plan.wait_layer()
        ck = plan.checksums()
    compare(m, d, ck, ref, "after a failed file load")
