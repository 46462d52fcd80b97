"""Segmented (multi-path) loading, section 4.2 "Optimization of Distributed Loading": every chunk
is cut into one equal segment per rank, each rank copies its own segment host->device, an
AllGather assembles the chunk in every rank's device slot (the chunk's Gathered state), and each
rank unpacks locally.

Without a GPU: the segment layout (cfa_segment_range), segmented host-only plans (what a rank
stages), the option checks, and the exchange itself as two gloo processes: each rank puts its
segments of every chunk into a host "slot" and the same AllGather hook the loader calls on GPUs
assembles them; every gathered chunk must equal the blob's bytes.

On one GPU (-m gpu): a segmented load of rank r of W whose gather step is stood in for by local
copies of the other ranks' segments out of a device copy of the blob (no rank waits on another),
compared with the oracle byte for byte, from pinned, pageable and callback sources."""
import multiprocessing as mp
import os
import socket
import sys

import numpy as np
import pytest

import paper_2607_18957_gb300 as cfa
import workloads
from paper_2607_18957_gb300 import _lib
from workloads.harness import entries_for

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _fake_dsts(m):
    # host-only plans never touch destination memory: distinct aligned fake addresses
    out, pos = [], 1 << 40
    for j in range(m.n_dsts):
        out.append((pos, str(m.d_dtype[j]), m.d_shape_tuple(j)))
        pos += (m.d_nbytes(j) + 4095) // 4096 * 4096 + 4096
    return out


def _noop(*args):
    return None


def small_model(seed=81, chunk_bytes=None):
    m = workloads.dense_config("seg_small", seed, layers=2, hidden=256, n_q=4, n_kv=2,
                               head_dim=64, inter=640, vocab=700, align=2, jitter=5)
    if chunk_bytes:
        m.chunk_bytes = chunk_bytes
    return m


def test_segment_range_cuts_every_chunk_into_equal_segments():
    B, S = 10 * 4096 + 1000, 4096
    for W in (1, 2, 4, 16):
        seg = S // W
        n_chunks = -(-B // S)
        for c in range(n_chunks):
            covered = 0
            for r in range(W):
                off, n = cfa.segment_range(B, S, W, r, c)
                assert off == c * S + r * seg
                assert n == max(0, min(seg, B - off))
                covered += n
            assert covered == min(S, B - c * S)  # the segments tile the chunk exactly
    # the last chunk is partial: rank 3 of 4 owns nothing past the blob's end
    assert cfa.segment_range(B, S, 4, 3, n_chunks - 1) == ((n_chunks - 1) * S + 3 * 1024, 0)
    for bad in [(B, S, 0, 0, 0), (B, S, 2, 2, 0), (B, S, 2, -1, 0), (B, 4096 + 256, 2, 0, 0),
                (B, S, 32, 0, 0), (B, S, 2, 0, 11)]:
        with pytest.raises(cfa.CfaError):
            cfa.segment_range(*bad)


def test_segmented_host_only_plan_stages_its_segments():
    m = small_model(chunk_bytes=64 << 10)
    B = m.blob_bytes
    dsts = _fake_dsts(m)
    whole = cfa.Plan(entries_for(m), dsts, B, chunk_bytes=m.chunk_bytes, host_only=True)
    st_whole = whole.stats()
    total = 0
    for W in (2, 4):
        for r in range(W):
            p = cfa.Plan(entries_for(m), dsts, B, chunk_bytes=m.chunk_bytes, host_only=True,
                         world=W, rank=r, gather=_noop)
            st = p.stats()
            want = sum(cfa.segment_range(B, m.chunk_bytes, W, r, c)[1]
                       for c in range(st["n_chunks"]))
            assert st["staged_bytes"] == want
            # the unpack work is the rank's whole plan, the same on every rank
            for k in ("n_pieces", "bytes_read", "bytes_written", "n_chunks"):
                assert st[k] == st_whole[k]
            if W == 4:
                total += st["staged_bytes"]
    assert total == B  # the ranks' segments together are the blob, each byte once


def test_segmented_plan_option_checks():
    m = small_model()
    dsts = _fake_dsts(m)
    bad = [dict(world=2, rank=2, gather=_noop), dict(world=2, rank=-1, gather=_noop),
           dict(world=2, rank=0, gather=None),                 # no gather step
           dict(world=3, rank=0, gather=_noop, chunk_bytes=4096)]  # 4096 % (256 * 3) != 0
    for kw in bad:
        kw.setdefault("chunk_bytes", 64 << 10)
        with pytest.raises(cfa.CfaError) as ei:
            cfa.Plan(entries_for(m), dsts, m.blob_bytes, host_only=True, **kw)
        assert ei.value.name == "CFA_ERR_INVAL", kw


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _gather_rank(rank, world, port, blob_bytes, chunk_bytes, seed, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import paper_2607_18957_gb300 as cfa
    from workloads import gen
    dist.init_process_group("gloo", rank=rank, world_size=world)
    blob = gen.fill("bits", seed, 0, blob_bytes)  # each rank's own copy of the checkpoint
    hook = cfa.AllGather(device="cpu")
    slot = np.full(chunk_bytes, 0xEE, dtype=np.uint8)
    n_chunks = -(-blob_bytes // chunk_bytes)
    bad = []
    for c in range(n_chunks):
        slot[:] = 0xEE
        seg = chunk_bytes // world
        off, n = cfa.segment_range(blob_bytes, chunk_bytes, world, rank, c)
        slot[rank * seg:rank * seg + n] = blob[off:off + n]  # this rank's H2D, on the host
        hook(slot.ctypes.data, seg, world, rank, c, 0)
        lo = c * chunk_bytes
        hi = min(blob_bytes, lo + chunk_bytes)
        if not np.array_equal(slot[:hi - lo], blob[lo:hi]):
            bad.append(c)
    dist.destroy_process_group()
    out.put((rank, n_chunks, bad))


@pytest.mark.parametrize("world", [2, 3])
def test_gathered_chunks_equal_the_blob_over_gloo(world):
    chunk = 256 * world * 16
    blob_bytes = 7 * chunk + 1234  # a partial last chunk: some ranks' segments are empty
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_gather_rank, args=(r, world, port, blob_bytes, chunk, 9, out))
             for r in range(world)]
    for p in procs:
        p.start()
    res = [out.get(timeout=180) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert sorted(r for r, _, _ in res) == list(range(world))
    for r, n, bad in res:
        assert n == 8 and not bad, (r, bad)


# ---- on one GPU --------------------------------------------------------------------------

class LocalGather:
    """Stands in for the AllGather on one GPU: fills the other ranks' segments of the slot from
    a device copy of the blob, on the loader's gather stream.  Records the chunks it saw."""

    def __init__(self, dev_blob, blob_bytes, chunk_bytes, fail_at=None):
        self.dev_blob = dev_blob
        self.B = blob_bytes
        self.S = chunk_bytes
        self.fail_at = fail_at
        self.chunks = []

    def __call__(self, chunk_ptr, seg, world, rank, chunk, stream):
        import torch
        self.chunks.append(chunk)
        if chunk == self.fail_at:
            raise RuntimeError("gather failed on purpose")
        slot = cfa.AllGather().slot(chunk_ptr, seg * world)
        with torch.cuda.stream(torch.cuda.ExternalStream(stream)):
            for r in range(world):
                if r == rank:
                    continue
                off, n = cfa.segment_range(self.B, self.S, world, r, chunk)
                if n:
                    slot[r * seg:r * seg + n].copy_(self.dev_blob[off:off + n],
                                                    non_blocking=True)


def _gpu_case(m, source_kind, world, rank, **kw):
    import torch

    import oracle
    from workloads.harness import CallbackSource, DeviceDsts, pinned_blob
    host = pinned_blob(m)
    dev_blob = host.to("cuda")
    ref = oracle.unpack(m, m.blob_range(0, m.blob_bytes))
    assert ref.status == 0
    d = DeviceDsts(m)
    g = LocalGather(dev_blob, m.blob_bytes, m.chunk_bytes)
    pageable = host.numpy().copy()
    cb = CallbackSource(m)
    src = {"pinned": cfa.Source.pinned(host.data_ptr()),
           "host": cfa.Source.host(pageable.ctypes.data),
           "callback": cb.source()}[source_kind]
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                  world=world, rank=rank, gather=g, **kw) as plan:
        for _ in range(2):  # twice: slots and events reused across loads
            d.buf.fill_(0xA5)
            g.chunks.clear()
            plan.load_async(src)
            plan.wait_layer()
            ck = plan.checksums()
            torch.cuda.synchronize()
            n_chunks = plan.info()["n_chunks"]
            assert g.chunks == list(range(n_chunks))  # every chunk, in order
            for j in range(m.n_dsts):
                assert np.array_equal(d.host_bytes(j), ref.dst[j]), (source_kind, m.d_name[j])
            assert np.array_equal(ck, ref.cksum)
            assert d.guards_intact()
        st = plan.stats()
        assert st["staged_bytes"] == sum(
            cfa.segment_range(m.blob_bytes, m.chunk_bytes, world, rank, c)[1]
            for c in range(n_chunks))


@pytest.mark.gpu
@pytest.mark.parametrize("source_kind,world,rank", [
    ("pinned", 2, 0), ("pinned", 2, 1), ("pinned", 4, 3), ("host", 2, 1), ("callback", 4, 2)])
def test_gpu_segmented_load_matches_the_oracle(source_kind, world, rank):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    m = small_model(chunk_bytes=256 * 4 * 64)  # 64 KiB chunks, last one partial
    _gpu_case(m, source_kind, world, rank, host_slots=2, dev_slots=2)


@pytest.mark.gpu
@pytest.mark.parametrize("source_kind", ["pinned", "host"])
def test_gpu_segmented_load_of_a_tensor_parallel_rank_with_conversions(source_kind):
    """A rank's plan with column slices (read by the column-slice kernel from the gathered slot)
    and fp32 -> bf16 conversions, over segments of 3 ranks."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    m = workloads.dense_config("seg_tp", 83, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                               inter=640, vocab=700, src_dtype="f32", align=4, jitter=3, tp=2,
                               rank=1)
    m.chunk_bytes = 256 * 3 * 128  # 96 KiB chunks: rows and tensors cross chunk boundaries
    _gpu_case(m, source_kind, 3, 2, host_slots=2, dev_slots=2)


@pytest.mark.gpu
def test_gpu_segmented_load_of_a_blob_shorter_than_one_chunk():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    m = small_model(chunk_bytes=8 << 20)  # one partial chunk; the slots are still 8 MiB
    _gpu_case(m, "pinned", 4, 1, host_slots=0)


@pytest.mark.gpu
def test_gpu_segmented_load_reports_a_failed_gather():
    import torch

    from workloads.harness import DeviceDsts, pinned_blob
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    m = small_model(chunk_bytes=64 << 10)
    host = pinned_blob(m)
    dev_blob = host.to("cuda")
    d = DeviceDsts(m)
    g = LocalGather(dev_blob, m.blob_bytes, m.chunk_bytes, fail_at=2)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                  host_slots=0, world=2, rank=0, gather=g) as plan:
        with pytest.raises(cfa.CfaError) as ei:
            plan.load_async(cfa.Source.pinned(host.data_ptr()))
        assert ei.value.name == "CFA_ERR_GATHER"
        assert g.chunks == [0, 1, 2]  # enqueueing stopped at the failed chunk
        assert _lib.STATUS[plan.try_wait_layer(timeout_ns=10_000_000_000)] == "CFA_ERR_GATHER"
        assert isinstance(plan.gather_error, RuntimeError)
        # the plan stays usable: the next load with a working gather is complete
        g.fail_at = None
        plan.load_async(cfa.Source.pinned(host.data_ptr()))
        plan.wait_layer()
        torch.cuda.synchronize()
    import oracle
    ref = oracle.unpack(m, m.blob_range(0, m.blob_bytes))
    for j in range(m.n_dsts):
        assert np.array_equal(d.host_bytes(j), ref.dst[j])


@pytest.mark.gpu
def test_gpu_segmented_plan_refuses_in_place_sources():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    from workloads.harness import DeviceDsts
    m = small_model()
    d = DeviceDsts(m)
    blob = torch.zeros(m.blob_bytes, dtype=torch.uint8, device="cuda")
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=64 << 10,
                  world=2, rank=0, gather=_noop) as plan:
        for src in (cfa.Source.device(blob.data_ptr()),):
            with pytest.raises(cfa.CfaError) as ei:
                plan.load_async(src)
            assert ei.value.name == "CFA_ERR_INVAL"
    assert d.guards_intact()
