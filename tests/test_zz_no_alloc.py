"""cfa_unpack_noalloc, the entry point that allocates nothing.

It exists for callers that cannot allocate device memory: an engine whose memory pool already
owns the whole GPU, a latency-critical path that cannot afford cudaFree's implicit device-wide
synchronisation, or a runtime without an allocator.  Here it is called through the C ABI
(ctypes).  Its destinations and checksums must equal, bit for bit, those of the oracle (the
plain CPU loader) and of the planned path (cfa_plan_create + cfa_load_async with a device
source) -- on two calls in a row, since every call reuses the same fixed scratch array -- and
the kernels' own status word must come back 0.  Collected last on purpose: it runs after every
other test, and also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2607_18957_gb300 as cfa
from paper_2607_18957_gb300 import _lib
from workloads import Manifest, dense_config, moe_config
from workloads.harness import DeviceDsts, entries_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def call_noalloc(m, d, blob, ck, status=None):
    lib = _lib.load()
    ents = entries_for(m)
    dsts = cfa.make_dsts(d.cfa_dsts)
    err = ctypes.create_string_buffer(512)
    st = lib.cfa_unpack_noalloc(ents.arr.ctypes.data, len(ents.arr), dsts.ctypes.data, len(dsts),
                                blob.data_ptr(), m.blob_bytes,
                                ck.data_ptr() if ck is not None else None,
                                status.data_ptr() if status is not None else None,
                                torch.cuda.current_stream().cuda_stream, err, len(err))
    return st, err.value.decode()


def planned(m, blob):
    d = DeviceDsts(m)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=1 << 20, dev_slots=0,
                  host_slots=0) as plan:
        plan.load_async(cfa.Source.device(blob.data_ptr()))
        plan.wait_layer()
        ck = plan.checksums()
    return d, ck


def check_against_oracle_and_planned(m):
    host_blob = m.blob_range(0, m.blob_bytes)
    ref = oracle.unpack(m, host_blob)
    assert ref.status == 0, ref.status_name
    blob = torch.from_numpy(host_blob).to("cuda")
    d_ref, ck_ref = planned(m, blob)
    d = DeviceDsts(m, fill=0x3C)
    ck = torch.full((m.n_entries,), -1, dtype=torch.int64, device="cuda")  # must be cleared
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")        # must be cleared
    st, msg = call_noalloc(m, d, blob, ck, status)
    assert st == 0, msg
    torch.cuda.synchronize()
    assert int(status.item()) == 0, "a kernel rejected a work item"
    got_ck = ck.cpu().numpy().view(np.uint64)
    for j in range(m.n_dsts):
        got = d.host_bytes(j)
        assert np.array_equal(got, ref.dst[j]), (m.name, m.d_name[j], "vs the oracle")
        assert torch.equal(d.view(j), d_ref.view(j)), (m.name, m.d_name[j], "vs the plan")
    assert np.array_equal(got_ck, ref.cksum), m.name
    assert np.array_equal(got_ck, ck_ref), m.name
    # nothing outside the destinations was written (guard bytes keep their fill)
    mask = torch.ones(d.total, dtype=torch.bool, device="cuda")
    for j in range(m.n_dsts):
        mask[d.offsets[j]:d.offsets[j] + m.d_nbytes(j)] = False
    assert bool((d.buf[mask] == 0x3C).all())
    return blob, d, ck


def edge_manifest():
    """Sizes at this entry point's own layout rules: entries of 8190, 8192 and 8194 destination
    bytes (the 8 KiB line between a warp-level item and 2 MiB block-level items), one of exactly
    2 MiB + 2 bytes (a slab split whose last item holds one element), one of 5 MiB + 6 bytes
    (three items), fused rows of two entries in one destination, and conversions: fp16 -> bf16,
    fp32 -> fp16 and bf16 -> fp32, with source offsets off the 16-byte grid."""
    rng = np.random.default_rng(75)
    specs = [  # (src dtype, dst dtype, destination elements, convert)
        ("bf16", "bf16", 8190 // 2, False), ("bf16", "bf16", 8192 // 2, False),
        ("bf16", "bf16", 8194 // 2, False), ("bf16", "bf16", (2 << 20) // 2 + 1, False),
        ("u8", "u8", 5 * (1 << 20) + 6, False), ("f16", "bf16", (3 << 20) // 2 + 3, True),
        ("f32", "f16", 4097, True), ("bf16", "f32", (2 << 20) // 4 + 5, True),
        ("f32", "f32", 2047, False), ("i64", "i64", 300_001, False)]
    size = {"u8": 1, "bf16": 2, "f16": 2, "f32": 4, "i64": 8}
    entries, dsts, off = [], [], 0
    for k, (s, dt, n, conv) in enumerate(specs):
        es = size[s]
        off = (off + es - 1) // es * es + es * int(rng.integers(0, 7))
        entries.append({"name": f"e{k}", "dtype": s, "shape": (n,), "offset": off, "dst": k,
                        "cast": conv})
        dsts.append({"name": f"d{k}", "dtype": dt, "shape": (n,)})
        off += n * es
    # a fused destination [2 rows + 3 rows, 4100 columns] written by two entries
    es = 2
    off = (off + 1) // 2 * 2 + 6
    k = len(dsts)
    dsts.append({"name": "fused", "dtype": "bf16", "shape": (5, 4100)})
    entries.append({"name": "top", "dtype": "bf16", "shape": (2, 4100), "offset": off, "dst": k,
                    "row": 0})
    off += 2 * 4100 * es + 2
    entries.append({"name": "bottom", "dtype": "bf16", "shape": (3, 4100), "offset": off,
                    "dst": k, "row": 2})
    off += 3 * 4100 * es
    return Manifest("noalloc_edges", entries, dsts, off + 64, "f16fin", 76)


def test_noalloc_matches_the_oracle_on_two_calls_in_a_row():
    # call 1: dense checkpoint with q/k/v and gate/up fusion, tensors at odd 2-byte offsets
    m1 = dense_config("noalloc_dense", 71, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                      inter=1536, vocab=1000, align=2, jitter=5)
    check_against_oracle_and_planned(m1)
    # call 2: a different checkpoint (MoE stacking, hundreds of tiny tensors) through the same
    # scratch; nothing from call 1 may leak into it
    m2 = moe_config("noalloc_moe", 72, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                    inter=512, n_experts=4, vocab=500, n_extra=600, align=2, jitter=3)
    blob, d, ck = check_against_oracle_and_planned(m2)
    # a third call on the same inputs leaves device memory where it was: nothing allocated
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    st, msg = call_noalloc(m2, d, blob, ck)
    torch.cuda.synchronize()
    assert st == 0, msg
    assert torch.cuda.mem_get_info()[0] == free0


def test_noalloc_multi_item_slabs_threshold_sizes_and_conversions():
    check_against_oracle_and_planned(edge_manifest())


def test_noalloc_fp32_to_bf16_cast():
    m = dense_config("noalloc_f32", 73, layers=1, hidden=256, n_q=4, n_kv=2, head_dim=64,
                     inter=768, vocab=300, src_dtype="f32", align=4, jitter=3)
    check_against_oracle_and_planned(m)


def test_noalloc_rejects_more_work_than_its_scratch_holds():
    n = 17000  # tiny tensors take one work item each; the scratch holds 16384
    ents = [{"name": f"t{k}", "dtype": "bf16", "shape": (4,), "offset": 8 * k, "dst": k}
            for k in range(n)]
    dsts = [{"name": f"d{k}", "dtype": "bf16", "shape": (4,)} for k in range(n)]
    m = Manifest("too_many", ents, dsts, 8 * n, "bits", 1)
    d = DeviceDsts(m, guard=0)
    blob = torch.zeros(m.blob_bytes, dtype=torch.uint8, device="cuda")
    st, msg = call_noalloc(m, d, blob, None)
    assert _lib.STATUS[st] == "CFA_ERR_INVAL"
    assert "16384" in msg
    # nothing was launched: the destinations still hold their fill
    torch.cuda.synchronize()
    assert bool((d.buf == 0xA5).all())
