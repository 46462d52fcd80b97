"""cfa_unpack_noalloc, the entry point that allocates nothing.

It exists for callers that cannot allocate device memory: an engine whose memory pool already
owns the whole GPU, a latency-critical path that cannot afford cudaFree's implicit device-wide
synchronisation, or a runtime without an allocator.  Here it is called through the C ABI (ctypes) and its
destinations and checksums must equal, bit for bit, those of the planned path (cfa_plan_create
+ cfa_load_async with a device source) -- on two calls in a row, since every call reuses the
same fixed scratch array.  Collected last on purpose: it runs after every other test, and also
passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

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


def call_noalloc(m, d, blob, ck):
    lib = _lib.load()
    ents = entries_for(m)
    dsts = cfa.make_dsts(d.cfa_dsts)
    err = ctypes.create_string_buffer(512)
    st = lib.cfa_unpack_noalloc(ents.arr.ctypes.data, len(ents.arr), dsts.ctypes.data, len(dsts),
                                blob.data_ptr(), m.blob_bytes,
                                ck.data_ptr() if ck is not None else None,
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


def check_against_planned(m):
    blob = torch.from_numpy(m.blob_range(0, m.blob_bytes)).to("cuda")
    d_ref, ck_ref = planned(m, blob)
    d = DeviceDsts(m, fill=0x3C)
    ck = torch.full((m.n_entries,), -1, dtype=torch.int64, device="cuda")  # must be cleared
    st, msg = call_noalloc(m, d, blob, ck)
    assert st == 0, msg
    torch.cuda.synchronize()
    for j in range(m.n_dsts):
        assert torch.equal(d.view(j), d_ref.view(j)), (m.name, m.d_name[j])
    assert np.array_equal(ck.cpu().numpy().view(np.uint64), ck_ref), m.name
    return blob, d, ck


def test_noalloc_matches_the_planned_path_on_two_calls_in_a_row():
    # call 1: dense checkpoint with q/k/v and gate/up fusion, tensors at odd 2-byte offsets
    m1 = dense_config("noalloc_dense", 71, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                      inter=1536, vocab=1000, align=2, jitter=5)
    check_against_planned(m1)
    # call 2: a different checkpoint (MoE stacking, hundreds of tiny tensors) through the same
    # scratch; nothing from call 1 may leak into it
    m2 = moe_config("noalloc_moe", 72, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                    inter=512, n_experts=4, vocab=500, n_extra=600, align=2, jitter=3)
    blob, d, ck = check_against_planned(m2)
    # a third call on the same inputs leaves device memory where it was: nothing allocated
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    st, msg = call_noalloc(m2, d, blob, ck)
    torch.cuda.synchronize()
    assert st == 0, msg
    assert torch.cuda.mem_get_info()[0] == free0


def test_noalloc_fp32_to_bf16_cast():
    m = dense_config("noalloc_f32", 73, layers=1, hidden=256, n_q=4, n_kv=2, head_dim=64,
                     inter=768, vocab=300, src_dtype="f32", align=4, jitter=3)
    check_against_planned(m)


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
