"""GPU parity on randomised manifests (the generator of test_plan_fuzz.py): destinations of
every dtype at random misalignments, sources at element alignment only, column slices with odd
strides, conversions over random bit patterns (NaNs, infinities, subnormals), random chunk,
slab and tiny thresholds, every source kind and the TMA bulk path, against the oracle byte for
byte and checksum for checksum."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_18957_gb300 as cfa
from workloads.harness import CallbackSource, DeviceDsts, entries_for

from test_plan_fuzz import random_manifest

pytestmark = pytest.mark.gpu

KINDS = ["device", "pinned", "host", "callback", "direct_pageable"]


@pytest.fixture(scope="module", autouse=True)
def cuda_device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def _aligned_pageable(blob, align=256):
    buf = np.empty(blob.size + align, dtype=np.uint8)
    off = (-buf.ctypes.data) % align
    h = buf[off:off + blob.size]
    h[:] = blob
    return h


@pytest.mark.parametrize("seed", range(80))
def test_random_manifest_on_the_gpu(seed):
    m = random_manifest(seed)
    blob = m.blob_range(0, m.blob_bytes)
    ref = oracle.unpack(m, blob)
    assert ref.status == 0
    rng = np.random.default_rng(seed + 11)
    kind = KINDS[seed % len(KINDS)]
    keep = []
    if kind == "device":
        t = torch.from_numpy(blob).to("cuda")
        keep.append(t)
        src = cfa.Source.device(t.data_ptr())
    elif kind == "pinned":
        t = torch.from_numpy(blob).pin_memory()
        keep.append(t)
        src = cfa.Source.pinned(t.data_ptr())
    elif kind == "host":
        keep.append(blob)
        src = cfa.Source.host(blob.ctypes.data)
    elif kind == "callback":
        cb = CallbackSource(m)
        keep.append(cb)
        src = cb.source()
    else:
        h = _aligned_pageable(blob)
        keep.append(h)
        src = cfa.Source.host_direct(h.ctypes.data)
    misalign = int(rng.choice([0, 2, 4, 6, 8, 14]))
    d = DeviceDsts(m, misalign=misalign)
    kw = dict(chunk_bytes=256 * int(rng.choice([1, 3, 17, 256, 4096])),
              slab_bytes=int(rng.choice([4096, 65536])),
              tiny_bytes=int(rng.choice([0, 256, 8192])),
              bulk=bool(rng.random() < 0.6))
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, **kw) as plan:
        for rep in range(2):  # twice: plan reuse must give the same state
            plan.load_async(src)
            plan.wait_layer()
            ck = plan.checksums()
            torch.cuda.synchronize()
            for j in range(m.n_dsts):
                got = d.host_bytes(j)
                if not np.array_equal(got, ref.dst[j]):
                    bad = np.nonzero(got != ref.dst[j])[0]
                    raise AssertionError(f"seed {seed} [{kind}, {kw}, misalign {misalign}] "
                                         f"{m.d_name[j]}: {bad.size} bytes differ, first at "
                                         f"{bad[0]}")
            assert np.array_equal(ck, ref.cksum), (seed, kind, kw)
            assert d.guards_intact(), (seed, kind, kw)
