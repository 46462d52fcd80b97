"""The oracle against its pins (CPU only).  See tests/_pins.py for what each pin fixes."""
import numpy as np
import pytest

import _pins
import oracle


@pytest.mark.parametrize("pin", _pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin()


def test_rne_exhaustive_vs_torch():
    """All 2^32 fp32 bit patterns: the oracle's fp32 -> bf16 and fp32 -> fp16 conversions equal
    torch's CPU conversions (NaNs as a class; the oracle's NaNs are 0x7FC0 and sign | 0x7E00)."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    step = 1 << 24

    def block(start):
        u = np.arange(start, start + step, dtype=np.uint32)
        _pins.check_rne_block(u)
        _pins.check_convert_block("f32", "f16", u)

    workers = min(8, len(os.sched_getaffinity(0)))
    with ThreadPoolExecutor(workers) as ex:
        for f in [ex.submit(block, s) for s in range(0, 1 << 32, step)]:
            f.result()


def test_empty_manifest():
    from workloads import Manifest
    m = Manifest("empty", [], [], 0, "bits", 0)
    r = oracle.unpack(m, np.zeros(0, np.uint8), cover=True)
    assert r.status == 0 and r.cksum.size == 0 and r.dst == {}


def test_zero_element_entry_and_destination():
    from workloads import Manifest
    ents = [{"name": "a", "dtype": "bf16", "shape": (0, 4), "offset": 0, "dst": 0, "row": 0},
            {"name": "b", "dtype": "bf16", "shape": (2,), "offset": 0, "dst": 1, "row": 0}]
    dsts = [{"name": "A", "dtype": "bf16", "shape": (0, 4)},
            {"name": "B", "dtype": "bf16", "shape": (2,)}]
    m = Manifest("zero", ents, dsts, 4, "bits", 0)
    blob = np.array([1, 2, 3, 4], np.uint8)
    r = oracle.unpack(m, blob, cover=True)
    assert r.status == 0
    assert r.dst[0].size == 0 and list(r.dst[1]) == [1, 2, 3, 4]
    assert list(r.cksum) == [0, 0x0201 + 0x0403]
    assert oracle.check_cover(r)[0] == 0
