"""Every input bit pattern through the GPU conversions, against the oracle: all 2^32 fp32
patterns to bf16 and to fp16, all 2^16 fp16 patterns to bf16 and fp32, all 2^16 bf16 patterns to
fp32 (NaN payloads, infinities, subnormals, signed zeros, the overflow thresholds included).
The source is one device-resident tensor holding the patterns in order (made by torch, not by
the loader); the checksum of each conversion is checked against the oracle's bits as well."""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
import paper_2607_18957_gb300 as cfa

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    yield
    torch.cuda.empty_cache()


def _threads():
    return max(1, min(16, len(os.sched_getaffinity(0))))


def _run(src_dtype, dst_dtype, n):
    """Loads patterns 0..n-1 of src_dtype as one converted 2-D entry; returns (dst, checksum)."""
    tdt = {"f32": torch.int32, "f16": torch.int16, "bf16": torch.int16}[src_dtype]
    es_s = 4 if src_dtype == "f32" else 2
    es_d = 4 if dst_dtype == "f32" else 2
    cols = 65536
    rows = n // cols
    src = torch.arange(0, n, dtype=torch.int64, device="cuda").to(tdt)  # wraps to the bit patterns
    dst = torch.empty(n * es_d, dtype=torch.uint8, device="cuda")
    ents = cfa.make_entries(dtype=[src_dtype], shape=[(rows, cols)], offset=[0], dst=[0],
                            cast=[True])
    with cfa.Plan(ents, [(dst.data_ptr(), dst_dtype, (rows, cols))], n * es_s,
                  chunk_bytes=1 << 30, dev_slots=0, host_slots=0) as plan:
        plan.load_async(cfa.Source.device(src.data_ptr()))
        plan.wait_layer()
        ck = int(plan.checksums()[0])
    del src
    return dst, ck


def _compare(src_dtype, dst_dtype, n):
    dst, ck = _run(src_dtype, dst_dtype, n)
    udt = np.uint32 if dst_dtype == "f32" else np.uint16
    sdt = np.uint32 if src_dtype == "f32" else np.uint16
    block = 1 << 26
    starts = list(range(0, n, block))

    def one(a):
        b = min(n, a + block)
        want = oracle.convert(src_dtype, dst_dtype, np.arange(a, b, dtype=np.uint64).astype(sdt))
        es = np.dtype(udt).itemsize
        got = dst[a * es:b * es].cpu().numpy().view(udt)
        bad = np.nonzero(got != want)[0]
        return (a + int(bad[0]), int(got[bad[0]]), int(want[bad[0]])) if bad.size else None, \
            int(want.astype(np.uint64).sum(dtype=np.uint64))

    with ThreadPoolExecutor(_threads()) as ex:
        res = list(ex.map(one, starts))
    for first_bad, _ in res:
        assert first_bad is None, (src_dtype, dst_dtype, "pattern 0x%x: gpu 0x%x oracle 0x%x"
                                   % first_bad)
    total = 0
    for _, s in res:
        total = (total + s) & 0xFFFFFFFFFFFFFFFF
    assert ck == total, (src_dtype, dst_dtype)


@pytest.mark.parametrize("dst_dtype", ["bf16", "f16"])
def test_every_fp32_pattern(dst_dtype):
    _compare("f32", dst_dtype, 1 << 32)


@pytest.mark.parametrize("src_dtype,dst_dtype", [("f16", "bf16"), ("f16", "f32"),
                                                 ("bf16", "f32")])
def test_every_16_bit_pattern(src_dtype, dst_dtype):
    _compare(src_dtype, dst_dtype, 1 << 16)
