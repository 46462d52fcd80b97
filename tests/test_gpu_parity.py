"""GPU parity: the loader (through the C ABI) against the oracle, byte for byte and checksum for
checksum, on seeded synthetic checkpoints at sizes the oracle finishes in seconds.  Every source
kind, several chunk sizes (down to 256 B, so tensors span many chunks and chunks end ragged),
misaligned blob offsets and destinations, the fp32 -> bf16 cast, fused layouts, thousands of
tiny tensors, readiness groups, and host-side failures (slow and failing sources)."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2607_18957_gb300 as cfa
from workloads import dense_config, fp8_block_config, moe_config, tiny_config
from workloads.harness import CallbackSource, DeviceDsts, entries_for, pinned_blob

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


_ORACLE_CACHE = {}


def reference(m):
    key = (m.name, m.seed, m.blob_bytes)
    if key not in _ORACLE_CACHE:
        blob = m.blob_range(0, m.blob_bytes)
        r = oracle.unpack(m, blob)
        assert r.status == 0, r.status_name
        _ORACLE_CACHE[key] = (blob, r)
    return _ORACLE_CACHE[key]


def make_source(kind, m, blob, keep):
    if kind == "device":
        d = torch.from_numpy(blob).to("cuda")
        keep.append(d)
        return cfa.Source.device(d.data_ptr())
    if kind == "pinned":
        h = torch.from_numpy(blob).pin_memory()
        keep.append(h)
        return cfa.Source.pinned(h.data_ptr())
    if kind == "host":
        h = np.ascontiguousarray(blob)
        keep.append(h)
        return cfa.Source.host(h.ctypes.data)
    if kind == "callback":
        cb = CallbackSource(m)
        keep.append(cb)
        return cb.source()
    if kind == "direct_pageable":
        h = aligned_host_copy(blob)
        keep.append(h)
        return cfa.Source.host_direct(h.ctypes.data)
    if kind == "direct_pinned":
        h = torch.from_numpy(blob).pin_memory()
        keep.append(h)
        return cfa.Source.host_direct(h.data_ptr())
    raise ValueError(kind)


def aligned_host_copy(blob, align=256):
    """A pageable copy of `blob` starting on an `align`-byte boundary."""
    buf = np.empty(blob.size + align, dtype=np.uint8)
    off = (-buf.ctypes.data) % align
    h = buf[off:off + blob.size]
    h[:] = blob
    return h


def load_and_compare(m, kind, chunk, misalign=0, **kw):
    blob, ref = reference(m)
    keep = []
    src = make_source(kind, m, blob, keep)
    d = DeviceDsts(m, misalign=misalign)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=chunk, **kw) as plan:
        plan.load_async(src)
        plan.wait_layer()
        ck = plan.checksums()
        stats = plan.stats()
    torch.cuda.synchronize()
    for j in range(m.n_dsts):
        got = d.host_bytes(j)
        if not np.array_equal(got, ref.dst[j]):
            bad = np.nonzero(got != ref.dst[j])[0]
            raise AssertionError(f"{m.name} [{kind}, chunk {chunk}] {m.d_name[j]}: "
                                 f"{bad.size} bytes differ, first at {bad[0]}")
    assert np.array_equal(ck, ref.cksum), f"{m.name} [{kind}, chunk {chunk}] checksums differ"
    assert d.guards_intact(), f"{m.name} [{kind}, chunk {chunk}] wrote outside a destination"
    return stats


def cfg_tiny():
    return tiny_config(seed=61, n=300, lo=2, hi=300_000, align=2, jitter=7, name="tiny_ragged")


def cfg_dense():
    return dense_config("dense_bf16", 62, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                        inter=1536, vocab=1000, align=2, jitter=5)


def cfg_dense_f32():
    return dense_config("dense_f32", 63, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                        inter=1536, vocab=1000, src_dtype="f32", align=4, jitter=3)


def cfg_moe():
    return moe_config("moe_bf16", 64, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                      inter=512, n_experts=4, vocab=500, n_extra=3000, align=2, jitter=3)


def cfg_dense_tp():
    return dense_config("dense_tp2r1", 68, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                        inter=1536, vocab=1000, align=2, jitter=5, tp=2, rank=1)


def cfg_f32_tp():
    return dense_config("dense_f32_tp4r3", 69, layers=2, hidden=512, n_q=8, n_kv=2,
                        head_dim=64, inter=1536, vocab=1000, src_dtype="f32", align=4,
                        jitter=3, tp=4, rank=3)


def cfg_moe_tp():
    return moe_config("moe_tp2r0", 70, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                      inter=512, n_experts=4, vocab=500, n_extra=300, align=2, jitter=3,
                      tp=2, rank=0)


def cfg_f32_to_f16():
    return dense_config("f32_to_f16", 71, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                        inter=1536, vocab=1000, src_dtype="f32", dst_dtype="f16", align=4,
                        jitter=3)


def cfg_f16_bits_to_bf16():
    # random 16-bit patterns: every NaN, infinity and subnormal of binary16 occurs; the norms
    # are widened to fp32
    return dense_config("f16bits_to_bf16", 72, layers=2, hidden=512, n_q=8, n_kv=2,
                        head_dim=64, inter=1536, vocab=1000, src_dtype="f16", norm_dtype="f32",
                        blob_kind="bits", align=2, jitter=5)


def cfg_bf16_f32_norms_tp():
    return dense_config("bf16_f32norm_tp2r0", 73, layers=2, hidden=512, n_q=8, n_kv=2,
                        head_dim=64, inter=1536, vocab=1000, norm_dtype="f32", align=2,
                        jitter=5, tp=2, rank=0)


def cfg_moe_ep():
    return moe_config("moe_ep4r2", 74, layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                      inter=512, n_experts=8, vocab=500, n_extra=300, align=2, jitter=3, ep=4,
                      rank=2)


def cfg_fp8_block():
    # 8-bit weights at odd byte offsets with fp32 block scales (scales fused like the weights)
    return fp8_block_config("fp8_block", 75, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                            inter=1536, vocab=1000, block=128, align=1, jitter=7)


CONFIGS = {"tiny": cfg_tiny, "dense": cfg_dense, "dense_f32": cfg_dense_f32, "moe": cfg_moe,
           "dense_tp": cfg_dense_tp, "f32_tp": cfg_f32_tp, "moe_tp": cfg_moe_tp,
           "f32_f16": cfg_f32_to_f16, "f16_bf16": cfg_f16_bits_to_bf16,
           "bf16_f32norm_tp": cfg_bf16_f32_norms_tp, "moe_ep": cfg_moe_ep,
           "fp8_block": cfg_fp8_block}


@pytest.mark.parametrize("cfg", list(CONFIGS))
@pytest.mark.parametrize("kind", ["device", "pinned", "host", "callback", "direct_pageable",
                                  "direct_pinned"])
def test_parity_sources(cfg, kind):
    m = CONFIGS[cfg]()
    load_and_compare(m, kind, chunk=1 << 20)


@pytest.mark.parametrize("cfg", list(CONFIGS))
@pytest.mark.parametrize("kind", ["pinned", "callback", "host"])
@pytest.mark.parametrize("pull,slots", [(0, 2), (50, 3), (100, 1)])
def test_parity_transfer_paths(cfg, kind, pull, slots):
    """Staged loads through the copy engine alone, split half and half with the pull kernel,
    and pulled alone through a single device slot (every transfer then waits for the previous
    chunk's unpack), at chunk sizes whose ranges go to both paths."""
    m = CONFIGS[cfg]()
    stats = load_and_compare(m, kind, chunk=(1 << 20) + 4096, pull_percent=pull, dev_slots=slots)
    assert stats["staged_bytes"] > 0


@pytest.mark.parametrize("cfg", list(CONFIGS))
@pytest.mark.parametrize("chunk", [256, 4096 + 256, 3 << 20, 1 << 30])
def test_parity_chunk_sizes(cfg, chunk):
    """Theorem 2: the chunking (any chunk length) must not change the loaded state."""
    m = CONFIGS[cfg]()
    load_and_compare(m, "device", chunk=chunk, no_merge=(chunk == 4096 + 256))
    if chunk in (256, 3 << 20):
        load_and_compare(m, "pinned", chunk=chunk)


@pytest.mark.parametrize("misalign", [2, 6, 14])
def test_parity_misaligned_destinations(misalign):
    for cfg in ("dense", "moe", "dense_f32", "f32_f16", "f16_bf16", "dense_tp"):
        m = CONFIGS[cfg]()
        load_and_compare(m, "device", chunk=1 << 20, misalign=misalign)


@pytest.mark.parametrize("slab,tiny", [(4096, 0), (1 << 20, 1 << 20), (65536, 512)])
def test_parity_work_splits(slab, tiny):
    """Slab and tiny thresholds only change how work is cut, never the result."""
    for cfg in ("dense", "moe", "dense_f32", "tiny"):
        m = CONFIGS[cfg]()
        load_and_compare(m, "device", chunk=1 << 20, slab_bytes=slab, tiny_bytes=tiny)


@pytest.mark.parametrize("cfg", list(CONFIGS))
@pytest.mark.parametrize("kind", ["device", "pinned", "callback"])
@pytest.mark.parametrize("chunk", [4096 + 256, 1 << 20])
def test_parity_vector_only_path(cfg, kind, chunk):
    """Without CFA_OPT_BULK every slab, aligned or not, goes through the vector kernel."""
    m = CONFIGS[cfg]()
    st = load_and_compare(m, kind, chunk=chunk, bulk=False)
    assert st["n_bulk"] == 0


def test_bulk_path_takes_every_aligned_slab():
    m = dense_config("dense_aligned", 67, layers=2, hidden=512, n_q=8, n_kv=2, head_dim=64,
                     inter=1536, vocab=1000, align=256)
    st = load_and_compare(m, "device", chunk=1 << 20)
    assert st["n_bulk"] > 0 and st["n_slabs"] == 0
    st = load_and_compare(m, "device", chunk=1 << 20, bulk=False)
    assert st["n_bulk"] == 0 and st["n_slabs"] > 0
    # conversions never take the bulk path
    st = load_and_compare(CONFIGS["dense_f32"](), "device", chunk=1 << 20)
    assert st["n_bulk"] == 0


@pytest.mark.parametrize("kind", ["direct_pageable", "direct_pinned", "device", "pinned"])
def test_aligned_slabs_from_host_memory(kind):
    """A 16-byte-aligned checkpoint (every slab a bulk item) of about 200 MB read in place from
    host memory takes the vector kernel for its bulk items; from device memory and staging slots
    the TMA kernel."""
    m = dense_config("aligned_200mb", 76, layers=2, hidden=2048, n_q=16, n_kv=4, head_dim=128,
                     inter=6144, vocab=8000, align=256)
    st = load_and_compare(m, kind, chunk=16 << 20)
    assert st["n_bulk"] > 0 and st["n_slabs"] == 0


def test_parity_aligned_full_tiny_workload():
    """The 1,000-tensor 256-byte-aligned workload at full size (about 125 MiB)."""
    m = tiny_config(seed=1)
    for kind in ("device", "pinned"):
        load_and_compare(m, kind, chunk=512 << 20)


def test_element_sizes_1_4_8():
    from workloads import Manifest
    rng = np.random.default_rng(5)
    ents, dsts, off = [], [], 0
    for k, (dt, es) in enumerate([("u8", 1), ("i32", 4), ("i64", 8), ("f64", 8), ("u8", 1)]):
        n = int(rng.integers(1, 70000))
        off = (off + es - 1) // es * es + int(rng.integers(0, 5)) * es
        dsts.append({"name": f"d{k}", "dtype": dt, "shape": (n,)})
        ents.append({"name": f"e{k}", "dtype": dt, "shape": (n,), "offset": off, "dst": k,
                     "row": 0, "layer": k})
        off += n * es
    m = Manifest("mixed_sizes", ents, dsts, off, "bits", 9)
    for chunk in (256, 1 << 20):
        load_and_compare(m, "device", chunk=chunk)
        load_and_compare(m, "pinned", chunk=chunk)


def _tiny_phase_manifest(n=3000, dst_phase=8, seed=17):
    """Only tiny pieces (below the 8 KiB line), of every element size: half at source offsets
    with the destinations' phase within 16 bytes (the tiny kernel's one-round path, partial first
    and last vectors included), half at other element-aligned offsets (its fallback)."""
    from workloads import Manifest
    rng = np.random.default_rng(seed)
    kinds = [("u8", 1), ("bf16", 2), ("f32", 4), ("i64", 8)]
    ents, dsts, off = [], [], 0
    for k in range(n):
        dt, es = kinds[k % 4]
        nel = max(1, int(rng.integers(1, 8000)) // es)
        off = (off + es - 1) // es * es
        if k % 2 == 0:
            off += (dst_phase - off) % 16          # the destination's phase
        else:
            off += es * int(rng.integers(0, 16 // es))
        dsts.append({"name": f"d{k}", "dtype": dt, "shape": (nel,)})
        ents.append({"name": f"e{k}", "dtype": dt, "shape": (nel,), "offset": off, "dst": k})
        off += nel * es
    return Manifest("tiny_phases", ents, dsts, off + 32, "bits", seed)


@pytest.mark.parametrize("kind", ["device", "pinned", "direct_pinned"])
def test_tiny_only_launches_at_every_phase(kind):
    m = _tiny_phase_manifest()
    # whole-blob chunks (one tiny-only launch), and 64 KiB chunks that cut pieces at chunk
    # starts (source phase 0) and ends
    for chunk in (1 << 30, 64 << 10):
        st = load_and_compare(m, kind, chunk=chunk, misalign=8, host_slots=0)
        assert st["n_slabs"] == 0 and st["n_bulk"] == 0 and st["n_tiny"] >= m.n_entries


def test_back_to_back_loads_and_reuse():
    """Loads on one plan run in order; the plan can be reused; the last load wins."""
    m = cfg_dense()
    blob, ref = reference(m)
    other = np.random.default_rng(1).integers(0, 256, size=blob.size, dtype=np.uint8)
    d = DeviceDsts(m)
    a = torch.from_numpy(other).to("cuda")
    b = torch.from_numpy(blob).pin_memory()
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=256 << 10) as plan:
        for _ in range(3):
            plan.load_async(cfa.Source.device(a.data_ptr()))
            plan.load_async(cfa.Source.pinned(b.data_ptr()))
        plan.wait_layer()
        ck = plan.checksums()
    for j in range(m.n_dsts):
        assert np.array_equal(d.host_bytes(j), ref.dst[j])
    assert np.array_equal(ck, ref.cksum)


def test_checksums_of_each_load_are_its_own():
    """A load accumulates into the checksum half cleared before it and clears the other one for
    the next load: read after each of several alternating loads, the checksums are that load's
    alone; cfa_reset_checksums then clears the current half for cfa_unpack_chunks_async."""
    m = cfg_dense()
    blob, ref = reference(m)
    other = np.random.default_rng(2).integers(0, 256, size=blob.size, dtype=np.uint8)
    ref_other = oracle.unpack(m, other)
    d = DeviceDsts(m)
    a = torch.from_numpy(other).to("cuda")
    b = torch.from_numpy(blob).pin_memory()
    S = 256 << 10
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=S) as plan:
        for k in range(5):
            if k % 2 == 0:
                plan.load_async(cfa.Source.device(a.data_ptr()))
                want = ref_other.cksum
            else:
                plan.load_async(cfa.Source.pinned(b.data_ptr()))
                want = ref.cksum
            assert np.array_equal(plan.checksums(), want), k
        plan.reset_checksums()
        stage = torch.empty(S, dtype=torch.uint8, device="cuda")
        for c in range(plan.info()["n_chunks"]):
            part = other[c * S:(c + 1) * S]
            stage[:part.size].copy_(torch.from_numpy(part))
            plan.unpack_chunks_async(c, c + 1, stage.data_ptr())
        torch.cuda.synchronize()
        assert np.array_equal(plan.checksums(), ref_other.cksum)
    for j in range(m.n_dsts):
        assert np.array_equal(d.host_bytes(j), ref_other.dst[j])


def test_layer_readiness_consumer_stream_and_host():
    m = dense_config("dense_layers", 65, layers=4, hidden=512, n_q=8, n_kv=2, head_dim=64,
                     inter=1536, vocab=1000)
    blob, ref = reference(m)
    h = torch.from_numpy(blob).pin_memory()
    d = DeviceDsts(m)
    consumer = torch.cuda.Stream()
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=1 << 20,
                  timing=True) as plan:
        groups = plan.info()["n_layers"]
        assert groups == m.n_groups() == 6
        plan.load_async(cfa.Source.pinned(h.data_ptr()))
        snaps = {}
        for g in range(groups):
            plan.wait_layer(g, stream=consumer)
            with torch.cuda.stream(consumer):
                for j in sorted(set(int(m.e_dst[i]) for i in np.nonzero(m.e_layer == g)[0])):
                    snaps[j] = d.view(j).clone()
        consumer.synchronize()
        for j, t in snaps.items():
            assert np.array_equal(t.cpu().numpy(), ref.dst[j]), m.d_name[j]
        assert len(snaps) == m.n_dsts
        # host waits
        plan.load_async(cfa.Source.pinned(h.data_ptr()))
        for g in range(groups):
            plan.wait_layer(g)
        plan.wait_layer()
        t = plan.layer_times()
        st = plan.stats()
    assert (t >= 0).all() and float(t.max()) <= st["load_ms"] + 1e-3
    assert st["h2d_ms"] > 0 and st["unpack_ms"] > 0


def test_wait_times_out_on_a_slow_source_then_completes():
    m = cfg_dense()
    blob, ref = reference(m)
    cb = CallbackSource(m, delay_us=300_000)  # every fill call sleeps 0.3 s on the host
    d = DeviceDsts(m)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=1 << 20) as plan:
        plan.load_async(cb.source())
        st = plan.try_wait_layer(cfa.ALL, timeout_ns=1_000_000)
        assert cfa._lib.STATUS[st] == "CFA_ERR_TIMEOUT"
        plan.wait_layer()  # no limit: completes
        ck = plan.checksums()
    for j in range(m.n_dsts):
        assert np.array_equal(d.host_bytes(j), ref.dst[j])
    assert np.array_equal(ck, ref.cksum)


def test_failing_source_is_reported_and_the_plan_recovers():
    m = cfg_dense()
    blob, ref = reference(m)
    bad = CallbackSource(m, fail_from=m.blob_bytes // 2)
    good = CallbackSource(m)
    d = DeviceDsts(m)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=256 << 10) as plan:
        plan.load_async(bad.source())
        with pytest.raises(cfa.CfaError) as e:
            plan.wait_layer()
        assert e.value.name == "CFA_ERR_SOURCE"
        plan.load_async(good.source())
        plan.wait_layer()
        ck = plan.checksums()
    for j in range(m.n_dsts):
        assert np.array_equal(d.host_bytes(j), ref.dst[j])
    assert np.array_equal(ck, ref.cksum)


def test_caller_managed_staging():
    """cfa_unpack_chunks_async: the caller stages chunks itself, one launch per chunk."""
    m = cfg_moe()
    blob, ref = reference(m)
    S = 1 << 20
    d = DeviceDsts(m)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=S, dev_slots=0,
                  host_slots=0) as plan:
        n = plan.info()["n_chunks"]
        plan.reset_checksums()
        stage = torch.empty(S, dtype=torch.uint8, device="cuda")
        for c in range(n):
            part = blob[c * S:(c + 1) * S]
            stage[:part.size].copy_(torch.from_numpy(part))
            plan.unpack_chunks_async(c, c + 1, stage.data_ptr())
        torch.cuda.synchronize()
        # the checksum buffer is read through a load-free path: compare destinations only,
        # then a normal load for the checksums
        for j in range(m.n_dsts):
            assert np.array_equal(d.host_bytes(j), ref.dst[j])


def test_periodic_source():
    """A blob defined as periodic is streamed from a pool of one period."""
    m = dense_config("dense_periodic", 66, layers=3, hidden=512, n_q=8, n_kv=2, head_dim=64,
                     inter=1536, vocab=1000, chunk_bytes=1 << 20, period=4 << 20)
    blob, ref = reference(m)
    pool_h = torch.from_numpy(m.blob_range(0, m.period)).pin_memory()
    pool_d = pool_h.to("cuda")
    pool_pg = aligned_host_copy(m.blob_range(0, m.period))
    for src in (cfa.Source.pinned(pool_h.data_ptr(), period=m.period),
                cfa.Source.device(pool_d.data_ptr(), period=m.period),
                cfa.Source.host_direct(pool_pg.ctypes.data, period=m.period),
                cfa.Source.host(pool_pg.ctypes.data, period=m.period)):
        d = DeviceDsts(m)
        with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=1 << 20) as plan:
            plan.load_async(src)
            plan.wait_layer()
            ck = plan.checksums()
        for j in range(m.n_dsts):
            assert np.array_equal(d.host_bytes(j), ref.dst[j])
        assert np.array_equal(ck, ref.cksum)


def test_empty_plan_loads():
    with cfa.Plan(cfa.make_entries([], [], [], []), [], 0) as plan:
        plan.load_async(cfa.Source.device(0))
        plan.wait_layer()
        assert plan.checksums().size == 0


def test_tma_wait_that_runs_out_ends_the_kernel_cleanly():
    """The TMA kernel's waits are bounded: with its loader issuing nothing, the first wait for a
    staged sub-block runs out, the kernel flags status 2 and returns, and the context loads
    correctly afterwards."""
    import ctypes
    lib = cfa._lib.load()
    word = ctypes.c_int(-1)
    assert lib.cfa_selftest_wait_timeout(-1, ctypes.byref(word)) == 0
    assert word.value == 2
    torch.cuda.synchronize()
    load_and_compare(CONFIGS["dense"](), "device", chunk=1 << 20)


def test_two_plans_load_at_once_from_two_threads():
    """Two plans (different checkpoints, sources and destinations) loading at the same time on
    their own streams from their own host threads: each matches the oracle."""
    import threading
    cases = []
    for name, kind in (("moe", "callback"), ("f32_tp", "pinned")):
        m = CONFIGS[name]()
        blob, ref = reference(m)
        keep = []
        src = make_source(kind, m, blob, keep)
        d = DeviceDsts(m)
        plan = cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=256 << 10)
        cases.append((m, ref, src, d, plan, keep, torch.cuda.Stream()))
    errors, results = [], {}

    def run(k):
        m, ref, src, d, plan, keep, stream = cases[k]
        try:
            torch.cuda.set_device(0)
            for _ in range(3):
                plan.load_async(src, stream)
                plan.wait_layer()
            results[k] = plan.checksums()
        except Exception as e:  # reported below
            errors.append(e)

    threads = [threading.Thread(target=run, args=(k,)) for k in range(len(cases))]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=300)
    assert not errors, errors
    torch.cuda.synchronize()
    for k, (m, ref, src, d, plan, keep, stream) in enumerate(cases):
        for j in range(m.n_dsts):
            assert np.array_equal(d.host_bytes(j), ref.dst[j]), (m.name, m.d_name[j])
        assert np.array_equal(results[k], ref.cksum), m.name
        assert d.guards_intact()
        plan.close()


@pytest.mark.parametrize("slots,pull", [(3, None), (2, None), (2, 0), (3, 50)])
def test_timeline_orders_copies_before_unpacks(slots, pull):
    """Per-chunk timeline of a staged load (the transfer's interval covers the copy engine's
    copies and the pull kernel's, whichever ran)."""
    m = CONFIGS["dense"]()
    blob, ref = reference(m)
    keep = []
    d = DeviceDsts(m)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=1 << 20,
                  timing=True, dev_slots=slots, pull_percent=pull) as plan:
        plan.load_async(make_source("pinned", m, blob, keep))
        plan.wait_layer()
        t = plan.timeline()
        n = plan.stats()["n_chunks"]
        assert t.shape == (n, 4)
        assert (t[:, 0] >= 0).all() and (t[:, 1] >= t[:, 0]).all()
        ran = t[:, 2] >= 0
        assert ran.sum() >= n - 1
        # a chunk is unpacked only after its copy into the device slot has finished
        assert (t[ran, 2] >= t[ran, 1] - 1e-3).all() and (t[ran, 3] >= t[ran, 2]).all()
        # with k device slots, chunk c + k's transfer waits for chunk c's unpack
        assert (t[slots:, 0] >= t[:-slots, 3] - 1e-3)[ran[:-slots]].all()
        # a device-resident source: no copies, one merged launch over every chunk
        plan.load_async(make_source("device", m, blob, keep))
        plan.wait_layer()
        t = plan.timeline()
        assert (t[:, 0] == -1).all() and (t[:, 1] == -1).all()
        assert len(set(t[:, 2].tolist())) == 1 and (t[:, 3] > t[:, 2]).all()
        ck = plan.checksums()
    assert np.array_equal(ck, ref.cksum)


@pytest.mark.parametrize("kind", ["pinned", "host", "callback"])
def test_staged_load_skips_chunks_no_piece_reads(kind):
    """An expert-parallel rank leaves whole chunks of other ranks' experts unread: a staged load
    neither fills, copies nor unpacks them, and they take no staging slot, so the busy chunks'
    copies follow one another with the two device slots alternating between busy chunks."""
    m = cfg_moe_ep()
    blob, ref = reference(m)
    keep = []
    d = DeviceDsts(m)
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=64 << 10,
                  timing=True, fill_threads=4, dev_slots=2) as plan:
        n = plan.info()["n_chunks"]
        busy = np.zeros(n, dtype=bool)
        busy[plan.pieces()["chunk"]] = True
        assert 0 < busy.sum() < n - 8  # whole chunks of other ranks' experts
        for _ in range(2):
            plan.load_async(make_source(kind, m, blob, keep))
            plan.wait_layer()
            ck = plan.checksums()
            for j in range(m.n_dsts):
                assert np.array_equal(d.host_bytes(j), ref.dst[j])
            assert np.array_equal(ck, ref.cksum)
            assert d.guards_intact()
            t = plan.timeline()
            assert (t[~busy] == -1).all()
            tb = t[busy]
            assert (tb[:, 0] >= 0).all() and (tb[:, 1] >= tb[:, 0]).all()
            assert (tb[:, 2] >= tb[:, 1] - 1e-3).all() and (tb[:, 3] >= tb[:, 2]).all()
            assert (tb[1:, 0] >= tb[:-1, 1] - 1e-3).all()  # transfers in chunk order
            # the slot of busy chunk k + 2 is the slot of busy chunk k
            assert (tb[2:, 0] >= tb[:-2, 3] - 1e-3).all()
            lt = plan.layer_times()
            assert (lt > 0).all() and (lt <= plan.stats()["load_ms"] + 1e-3).all()


def test_destroy_while_a_load_is_in_flight():
    """Closing a plan with a load still running (a slow callback source) waits for the load and
    frees everything; the destinations hold the complete load."""
    m = CONFIGS["moe"]()
    blob, ref = reference(m)
    cb = CallbackSource(m, delay_us=300)
    d = DeviceDsts(m)
    plan = cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=256 << 10)
    plan.load_async(cb.source())
    timeout = {v: k for k, v in cfa._lib.STATUS.items()}["CFA_ERR_TIMEOUT"]
    assert plan.try_wait_layer(timeout_ns=0) == timeout
    plan.close()
    torch.cuda.synchronize()
    for j in range(m.n_dsts):
        assert np.array_equal(d.host_bytes(j), ref.dst[j]), m.d_name[j]
    assert d.guards_intact()


@pytest.mark.parametrize("stage_slices", [False, True])
@pytest.mark.parametrize("chunk", [256, 64 << 10, 1 << 20])
@pytest.mark.parametrize("cfg", ["dense_tp", "f32_tp", "moe_tp", "bf16_f32norm_tp"])
def test_column_slices_from_pinned_memory(cfg, chunk, stage_slices):
    """Pinned sources read column slices in place beside the copy ring (default), or copy them
    through the slots as strided 2-D copies (stage_slices)."""
    m = CONFIGS[cfg]()
    st = load_and_compare(m, "pinned", chunk=chunk, stage_slices=stage_slices)
    if chunk >= 64 << 10:  # with 256-byte chunks every slice row is cut into contiguous pieces
        assert st["n_strided"] > 0


def test_layer_readiness_waits_for_column_slices_read_in_place():
    """A readiness group of a tensor-parallel rank is signalled only after its column slices,
    read in place on their own stream, are written: snapshots taken on a consumer stream right
    after each group's event equal the oracle."""
    m = dense_config("tp_layers", 66, layers=4, hidden=512, n_q=8, n_kv=2, head_dim=64,
                     inter=1536, vocab=1000, tp=2, rank=1)
    blob, ref = reference(m)
    h = torch.from_numpy(blob).pin_memory()
    d = DeviceDsts(m)
    consumer = torch.cuda.Stream()
    with cfa.Plan(entries_for(m), d.cfa_dsts, m.blob_bytes, chunk_bytes=256 << 10) as plan:
        groups = plan.info()["n_layers"]
        for rep in range(3):
            d.buf.fill_(0xA5)
            plan.load_async(cfa.Source.pinned(h.data_ptr()))
            snaps = {}
            for g in range(groups):
                plan.wait_layer(g, stream=consumer)
                with torch.cuda.stream(consumer):
                    for j in sorted(set(int(m.e_dst[i]) for i in np.nonzero(m.e_layer == g)[0])):
                        snaps[j] = d.view(j).clone()
            consumer.synchronize()
            for j, t in snaps.items():
                assert np.array_equal(t.cpu().numpy(), ref.dst[j]), (rep, m.d_name[j])
            assert len(snaps) == m.n_dsts
