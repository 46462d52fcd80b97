#!/usr/bin/env python3
"""Benchmark of the GB300 checkpoint loader.

One step = one complete load of a synthetic checkpoint into its final per-parameter layout, i.e.
every stage of the path: chunked staging, host->device transfer (e2e only), the unpack kernels
with fused layouts and per-tensor checksums, readiness events, and the checksum read-back (e2e
only).  The headline workload is the largest one that fits one GPU: a Llama-3-70B-shaped bf16
checkpoint (80 layers, q/k/v and gate/up fused; 141.1 GB) streamed in 1 GiB chunks from an
8 GiB pool (the blob is defined periodic with that period).

Printed on one JSON line (rank 0):
  value      unpacked GB/s into the final layout, kernel only: the blob already sits in HBM
             (device source); algorithmic bytes = every source byte read once + every
             destination byte written once, over the device time of K steps
  e2e        the same metric end to end through the C ABI with a pinned HOST blob: every step
             copies the whole checkpoint host->device (cudaMemcpyAsync on the loader's copy
             stream) and reads the checksums back; also seconds per model, the fraction of the
             measured host->device bandwidth, and the per-layer ready times of one load
  roofline   the unpack kernels against the measured HBM copy bandwidth
  cpu_baseline  the oracle (plain CPU loader) on a bounded sample, on this host's cores
  configs    the same kernel-only and end-to-end figures for the other workloads: 1,000 tiny
             tensors and the Mixtral workload's 200k extras alone (L2 flushed between steps),
             Llama-3-8B bf16 (with the end-to-end attribution), Llama-3-8B fp32 -> bf16 (the
             oracle over the whole model on all host cores), Mixtral-8x7B bf16

--impl reference times the oracle as the reference arm.  --gpus N runs N independent replicas
(one process per GPU under torchrun); nothing in the path is sharded or exchanged.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "unpacked GB/s into final layout (% of HBM peak); end-to-end H2D load s per model"
UNIT = "GB/s"
HBM_FALLBACK_GBS = 6800.0
L2_BYTES = 129e6
HEADLINE = "llama3_70b_bf16"
CONFIGS = ("tiny_1000", "mixtral_extras_200k", "llama3_8b_bf16", "llama3_8b_f32_rne",
           "mixtral_8x7b_bf16")
# workloads whose inputs fit in L2: the kernel-only steps flush it (a 1 GiB write) in between
L2_FLUSHED = ("tiny_1000", "mixtral_extras_200k")
# the oracle over every tensor (on all host cores) for these; a bounded sample for the others
CPU_FULL = ("tiny_1000", "llama3_8b_f32_rne")


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=HEADLINE)
    ap.add_argument("--configs", default=",".join(CONFIGS),
                    help="comma-separated workloads measured after the headline one, or 'none'")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-attribution", action="store_true",
                    help="skip the end-to-end attribution measurements")
    ap.add_argument("--timeline", default=None, metavar="PATH",
                    help="write the per-chunk timeline (copy and unpack intervals) of the timed "
                         "pinned load of the attribution to PATH as JSON")
    ap.add_argument("--stage-slices", action="store_true",
                    help="pinned sources: copy column slices through the device slots instead of "
                         "reading them in place (for comparison)")
    ap.add_argument("--vector-only", dest="bulk", action="store_false",
                    help="copy every slab with the 16-byte vector kernel instead of the TMA bulk "
                         "kernel (for comparison)")
    ap.add_argument("--slab-kib", type=int, default=None,
                    help="destination KiB per block-level work item (default: the library's)")
    ap.add_argument("--dst-order", default="index", choices=["index", "blob"],
                    help="destinations laid out in index order (default) or in blob order, so "
                         "that a load writes them front to back (for comparison)")
    ap.add_argument("--e2e-steps", type=int, default=None,
                    help="steps of the end-to-end measurement (default: min(steps, 20))")
    return ap.parse_args()


# ------------------------------------------------------------------------------------------
# Small cases of the workloads' kernel classes for ncu captures (a few GB on the device, inputs
# larger than L2): 2 layers and a 32k vocabulary of the 8B and 70B shapes.
_SMALL = {
    "llama3_8b_bf16_2layer_v32k": dict(seed=2, layers=2, hidden=4096, n_q=32, n_kv=8,
                                       head_dim=128, inter=14336, vocab=32000),
    # fp32 -> bf16 class, 256-byte aligned tensors (~2.8 GB blob)
    "llama3_8b_f32_rne_2layer_v32k": dict(seed=3, layers=2, hidden=4096, n_q=32, n_kv=8,
                                          head_dim=128, inter=14336, vocab=32000,
                                          src_dtype="f32"),
    # the same packed at 4-byte offsets with gaps: sources off the 16-byte grid
    "llama3_8b_f32_rne_2layer_v32k_odd": dict(seed=8, layers=2, hidden=4096, n_q=32, n_kv=8,
                                              head_dim=128, inter=14336, vocab=32000,
                                              src_dtype="f32", align=4, jitter=3),
    # the 70B layer shapes, 1 GiB chunks (~4.5 GB blob): the headline's TMA kernel
    "llama3_70b_bf16_2layer_v32k": dict(seed=5, layers=2, hidden=8192, n_q=64, n_kv=8,
                                        head_dim=128, inter=28672, vocab=32000,
                                        chunk_bytes=1 << 30),
    # tensor-parallel rank 3 of 8 of the 70B shape: column slices of o and down
    "llama3_70b_bf16_2layer_v32k_tp8r3": dict(seed=5, layers=2, hidden=8192, n_q=64, n_kv=8,
                                              head_dim=128, inter=28672, vocab=32000, tp=8,
                                              rank=3, chunk_bytes=1 << 30),
}


def make_workload(name):
    import workloads
    if name in _SMALL:
        return workloads.dense_config(name, **_SMALL[name])
    try:
        return workloads.named_config(name)
    except KeyError:
        raise SystemExit(f"unknown workload {name}")


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": HBM_FALLBACK_GBS}, "fallback"


KERNEL_SOURCES = ("cfa_unpack.cu", "cfa_bulk.cu", "cfa_device.cuh")


def kernel_source_hash(files=KERNEL_SOURCES):
    """sha256 over the named kernel source files (csrc/), in order."""
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2607_18957_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def recorded_traffic(workload):
    """DRAM bytes per launch from the committed ncu summary, if the sources of the captured
    kernel (the record's `sources`, else all kernel sources) are unchanged since."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except OSError:
        return None
    r = rec.get(workload)
    if not r or r.get("kernel_sha256") != kernel_source_hash(tuple(r.get("sources",
                                                                          KERNEL_SOURCES))):
        return None
    return r.get("dram_bytes_per_launch")


def kernel_names(st):
    """The unpack kernels one load of a plan with these stats launches."""
    out = []
    if st["n_bulk"]:
        out.append("cfa_bulk_kernel (TMA bulk copies)")
    if st["n_slabs"]:
        out.append("cfa_unpack_kernel (16-byte vector slabs" + (", tiny pieces interleaved)"
                                                               if st["n_tiny"] else ")"))
    elif st["n_tiny"]:
        out.append("cfa_tiny_kernel (tiny pieces)")
    if st["n_strided"]:
        out.append("cfa_strided_kernel (column slices)")
    return " + ".join(out)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled while the timed region runs."""

    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 10:
                    continue
                if self.uuid and parts[1] != self.uuid and not self.uuid.endswith(parts[1]) \
                        and not parts[1].endswith(self.uuid):
                    continue
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        mhz = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        maxs = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for k, nm in enumerate(names):
                if r[6 + k].lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(mhz) if mhz else None,
                "sm_max_mhz": max(maxs) if maxs else None,
                "samples": len(rows), "reasons": sorted(reasons)}


# ------------------------------------------------------------------------------------------
def attribution_sizes(source_bytes, threads):
    """Bytes of the pageable source copied to the device (1 GiB) and bytes per thread of the
    host memcpy (4 GiB split evenly), both capped by the source for a smaller checkpoint."""
    gib = 1 << 30
    return min(gib, source_bytes), min(4 * gib, source_bytes) // max(1, threads)


def attribution(m, host, dsts, entries, stream, args, h2d_gbs, sweep=False):
    """Where end-to-end time goes: (CFA_OPT_TIMING) per-layer readiness of one pinned load, the
    pinned blob read in place by the kernels (no copy engine), the host link for pinned and
    pageable memory, host memcpy with the loader's fill threads, a load from a pageable copy of
    the checkpoint through the pinned staging ring and the same copy read in place, and a load
    from a safetensors file."""
    from concurrent.futures import ThreadPoolExecutor

    import numpy as np
    import torch

    import paper_2607_18957_gb300 as cfa
    out = {"h2d_pinned_gbs": round(h2d_gbs, 2)}
    # first, next to the end-to-end steps: per-layer readiness of one timed pinned load
    plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                    dev_slots=3, host_slots=0, timing=True, bulk=args.bulk,
                    stage_slices=args.stage_slices)
    plan.load_async(cfa.Source.pinned(host.data_ptr(), period=m.period or 0), stream)
    plan.wait_layer()
    t = plan.layer_times()
    st = plan.stats()
    if args.timeline:
        tl = plan.timeline()
        with open(args.timeline, "w") as f:
            json.dump({"workload": m.name, "chunk_bytes": m.chunk_bytes,
                       "source": "pinned host blob, 3 device staging slots",
                       "columns": ["h2d_begin_ms", "h2d_end_ms", "unpack_begin_ms",
                                   "unpack_end_ms"],
                       "chunks": [[round(float(x), 4) for x in row] for row in tl],
                       "layer_ready_ms": [round(float(x), 4) for x in t]}, f)
    plan.close()
    # the same staged load with each chunk's ranges split half and half between the copy engine
    # and the SM pull kernel (the default pulls all of it; the copy engine alone is in every
    # workload's e2e record)
    for pct, key in ((50, "e2e_half_copy_engine"),):
        plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                        dev_slots=3, host_slots=0, bulk=args.bulk,
                        stage_slices=args.stage_slices, pull_percent=pct)
        src = cfa.Source.pinned(host.data_ptr(), period=m.period or 0)
        plan.load_async(src, stream)
        plan.checksums()
        steps = [_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                 for _ in range(3)]
        plan.close()
        out[key + "_step_ms"] = [round(x, 1) for x in steps]
    out["layer_ready_ms"] = {"first_group": round(float(t[0]), 2),
                             "median_group": round(float(np.median(t)), 2),
                             "last_group": round(float(t[-1]), 2),
                             "groups": int(t.size), "load_ms": round(st["load_ms"], 2),
                             "all": [round(float(x), 2) for x in t],
                             "h2d_ms": round(st["h2d_ms"], 2),
                             "unpack_ms": round(st["unpack_ms"], 2)}
    # the same pinned blob read in place by the unpack kernels over NVLink-C2C (no copy
    # engine, no slots): every step, to show step-to-step spread beside the staged steps
    plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                    dev_slots=0, host_slots=0, bulk=args.bulk)
    src = cfa.Source.host_direct(host.data_ptr(), period=m.period or 0)
    try:
        plan.load_async(src, stream)
        plan.checksums()
        steps = [_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                 for _ in range(6)]
        out["e2e_direct_pinned_s_per_model"] = round(statistics.mean(steps) / 1e3, 4)
        out["e2e_direct_pinned_step_ms"] = [round(x, 1) for x in steps]
    except cfa.CfaError as e:
        out["e2e_direct_pinned"] = f"unavailable: {e}"
    plan.close()
    gib = 1 << 30
    threads = max(1, len(os.sched_getaffinity(0)))
    raw = np.empty(m.source_bytes() + 256, dtype=np.uint8)
    pageable = raw[(-raw.ctypes.data) % 256:][:m.source_bytes()]  # 256-byte aligned view
    pageable[:] = host.numpy()                                   # the same bytes, pageable
    n_h2d, part = attribution_sizes(pageable.size, threads)
    dtmp = torch.empty(n_h2d, dtype=torch.uint8, device="cuda")
    src_t = torch.from_numpy(pageable[:n_h2d])
    best = min(_timed(lambda: dtmp.copy_(src_t), stream) for _ in range(5))
    out["h2d_pageable_gbs"] = round(n_h2d / best / 1e6, 2)
    del dtmp
    dst = np.empty(part * threads, dtype=np.uint8)

    def cp(k):
        np.copyto(dst[k * part:(k + 1) * part], pageable[k * part:(k + 1) * part])
    with ThreadPoolExecutor(threads) as ex:
        list(ex.map(cp, range(threads)))                         # warm
        t0 = time.perf_counter()
        list(ex.map(cp, range(threads)))
        out["host_memcpy_gbs"] = round(dst.size / (time.perf_counter() - t0) / 1e9, 2)
    out["host_threads"] = threads
    del dst
    # a pageable copy of the checkpoint as a HOST source: by default the SM pull kernel reads it
    # straight into the device slots; with pull_percent 0 the fill threads copy it into the
    # pinned ring and the copy engine takes it from there
    for pct, key in ((None, "e2e_pageable"), (0, "e2e_pageable_ring")):
        kw = {} if pct is None else {"pull_percent": pct}
        plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                        dev_slots=3, host_slots=2, fill_threads=threads, bulk=args.bulk, **kw)
        src = cfa.Source.host(pageable.ctypes.data, period=m.period or 0)
        plan.load_async(src, stream)
        plan.checksums()
        ms = min(_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                 for _ in range(2))
        plan.close()
        out[key + "_s_per_model"] = round(ms / 1e3, 4)
        out[key + "_gbs"] = round(m.blob_bytes / ms / 1e6, 2)
    if sweep:
        out["fill_threads_sweep"] = fill_thread_sweep(m, pageable, dsts, entries, stream, args,
                                                      part * threads)
    # the same pageable bytes read in place by the unpack kernel over NVLink-C2C (no staging)
    plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                    dev_slots=0, host_slots=0, bulk=args.bulk)
    src = cfa.Source.host_direct(pageable.ctypes.data, period=m.period or 0)
    try:
        plan.load_async(src, stream)
        plan.checksums()
        ms = min(_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                 for _ in range(2))
        out["e2e_direct_pageable_s_per_model"] = round(ms / 1e3, 4)
        # the kernel reads only the bytes the entries cover (a tensor-parallel rank: its shard)
        out["e2e_direct_pageable_link_gbs"] = round(plan.stats()["bytes_read"] / ms / 1e6, 2)
    except cfa.CfaError as e:
        out["e2e_direct_pageable"] = f"unavailable: {e}"
    plan.close()
    # last: writing the file leaves the host busy with write-back for a while
    out.update(file_attribution(m, pageable, dsts, stream, args, threads))
    del pageable, raw
    return out


def fill_thread_sweep(m, pageable, dsts, entries, stream, args, memcpy_bytes):
    """Host memcpy rate and the pageable load through the pinned ring, per fill thread count:
    where the host side of the staged path saturates on this machine."""
    from concurrent.futures import ThreadPoolExecutor

    import numpy as np

    import paper_2607_18957_gb300 as cfa
    rows = []
    dst = np.empty(memcpy_bytes, dtype=np.uint8)
    for t in (4, 8, 16, 32, 48, 64):
        part = memcpy_bytes // t

        def cp(k):
            np.copyto(dst[k * part:(k + 1) * part], pageable[k * part:(k + 1) * part])
        with ThreadPoolExecutor(t) as ex:
            list(ex.map(cp, range(t)))
            t0 = time.perf_counter()
            list(ex.map(cp, range(t)))
            memcpy_gbs = part * t / (time.perf_counter() - t0) / 1e9
        plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                        dev_slots=3, host_slots=2, fill_threads=t, bulk=args.bulk,
                        pull_percent=0)  # the fill threads' ring, not the SM pull
        src = cfa.Source.host(pageable.ctypes.data, period=m.period or 0)
        plan.load_async(src, stream)
        plan.checksums()
        ms = min(_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                 for _ in range(2))
        plan.close()
        rows.append({"threads": t, "host_memcpy_gbs": round(memcpy_gbs, 2),
                     "e2e_pageable_s_per_model": round(ms / 1e3, 4),
                     "e2e_pageable_gbs": round(m.blob_bytes / ms / 1e6, 2)})
    del dst
    return rows


def file_attribution(m, pageable, dsts, stream, args, threads):
    """A load from a safetensors file of the checkpoint (its header read by the library, the
    data section read by the fill threads into the pinned ring: with pread, or copied from a
    read-only mapping of the file; or the mapping read in place by the unpack kernels).  The file is written just before, so buffered reads come
    from the page cache; O_DIRECT reads (data section at a 4 KiB boundary, so whole blocks land
    in the pinned slots) come from the storage under the temporary directory.  The file is
    removed afterwards."""
    import shutil
    import struct
    import tempfile

    import paper_2607_18957_gb300 as cfa
    from workloads.stfile import file_tensors, header_bytes, targets_for
    if m.period is not None:
        return {"e2e_file": "not measured: the blob is defined by a period, no file of it"}
    d = tempfile.mkdtemp(prefix="cfa_bench_")
    try:
        if shutil.disk_usage(d).free < m.blob_bytes * 1.2:
            return {"e2e_file": f"not measured: under {m.blob_bytes * 1.2 / 1e9:.0f} GB free"}
        path = os.path.join(d, "model.safetensors")
        hdr = header_bytes(file_tensors(m), data_align=4096)
        t0 = time.perf_counter()
        with open(path, "wb") as f:
            f.write(struct.pack("<Q", len(hdr)))
            f.write(hdr)
            f.write(memoryview(pageable))
            f.flush()
            os.fsync(f.fileno())
        write_s = time.perf_counter() - t0
        st = cfa.Safetensors.open(path)
        plan = cfa.Plan(st.entries(targets_for(m)), dsts.cfa_dsts, st.data_bytes,
                        chunk_bytes=m.chunk_bytes, dev_slots=3, host_slots=2,
                        fill_threads=threads, bulk=args.bulk)
        with cfa.Source.file(path, st.data_offset) as src:
            plan.load_async(src, stream)
            plan.checksums()
            ms = min(_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                     for _ in range(2))
        out = {"e2e_file_s_per_model": round(ms / 1e3, 4),
               "e2e_file_gbs": round(m.blob_bytes / ms / 1e6, 2),
               "file": f"safetensors, {len(st.tensors)} tensors, page cache (written and "
                       f"synced in {write_s:.1f} s just before)"}
        with cfa.Source.file(path, st.data_offset, mapped=True) as src:
            plan.load_async(src, stream)
            plan.checksums()
            ms = min(_timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
                     for _ in range(2))
        out["e2e_file_mapped_s_per_model"] = round(ms / 1e3, 4)
        out["e2e_file_mapped_gbs"] = round(m.blob_bytes / ms / 1e6, 2)
        try:  # the mapping read in place by the unpack kernels over the host link
            with cfa.Source.file(path, st.data_offset, in_place=True) as src:
                plan.load_async(src, stream)
                plan.checksums()
                ms = min(_timed(lambda: (plan.load_async(src, stream), plan.checksums()),
                                stream) for _ in range(2))
            out["e2e_file_in_place_s_per_model"] = round(ms / 1e3, 4)
            out["e2e_file_in_place_gbs"] = round(m.blob_bytes / ms / 1e6, 2)
        except cfa.CfaError as e:
            out["e2e_file_in_place"] = f"unavailable: {e}"
        try:
            with cfa.Source.file(path, st.data_offset, direct=True) as src:
                plan.load_async(src, stream)
                plan.checksums()
                ms = _timed(lambda: (plan.load_async(src, stream), plan.checksums()), stream)
            out["e2e_file_direct_s_per_model"] = round(ms / 1e3, 4)
            out["e2e_file_direct_gbs"] = round(m.blob_bytes / ms / 1e6, 2)
        except cfa.CfaError as e:
            out["e2e_file_direct"] = f"unavailable: {e}"
        plan.close()
        return out
    finally:
        shutil.rmtree(d, ignore_errors=True)


_COPY = {1: "u8", 2: "u16", 4: "u32", 8: "u64"}
_CONV_CLASS = {("f32", "bf16"): 4, ("f32", "f16"): 5, ("f16", "bf16"): 6, ("bf16", "f32"): 7,
               ("f16", "f32"): 8}
_BLOB_KIND = {"bits": "random bit patterns",
              "f32mix": "fp32 normal(0, 0.02) with ties and subnormals",
              "f16fin": "finite fp16 values"}


def path_types(m):
    """(dtype string, dominant work class, its description) of a manifest: the element types
    the unpack moves (copies by size, conversions by name) and the class with the most bytes."""
    from workloads import DTYPE_SIZE
    kinds, by_class = set(), {}
    for i in range(m.n_entries):
        s, d = str(m.e_dtype[i]), str(m.d_dtype[int(m.e_dst[i])])
        n = m.e_numel(i)
        if m.e_cast[i]:
            kinds.add(f"{s}->{d}")
            cls, desc = _CONV_CLASS[(s, d)], f"{s} -> {d} conversion class"
        else:
            es = DTYPE_SIZE[s]
            kinds.add(_COPY[es])
            cls, desc = es.bit_length() - 1, f"{8 * es}-bit copy class"
        b = by_class.setdefault(cls, [0, desc])
        b[0] += n * (DTYPE_SIZE[s] + DTYPE_SIZE[d])
    cls = max(by_class, key=lambda c: by_class[c][0])
    return "+".join(sorted(kinds)), cls, by_class[cls][1]


def _timed(fn, stream):
    import torch
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    fn()
    b.record(stream)
    b.synchronize()
    return a.elapsed_time(b)


def host_cores():
    """Cores this process may run on (the box's own count, not this container's)."""
    return len(os.sched_getaffinity(0))


def _dst_order(m):
    """Destinations in blob order (by the first blob byte any of their entries reads)."""
    return sorted(range(m.n_dsts),
                  key=lambda j: min(int(m.e_offset[i]) for i in m.entries_of_dst(j)))


def _oracle_one(m, j):
    """Destination j through the oracle: (unpack seconds, algorithmic bytes).  Generating the
    source window is outside the timed call."""
    import oracle
    es = m.entries_of_dst(j)
    lo = min(int(m.e_offset[i]) for i in es)
    hi = max(int(m.e_offset[i]) + m.e_extent(i) for i in es)
    window = m.blob_range(lo, hi - lo)
    t0 = time.perf_counter()
    r = oracle.unpack(m, window, blob_begin=lo, dsts=[j])
    dt = time.perf_counter() - t0
    assert r.status == 0
    return dt, sum(m.e_nbytes(i) for i in es) + m.d_nbytes(j)


def cpu_baseline(m, seconds, steps=None):
    """The oracle, as it stands, on destinations in blob order until `seconds` of CPU time (or
    one destination per step for the reference arm; seconds=None: every destination).
    Generation of the sample's blob bytes is outside the timed region.  Returns (GB/s, bytes,
    secs, description, per-step times)."""
    order = _dst_order(m)
    done_bytes, busy, used, step_times = 0, 0.0, [], []
    k = 0
    while True:
        j = order[k % len(order)]
        k += 1
        dt, nb = _oracle_one(m, j)
        done_bytes += nb
        busy += dt
        used.append(m.d_name[j])
        step_times.append((dt, nb))
        if steps is not None:
            if len(step_times) >= steps:
                break
        elif (seconds is not None and busy >= seconds) or k >= len(order):
            break
    whole = seconds is None and steps is None
    desc = (f"{'all ' if whole else ''}{len(used)} destination tensor(s) of {m.name} in blob "
            f"order ({used[0]} ...), {done_bytes / 1e9:.2f} GB of algorithmic bytes, single "
            "thread")
    return done_bytes / busy / 1e9, done_bytes, busy, desc, step_times


_POOL_MANIFESTS = {}


def _pool_task(args):
    key, j = args
    if key not in _POOL_MANIFESTS:  # a plain exception (not SystemExit) reaches the parent
        import workloads
        _POOL_MANIFESTS[key] = workloads.named_config(key)
    return _oracle_one(_POOL_MANIFESTS[key], j)


def cpu_baseline_all_cores(m, key, workers):
    """The oracle over every destination of `m`, one destination per task, on `workers` spawned
    processes (each runs the single-threaded oracle as it stands).  Returns the whole-model rate
    over the wall time of the pool (blob windows generated inside it, in each worker) and the
    single-thread rate over the oracle calls alone."""
    import multiprocessing as mp
    order = _dst_order(m)
    # largest first, so that the pool does not end on one big tensor
    order.sort(key=lambda j: -m.d_nbytes(j))
    ctx = mp.get_context("spawn")
    with ctx.Pool(workers) as pool:
        t0 = time.perf_counter()
        res = pool.map(_pool_task, [(key, j) for j in order], chunksize=1)
        wall = time.perf_counter() - t0
    nb = sum(b for _, b in res)
    busy = sum(t for t, _ in res)
    return {"value": round(nb / wall / 1e9, 4), "unit": UNIT, "cores": workers,
            "host_cores": host_cores(), "kind": "oracle",
            "single_thread_gbs": round(nb / busy / 1e9, 4),
            "sample": f"all {len(order)} destinations of {m.name} ({nb / 1e9:.2f} GB of "
                      f"algorithmic bytes) on {workers} processes, one destination per task; "
                      f"wall {wall:.1f} s including each task's blob-window generation"}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    m = make_workload(args.workload)
    cores = 1
    # warm-up steps, then K timed steps, each one destination tensor through the oracle
    cpu_baseline(m, 0, steps=max(args.warmup, 1))
    gbs, nbytes, busy, desc, times = cpu_baseline(m, 0, steps=args.steps)
    ms = 1e3 * sum(t for t, _ in times) / len(times)
    line = {
        "impl": "reference", "metric": METRIC, "value": round(gbs, 4), "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": path_types(m)[0],
        "data": f"synthetic (seeded counter-based generator; {_BLOB_KIND[m.blob_kind]})",
        "config": {"workload": m.name, "step": "one destination tensor per step, in blob order",
                   "parallelism": "rank 0 of replicas" if args.gpus > 1 else "single host"},
        "cpu_baseline": {"value": round(gbs, 4), "unit": UNIT, "cores": cores,
                         "host_cores": host_cores(), "kind": "oracle", "sample": desc},
        "e2e": {"value": round(gbs, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------
class Ranks:
    """The job's processes: one per GPU under torchrun (RANK / LOCAL_RANK / WORLD_SIZE /
    MASTER_* from the environment), each loading its own replica of the checkpoint.  The
    collectives only serve the timing: a barrier on both sides of the timed region, the maximum
    of the ranks' times and the sum of their units.  NCCL on GPUs; gloo on the host (tests)."""

    def __init__(self, backend="nccl", device="cuda"):
        import torch.distributed as dist
        self.dist = dist
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.device = device
        if self.world > 1:
            dist.init_process_group(backend)

    def _reduce(self, x, op):
        if self.world == 1:
            return float(x)
        import torch
        t = torch.tensor([float(x)], dtype=torch.float64, device=self.device)
        self.dist.all_reduce(t, op=op)
        return float(t.item())

    def barrier(self):
        if self.world > 1:
            self.dist.barrier()

    def max(self, x):
        return self._reduce(x, self.dist.ReduceOp.MAX)

    def sum(self, x):
        return self._reduce(x, self.dist.ReduceOp.SUM)

    def close(self):
        if self.world > 1:
            self.dist.destroy_process_group()


def whole_job_gbs(ranks, bytes_this_rank, ms_this_rank):
    """Whole-job throughput: the bytes all ranks moved over the slowest rank's time."""
    return ranks.sum(bytes_this_rank) / (ranks.max(ms_this_rank) / 1e3) / 1e9


def free_memory():
    """Returns device memory and cached page-locked host memory between workloads."""
    import gc

    import torch
    gc.collect()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if hasattr(torch._C, "_host_emptyCache"):
        torch._C._host_emptyCache()


def measure_kernel(m, plan, src, stream, ranks, steps, warmup, l2_flush, clean_l2=False):
    """Kernel-only steps: `warmup` untimed loads, then `steps` timed ones between a barrier and a
    synchronize on both sides; with l2_flush a 1 GiB write runs between loads, outside the
    per-load events, and with clean_l2 a 256 MiB read follows it, so that L2 holds clean lines
    only and the timed load does not write back the flush's dirty ones.  Returns (total ms,
    per-load ms list, checksums of the last load)."""
    import torch
    flush = torch.empty(1 << 30, dtype=torch.uint8, device="cuda") if l2_flush else None
    clean = torch.ones(1 << 25, dtype=torch.int64, device="cuda") if clean_l2 else None

    def flush_l2(k):
        if flush is not None:
            flush.fill_(k & 255)
        if clean is not None:
            clean.sum()

    for k in range(warmup):
        flush_l2(k)
        plan.load_async(src, stream)
    torch.cuda.synchronize()
    ranks.barrier()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for k in range(steps):
        flush_l2(k + 1)
        ev[k][0].record(stream)
        plan.load_async(src, stream)
        ev[k][1].record(stream)
    t1.record(stream)
    torch.cuda.synchronize()
    ranks.barrier()
    per_load = [a.elapsed_time(b) for a, b in ev]
    total = sum(per_load) if l2_flush else t0.elapsed_time(t1)
    return total, per_load, plan.checksums()


def measure_h2d(host, stream):
    """Host->device copy bandwidth of this machine: 1 GiB from page-locked memory, best of 12."""
    import torch
    gib = 1 << 30
    hsrc = host[:gib] if host.numel() >= gib else torch.empty(gib, dtype=torch.uint8,
                                                             pin_memory=True)
    dtmp = torch.empty(gib, dtype=torch.uint8, device="cuda")
    best = min(_timed(lambda: dtmp.copy_(hsrc, non_blocking=True), stream) for _ in range(12))
    return gib / (best / 1e3) / 1e9


def host_buffer_rate(host, stream, passes=2):
    """GB/s of plain 512 MiB host->device copies over the whole page-locked source buffer, per
    pass: the rate the copy engine gets from this particular buffer, beside the loader's."""
    import torch
    ch = 512 << 20
    n = host.numel() // ch
    if n == 0:
        return []
    dev = torch.empty(ch, dtype=torch.uint8, device="cuda")
    out = []
    for _ in range(passes):
        ms = _timed(lambda: [dev.copy_(host[k * ch:(k + 1) * ch], non_blocking=True)
                             for k in range(n)], stream)
        out.append(round(n * ch / ms / 1e6, 1))
    return out


def measure_e2e(m, entries, dsts, host, stream, ranks, steps, warmup, args, ck_want,
                pull_percent=None):
    """End-to-end steps through the C ABI from the pinned host blob: every step copies the
    staged bytes host->device through three device slots, unpacks, and reads the checksums
    back.  Returns (ms per step over the slowest rank, per-step ms, staged bytes)."""
    import numpy as np
    import torch

    import paper_2607_18957_gb300 as cfa
    plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                    dev_slots=3, host_slots=0, bulk=args.bulk, stage_slices=args.stage_slices,
                    pull_percent=pull_percent)
    src = cfa.Source.pinned(host.data_ptr(), period=m.period or 0)
    for _ in range(warmup):
        plan.load_async(src, stream)
        plan.checksums()
    ranks.barrier()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    marks = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    a.record(stream)
    for k in range(steps):
        plan.load_async(src, stream)   # H2D of the whole checkpoint + unpack
        ck = plan.checksums()           # D2H of the step's result
        marks[k].record(stream)
    b.record(stream)
    torch.cuda.synchronize()
    ranks.barrier()
    ms = ranks.max(a.elapsed_time(b)) / steps
    step_ms = [a.elapsed_time(marks[0])] + [marks[k - 1].elapsed_time(marks[k])
                                            for k in range(1, steps)]
    assert np.array_equal(ck, ck_want), f"{m.name}: end-to-end checksums differ from the " \
                                        "kernel-only run"
    staged = plan.stats()["staged_bytes"]
    plan.close()
    return ms, step_ms, staged


def measure_workload(name, args, ranks, stream, peak, e2e_steps, attribution_on=False,
                     h2d_gbs=None):
    """Kernel-only and end-to-end figures of one workload; frees its memory before returning.
    Returns a record (dict) plus the manifest."""
    import torch

    import paper_2607_18957_gb300 as cfa
    from workloads.harness import DeviceDsts, entries_for, pinned_blob

    m = make_workload(name)
    t_setup = time.time()
    host = pinned_blob(m)                      # the checkpoint (or its period) page-locked
    dev_blob = torch.empty(m.source_bytes(), dtype=torch.uint8, device="cuda")
    dev_blob.copy_(host)
    dsts = DeviceDsts(m, order=args.dst_order)
    entries = entries_for(m)
    setup_s = time.time() - t_setup
    l2_flush = name in L2_FLUSHED

    # ---------------- kernel only: the blob already resident in HBM -------------------------
    slab = {} if args.slab_kib is None else {"slab_bytes": args.slab_kib << 10}
    plan = cfa.Plan(entries, dsts.cfa_dsts, m.blob_bytes, chunk_bytes=m.chunk_bytes,
                    dev_slots=0, host_slots=0, bulk=args.bulk, **slab)
    st = plan.stats()
    algo = st["bytes_read"] + st["bytes_written"]
    src = cfa.Source.device(dev_blob.data_ptr(), period=m.period or 0)
    total_ms, per_load, ck_dev = measure_kernel(m, plan, src, stream, ranks, args.steps,
                                                args.warmup, l2_flush)
    clean_ms = None
    if l2_flush:  # the same loads after a flush that leaves no dirty lines (for attribution)
        clean_ms = measure_kernel(m, plan, src, stream, ranks, args.steps, args.warmup, True,
                                  clean_l2=True)[1]
    launches = plan.stats()["kernel_launches"]
    plan.close()
    del dev_blob
    torch.cuda.empty_cache()
    mean_ms = statistics.mean(per_load)
    achieved = algo / (mean_ms / 1e3) / 1e9
    rec = {"workload": m.name, "blob_bytes": m.blob_bytes, "tensors": m.n_entries,
           "destinations": m.n_dsts, "algorithmic_bytes": algo, "chunk_bytes": m.chunk_bytes,
           "total_ms": total_ms, "steps": args.steps,
           "value_gbs": whole_job_gbs(ranks, algo * args.steps, total_ms),
           "kernel_ms": round(mean_ms, 4), "kernel_ms_median": round(statistics.median(per_load), 4),
           "kernel_ms_min": round(min(per_load), 4), "kernel_gbs": round(achieved, 1),
           "frac": round(achieved / peak, 4), "launches_per_load": launches,
           "work_items": {"tma": st["n_bulk"], "slabs": st["n_slabs"], "tiny": st["n_tiny"],
                          "column_blocks": st["n_strided"]},
           "pieces": st["n_pieces"],
           "pieces_per_s": round(st["n_pieces"] / (mean_ms / 1e3), 1),
           "l2": ("flushed between steps (1 GiB write outside the timed loads)" if l2_flush
                  else f"no flush: inputs {m.blob_bytes / 1e9:.2f} GB > L2 "
                       f"{L2_BYTES / 1e6:.0f} MB"),
           "kernels": kernel_names(st),
           "setup_s": round(setup_s, 2), "_n_bulk": st["n_bulk"]}
    if clean_ms:
        # attribution only: the flush's own dirty lines, written back during the timed load,
        # are part of the figures above; these are the same loads without them
        c_ms = statistics.mean(clean_ms)
        rec["clean_l2"] = {"kernel_ms": round(c_ms, 4),
                           "frac": round(algo / (c_ms / 1e3) / 1e9 / peak, 4),
                           "flush": "1 GiB write, then a 256 MiB read"}

    # ---------------- end to end: pinned host blob -> final layout through the C ABI ---------
    if e2e_steps:
        if h2d_gbs is None:
            h2d_gbs = measure_h2d(host, stream)
        buffer_gbs = host_buffer_rate(host, stream)
        ms, step_ms, staged = measure_e2e(m, entries, dsts, host, stream, ranks, e2e_steps,
                                          min(args.warmup, 3), args, ck_dev)
        print(f"{m.name} e2e step ms:", [round(x, 1) for x in step_ms], file=sys.stderr)
        rec["e2e"] = {
            "value": round(ranks.sum(algo) / (ms / 1e3) / 1e9, 3), "unit": UNIT,
            "h2d_bytes_per_step": staged, "d2h_bytes_per_step": 8 * m.n_entries,
            "seconds_per_model": round(ms / 1e3, 5), "h2d_gbs_measured": round(h2d_gbs, 2),
            "frac_of_h2d": round((staged / (ms / 1e3) / 1e9) / h2d_gbs, 4),
            "steps": e2e_steps, "step_ms_median": round(statistics.median(step_ms), 2),
            "step_ms_max": round(max(step_ms), 2),
            "host_buffer_h2d_gbs": buffer_gbs,
            "source": f"pinned host {'pool of ' + str(m.period >> 30) + ' GiB (periodic blob)' if m.period else 'blob'}, "
                      f"3 device staging slots of {m.chunk_bytes >> 20} MiB"}
        # the same staged load with every transfer on the copy engine (`cudaMemcpyAsync` on the
        # plan's copy stream, pull_percent 0) instead of the default pull kernel
        ce_ms, ce_steps, _ = measure_e2e(m, entries, dsts, host, stream, ranks, 3, 1, args,
                                         ck_dev, pull_percent=0)
        rec["e2e"]["copy_engine_only"] = {
            "seconds_per_model": round(ce_ms / 1e3, 5),
            "frac_of_h2d": round((staged / (ce_ms / 1e3) / 1e9) / h2d_gbs, 4),
            "step_ms": [round(x, 1) for x in ce_steps]}
        if attribution_on and not args.no_attribution:
            rec["e2e"]["attribution"] = attribution(m, host, dsts, entries, stream, args,
                                                    h2d_gbs, sweep=(name == "llama3_8b_bf16"))
    rec["_h2d_gbs"] = h2d_gbs
    del host, dsts, entries
    free_memory()
    return rec, m


def _config_record(rec):
    """The per-workload entry of the `configs` object: kernel-only and end-to-end figures."""
    out = {k: v for k, v in rec.items() if not k.startswith("_") and
           k not in ("total_ms", "value_gbs", "steps")}
    e2e = rec.get("e2e")
    if e2e:
        out["e2e"] = {k: e2e[k] for k in ("seconds_per_model", "frac_of_h2d", "h2d_gbs_measured",
                                          "h2d_bytes_per_step", "step_ms_median", "step_ms_max",
                                          "host_buffer_h2d_gbs", "steps", "source",
                                          "copy_engine_only")}
        if "attribution" in e2e:
            out["e2e"]["attribution"] = e2e["attribution"]
    return out


def run_ours(args):
    import torch

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    ranks = Ranks("nccl", "cuda")
    world, rank = ranks.world, ranks.rank
    stream = torch.cuda.current_stream()
    peaks, peak_kind = measured_peaks()
    peak = float(peaks.get("hbm_gbs", HBM_FALLBACK_GBS))

    props = torch.cuda.get_device_properties(local)
    uuid = str(getattr(props, "uuid", "") or "")
    if uuid and not uuid.startswith("GPU-"):
        uuid = "GPU-" + uuid
    sampler = ClockSampler(uuid)
    sampler.start()
    time.sleep(0.3)
    # context for the roofline: this GPU's own device copy, taken the way the measured peak was
    # (torch copy_ of 1 Gi bf16 elements, read + write bytes, best of 10)
    ca = torch.empty(1 << 30, dtype=torch.bfloat16, device="cuda")
    cb = torch.empty_like(ca)
    cb.copy_(ca)
    copy_ms = min(_timed(lambda: cb.copy_(ca), stream) for _ in range(10))
    same_box_copy_gbs = 2 * ca.numel() * 2 / (copy_ms / 1e3) / 1e9
    del ca, cb
    torch.cuda.empty_cache()

    e2e_steps = 0 if args.no_e2e else (args.e2e_steps or min(args.steps, 20))
    # the attribution (pageable copies, a safetensors file of the 8B, fill-thread sweeps) is a
    # single-GPU diagnostic: replicas would multiply its host memory and disk use by N
    head, m = measure_workload(args.workload, args, ranks, stream, peak, e2e_steps,
                               attribution_on=(world == 1))
    h2d_gbs = head["_h2d_gbs"]
    names = [] if args.configs in ("", "none") else \
        [n for n in args.configs.split(",") if n and n != args.workload]
    configs, manifests = {}, {}
    for name in names:
        try:
            rec, mc = measure_workload(name, args, ranks, stream, peak,
                                       0 if args.no_e2e else min(e2e_steps, 8),
                                       attribution_on=(name == "llama3_8b_bf16" and
                                                       world == 1),
                                       h2d_gbs=h2d_gbs)
        except Exception as e:  # noqa: BLE001 -- one workload must not cost the whole line
            if world > 1:
                raise  # the ranks' collectives would no longer match
            print(f"{name}: {type(e).__name__}: {e}", file=sys.stderr, flush=True)
            configs[name] = {"error": f"{type(e).__name__}: {e}"[:300]}
            free_memory()
            continue
        configs[name] = _config_record(rec)
        manifests[name] = mc
    clocks = sampler.stop()

    # ---------------- the oracle on this host -------------------------------------------------
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        gbs, nb, busy, desc, _ = cpu_baseline(m, args.cpu_seconds)
        cpu = {"value": round(gbs, 4), "unit": UNIT, "cores": 1, "host_cores": host_cores(),
               "kind": "oracle", "sample": desc}
        for name, mc in manifests.items():
            try:
                if name == "llama3_8b_f32_rne":
                    configs[name]["cpu_baseline"] = cpu_baseline_all_cores(mc, name,
                                                                           host_cores())
                    continue
                whole = name in CPU_FULL
                gbs, nb, busy, desc, _ = cpu_baseline(mc, None if whole else 2.0)
                configs[name]["cpu_baseline"] = {"value": round(gbs, 4), "unit": UNIT,
                                                 "cores": 1, "host_cores": host_cores(),
                                                 "kind": "oracle", "sample": desc}
            except Exception as e:  # noqa: BLE001 -- reported in the line, not fatal
                configs[name]["cpu_baseline"] = {"error": f"{type(e).__name__}: {e}"[:300]}

    if rank != 0:
        ranks.close()
        return
    dtype, cls, cls_desc = path_types(m)
    kernel_name = f"{head['kernels']}; dominant work class: {cls_desc}"
    line = {
        "metric": METRIC, "value": round(head["value_gbs"], 3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ranks.max(head["total_ms"]) / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": dtype,
        "data": f"synthetic (seeded counter-based generator; {_BLOB_KIND[m.blob_kind]})",
        "config": {"workload": m.name, "blob_bytes": m.blob_bytes, "tensors": m.n_entries,
                   "destinations": m.n_dsts, "algorithmic_bytes_per_step":
                       head["algorithmic_bytes"],
                   "chunk_bytes": m.chunk_bytes,
                   "kernel_source": "device-resident blob" + (
                       f" (periodic: an {m.period >> 30} GiB pool)" if m.period else ""),
                   "l2": head["l2"],
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "achieved": head["kernel_gbs"], "peak": peak,
                     "unit": "GB/s", "frac": head["frac"],
                     "traffic": recorded_traffic(m.name),
                     "peak_source": peak_kind, "kernel": kernel_name,
                     "launch_ms": head["kernel_ms"],
                     "same_box_copy_gbs": round(same_box_copy_gbs, 1),
                     "frac_of_same_box_copy": round(head["kernel_gbs"] / same_box_copy_gbs, 4),
                     **({"clean_l2": head["clean_l2"]} if "clean_l2" in head else {})},
        "e2e": head.get("e2e"),
        "cpu_baseline": cpu,
        "configs": configs,
        "gpu_launches": int(head["launches_per_load"] * args.steps),
        "clocks": clocks,
        "setup_s": head["setup_s"],
    }
    print(json.dumps(line), flush=True)
    ranks.close()



def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
