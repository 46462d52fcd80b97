"""Randomised manifests through the host plan builder (no GPU): destinations of every dtype, 1-D
and 2-D, filled by row blocks or element ranges whose sources sit anywhere in the blob (random
gaps, element alignment only), some of them column slices of wider source tensors, some
converting between dtypes; chunk lengths from 256 B up.  The plan's pieces, applied with numpy,
must give the oracle's destination bytes, each piece must lie inside one chunk, and the
staged copy ranges must cover every byte a piece reads."""
import numpy as np
import pytest

import oracle
import paper_2607_18957_gb300 as cfa
from workloads import DTYPE_SIZE, Manifest
from workloads.harness import entries_for

from test_lib_host import fake_dsts

DTYPES = ["u8", "i16", "bf16", "f16", "f32", "i32", "i64", "f64"]
CONVERT_FROM = {"bf16": ["f32", "f16"], "f16": ["f32"], "f32": ["bf16", "f16"]}


def random_manifest(seed):
    rng = np.random.default_rng(seed)
    dsts, ents = [], []
    for j in range(int(rng.integers(1, 9))):
        ddt = str(rng.choice(DTYPES))
        two_d = rng.random() < 0.6
        if two_d:
            R, C = int(rng.integers(1, 24)), int(rng.integers(1, 200))
            dsts.append({"name": f"d{j}", "dtype": ddt, "shape": (R, C)})
            n_rows = R
        else:
            n_rows = int(rng.integers(0, 3000))
            dsts.append({"name": f"d{j}", "dtype": ddt, "shape": (n_rows,)})
        cuts = sorted(set(rng.integers(0, n_rows + 1, size=int(rng.integers(0, 5))).tolist()))
        bounds = [0] + [c for c in cuts if 0 < c < n_rows] + [n_rows]
        for k, (r0, r1) in enumerate(zip(bounds[:-1], bounds[1:])):
            sdt, cast = ddt, False
            if ddt in CONVERT_FROM and rng.random() < 0.35:
                sdt, cast = str(rng.choice(CONVERT_FROM[ddt])), True
            e = {"name": f"d{j}.p{k}", "dtype": sdt, "dst": j, "row": r0, "cast": cast,
                 "cksum": bool(rng.random() < 0.8), "layer": int(rng.integers(0, 4))}
            if two_d:
                e["shape"] = (r1 - r0, C)
                if r1 - r0 > 1 and rng.random() < 0.4:  # a column slice of a wider tensor
                    full = C + int(rng.integers(1, 64))
                    e["stride"] = full
                    e["lead"] = int(rng.integers(0, full - C + 1))
            else:
                e["shape"] = (r1 - r0,)
            ents.append(e)
    # place the source tensors in a random order with random gaps
    off = 0
    for i in rng.permutation(len(ents)):
        e = ents[i]
        es = DTYPE_SIZE[e["dtype"]]
        off = -(-off // es) * es + es * int(rng.integers(0, 9))
        nel = int(np.prod(e["shape"], dtype=np.int64))
        if e.get("stride"):
            rows, cols = e["shape"]
            e["offset"] = off + e.pop("lead") * es
            off += es * rows * e["stride"]
        else:
            e["offset"] = off
            off += es * nel
    blob = off + int(rng.integers(0, 300))
    return Manifest(f"fuzz{seed}", ents, dsts, blob, "bits", 1000 + seed)


def apply_pieces(m, pieces, blob):
    out = {j: np.zeros(m.d_nbytes(j), np.uint8) for j in range(m.n_dsts)}
    for pc in pieces:
        i = int(pc["entry"])
        s_dt, d_dt = str(m.e_dtype[i]), str(m.d_dtype[int(pc["dst_index"])])
        es_s = DTYPE_SIZE[s_dt]
        rows = int(pc["rows"])
        cols = int(pc["n_elems"]) // rows
        step = int(pc["src_row_stride"]) * es_s if rows > 1 else cols * es_s
        o = int(pc["dst_offset"])
        for k in range(rows):
            a = int(pc["src_offset"]) + k * step
            src = blob[a:a + cols * es_s]
            if pc["conv"]:
                bits = src.view(np.uint16 if es_s == 2 else np.uint32)
                src = oracle.convert(s_dt, d_dt, bits).view(np.uint8)
            out[int(pc["dst_index"])][o:o + src.size] = src
            o += src.size
    return out


@pytest.mark.parametrize("seed", range(200))
def test_random_manifest_pieces_reproduce_the_oracle(seed):
    m = random_manifest(seed)
    blob = m.blob_range(0, m.blob_bytes)
    ref = oracle.unpack(m, blob)
    assert ref.status == 0, (seed, ref.status_name, ref.bad_entry)
    rng = np.random.default_rng(seed + 7)
    chunks = {256, 256 * int(rng.integers(2, 40)), 256 * int(rng.integers(40, 400)), 1 << 30}
    for chunk in sorted(chunks):
        with cfa.Plan(entries_for(m, with_names=True), fake_dsts(m), m.blob_bytes,
                      chunk_bytes=chunk, host_only=True,
                      tiny_bytes=int(rng.choice([0, 64, 8192])),
                      slab_bytes=int(rng.choice([4096, 8192, 65536]))) as p:
            pcs = p.pieces()
            st = p.stats()
        es = np.array([DTYPE_SIZE[str(m.e_dtype[int(i)])] for i in pcs["entry"]], np.int64)
        start = pcs["src_offset"].astype(np.int64)
        rows = pcs["rows"].astype(np.int64)
        cols = pcs["n_elems"].astype(np.int64) // np.maximum(rows, 1)
        step = np.where(rows > 1, pcs["src_row_stride"].astype(np.int64), cols)
        end = start + ((rows - 1) * step + cols) * es
        assert (start // chunk == pcs["chunk"]).all(), (seed, chunk)
        assert ((end - 1) // chunk == pcs["chunk"]).all(), (seed, chunk)
        got = apply_pieces(m, pcs, blob)
        for j in range(m.n_dsts):
            assert np.array_equal(got[j], ref.dst[j]), (seed, chunk, m.d_name[j])
        # staged bytes: at least every byte a piece reads, at most the blob
        read = np.zeros(m.blob_bytes, bool)
        for a, r, c, s, e in zip(start, rows, cols, step, es):
            for k in range(int(r)):
                read[a + k * s * e:a + k * s * e + c * e] = True
        assert int(read.sum()) <= st["staged_bytes"] <= m.blob_bytes


def _corrupt(rng, ents, dsts, opts):
    """One field of one entry or destination, or one option, set to an extreme value."""
    big = [-1, 0, 1, 3, 1 << 31, (1 << 32) + 1, 1 << 62, (1 << 63) - 1]
    what = int(rng.integers(0, 14))
    i = int(rng.integers(0, len(ents))) if len(ents) else 0
    j = int(rng.integers(0, len(dsts)))
    pick = lambda vals: vals[int(rng.integers(0, len(vals)))]
    if what == 0 and len(ents):
        ents["shape"][i][int(rng.integers(0, 8))] = pick(big)
    elif what == 1 and len(ents):
        ents["ndim"][i] = pick([-1, 0, 1, 3, 8, 9])
    elif what == 2 and len(ents):
        ents["blob_offset"][i] = pick([1, opts[0] - 1, opts[0], 1 << 40, (1 << 64) - 2])
    elif what == 3 and len(ents):
        ents["dst_index"][i] = pick([-1, len(dsts), 1 << 30])
    elif what == 4 and len(ents):
        ents["dst_row_offset"][i] = pick(big)
    elif what == 5 and len(ents):
        ents["flags"][i] = pick([0, 1, 4, 0xFF, 1 << 31])
    elif what == 6 and len(ents):
        ents["src_row_stride"][i] = pick([1, 2, 7, 1 << 20, (1 << 32) - 1])
    elif what == 7 and len(ents):
        ents["layer"][i] = pick([-1, 1 << 20, (1 << 31) - 1])
    elif what == 8 and len(ents):
        ents["src_dtype"][i] = pick([0, 9, -3, 4])
    elif what == 9:
        dsts["dtype"][j] = pick([0, 9, 1, 7])
    elif what == 10:
        dsts["ndim"][j] = pick([-1, 0, 1, 3, 9])
    elif what == 11:
        dsts["shape"][j][int(rng.integers(0, 2))] = pick(big)
    elif what == 12:
        dsts["dev_ptr"][j] = pick([0, 1, int(dsts["dev_ptr"][j]) + 1, int(dsts["dev_ptr"][0])])
    else:
        opts[int(rng.integers(0, 4))] = pick([0, 1, 100, 256, 4096, 1 << 20, (1 << 64) - 256])


def test_plan_builder_under_address_sanitizer(tmp_path):
    """The 200 random manifests (several chunk, slab and tiny sizes each) and 1,600 single-field
    corruptions of them through the plan builder built with AddressSanitizer and UBSan; every
    accepted plan's pieces and work items are checked to stay inside their chunk, the blob and
    one destination (tests/plan_fuzz_asan.c)."""
    import os
    import struct
    import subprocess

    from test_lib_host import ROOT
    exe = tmp_path / "plan_fuzz_asan"
    csrc = os.path.join(ROOT, "paper_2607_18957_gb300", "csrc")
    r = subprocess.run(["gcc", "-g", "-O1", "-std=c11", "-fsanitize=address,undefined",
                        "-fno-sanitize-recover=all", "-I", csrc,
                        "-I", os.path.join(ROOT, "include"),
                        os.path.join(ROOT, "tests", "plan_fuzz_asan.c"),
                        os.path.join(csrc, "cfa_plan.c"), "-o", str(exe)],
                       capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("no AddressSanitizer runtime for gcc here: " + r.stderr[-200:])
    path = tmp_path / "manifests.bin"
    with open(path, "wb") as f:
        for seed in range(200):
            m = random_manifest(seed)
            rng = np.random.default_rng(10_000 + seed)
            base_e = entries_for(m).arr.copy()
            base_e["name"] = 0
            base_d = cfa.make_dsts(fake_dsts(m))
            for variant in range(10):
                ents, dsts = base_e.copy(), base_d.copy()
                # blob bytes, chunk bytes, slab bytes, tiny bytes
                opts = [m.blob_bytes, 256 * int(rng.integers(1, 64)),
                        int(rng.choice([4096, 8192, 65536])), int(rng.choice([0, 64, 8192]))]
                if variant >= 2:
                    _corrupt(rng, ents, dsts, opts)
                flags = 0x1 | 0x8 if variant % 3 else 0x8  # strict coverage on most
                f.write(struct.pack("<QQQQIIII", len(ents), len(dsts), opts[0] % (1 << 64),
                                    opts[1] % (1 << 64), opts[2] % (1 << 32),
                                    opts[3] % (1 << 32), flags, 0))
                f.write(ents.tobytes())
                f.write(dsts.tobytes())
    r = subprocess.run([str(exe), str(path)], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr[-3000:]
