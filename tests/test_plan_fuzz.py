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
