"""Pins of the oracle: checks against what the paper and the mathematics fix, not against the
oracle's own formulas.  Each function raises AssertionError on a mismatch.  They take `lib` so
that test_oracle_mutants.py can run them against deliberately broken builds of the oracle.

What pins what:
  rne_golden          hand-derived IEEE roundTiesToEven cases (tests/golden/rne_cases.txt)
  rne_vs_torch        a library routine: torch's CPU float32 -> bfloat16 conversion
  rne_vs_nearest      the definition of round-to-nearest-even, evaluated in fp64
  golden_manifests    hand-written manifests with their loaded bytes typed out by hand
  one_to_one          closed form: a 1:1 cast-free load copies blob slices (numpy sum checksums)
  concat_reference    fused layouts equal numpy/torch concatenation and stacking of the parts
                      (bf16, MoE expert stacks, 8-bit weights with per-block fp32 scales)
  cast_reference      cast entries equal torch's conversion of the source values
  invariants          exact-once coverage, byte conservation, repack(unpack(blob)) == blob,
                      entry-order invariance (Theorem 2), padding independence
  validation          malformed manifests are rejected with the right class of error
  tp_shards           tensor-parallel shards: each equals numpy slicing of the full tensor, and
                      the shards of all ranks reassemble (numpy concatenate) into the unsharded
                      load
  ep_shards           expert-parallel ranks: whole experts of the unchanged blob; the ranks'
                      expert stacks concatenate into the unsharded ones, the rest is replicated
  f16_golden          hand-derived binary16 conversion cases (tests/golden/f16_cases.txt)
  convert_vs_torch    torch's CPU conversions float16 <-> float32, float16 / float32 ->
                      bfloat16, bfloat16 -> float32 (exhaustive over 16-bit inputs)
  f16_vs_nearest      the definition of round-to-nearest-even into binary16, in fp64
"""
import numpy as np
import torch

import oracle
from workloads import (DTYPE_SIZE, Manifest, dense_config, fp8_block_config, moe_config,
                       tiny_config)

from _golden import f16_cases, manifest_case, rne_cases


# ---------------------------------------------------------------------------------------------
# the cast
# ---------------------------------------------------------------------------------------------
def _torch_bf16_bits(u32):
    f = torch.from_numpy(np.ascontiguousarray(u32, dtype=np.uint32).view(np.float32))
    return f.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


_TORCH = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}
_BITS = {"f32": (np.uint32, torch.int32), "bf16": (np.uint16, torch.int16),
         "f16": (np.uint16, torch.int16)}


def torch_convert_bits(src, dst, bits):
    """torch's CPU conversion of src-dtype bit patterns to dst-dtype bit patterns."""
    np_s, t_s = _BITS[src]
    np_d, t_d = _BITS[dst]
    t = torch.from_numpy(np.ascontiguousarray(bits, dtype=np_s).view(
        {np.uint32: np.int32, np.uint16: np.int16}[np_s])).view(_TORCH[src])
    return t.to(_TORCH[dst]).view(t_d).numpy().view(np_d)


def _nan_mask(dtype, bits):
    bits = np.asarray(bits)
    if dtype == "f32":
        b = bits.astype(np.uint32)
        return ((b & 0x7F800000) == 0x7F800000) & ((b & 0x7FFFFF) != 0)
    b = bits.astype(np.uint32)
    if dtype == "bf16":
        return ((b & 0x7F80) == 0x7F80) & ((b & 0x7F) != 0)
    return ((b & 0x7C00) == 0x7C00) & ((b & 0x3FF) != 0)


def check_convert_block(src, dst, bits, lib=None):
    """Oracle conversion vs torch: bit-equal unless the input is NaN; then both are NaN."""
    got = oracle.convert(src, dst, bits, lib=lib)
    ref = torch_convert_bits(src, dst, bits)
    nan = _nan_mask(src, bits)
    bad = (~nan) & (got != ref)
    assert not bad.any(), f"{src}->{dst}({int(np.asarray(bits)[bad][0]):#x}): " \
                          f"{int(got[bad][0]):#x} vs torch {int(ref[bad][0]):#x}"
    if nan.any():
        assert _nan_mask(dst, got[nan]).all() and _nan_mask(dst, ref[nan]).all()


def _is_nan32(u32):
    u32 = np.asarray(u32, dtype=np.uint32)
    return ((u32 & 0x7F800000) == 0x7F800000) & ((u32 & 0x007FFFFF) != 0)


def check_rne_block(u32, lib=None):
    """Oracle cast of u32 vs torch: equal on non-NaN inputs; NaN -> 0x7FC0 (torch: any NaN)."""
    got = oracle.rne_bf16(u32, lib=lib)
    ref = _torch_bf16_bits(u32)
    nan = _is_nan32(u32)
    bad = (~nan) & (got != ref)
    assert not bad.any(), f"rne differs from torch at {hex(int(u32[bad][0]))}: " \
                          f"{hex(int(got[bad][0]))} vs {hex(int(ref[bad][0]))}"
    if nan.any():
        assert (got[nan] == 0x7FC0).all(), "NaN must map to 0x7FC0"
        r = ref[nan]
        assert (((r & 0x7F80) == 0x7F80) & ((r & 0x007F) != 0)).all()


def rne_golden(lib=None):
    for u, want in rne_cases():
        got = oracle.rne_bf16_scalar(u, lib=lib)
        assert got == want, f"rne({u:#010x}) = {got:#06x}, want {want:#06x}"


def rne_vs_torch(lib=None):
    """Every upper half x the lower halves that decide rounding (0, 1, 0x7FFF, 0x8000, 0x8001,
    0xFFFF) plus random patterns."""
    hi = np.arange(1 << 16, dtype=np.uint32) << 16
    lows = np.array([0, 1, 0x7FFF, 0x8000, 0x8001, 0xFFFF], dtype=np.uint32)
    u = (hi[:, None] | lows[None, :]).ravel()
    check_rne_block(u, lib)
    rng = np.random.default_rng(11)
    check_rne_block(rng.integers(0, 1 << 32, size=1 << 20, dtype=np.uint64).astype(np.uint32),
                    lib)


def _bf16_value(b16):
    return np.asarray(b16, dtype=np.uint32).__lshift__(16).view(np.float32).astype(np.float64)


def rne_vs_nearest(lib=None):
    """For finite x the result must be the nearer of the two bf16 neighbours that bracket x
    (truncation toward zero and one unit further out, the latter possibly infinity as the
    overflow threshold), the even one on a tie."""
    rng = np.random.default_rng(12)
    u = rng.integers(0, 1 << 32, size=1 << 20, dtype=np.uint64).astype(np.uint32)
    u = np.concatenate([u, (u & 0xFFFF0000) | 0x8000, np.arange(1 << 16, dtype=np.uint32)])
    u = u[~_is_nan32(u) & ((u & 0x7F800000) != 0x7F800000)]  # finite only
    x = u.view(np.float32).astype(np.float64)
    lo = (u >> 16).astype(np.uint32)                       # toward zero
    hi = lo + 1                                            # one bf16 unit further from zero
    vlo = _bf16_value(lo)
    # value of `hi` as if the exponent were unbounded (2^128 for the step past the max)
    ulp = np.abs(_bf16_value(lo | 1) - _bf16_value(lo & ~np.uint32(1)))
    ulp = np.where(ulp == 0, np.ldexp(1.0, -133), ulp)     # subnormal/zero spacing is 2^-133
    vhi = vlo + np.sign(x + (x == 0)) * ulp
    dlo, dhi = np.abs(x - vlo), np.abs(vhi - x)
    want = np.where(dlo < dhi, lo, np.where(dhi < dlo, hi, np.where(lo & 1, hi, lo)))
    got = oracle.rne_bf16(u, lib=lib).astype(np.uint32)
    bad = got != want.astype(np.uint32)
    assert not bad.any(), f"rne({int(u[bad][0]):#010x}) = {int(got[bad][0]):#06x}, " \
                          f"nearest-even gives {int(want[bad][0]):#06x}"


# ---------------------------------------------------------------------------------------------
# unpacking
# ---------------------------------------------------------------------------------------------
def golden_manifests(lib=None):
    for name in ("fused_tiny.txt", "moe_tiny.txt", "tp_shard_tiny.txt"):
        m, blob, exp_dst, exp_ck = manifest_case(name)
        r = oracle.unpack(m, blob, lib=lib, fill=0xEE)
        assert r.status == 0, (name, r.status_name, r.bad_entry)
        for j, want in exp_dst.items():
            assert np.array_equal(r.dst[j], want), (name, j, r.dst[j], want)
        assert np.array_equal(r.cksum, exp_ck), (name, r.cksum, exp_ck)


def _blob(m):
    return m.blob_range(0, m.blob_bytes)


def _elem_view(buf, dtype):
    es = DTYPE_SIZE[dtype]
    return buf.view({1: np.uint8, 2: np.uint16, 4: np.uint32, 8: np.uint64}[es])


def one_to_one(lib=None):
    m = tiny_config(seed=21, n=60, lo=2, hi=6000, align=2, jitter=5)
    blob = _blob(m)
    r = oracle.unpack(m, blob, lib=lib)
    assert r.status == 0
    for i in range(m.n_entries):
        off, nb = int(m.e_offset[i]), m.e_nbytes(i)
        sl = blob[off:off + nb]
        assert np.array_equal(r.dst[int(m.e_dst[i])], sl), i
        assert int(r.cksum[i]) == int(sl.view(np.uint16).astype(np.uint64).sum()), i


def _source_elements(m, blob, i):
    """Entry i's source bytes in element order: the blob slice, or for a column slice the
    leading columns of a (rows, stride) numpy view of the bytes it spans."""
    off, nb = int(m.e_offset[i]), m.e_nbytes(i)
    stride = int(m.e_stride[i])
    if stride == 0:
        return blob[off:off + nb]
    es = DTYPE_SIZE[str(m.e_dtype[i])]
    cols = int(m.e_shape[i, m.e_ndim[i] - 1])
    rows = nb // es // cols
    span = np.zeros(rows * stride * es, dtype=np.uint8)
    ext = m.e_extent(i)
    span[:ext] = blob[off:off + ext]
    return np.ascontiguousarray(span.reshape(rows, stride * es)[:, :cols * es]).ravel()


def _expected_by_concat(m, blob):
    """Destination bytes built by concatenating each destination's parts in row order, with
    torch doing the casts: no offsets are computed."""
    out = {}
    for j in range(m.n_dsts):
        parts = []
        for i in sorted(m.entries_of_dst(j), key=lambda i: int(m.e_row[i])):
            sl = _source_elements(m, blob, i)
            if m.e_cast[i]:
                src, dst = str(m.e_dtype[i]), str(m.d_dtype[j])
                sl = torch_convert_bits(src, dst, sl.view(_BITS[src][0])).view(np.uint8)
            parts.append(sl)
        out[j] = np.concatenate(parts) if parts else np.zeros(0, np.uint8)
        assert out[j].size == m.d_nbytes(j)
    return out


def _mini_dense(src="bf16", seed=31, **kw):
    kw.setdefault("align", 2 if src == "bf16" else 4)
    kw.setdefault("jitter", 3)
    return dense_config("mini_dense", seed, layers=2, hidden=64, n_q=4, n_kv=2, head_dim=16,
                        inter=96, vocab=100, src_dtype=src, **kw)


def _mini_moe(seed=41, n_experts=3, **kw):
    kw.setdefault("align", 2)
    kw.setdefault("jitter", 3)
    return moe_config("mini_moe", seed, layers=2, hidden=32, n_q=4, n_kv=2, head_dim=8,
                      inter=48, n_experts=n_experts, vocab=52, n_extra=25, **kw)


def _check_against_concat(m, lib):
    blob = _blob(m)
    r = oracle.unpack(m, blob, lib=lib, fill=0x5A)
    assert r.status == 0, (r.status_name, r.bad_entry)
    exp = _expected_by_concat(m, blob)
    for j in range(m.n_dsts):
        assert np.array_equal(r.dst[j], exp[j]), (m.name, m.d_name[j])
    # checksums: sum of each entry's destination elements, cut out of the expected bytes in the
    # same row order
    for j in range(m.n_dsts):
        pos = 0
        for i in sorted(m.entries_of_dst(j), key=lambda i: int(m.e_row[i])):
            nb = m.e_numel(i) * DTYPE_SIZE[str(m.d_dtype[j])]
            want = int(_elem_view(exp[j][pos:pos + nb], str(m.d_dtype[j])).astype(np.uint64)
                       .sum(dtype=np.uint64))
            assert int(r.cksum[i]) == want, (m.name, m.e_name[i])
            pos += nb


def concat_reference(lib=None):
    m = _mini_dense()
    # the fused layout itself: q, k, v rows and gate, up rows in that order
    for j in range(m.n_dsts):
        names = [m.e_name[i].rsplit(".", 2)[-2]
                 for i in sorted(m.entries_of_dst(j), key=lambda i: int(m.e_row[i]))]
        if m.d_name[j].endswith("qkv_proj.weight"):
            assert names == ["q_proj", "k_proj", "v_proj"]
        if m.d_name[j].endswith("gate_up_proj.weight"):
            assert names == ["gate_proj", "up_proj"]
    _check_against_concat(m, lib)
    mm = _mini_moe()
    _check_against_concat(mm, lib)
    # stacking: w13[e] == cat(w1_e, w3_e), w2[e] == w2_e, through numpy reshapes
    blob = _blob(mm)
    r = oracle.unpack(mm, blob, lib=lib)
    for j in range(mm.n_dsts):
        if not mm.d_name[j].endswith("w13_weight"):
            continue
        E, I2, H = mm.d_shape_tuple(j)
        w13 = r.dst[j].view(np.uint16).reshape(E, I2, H)
        pre = mm.d_name[j].rsplit("experts.", 1)[0] + "experts."
        idx = {mm.e_name[i]: i for i in mm.entries_of_dst(j)}
        for e in range(E):
            parts = []
            for w in ("w1", "w3"):
                i = idx[f"{pre}{e}.{w}.weight"]
                off = int(mm.e_offset[i])
                parts.append(blob[off:off + mm.e_nbytes(i)].view(np.uint16).reshape(I2 // 2, H))
            assert np.array_equal(w13[e], np.concatenate(parts, axis=0)), (j, e)
    # 8-bit weights with per-block fp32 scales: both passed through; fused weights and fused
    # scales keep the same part order, one scale row per `block` weight rows
    for fuse in (True, False):
        m8 = fp8_block_config("mini_fp8", 37, layers=2, hidden=48, n_q=4, n_kv=2, head_dim=16,
                              inter=80, vocab=30, block=16, fuse=fuse, align=1, jitter=5)
        _check_against_concat(m8, lib)
        for j, name in enumerate(m8.d_name):
            if name.endswith("_scale_inv"):
                jw = m8.d_name.index(name[:-len("_scale_inv")])
                rw, cw = m8.d_shape_tuple(jw)
                assert m8.d_shape_tuple(j) == (-(-rw // 16), -(-cw // 16)), name
                assert str(m8.d_dtype[j]) == "f32" and str(m8.d_dtype[jw]) == "u8"


def cast_reference(lib=None):
    m = _mini_dense("f32", seed=32)
    assert m.e_cast.all()
    _check_against_concat(m, lib)
    # the other conversions: fp32 -> fp16, fp16 -> bf16 with fp32 norms, bf16 -> fp32 norms
    for src, dst, norm in (("f32", "f16", None), ("f16", "bf16", "f32"), ("bf16", "bf16", "f32")):
        m = _mini_dense(src, seed=33, dst_dtype=dst, norm_dtype=norm)
        assert m.e_cast.any()
        _check_against_concat(m, lib)


def invariants(lib=None):
    m = _mini_moe(seed=43)
    blob = _blob(m)
    r = oracle.unpack(m, blob, lib=lib, cover=True)
    assert r.status == 0
    # exactly-once coverage
    st, bad = oracle.check_cover(r, lib=lib)
    assert st == 0, (oracle.STATUS_NAME[st], bad)
    assert all((c == 1).all() for c in r.cover.values())
    # bytes conserved (cast-free: source bytes == destination bytes)
    assert m.total_src_bytes() == sum(v.size for v in r.dst.values())
    # repack(unpack(blob)) == blob on the bytes entries cover; positions come from summing
    # part sizes in row order, not from the row-offset formula
    back = np.zeros_like(blob)
    covered = np.zeros(blob.size, dtype=bool)
    for j in range(m.n_dsts):
        pos = 0
        for i in sorted(m.entries_of_dst(j), key=lambda i: int(m.e_row[i])):
            off, nb = int(m.e_offset[i]), m.e_nbytes(i)
            back[off:off + nb] = r.dst[j][pos:pos + nb]
            covered[off:off + nb] = True
            pos += nb
    assert np.array_equal(back[covered], blob[covered])
    # entry-order invariance (Theorem 2: any order reaching the same per-tensor states)
    perm = np.random.default_rng(5).permutation(m.n_entries)
    mp = _permuted(m, perm)
    rp = oracle.unpack(mp, blob, lib=lib)
    assert rp.status == 0
    for j in range(m.n_dsts):
        assert np.array_equal(rp.dst[j], r.dst[j])
    assert np.array_equal(rp.cksum, r.cksum[perm])
    # padding independence: bytes no entry covers do not matter
    noisy = blob.copy()
    noisy[~covered] ^= 0xA5
    rn = oracle.unpack(m, noisy, lib=lib)
    for j in range(m.n_dsts):
        assert np.array_equal(rn.dst[j], r.dst[j])
    # a window of the blob that holds every byte of the selected destinations is enough
    j = max(range(m.n_dsts), key=m.d_nbytes)
    es = m.entries_of_dst(j)
    lo = min(int(m.e_offset[i]) for i in es)
    hi = max(int(m.e_offset[i]) + m.e_nbytes(i) for i in es)
    rw = oracle.unpack(m, blob[lo:hi], blob_begin=lo, dsts=[j], lib=lib)
    assert rw.status == 0 and np.array_equal(rw.dst[j], r.dst[j])
    assert all(int(rw.cksum[i]) == int(r.cksum[i]) for i in es)


def _permuted(m, perm):
    ents = []
    for i in perm:
        i = int(i)
        ents.append({"name": m.e_name[i], "dtype": str(m.e_dtype[i]),
                     "shape": m.e_shape_tuple(i), "offset": int(m.e_offset[i]),
                     "dst": int(m.e_dst[i]), "row": int(m.e_row[i]),
                     "cast": bool(m.e_cast[i]), "cksum": bool(m.e_cksum[i]),
                     "layer": int(m.e_layer[i]), "stride": int(m.e_stride[i])})
    dsts = [{"name": m.d_name[j], "dtype": str(m.d_dtype[j]), "shape": m.d_shape_tuple(j)}
            for j in range(m.n_dsts)]
    return Manifest(m.name, ents, dsts, m.blob_bytes, m.blob_kind, m.seed, m.period,
                    m.chunk_bytes)


def _variant(m, i, **change):
    ents = []
    for k in range(m.n_entries):
        e = {"name": m.e_name[k], "dtype": str(m.e_dtype[k]), "shape": m.e_shape_tuple(k),
             "offset": int(m.e_offset[k]), "dst": int(m.e_dst[k]), "row": int(m.e_row[k]),
             "cast": bool(m.e_cast[k]), "cksum": bool(m.e_cksum[k]),
             "layer": int(m.e_layer[k]), "stride": int(m.e_stride[k])}
        if k == i:
            e.update(change)
        ents.append(e)
    dsts = [{"name": m.d_name[j], "dtype": str(m.d_dtype[j]), "shape": m.d_shape_tuple(j)}
            for j in range(m.n_dsts)]
    return Manifest(m.name, ents, dsts, m.blob_bytes, m.blob_kind, m.seed)


def validation(lib=None):
    m, blob, _, _ = manifest_case("fused_tiny.txt")
    # q is entry 0 (bf16 [2, 2] at offset 4 into qkv rows 0..1); norm is entry 3 (cast)
    cases = [
        (_variant(m, 0, offset=32), oracle.ORC_E_OOB),         # reads past the 34-byte blob
        (_variant(m, 0, offset=5), oracle.ORC_E_ALIGN),        # not a multiple of 2
        (_variant(m, 0, row=3), oracle.ORC_E_OOB),             # rows 3..4 of a 4-row dst
        (_variant(m, 0, dtype="f16"), oracle.ORC_E_DTYPE),     # bf16 destination
        (_variant(m, 3, cast=False), oracle.ORC_E_DTYPE),      # f32 into bf16 without cast
        (_variant(m, 0, shape=(1, 4)), oracle.ORC_E_SHAPE),    # last dim 4 != row length 2
        (_variant(m, 5, row=2), oracle.ORC_E_OOB),             # bias[2:4] of a 3-element dst
    ]
    for mv, code in cases:
        r = oracle.unpack(mv, blob, lib=lib)
        assert r.status == code, (oracle.STATUS_NAME[r.status], oracle.STATUS_NAME[code])
    # overlap and gap are decided by coverage
    r = oracle.unpack(_variant(m, 1, row=1), blob, cover=True, lib=lib)   # k onto q's row 1
    assert r.status == 0
    assert oracle.check_cover(r, lib=lib)[0] == oracle.ORC_E_OVERLAP
    r = oracle.unpack(_variant(m, 4, shape=(0,)), blob, cover=True, lib=lib)  # bias[0] unset
    assert r.status == 0
    assert oracle.check_cover(r, lib=lib)[0] == oracle.ORC_E_COVERAGE


def tp_shards(lib=None):
    """Rank shards against numpy slicing, and the ranks together against the unsharded load."""
    for build, src in ((_mini_dense, "bf16"), (_mini_dense, "f32"), (_mini_moe, None)):
        for tp in (2, 4):
            kw = {} if src is None else {"src": src}
            full = build(seed=35, **kw)
            blob = _blob(full)
            rf = oracle.unpack(full, blob, lib=lib)
            assert rf.status == 0
            ranks = []
            for rank in range(tp):
                m = build(seed=35, tp=tp, rank=rank, **kw)
                assert m.blob_bytes == full.blob_bytes
                r = oracle.unpack(m, blob, lib=lib)
                assert r.status == 0, (m.name, tp, rank, r.status_name)
                exp = _expected_by_concat(m, blob)
                for j in range(m.n_dsts):
                    assert np.array_equal(r.dst[j], exp[j]), (tp, rank, m.d_name[j])
                ranks.append((m, r))
            _check_reassembly(full, rf, ranks, tp)


def _check_reassembly(full, rf, ranks, tp):
    """Shards of all ranks, concatenated the way the split cut them, give the unsharded
    destinations: row-parallel weights along columns, vocabulary and column-parallel weights
    (each fused part separately) along rows."""
    def dst(m, r, name):
        j = m.d_name.index(name)
        return r.dst[j].view(np.uint16).reshape(m.d_shape_tuple(j))

    names = full.d_name
    for name in names:
        jf = names.index(name)
        want = rf.dst[jf].view(np.uint16).reshape(full.d_shape_tuple(jf))
        parts = [dst(m, r, name) for m, r in ranks]
        if name.endswith("gate_up_proj.weight"):
            halves = [np.split(p, 2, axis=0) for p in parts]
            got = np.concatenate([h[0] for h in halves] + [h[1] for h in halves], axis=0)
        elif name.endswith(("o_proj.weight", "down_proj.weight", "w2_weight")):
            got = np.concatenate(parts, axis=-1)
        elif name.endswith(("embed_tokens.weight", "lm_head.weight", "q_proj.weight",
                            "gate_proj.weight", "up_proj.weight")):
            got = np.concatenate(parts, axis=0)
        elif name.endswith("w13_weight"):
            halves = [np.split(p, 2, axis=1) for p in parts]
            got = np.concatenate([h[0] for h in halves] + [h[1] for h in halves], axis=1)
        elif name.endswith("qkv_proj.weight"):
            continue  # checked below, per part
        else:
            got = parts[0]  # replicated: norms, router, extras
            for p in parts[1:]:
                assert np.array_equal(p, got), name
        assert np.array_equal(got, want), name
    # fused qkv: q rows split over ranks; k and v split, or replicated per kv head
    m0 = ranks[0][0]
    qkv = [n for n in names if n.endswith("qkv_proj.weight")]
    for name in qkv:
        jf = names.index(name)
        want = rf.dst[jf].view(np.uint16).reshape(full.d_shape_tuple(jf))
        parts = [dst(m, r, name) for m, r in ranks]
        rows_r = parts[0].shape[0]
        q_rows_r = (want.shape[0] - 2 * _kv_rows(full, name)) // tp
        kv_r = (rows_r - q_rows_r) // 2
        q = np.concatenate([p[:q_rows_r] for p in parts], axis=0)
        assert np.array_equal(q, want[:q_rows_r * tp]), name
        kv_full = _kv_rows(full, name)
        for which, base in (("k", q_rows_r * tp), ("v", q_rows_r * tp + kv_full)):
            off = q_rows_r if which == "k" else q_rows_r + kv_r
            shards = [p[off:off + kv_r] for p in parts]
            if kv_r * tp == kv_full:
                got = np.concatenate(shards, axis=0)
                assert np.array_equal(got, want[base:base + kv_full]), (name, which)
            else:  # replicated heads: every shard is one of the full kv heads
                for s in shards:
                    heads = want[base:base + kv_full].reshape(-1, kv_r, want.shape[1])
                    assert any(np.array_equal(s, h) for h in heads), (name, which)
    del m0


def ep_shards(lib=None):
    """Expert-parallel ranks read whole experts out of the unchanged blob: each rank's
    destinations equal concatenation of its parts, and the ranks' w13 / w2 stacked along the
    expert axis give the unsharded ones; every other destination equals the unsharded load."""
    full = _mini_moe(seed=36, n_experts=4)
    blob = _blob(full)
    rf = oracle.unpack(full, blob, lib=lib)
    assert rf.status == 0
    for ep in (2, 4):
        ranks = []
        for rank in range(ep):
            m = _mini_moe(seed=36, n_experts=4, ep=ep, rank=rank)
            assert m.blob_bytes == full.blob_bytes
            for i, name in enumerate(m.e_name):
                assert m.e_offset[i] == full.e_offset[full.e_name.index(name)], name
            r = oracle.unpack(m, blob, lib=lib)
            assert r.status == 0, (ep, rank, r.status_name)
            exp = _expected_by_concat(m, blob)
            for j in range(m.n_dsts):
                assert np.array_equal(r.dst[j], exp[j]), (ep, rank, m.d_name[j])
            ranks.append((m, r))
        for jf, name in enumerate(full.d_name):
            want = rf.dst[jf].view(np.uint16).reshape(full.d_shape_tuple(jf))
            parts = []
            for m, r in ranks:
                j = m.d_name.index(name)
                parts.append(r.dst[j].view(np.uint16).reshape(m.d_shape_tuple(j)))
            if name.endswith(("w13_weight", "w2_weight")):
                assert all(p.shape[0] == want.shape[0] // ep for p in parts), name
                assert np.array_equal(np.concatenate(parts, axis=0), want), name
            else:
                for p in parts:
                    assert np.array_equal(p, want), name


def _kv_rows(full, qkv_name):
    prefix = qkv_name.rsplit("qkv_proj", 1)[0]
    i = full.e_name.index(prefix + "k_proj.weight")
    return int(full.e_shape[i, 0])


def f16_golden(lib=None):
    for direction, x, want in f16_cases():
        if direction == "f32>f16":
            got = oracle.f32_to_f16_scalar(x, lib=lib)
        else:
            got = int(oracle.convert("f16", "f32", np.array([x], np.uint16), lib=lib)[0])
        assert got == want, f"{direction}({x:#x}) = {got:#x}, want {want:#x}"


def convert_vs_torch(lib=None):
    all16 = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    for src, dst in (("f16", "f32"), ("f16", "bf16"), ("bf16", "f32")):
        check_convert_block(src, dst, all16, lib)
    # f32 -> f16: every sign/exponent/upper fraction pattern with the low 13 bits that decide
    # the rounding, plus random patterns (all 2^32 in test_convert_exhaustive_vs_torch)
    hi = np.arange(1 << 19, dtype=np.uint32) << 13
    lows = np.array([0, 1, 0xFFF, 0x1000, 0x1001, 0x1FFF], dtype=np.uint32)
    check_convert_block("f32", "f16", (hi[:, None] | lows[None, :]).ravel(), lib)
    rng = np.random.default_rng(13)
    check_convert_block("f32", "f16",
                        rng.integers(0, 1 << 32, size=1 << 20, dtype=np.uint64).astype(np.uint32),
                        lib)


def _f16_value(b16):
    b = np.asarray(b16, dtype=np.uint32)
    e = (b >> 10) & 31
    m = (b & 1023).astype(np.float64)
    v = np.where(e == 0, np.ldexp(m, -24), np.ldexp(1024.0 + m, e.astype(np.int64) - 25))
    return np.where(b & 0x8000, -v, v)


def f16_vs_nearest(lib=None):
    """For finite x below the overflow threshold the result must be the nearer of the two
    binary16 values bracketing x (candidates from a sorted table of all finite halves), the
    one with an even last fraction bit on a tie."""
    rng = np.random.default_rng(14)
    u = rng.integers(0, 1 << 32, size=1 << 18, dtype=np.uint64).astype(np.uint32)
    mant = rng.integers(0, 1 << 23, size=1 << 18, dtype=np.uint64).astype(np.uint32)
    expo = rng.integers(100, 145, size=1 << 18, dtype=np.uint64).astype(np.uint32)
    u = np.concatenate([u, (expo << 23) | mant, ((expo << 23) | (mant & ~np.uint32(0x1FFF)) |
                                                 0x1000)])
    x = u.view(np.float32).astype(np.float64)
    keep = np.isfinite(x) & (np.abs(x) < 65520.0)
    u, x = u[keep], x[keep]
    pos = np.arange(0x7C00, dtype=np.uint32)            # every finite non-negative half
    vals = _f16_value(pos)                               # increasing
    ax = np.abs(x)
    k = np.searchsorted(vals, ax, side="right") - 1      # vals[k] <= ax < vals[k + 1]
    lo = pos[k]
    hi_v = np.where(k + 1 < pos.size, vals[np.minimum(k + 1, pos.size - 1)], 65536.0)
    dlo, dhi = ax - vals[k], hi_v - ax
    pick = np.where(dlo < dhi, lo, np.where(dhi < dlo, lo + 1, np.where(lo & 1, lo + 1, lo)))
    want = (pick | np.where(np.signbit(x), 0x8000, 0)).astype(np.uint32)
    got = oracle.convert("f32", "f16", u, lib=lib).astype(np.uint32)
    bad = got != want
    assert not bad.any(), f"f16({int(u[bad][0]):#010x}) = {int(got[bad][0]):#06x}, " \
                          f"nearest-even gives {int(want[bad][0]):#06x}"


ALL_PINS = [rne_golden, rne_vs_torch, rne_vs_nearest, golden_manifests, one_to_one,
            concat_reference, cast_reference, invariants, validation, tp_shards, ep_shards,
            f16_golden, convert_vs_torch, f16_vs_nearest]
