"""The seeded input generator and the manifest builders (CPU only)."""
import numpy as np

import workloads
from workloads import gen


def _splitmix64_np(seed, w):
    M = np.uint64(0xFFFFFFFFFFFFFFFF)
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (np.asarray(w, dtype=np.uint64) + np.uint64(1)) * \
            np.uint64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return (z ^ (z >> np.uint64(31))) & M


def test_splitmix64_published_vector():
    # first outputs of SplitMix64 seeded with 1234567 (Vigna's reference splitmix64.c)
    want = [6457827717110365317, 3203168211198807973, 9817491932198370423,
            4593380528125082431, 16408922859458223821]
    assert [gen.splitmix64_word(1234567, w) for w in range(5)] == want


def test_bits_matches_numpy_and_ranges_are_independent():
    words = _splitmix64_np(7, np.arange(4096))
    ref = words.view(np.uint8)
    full = gen.fill("bits", 7, 0, ref.size, threads=1)
    assert np.array_equal(full, ref)
    for off, ln in [(3, 1000), (8, 8), (4095, 17), (1, 0), (100, 32000)]:
        assert np.array_equal(gen.fill("bits", 7, off, ln), ref[off:off + ln])
    # threaded fill across a 64 MiB boundary equals the single-thread fill
    a = gen.fill("bits", 9, (64 << 20) - 1000, 3000, threads=4)
    b = gen.fill("bits", 9, (64 << 20) - 1000, 3000, threads=1)
    assert np.array_equal(a, b)


def test_f32mix_statistics():
    n = 1 << 22
    u = gen.fill("f32mix", 3, 0, 4 * n).view(np.uint32)
    f = u.view(np.float32)
    assert np.isfinite(f).all()
    exp = u & 0x7F800000
    sub = (exp == 0) & ((u & 0x7FFFFF) != 0)
    ties = ((u & 0xFFFF) == 0x8000) & (exp != 0)
    assert 0.004 < sub.mean() < 0.006
    assert 0.004 < ties.mean() < 0.006
    norm = (exp != 0)
    assert abs(float(f[norm].std()) - 0.02) < 0.001
    assert abs(float(f[norm].mean())) < 0.001
    # both parities of the kept bit occur among ties
    lsb = (u[ties] >> 16) & 1
    assert 0.3 < lsb.mean() < 0.7
    # range independence
    assert np.array_equal(gen.fill("f32mix", 3, 4 * 1001, 4 * 77).view(np.uint32),
                          u[1001:1078])


def test_named_configs_match_published_shapes():
    m = workloads.named_config("llama3_8b_bf16")
    assert m.n_entries == 291 and m.n_dsts == 195
    assert m.blob_bytes == 16_060_522_496
    assert m.total_dst_bytes() == m.total_src_bytes()
    names = {m.d_name[j]: m.d_shape_tuple(j) for j in range(m.n_dsts)}
    assert names["model.layers.0.self_attn.qkv_proj.weight"] == (6144, 4096)
    assert names["model.layers.31.mlp.gate_up_proj.weight"] == (28672, 4096)
    m3 = workloads.named_config("llama3_8b_f32_rne")
    assert m3.blob_bytes == 2 * m.blob_bytes and m3.e_cast.all()
    m5 = workloads.named_config("llama3_70b_bf16")
    assert m5.n_entries == 723 and m5.n_dsts == 483
    assert m5.chunk_bytes == 1 << 30 and m5.period == 8 << 30
    names5 = {m5.d_name[j]: m5.d_shape_tuple(j) for j in range(m5.n_dsts)}
    assert names5["model.layers.0.self_attn.qkv_proj.weight"] == (10240, 8192)
    assert names5["model.layers.0.mlp.gate_up_proj.weight"] == (57344, 8192)
    t = workloads.named_config("tiny_1000")
    assert t.n_entries == 1000 and (t.e_offset % 256 == 0).all()


def test_offsets_are_aligned_and_disjoint():
    for m in [workloads.tiny_config(seed=2, n=200),
              workloads.dense_config("d", 3, 2, 64, 4, 2, 16, 96, 100, jitter=3, align=2)]:
        order = np.argsort(m.e_offset)
        end = 0
        for i in order:
            es = workloads.DTYPE_SIZE[str(m.e_dtype[i])]
            assert int(m.e_offset[i]) % es == 0
            assert int(m.e_offset[i]) >= end
            end = int(m.e_offset[i]) + m.e_nbytes(i)
        assert end <= m.blob_bytes
