"""Host-side checks of the seeded input generator (mlkv_synth.gen)."""
import numpy as np

from mlkv_synth import gen, workloads


def test_splitmix64_published_vectors():
    # first outputs of SplitMix64 seeded with 0 and with 1234567 (reference test vectors)
    assert [gen.out_int(0, n) for n in range(3)] == [
        0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    assert [gen.out_int(1234567, n) for n in range(3)] == [
        6457827717110365317, 3203168211198807973, 9817491932198370423]


def test_c_generator_matches_numpy_bits():
    for sigma in (1.0, 0.5):
        a = gen.gen_bf16(7, 0x305, [0, 3, 1 << 20], 5000, sigma=sigma, col0=11, impl="numpy")
        b = gen.gen_bf16(7, 0x305, [0, 3, 1 << 20], 5000, sigma=sigma, col0=11, impl="c")
        assert np.array_equal(a, b)


def test_vectorised_generator_matches_scalar_definition():
    seed, tid, row, ncols = 99, 0x201, 5, 17
    bits = gen.gen_bf16(seed, tid, [row], ncols, sigma=0.5, col0=3, impl="numpy")[0]
    s = gen.row_seed(seed, tid, row)
    for c in range(ncols):
        col = 3 + c
        total = 0
        for k in range(3):
            x = gen.out_int(s, 3 * col + k)
            total += sum((x >> (16 * q)) & 0xFFFF for q in range(4))
        z = np.float32(total - 6 * 65536) * np.float32(1 / 65536)
        assert gen.f32_to_bf16_bits(np.float32(0.5) * z) == bits[c]


def test_bf16_rounding_is_nearest_even():
    v = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-3], dtype=np.float32)
    bits = gen.f32_to_bf16_bits(v)
    back = gen.bf16_bits_to_f32(bits)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: even mantissa (1.0) wins
    assert back[1] == np.float32(1.0)
    # 1 + 3*2^-8 is a tie between 1 + 2^-7 and 1 + 2^-6: even (1 + 2^-6) wins
    assert back[2] == np.float32(1.015625)
    assert back[3] == np.float32(-2.5)
    assert abs(back[4] - 3.0e-3) <= 3.0e-3 * 2 ** -8


def test_distribution_moments():
    v = gen.bf16_bits_to_f64(gen.gen_bf16(1, 2, [0, 1, 2, 3], 1 << 15))
    assert abs(v.mean()) < 0.01
    assert abs(v.std() - 1.0) < 0.01
    assert np.abs(v).max() <= 6.0


def test_seq_lens_uniform_range():
    sl = gen.gen_seq_lens(1003, 128, 4096)
    assert sl.min() >= 1 and sl.max() <= 4096 and len(sl) == 128
    assert 1500 < sl.mean() < 2600


def test_workloads_well_formed():
    import oracle
    for name in workloads.all_names():
        w = workloads.by_name(name)
        assert len(w.owner) == w.l
        assert oracle.validate(w.owner, w.h, w.g, w.d) == 0, name
    assert workloads.config(2).owners() == [0, 6]
    assert workloads.config(4).owners() == [0, 4, 8, 12, 16, 20, 24, 28]
