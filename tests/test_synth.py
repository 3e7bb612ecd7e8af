"""The seeded input generators pinned to their published definitions and to
the distribution the input recipe states (CPU)."""
import numpy as np

import synth

M64 = (1 << 64) - 1


def test_splitmix64_reference_sequence():
    """SplitMix64 (Steele, Lea and Flood 2014) started from state 0: the
    reference implementation's first outputs."""
    z = synth.mix64(np.array([(k * synth.GAMMA) & M64 for k in (1, 2, 3)], dtype=np.uint64))
    assert [int(v) for v in z] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_draws_are_counter_based():
    """Output i of a stream depends on i alone: any window equals the same
    slice of a longer run, and streams / seeds are distinct."""
    long = synth.draws(7, 3, 0, 1000)
    assert np.array_equal(synth.draws(7, 3, 123, 77), long[123:200])
    assert not np.array_equal(synth.draws(7, 4, 0, 1000), long)
    assert not np.array_equal(synth.draws(8, 3, 0, 1000), long)


def test_weights_irwin_hall_sigma_002():
    """N(0, 0.02) read as Irwin-Hall(4) of 16-bit lanes: mean 0, standard
    deviation 0.02, bounded by 2 x 65535 lanes' worth of deviation (3.46 sigma)."""
    w = synth.bf16_bits_to_f32(synth.weight_bf16(0, 0, 0, (1000, 1000))).astype(np.float64)
    n = w.size
    assert abs(w.mean()) < 5 * 0.02 / np.sqrt(n)
    assert abs(w.std() / 0.02 - 1) < 5e-3
    bound = 2 * 65535 * synth.WEIGHT_SCALE_002
    assert np.abs(w).max() <= bound * (1 + 2 ** -8)
    # the scale is the exact fp64 value of sigma over the sum's standard deviation
    assert abs(synth.WEIGHT_SCALE_002 * np.sqrt(4 * (65536.0 ** 2 - 1) / 12) - 0.02) < 1e-17


def test_tokens_in_range_and_uniform():
    v = 32000
    t = synth.tokens(1, 320000, v)
    assert t.dtype == np.int32 and t.min() >= 0 and t.max() < v
    counts = np.bincount(t // 1000, minlength=32)  # 32 bins of 1000 ids, 10000 expected each
    chi2 = ((counts - 10000.0) ** 2 / 10000.0).sum()
    assert chi2 < 80  # 31 degrees of freedom: 80 is far in the tail


def test_bf16_rounding_nearest_even():
    x = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -8 + 2.0 ** -20, -2.5, 65504.0],
                 dtype=np.float32)
    got = synth.f32_to_bf16_bits(x)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: to the even mantissa (1.0);
    # 1 + 3 * 2^-8 ties between 1 + 2^-7 and 1 + 2^-6: to 1 + 2^-6 (even)
    assert [hex(int(b)) for b in got] == ["0x3f80", "0x3f80", "0x3f82", "0x3f81", "0xc020", "0x4780"]


def test_act_order_is_a_seeded_permutation():
    """Fisher-Yates over counter-based draws: a permutation, a function of
    (seed, layer, matrix) alone, and uniform over the 6 orders of 3 items."""
    p = synth.act_order(0, 1, 2, 1000)
    assert p.dtype == np.int32 and sorted(p.tolist()) == list(range(1000))
    assert np.array_equal(p, synth.act_order(0, 1, 2, 1000))
    assert not np.array_equal(p, synth.act_order(0, 1, 3, 1000))
    assert not np.array_equal(p, synth.act_order(1, 1, 2, 1000))
    counts = {}
    for seed in range(3000):
        t = tuple(synth.act_order(seed, 0, 0, 3).tolist())
        counts[t] = counts.get(t, 0) + 1
    assert len(counts) == 6
    chi2 = sum((c - 500.0) ** 2 / 500.0 for c in counts.values())
    assert chi2 < 25  # 5 degrees of freedom


def test_act_order_first_swaps_by_hand():
    """K = 2: one swap, j = multiply-shift of draw 0's high 32 bits onto [0, 1]."""
    hi = int(synth.draws(7, synth.perm_stream(0, 0), 0, 1)[0]) >> 32
    want = [1, 0] if (hi * 2) >> 32 == 0 else [0, 1]
    assert synth.act_order(7, 0, 0, 2).tolist() == want
