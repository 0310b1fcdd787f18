"""Pins for the oracle's seeded weight generator and bf16 helpers."""
import fractions

import numpy as np
import torch

from paper_2512_21835_gb300 import inputs


def test_splitmix64_published_outputs(orc):
    # Reference outputs of SplitMix64 (Steele, Lea & Flood 2014; Vigna's splitmix64.c)
    # for seed 1234567 and for seed 1477776061723855037.
    assert [orc.splitmix64(1234567, k) for k in range(5)] == [
        6457827717110365317, 3203168211198807973, 9817491932198370423, 4593380528125082431,
        16408922859458223821]
    assert [orc.splitmix64(1477776061723855037, k) for k in range(3)] == [
        1985237415132408290, 2979275885539914483, 13511426838097143398]


def test_f32_to_bf16_round_to_nearest_even(orc):
    L = orc.lib()
    assert L.orc_f32_to_bf16(1.0) == 0x3F80
    assert L.orc_f32_to_bf16(1.0 + 2 ** -8) == 0x3F80          # tie -> even
    assert L.orc_f32_to_bf16(1.0 + 3 * 2 ** -8) == 0x3F82      # tie -> even (up)
    assert L.orc_f32_to_bf16(1.0 + 2 ** -8 + 2 ** -20) == 0x3F81
    assert L.orc_f32_to_bf16(-2.0) == 0xC000
    # agrees with torch's fp32 -> bf16 conversion on random values
    f = inputs.normal_f32(5, 20000, 3.0)
    ours = np.array([L.orc_f32_to_bf16(float(v)) for v in f], dtype=np.uint16)
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def _nearest_bf16_exact(v: float) -> float:
    """Brute force: the bf16 value nearest to v (ties to even mantissa), exact rationals."""
    import math
    m, e = math.frexp(v)
    ulp = 2.0 ** (e - 8)
    lo = math.floor(v / ulp) * ulp
    hi = lo + ulp
    fv, flo, fhi = fractions.Fraction(v), fractions.Fraction(lo), fractions.Fraction(hi)
    if fv - flo < fhi - fv:
        return lo
    if fhi - fv < fv - flo:
        return hi
    return lo if int(lo / ulp) % 2 == 0 else hi


def test_round_bf16_from_f64_brute_force(orc):
    rng = np.random.default_rng(7)
    vals = list(rng.standard_normal(3000) * 10.0 ** rng.integers(-6, 6, 3000))
    vals += [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8), 0.0, 3.0 + 2 ** -7]
    for v in vals:
        assert orc.lib().orc_round_bf16(float(v)) == _nearest_bf16_exact(float(v)), v


def test_generator_slices_and_statistics(orc):
    a = orc.gen_tensor(99, orc.tensor_id(3, 6), 5000, 0)
    b = orc.gen_tensor(99, orc.tensor_id(3, 6), 1000, 0, first=4000)
    assert np.array_equal(a[4000:], b)
    w = orc.bf16_bits_to_f64(orc.gen_tensor(0x10A1B, orc.tensor_id(0, 1), 400_000, 0))
    assert abs(w.mean()) < 2e-4
    assert abs(w.std() - 0.02) < 0.02 * 0.01
    g = orc.bf16_bits_to_f64(orc.gen_tensor(0x10A1B, orc.tensor_id(0, 0), 100_000, 1))
    assert abs(g.mean() - 1.0) < 1e-3 and abs(g.std() - 0.02) < 0.02 * 0.05
    # distinct tensors and seeds give different streams
    c = orc.gen_tensor(100, orc.tensor_id(3, 6), 5000, 0)
    assert np.mean(a == c) < 0.05
    # every value is a bf16 pattern of a value in [-4*sqrt(3)*0.02, +] (Irwin-Hall support)
    assert np.abs(w).max() <= 2 * 0.0347 + 1e-6


def test_tensor_ids_distinct(orc):
    ids = [orc.tensor_id(-1, w) for w in range(3)] + [orc.tensor_id(l, w) for l in range(80) for w in range(9)]
    assert len(set(ids)) == len(ids)
