"""Pins for the oracle's storage rounding (double -> bf16 / fp32, one rounding)."""
import numpy as np
import torch


def test_bf16_roundtrip_exhaustive(oracle):
    # Every non-NaN bf16 value survives widening and re-rounding unchanged.
    for h in range(1 << 16):
        if (h & 0x7F80) == 0x7F80 and (h & 0x7F):
            continue  # NaN payloads
        assert oracle.bf16_from_double(oracle.bf16_to_double(h)) == h, hex(h)


def test_bf16_matches_torch_round_to_nearest_even(oracle):
    # For float32 inputs (exact in double) one rounding to bf16 is torch's
    # float -> bfloat16 conversion (round to nearest, ties to even).
    rng = np.random.default_rng(123)
    bits = rng.integers(0, 2**32, size=60000, dtype=np.uint64).astype(np.uint32)
    # force ties and near-ties: low 16 bits 0x8000 / 0x7FFF / 0x8001
    bits[:6000] = (bits[:6000] & 0xFFFF0000) | 0x8000
    bits[6000:9000] = (bits[6000:9000] & 0xFFFF0000) | 0x7FFF
    bits[9000:12000] = (bits[9000:12000] & 0xFFFF0000) | 0x8001
    bits[12000:14000] &= 0x807FFFFF      # float subnormals
    bits[14000:15000] |= 0x7F7F0000      # near overflow
    bits = bits[~(((bits & 0x7F800000) == 0x7F800000) & ((bits & 0x7FFFFF) != 0))]
    f = bits.view(np.float32)
    want = torch.from_numpy(f.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.bf16_from_double(float(v)) for v in f], dtype=np.uint16)
    assert np.array_equal(got, want)


def test_bf16_single_rounding_closed_forms(oracle):
    one = 0x3F80
    # exactly halfway between 1 and 1 + 2^-7: ties to even -> 1
    assert oracle.bf16_from_double(1.0 + 2.0**-8) == one
    # just above halfway by less than a float ulp: one rounding goes up,
    # rounding through float first would tie back down to 1
    assert oracle.bf16_from_double(1.0 + 2.0**-8 + 2.0**-40) == one + 1
    assert oracle.bf16_from_double(-(1.0 + 2.0**-8 + 2.0**-40)) == 0x8000 | (one + 1)
    # halfway between 1 + 2^-7 and 1 + 2^-6: ties to even -> 1 + 2^-6
    assert oracle.bf16_from_double(1.0 + 3 * 2.0**-8) == one + 2
    # overflow and the largest finite value
    assert oracle.bf16_from_double(2.0**128) == 0x7F80
    assert oracle.bf16_from_double(-3.5e38) == 0xFF80
    assert oracle.bf16_from_double((2 - 2.0**-7) * 2.0**127) == 0x7F7F
    # bf16 subnormals (spacing 2^-133) and underflow to signed zero
    assert oracle.bf16_from_double(2.0**-133) == 0x0001
    assert oracle.bf16_from_double(2.0**-134) == 0x0000          # tie -> even (0)
    assert oracle.bf16_from_double(1.5 * 2.0**-133) == 0x0002    # tie -> even (2)
    assert oracle.bf16_from_double(-(2.0**-140)) == 0x8000
    assert (oracle.bf16_from_double(float("nan")) & 0x7FFF) > 0x7F80


def test_f32_rounding_is_round_to_nearest_even(oracle):
    assert oracle.lib().oracle_f32_from_double(1.0 + 2.0**-24) == 1.0
    assert oracle.lib().oracle_f32_from_double(1.0 + 2.0**-24 + 2.0**-40) == np.float32(1.0 + 2.0**-23)
    assert oracle.lib().oracle_f32_from_double(1.0 + 3 * 2.0**-24) == np.float32(1.0 + 2.0**-22)
