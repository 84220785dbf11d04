"""The parity checker itself (host logic, no GPU): the per-unit and per-row
bounds catch what the whole-output norm lets through."""
import numpy as np
import pytest

from parity_util import Parity, assert_parity, lbthw_units


def _noisy(shape, seed, rel=3e-3):
    g = np.random.default_rng(seed)
    ref = g.standard_normal(shape)
    out = ref + rel * g.standard_normal(shape) / np.sqrt(3.0)
    return out, ref


def test_rounding_level_noise_passes():
    out, ref = _noisy((6, 4096, 64), 1)
    r = assert_parity("noise", out, ref, "bf16")
    assert r["rel_l2"] < 5e-3 and r["worst_row"] < 2e-2 and r["units"] == 6


def test_one_wrong_row_fails_though_the_norm_passes():
    out, ref = _noisy((3, 8192, 64), 2)
    out[1, 5000] = ref[1, 4999]                  # another token's row
    p = Parity("planted row", "bf16").add(out, ref)
    assert p.whole() < 2e-2                      # the norm alone would pass
    with pytest.raises(AssertionError, match="per-row"):
        p.check()


def test_one_wrong_unit_fails_though_the_norm_passes():
    out, ref = _noisy((200, 256, 16), 3)
    out[117] *= 1.1                              # one unit 10% off
    p = Parity("planted unit", "bf16")
    for lo in range(0, 200, 64):                 # added in batches, as by layer
        p.add(out[lo:lo + 64], ref[lo:lo + 64])
    assert p.whole() < 2e-2
    with pytest.raises(AssertionError, match="unit 117"):
        p.check()


def test_small_rows_are_measured_against_the_unit_scale():
    """A row whose reference is near zero is not failed for rounding noise that is
    small against the unit's typical row."""
    out, ref = _noisy((2, 512, 32), 4)
    ref[0, 10] = 1e-9
    out[0, 10] = 1e-3
    assert_parity("small row", out, ref, "bf16")


def test_scalar_rows_and_non_finite():
    g = np.random.default_rng(5)
    ref = g.standard_normal((4, 100))
    assert_parity("scalars", ref * (1 + 1e-6), ref, "f32")
    bad = ref.copy()
    bad[2, 7] = np.nan
    with pytest.raises(AssertionError, match="non-finite"):
        assert_parity("nan", bad, ref, "bf16")


def test_lbthw_units_order():
    a = np.arange(2 * 3 * 5 * 4 * 2, dtype=np.float64).reshape(2, 3, 5, 4, 2)
    u = lbthw_units(a)
    assert u.shape == (24, 5, 2)
    assert np.array_equal(u[(1 * 3 + 2) * 4 + 3], a[1, 2, :, 3])
    s = lbthw_units(a[..., 0])
    assert s.shape == (24, 5) and np.array_equal(s[5], a[0, 1, :, 1, 0])
