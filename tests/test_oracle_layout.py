"""Exhaustive checks of the digit-plane layout (§2.5), one modulus at a time.

For every modulus of S and of the r > 12 extension, over every centred
residue and every ordered pair of centred residues:
  * each stored plane is an E4M3-exact integer,
  * the digits reconstruct the residue,
  * the plane products recombine to d·e (mod m), unmerged and merged,
  * each accumulator term stays under the bound that Eq. (accum-exact) uses.
The E4M3 encoder is pinned to the format definition and to torch's float8.
"""
import numpy as np
import pytest
import torch

from oracle import ozaki2 as oz

ALL_MODULI = oz.moduli(oz.MAX_MODULI)


def centred_range(m):
    return np.arange(-(m // 2), m - m // 2)


def test_e4m3_encoder_against_format_definition_and_torch():
    codes = np.arange(256, dtype=np.uint8)
    ours = np.array([oz.e4m3_decode(int(c)) for c in codes])
    theirs = torch.from_numpy(codes.copy()).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    same = (ours == theirs) | (np.isnan(ours) & np.isnan(theirs))
    assert same.all()
    # every finite integer value has exactly the codes the encoder produces
    ints = {}
    for c, v in zip(codes, ours):
        if np.isfinite(v) and v == int(v):
            ints.setdefault(int(v), set()).add(int(c))
    members = [v for v in range(-448, 449) if oz.e4m3_exact_integer(v)]
    assert set(members) == set(ints)
    for v in members:
        code = oz.e4m3_encode_integer(v)
        assert code in ints[v]
        if v != 0:
            assert oz.e4m3_decode(code) == v
    assert oz.e4m3_encode_integer(0) == 0
    for v in (17, 19, 21, 23, 33, 450, -17):
        assert not oz.e4m3_exact_integer(v)
    for q in range(-9, 9):
        assert oz.e4m3_decode(oz.e4m3_encode_power_of_two(q)) == 2.0 ** q


@pytest.mark.parametrize("m", ALL_MODULI)
def test_digits_reconstruct_and_are_e4m3(m):
    d = centred_range(m)
    ok = np.vectorize(oz.e4m3_exact_integer)
    for merged in (False, True):
        planes = oz.digit_planes(d, m, merged=merged)
        for p in planes:
            assert ok(p).all()
        s = oz.square_base(m)
        if s:
            assert np.array_equal(planes[0] + s * planes[1], d)
            assert planes[0].min() >= -(s // 2) and planes[0].max() <= s - 1 - s // 2
        else:
            d0, d1 = planes[1], (planes[2] // -16 if merged else planes[2])
            assert np.array_equal(d0 + 16 * d1, d)
            assert np.array_equal(planes[0], d0 + d1)


@pytest.mark.parametrize("m", ALL_MODULI)
def test_plane_identity_all_pairs(m):
    d = centred_range(m)
    for merged in (False, True):
        pa = [p[:, None] for p in oz.digit_planes(d, m, merged=merged)]
        pb = [p[None, :] for p in oz.digit_planes(d, m, merged=False)]
        v = oz.plane_product_value(pa, pb, m, merged=merged)
        want = d[:, None] * d[None, :]
        if oz.square_base(m):
            assert np.all(np.mod(v - want, m) == 0)
        else:
            # Eq. (kar) is an identity over the integers, not only mod m
            assert np.array_equal(v, want)


@pytest.mark.parametrize("m", ALL_MODULI)
def test_accumulator_term_bounds(m):
    d = centred_range(m)
    s = oz.square_base(m)
    if s:
        d0, d1 = oz.square_digits(d, s)
        t0 = np.abs(d0[:, None] * d0[None, :]).max()
        t1 = np.abs(d1[:, None] * d0[None, :] + d0[:, None] * d1[None, :]).max()
        assert t0 <= 256 and t1 <= 512
        # K_slab × max|term| ≤ 2^24 (Eq. accum-exact) for the kernel's slab
        assert 32768 * t1 <= 2**24
    else:
        d0, d1 = oz.nonsquare_digits(d)
        ts = np.abs((d0 + d1)[:, None] * (d0 + d1)[None, :]).max()
        t0 = np.abs(d0[:, None] * d0[None, :]).max()
        t1 = np.abs(d1[:, None] * d1[None, :]).max()
        tm = np.abs(d0[:, None] * d0[None, :] - 16 * d1[:, None] * d1[None, :]).max()
        assert ts <= 484 and t0 <= 196 and t1 <= 256 and tm <= 4095
        assert 4096 * tm < 2**24


def test_mutation_diagonal_pairing_is_caught():
    """A diagonal plane pairing (d1·e1 in place of the cross terms) must fail."""
    m, s = 1089, 33
    d = centred_range(m)
    d0, d1 = oz.square_digits(d, s)
    wrong = d0[:, None] * d0[None, :] + s * (d1[:, None] * d1[None, :])
    want = d[:, None] * d[None, :]
    assert not np.all(np.mod(wrong - want, m) == 0)


def test_mutation_uncorrected_split_is_caught():
    """Without the carry correction some sum planes leave E4M3 (§2.5)."""
    d = centred_range(511)
    d0 = np.mod(d + 8, 16) - 8
    d1 = (d - d0) // 16
    ok = np.vectorize(oz.e4m3_exact_integer)
    assert not ok(d0 + d1).all()
