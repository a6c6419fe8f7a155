"""Pin the oracle's layout and constants to the numbers the paper prints.

Fixture: tests/golden/paper_constants.txt (each value cites its passage).
"""
import math

import numpy as np
import pytest

from conftest import golden
from oracle import ozaki2 as oz


def load_constants():
    out = {}
    with open(golden("paper_constants.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            name, value = line.split()[:2]
            out[name] = float(value)
    return out


K = load_constants()


def centred_range(m):
    return np.arange(-(m // 2), m - m // 2)


def test_modulus_set_is_pairwise_coprime_and_log2M():
    S = oz.moduli(12)
    assert S == oz.MODULI_S
    allm = oz.moduli(16)
    for i in range(len(allm)):
        for j in range(i + 1, len(allm)):
            assert math.gcd(allm[i], allm[j]) == 1
    assert round(math.log2(oz.modulus_product(S)), 1) == K["log2_M_S"]
    assert round(sum(math.log2(j) for j in range(243, 257)), 1) == K["log2_M_bytes14"]
    assert 3 * 12 + 1 == K["alpha_r12"]
    assert round(5.0e15 / K["alpha_r12"] / 1e12) == K["emulated_ceiling_tflops"]


def test_three_counts():
    p_store, p_mma, n_acc = oz.plane_counts(oz.MODULI_S)
    assert (p_store, p_mma, n_acc) == (K["p_store_S"], K["p_mma_S"], K["n_acc_S"])


def test_tail_digit_extremes_and_correction_rate():
    tot = corr = 0
    mx0 = mx1 = mxs = 0
    for m in oz.MODULI_S[6:]:
        d = centred_range(m)
        d0, d1 = oz.nonsquare_digits(d)
        b0 = np.mod(d + 8, 16) - 8
        corr += int(np.sum(d0 != b0))
        tot += d.size
        mx0 = max(mx0, int(np.abs(d0).max()))
        mx1 = max(mx1, int(np.abs(d1).max()))
        mxs = max(mxs, int(np.abs(d0 + d1).max()))
    assert (mx0, mx1, mxs) == (K["tail_max_d0"], K["tail_max_d1"], K["tail_max_d0_plus_d1"])
    assert abs(corr / tot - K["tail_correction_fraction"]) < 0.01
    assert mxs * mxs == K["tail_unmerged_max_product"]


def test_tail_merged_term_maximum():
    best = 0
    for m in oz.MODULI_S[6:]:
        d0, d1 = oz.nonsquare_digits(centred_range(m))
        t = np.abs(d0[:, None] * d0[None, :] - 16 * d1[:, None] * d1[None, :])
        best = max(best, int(t.max()))
        # the pre-scaled plane is E4M3-exact and reaches -256 = -2^8
        assert all(oz.e4m3_exact_integer(v) for v in np.unique(-16 * d1))
        assert int(np.abs(16 * d1).max()) == 256
    assert best == K["tail_merged_max_term"]
    # exact at K_slab = 4096 by a single term
    assert 4096 * best < 2**24 <= 4097 * best + best


def _canonical_ok(m, B):
    d = centred_range(m)
    h = B // 2
    d0 = np.mod(d + h, B) - h
    d1 = (d - d0) // B
    ok = np.vectorize(oz.e4m3_exact_integer)
    return bool(ok(d0).all() and ok(d1).all() and ok(d0 + d1).all())


def test_canonical_envelope():
    def largest(B):
        m = 2
        while _canonical_ok(m + 1, B):
            m += 1
        return m
    assert largest(16) == K["envelope_canonical_B16"]
    assert largest(17) == K["envelope_canonical_B17"]
    assert max(largest(B) for B in range(4, 40)) == K["envelope_canonical_B17"]
    m, B = int(K["envelope_canonical_B17"]), 17
    d = centred_range(m)
    d0 = np.mod(d + 8, B) - 8
    d1 = (d - d0) // B
    assert int(np.abs(d0).max()) == K["canonical_B17_digit_max"]
    assert int(np.abs(d1).max()) == K["canonical_B17_high_max"]
    assert int(np.abs(d0 + d1).max()) == K["canonical_B17_sum_max"]
    assert 17 * 19 >= m


def test_square_envelope_is_tight_at_33():
    ok = np.vectorize(oz.e4m3_exact_integer)
    for s in range(2, 34):
        d0, d1 = oz.square_digits(centred_range(s * s), s)
        assert ok(d0).all() and ok(d1).all()
    d0, d1 = oz.square_digits(centred_range(34 * 34), 34)
    assert not (ok(d0).all() and ok(d1).all())
    assert 33 * 33 == K["envelope_square"]


def test_accumulation_constants():
    assert 16 * 16 == K["max_term_square_d0e0"]
    assert 2 * 16 * 16 == K["max_term_square_cross"]
    assert 2**24 // int(K["max_term_merged"]) == K["kslab_limit"]
    assert K["max_term_merged"] * K["kslab_design"] == K["acc_at_design"]
    assert round(2**24 / K["acc_at_design"], 2) == K["acc_margin"]


def test_n_gamma():
    r = 12
    assert r * (r - 1) // 2 + 2 * r == K["n_gamma_r12"]
