"""The library's own planning logic, through oz2_plan, on the host (no GPU):
the residue GEMM's split of k and the host entry's column blocks."""
import numpy as np
import pytest

from helpers import ensure_built

PAIRS = 76  # CTA pairs of a GB300 (152 SMs)


@pytest.fixture(scope="module")
def oz():
    ensure_built()
    import paper_2606_06510_gb300 as oz
    oz.lib()
    return oz


def tiles(m, n):
    return -(-m // 256) * -(-n // 256)


@pytest.mark.parametrize("shape,kparts", [
    ((4096, 4096, 4096, 12), 1),      # 3072 units: many waves
    ((16384, 16384, 16384, 13), 1),
    ((1024, 1024, 65536, 12), 1),     # 192 units, balanced by the schedule
    ((1536, 1280, 1536, 12), 1),      # 360 units: at least four waves
    ((256, 256, 65536, 12), 12),      # 12 units on 76 pairs
    ((512, 512, 65536, 12), 3),
    ((9, 7, 262144, 12), 12),
    ((200, 136, 300, 12), 1),         # k too short to split
])
def test_split_choice(oz, shape, kparts):
    assert oz.oz2_plan(*shape, cta_pairs=PAIRS)["kparts"] == kparts


def test_split_invariants(oz):
    """Over seeded shapes: a split happens only for problems under four
    waves of units, every part is non-empty and at least 4 k-blocks long,
    there are at most 16, and the partial residues fit in the magnitude-plane
    region of the workspace."""
    rng = np.random.default_rng(17)
    splits = 0
    for _ in range(3000):
        m, n = (int(x) for x in rng.integers(1, 1600, size=2))
        k = int(rng.integers(1, 300000))
        r = int(rng.integers(1, 17))
        pairs = int(rng.choice([1, 8, 76, 100]))
        p = oz.oz2_plan(m, n, k, r, cta_pairs=pairs)["kparts"]
        assert 1 <= p <= 16
        if p == 1:
            continue
        splits += 1
        ksteps = -(-k // 128)
        s = -(-ksteps // p)
        assert tiles(m, n) * r < 4 * pairs
        assert s >= 4 and (p - 1) * s < ksteps
        L = oz.oz2_workspace_layout(m, n, k, r)
        assert p * r * n * L["res_ld"] * 2 <= L["planes_a"] - L["mag_a"]
    assert splits > 300


def test_host_blocks(oz):
    """oz2_dgemm_host's column blocks: the documented 4096² blocking, and over
    seeded shapes widths that cover n, multiples of 256 but the last, which
    is the last tile column."""
    P = oz.oz2_plan(4096, 4096, 4096, 12, cta_pairs=PAIRS)
    assert P["host_widths"] == [1280, 1280, 1280, 256]
    assert oz.oz2_plan(300, 1000, 64, 12)["host_widths"] == [1000]  # narrow C: one block
    rng = np.random.default_rng(18)
    for _ in range(2000):
        m, n = int(rng.integers(1, 20000)), int(rng.integers(1, 40000))
        r = int(rng.integers(1, 17))
        w = oz.oz2_plan(m, n, 1024, r, cta_pairs=PAIRS)["host_widths"]
        assert 1 <= len(w) <= 8 and sum(w) == n
        if len(w) > 1:
            assert all(x % 256 == 0 and x >= 768 for x in w[:-1])
            assert w[-1] == n - 256 * (-(-n // 256) - 1)


def test_plan_argument_errors(oz):
    with pytest.raises(oz.Oz2Error):
        oz.oz2_plan(8, 8, 8, 12, cta_pairs=0)
    with pytest.raises(oz.Oz2Error):
        oz.oz2_plan(-1, 8, 8, 12)
    with pytest.raises(oz.Oz2Error):
        oz.oz2_plan(8, 8, 8, 17)
