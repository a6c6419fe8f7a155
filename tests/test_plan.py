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


# The host entry's block model (rates of the residue GEMM per CTA pair, of
# the reconstruction and of the host link, with per-unit, per-block and
# per-copy overheads), restated here to check the planner's optimisation.
MODEL = dict(pair_flops=46e12, unit_extra=2e-6, crt_bytes=4.0e12, link=190e9, block_extra=8e-6,
             copy_extra=5e-6)


def model_end(widths, m, k, r, pairs):
    """End of the last copy back for column blocks of these widths: each
    block's compute (its residue GEMM's waves of units, then its
    reconstruction) follows the previous block's; its copy follows both the
    block and the previous copy."""
    M = MODEL
    k_pad = -(-k // 128) * 128
    t_unit = 3 * 2 * 256 * 256 * k_pad / M["pair_flops"] + M["unit_extra"]
    per_tile = -(-m // 256) * r
    ce = cp = 0.0
    for w in widths:
        waves = -(-per_tile * -(-w // 256) // pairs)
        ce += waves * t_unit + w * m * (2 * r + 8) / M["crt_bytes"] + M["block_extra"]
        cp = max(ce, cp) + w * m * 8 / M["link"] + M["copy_extra"]
    return cp


def compositions(total, parts_max):
    import itertools
    for p in range(1, parts_max + 1):
        for cuts in itertools.combinations(range(1, total), p - 1):
            b = (0,) + cuts + (total,)
            yield [b[i + 1] - b[i] for i in range(p)]


def test_host_blocks(oz):
    """oz2_dgemm_host's column blocks: the 4096³ blocking, the shape of the
    plan at both ends of k (long k: a narrow last block, whose copy is the
    one left exposed; short k, where the link is the bottleneck: a narrow
    first block, which starts the copies early), and widths that cover n in
    multiples of 256 but the last, at most 8 of them."""
    P = oz.oz2_plan(4096, 4096, 4096, 12, cta_pairs=PAIRS)
    assert P["host_widths"] == [2304, 768, 768, 256]
    w = oz.oz2_plan(16384, 16384, 16384, 13, cta_pairs=PAIRS)["host_widths"]
    assert w[-1] == 256 and w[0] > 8192
    w = oz.oz2_plan(16384, 16384, 64, 12, cta_pairs=PAIRS)["host_widths"]
    assert w[0] == 256 and w == sorted(w)
    assert oz.oz2_plan(300, 1000, 64, 12)["host_widths"] == [1000]  # narrow C: one block
    rng = np.random.default_rng(18)
    for _ in range(300):
        m, n = int(rng.integers(1, 20000)), int(rng.integers(1, 40000))
        r = int(rng.integers(1, 17))
        w = oz.oz2_plan(m, n, int(rng.integers(1, 40000)), r, cta_pairs=PAIRS)["host_widths"]
        assert 1 <= len(w) <= 8 and sum(w) == n
        assert all(x % 256 == 0 and x > 0 for x in w[:-1])


def test_host_blocks_are_the_model_optimum(oz):
    """For C up to 12 tile columns wide, the planner's blocks end the last
    copy as early as the best of all partitions into at most 8 blocks of
    whole tile columns (by exhaustion) under the same model."""
    rng = np.random.default_rng(19)
    for _ in range(40):
        m = int(rng.integers(1, 20000))
        n = int(rng.integers(257, 12 * 256 + 1))
        k = int(rng.integers(1, 30000))
        r = int(rng.integers(1, 17))
        pairs = int(rng.integers(1, 80))
        w = oz.oz2_plan(m, n, k, r, cta_pairs=pairs)["host_widths"]
        tiles_n = -(-n // 256)
        best = min(model_end([256 * t for t in c[:-1]] + [n - 256 * (tiles_n - c[-1])], m, k, r, pairs)
                   for c in compositions(tiles_n, 8))
        assert model_end(w, m, k, r, pairs) <= best * (1 + 1e-9), (m, n, k, r, pairs, w)


def test_magnitude_gemm_split(oz):
    """The "+1" GEMM splits k only when its 256×256 tiles fill less than half
    a wave of the CTA pairs: none at 4096³; 4 parts for 16 tiles at
    k = 65536 (64 units on 76 pairs); 64 for a single tile; none when k is
    too short for two parts of 512 entries or the planes' scratch cannot
    hold m×n FP32 sums."""
    assert oz.oz2_plan(4096, 4096, 4096, 12, cta_pairs=PAIRS)["mag_kparts"] == 1
    assert oz.oz2_plan(1024, 1024, 65536, 12, cta_pairs=PAIRS)["mag_kparts"] == 4
    assert oz.oz2_plan(256, 256, 65536, 12, cta_pairs=PAIRS)["mag_kparts"] == 64
    assert oz.oz2_plan(1536, 1280, 1536, 12, cta_pairs=PAIRS)["mag_kparts"] == 2   # 30 tiles
    assert oz.oz2_plan(1024, 1024, 1000, 12, cta_pairs=PAIRS)["mag_kparts"] == 2   # 8 k-blocks: 2 parts of 4
    assert oz.oz2_plan(256, 256, 512, 12, cta_pairs=PAIRS)["mag_kparts"] == 1      # 4 k-blocks: one part
    rng = np.random.default_rng(20)
    for _ in range(500):
        m, n, k = int(rng.integers(1, 6000)), int(rng.integers(1, 6000)), int(rng.integers(1, 200000))
        pairs = int(rng.integers(1, 80))
        p = oz.oz2_plan(m, n, k, 12, cta_pairs=pairs)["mag_kparts"]
        t = tiles(m, n)
        ksteps = -(-k // 128)
        if p > 1:
            assert 2 * t < pairs and p <= 64 and p * t <= pairs
            s = -(-ksteps // p)
            assert s >= 4 and (p - 1) * s < ksteps         # parts of at least 4 k-blocks, none empty
        else:
            assert 2 * t >= pairs or min(64, pairs // t, ksteps // 4) < 2


def test_plan_argument_errors(oz):
    with pytest.raises(oz.Oz2Error):
        oz.oz2_plan(8, 8, 8, 12, cta_pairs=0)
    with pytest.raises(oz.Oz2Error):
        oz.oz2_plan(-1, 8, 8, 12)
    with pytest.raises(oz.Oz2Error):
        oz.oz2_plan(8, 8, 8, 17)
