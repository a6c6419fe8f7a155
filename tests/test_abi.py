"""The C-ABI library loads, exports every symbol its header declares, and
rejects invalid arguments on the host (no GPU compute is issued)."""
import ctypes

import pytest

from helpers import ensure_built, header_functions


@pytest.fixture(scope="module")
def oz():
    ensure_built()
    import paper_2606_06510_gb300 as oz
    oz.lib()
    return oz


def test_every_header_symbol_is_exported(oz):
    names = header_functions()
    assert len(names) == 22
    raw = ctypes.CDLL(oz.LIB_PATH)
    missing = [n for n in names if not hasattr(raw, n)]
    assert not missing
    assert set(names) <= set(oz.exported_symbols())


def test_status_strings(oz):
    for code, name in oz.STATUS.items():
        assert oz.oz2_status_string(code) == name


def test_host_argument_errors(oz):
    L = oz.lib()
    null = None
    # lda < m
    assert L.oz2_dgemm(8, 8, 8, null, 4, null, 8, null, 8, 12, null) == -1
    # ldb < k, ldc < m, negative sizes
    assert L.oz2_dgemm(8, 8, 8, null, 8, null, 4, null, 8, 12, null) == -1
    assert L.oz2_dgemm(8, 8, 8, null, 8, null, 8, null, 4, 12, null) == -1
    assert L.oz2_dgemm(-1, 8, 8, null, 8, null, 8, null, 8, 12, null) == -1
    # unsupported moduli counts
    assert L.oz2_dgemm(8, 8, 8, null, 8, null, 8, null, 8, 0, null) == -2
    assert L.oz2_dgemm(8, 8, 8, null, 8, null, 8, null, 8, 17, null) == -2
    # k beyond the exact "+1" pass limit
    assert L.oz2_dgemm(8, 8, (1 << 24) + 1, null, 8, null, (1 << 24) + 1, null, 8, 12, null) == -6
    # empty problems are no-ops
    assert L.oz2_dgemm(0, 8, 8, null, 1, null, 8, null, 1, 12, null) == 0
    assert L.oz2_dgemm(8, 0, 8, null, 8, null, 8, null, 8, 12, null) == 0
    # _ex: bad variant, missing/misaligned workspace
    assert L.oz2_dgemm_ex(8, 8, 8, 1, 8, 1, 8, 1, 8, 12, 5, 0, 0, null, 0, null) == -1
    assert L.oz2_dgemm_ex(8, 8, 8, 1, 8, 1, 8, 1, 8, 12, 0, 0, 0, null, 0, null) == -3
    assert L.oz2_dgemm_ex(8, 8, 8, 1, 8, 1, 8, 1, 8, 12, 0, 0, 0, 3, 1 << 30, null) == -3
    # failure-path self-test: limit out of range
    assert L.oz2_selftest_timeout(10, null) == -1
    # stage entries: residue leading dimension below m
    assert L.oz2_residue_gemm(8, 8, 8, 12, 1, 1, 1, 7, null) == -1
    assert L.oz2_reconstruct(8, 8, 12, 1, 7, 1, 1, 1, 8, null) == -1


def test_layout_queries(oz):
    offs, total = oz.oz2_plane_layout(12)
    assert total == 30 and offs == [0, 2, 4, 6, 8, 10, 12, 15, 18, 21, 24, 27]
    assert oz.oz2_plane_layout(16)[1] == 42
    L = oz.oz2_workspace_layout(300, 200, 129, 12)
    assert L["k_pad"] == 256 and L["num_planes"] == 30
    keys = ["ra", "cb", "row_flag", "col_flag", "d", "e", "urow", "misc", "mag_a", "mag_b", "planes_a",
            "planes_b", "residues", "total"]
    offs = [L[k] for k in keys]
    assert offs == sorted(offs) and all(o % 256 == 0 for o in offs)
    assert L["planes_b"] - L["planes_a"] >= 30 * 300 * 256
    assert L["res_ld"] == 304 and L["total"] - L["residues"] >= 2 * 12 * 304 * 200
    assert oz.oz2_workspace_layout(301, 5, 1, 3)["res_ld"] == 304
    assert oz.oz2_workspace_size(300, 200, 129, 12) == L["total"]
