"""Workspace canaries: every intermediate the call must write is written in
full, and nothing is written outside it.

The workspace, 64 KiB of guard bytes on each side of it and the pad rows of
C are filled with 0x7F bytes, a value no stage produces in any region (an
E4M3 NaN in the planes, 32639 as a residue, 0x7F7F7F7F as a scale or scan
key, 3.4e38 as a row maximum of U, 0x7F as a flag byte; C gets a NaN of a
payload the reconstruction never writes).  After the call the regions the
path writes must hold no canary element, and the guard bytes, the gaps
between the 256-byte aligned regions and C's pad rows must hold nothing
else.  (compute-sanitizer is closed on this machine; this checks the same
write bounds from the outside.)
"""
import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built, to_dev

pytestmark = pytest.mark.gpu

GUARD = 64 * 1024
CANARY = 0x7F
C_CANARY = 0x7FF7CA11CA11CA11


@pytest.fixture(scope="module")
def oz():
    ensure_built()
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_06510_gb300 as oz
    oz.lib()
    return oz


def regions(L, m, n, r, k_pad, planes_a_written, residues_written, mag_written):
    """(name, offset, bytes, element size) of what the call must write."""
    P = L["num_planes"]
    out = [("ra", L["ra"], 4 * m, 4), ("cb", L["cb"], 4 * n, 4), ("row_flag", L["row_flag"], m, 1),
           ("col_flag", L["col_flag"], n, 1), ("d", L["d"], 4 * m, 4), ("e", L["e"], 4 * n, 4),
           ("urow", L["urow"], 4 * m, 4),
           ("planes_b", L["planes_b"], P * ((n + 127) // 128 * 128) * k_pad, 1)]
    if mag_written:
        out += [("mag_a", L["mag_a"], m * k_pad, 1), ("mag_b", L["mag_b"], n * k_pad, 1)]
    if planes_a_written:
        out.append(("planes_a", L["planes_a"], P * ((m + 127) // 128 * 128) * k_pad, 1))
    if residues_written:
        out.append(("residues", L["residues"], 2 * r * n * L["res_ld"], 2))
    return out


def extents(L, m, n, r, k_pad):
    """Every region's full extent (written or not), to find the gaps between them."""
    P = L["num_planes"]
    return sorted([(L["ra"], 4 * m), (L["cb"], 4 * n), (L["row_flag"], m), (L["col_flag"], n), (L["d"], 4 * m),
                   (L["e"], 4 * n), (L["urow"], 4 * m), (L["misc"], 4 * (m + n + 2)), (L["mag_a"], m * k_pad),
                   (L["mag_b"], n * k_pad), (L["planes_a"], P * ((m + 127) // 128 * 128) * k_pad),
                   (L["planes_b"], P * ((n + 127) // 128 * 128) * k_pad), (L["residues"], 2 * r * n * L["res_ld"])])


@pytest.mark.parametrize("shape,r,flags,path", [
    ((77, 45, 131), 12, 0, "stored"),
    ((300, 7, 1500), 12, "ON_THE_FLY", "on_the_fly"),
    ((300, 7, 1500), 12, 0, "stored"),
    ((130, 33, 100), 12, "FUSED", "fused"),
    ((9, 7, 9000), 16, 0, "split"),          # the residue GEMM splits k
    ((129, 257, 300), 5, 0, "stored"),
])
def test_intermediates_written_in_full_and_nothing_outside(oz, shape, r, flags, path):
    import torch
    m, n, k = shape
    fl = getattr(oz, f"FLAG_{flags}") if flags else 0
    A = wl.random_matrix(m, k, 1.0, 9300 + m)
    B = wl.random_matrix(k, n, 1.0, 9400 + n)
    size = oz.oz2_workspace_size(m, n, k, r)
    buf = torch.full((size + 2 * GUARD,), CANARY, dtype=torch.uint8, device="cuda")
    ws = buf[GUARD:GUARD + size]
    assert ws.data_ptr() % 256 == 0
    ldc = m + 3
    Cbuf = torch.full((n, ldc), 0, dtype=torch.int64, device="cuda")
    Cbuf.fill_(C_CANARY)
    C = Cbuf.view(torch.float64).t()[:m, :]
    oz.oz2_dgemm_ex(to_dev(A), to_dev(B), C=C, num_moduli=r, flags=fl, workspace=ws)
    torch.cuda.synchronize()
    assert oz.oz2_check_device_status() == 0
    host = buf.cpu().numpy()
    assert (host[:GUARD] == CANARY).all() and (host[GUARD + size:] == CANARY).all(), "write outside the workspace"
    w = host[GUARD:GUARD + size]
    L = oz.oz2_workspace_layout(m, n, k, r)
    k_pad = L["k_pad"]
    # gaps between the aligned regions stay untouched
    ext = extents(L, m, n, r, k_pad)
    for (o0, b0), (o1, _) in zip(ext, ext[1:]):
        assert (w[o0 + b0:o1] == CANARY).all(), f"write into the gap after offset {o0}"
    assert (w[ext[-1][0] + ext[-1][1]:] == CANARY).all()
    # every element of the written regions was written
    # A residue GEMM that splits k keeps its partial residues (any bytes) in
    # the magnitude-plane region; that path is checked through the residues.
    split = path in ("stored", "split") and oz.oz2_plan(m, n, k, r, 76)["kparts"] > 1
    for name, off, nbytes, esz in regions(L, m, n, r, k_pad, planes_a_written=path != "on_the_fly",
                                          residues_written=path != "fused", mag_written=not split):
        v = w[off:off + nbytes]
        if name == "residues":   # the rows < m of every column of every modulus
            v = v.view(np.int16).reshape(r, n, L["res_ld"])[:, :, :m]
            assert not (v == 0x7F7F).any(), "residue entry left unwritten"
            continue
        if esz == 4:
            assert not (v.view(np.uint32) == 0x7F7F7F7F).any(), f"{name}: entry left unwritten"
        else:
            assert not (v == CANARY).any(), f"{name}: byte left unwritten"
    Ch = Cbuf.cpu().numpy()
    assert (Ch[:, m:] == C_CANARY).all(), "write into C's pad rows"
    assert not (Ch[:, :m] == C_CANARY).any(), "entry of C left unwritten"
