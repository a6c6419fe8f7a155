"""Shared helpers for the GPU parity tests (marshalling only, no method arithmetic)."""
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "oz2.h")


def header_functions():
    txt = open(HEADER).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(oz2_\w+)\s*\(", txt, flags=re.M)))


def ensure_built():
    from paper_2606_06510_gb300 import LIB_PATH
    if not os.path.exists(LIB_PATH):
        from paper_2606_06510_gb300 import build
        build.build()


def to_dev(x, dtype=None):
    """numpy matrix -> column-major CUDA tensor."""
    import torch
    import paper_2606_06510_gb300 as oz
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return oz.colmajor(t.cuda()) if t.dim() == 2 else t.cuda()


def planes_from_residues(resid, mods, oz_oracle, k_pad, merged=False):
    """Oracle digit planes (E4M3 codes) of centred residue matrices, in the
    library's storage layout.

    resid: list over moduli of (rows, k) int arrays of centred residues.
    Returns a uint8 array (⌈rows/128⌉, k_pad/128, P, 128, 128): 128 × 128-byte
    blocks (row block, k-block, plane, row in block, byte), pad rows zero.
    """
    rows, k = resid[0].shape
    planes = []
    for d, m in zip(resid, mods):
        for p in oz_oracle.digit_planes(d, m, merged=merged):
            buf = np.zeros((rows, k_pad), dtype=np.uint8)
            buf[:, :k] = oz_oracle.e4m3_encode_array(p)
            planes.append(buf)
    P = len(planes)
    rows_pad = (rows + 127) // 128 * 128
    full = np.zeros((P, rows_pad, k_pad), dtype=np.uint8)
    full[:, :rows] = np.stack(planes)
    blocks = full.reshape(P, rows_pad // 128, 128, k_pad // 128, 128).transpose(1, 3, 0, 2, 4)
    return np.ascontiguousarray(blocks)
