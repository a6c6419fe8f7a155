"""CPU oracle for Ozaki Scheme II DGEMM emulation on an FP8 substrate.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
execute this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` use it.  It shares no code, tables or
constants with the CUDA library; the two meet only through the seeded input
generator in ``workloads.py``.

Modules
-------
ozaki2   the method, step by step (scale, quantise, residues, modular GEMMs,
         Garner, unscale, native fallback) plus the FP8 digit-plane layout.
cref     an independent high-accuracy reference product (Dot2 and exact
         integer dot products) used to measure error, not to define results.
"""
from . import ozaki2, cref  # noqa: F401
