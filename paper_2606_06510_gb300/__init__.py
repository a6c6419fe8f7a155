"""GB300-native Ozaki Scheme II DGEMM on FP8 tensor cores -- Python binding.

A thin ctypes layer over ``liboz2.so`` (include/oz2.h): every function here
marshals torch CUDA tensors into pointers, sizes and the current stream and
calls the C entry point of the same name.  All arithmetic happens in the
library's CUDA kernels; if the library is not built, every call raises.

Matrices follow the BLAS convention of the C ABI: column-major, i.e. a torch
tensor of shape (rows, cols) with stride(0) == 1.  ``colmajor(t)`` makes one.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liboz2.so")

OZ2_OK = 0
STATUS = {0: "OZ2_OK", -1: "OZ2_ERR_INVALID_ARG", -2: "OZ2_ERR_UNSUPPORTED_R", -3: "OZ2_ERR_ALLOC",
          -4: "OZ2_ERR_CUDA", -5: "OZ2_ERR_TIMEOUT", -6: "OZ2_ERR_UNSUPPORTED"}
QUANT = {"tz": 0, "rn": 1}
SCALE = {"r2": 0, "r1": 1}
FLAG_NO_FALLBACK = 0x1
FLAG_TIMING = 0x2
FLAG_FUSED = 0x4
FLAG_ON_THE_FLY = 0x8
FLAG_DEBUG_SIMT_GEMM = 0x100
STAGES = ("scan", "magnitude", "plus_one_gemm", "scale", "deconstruct", "residue_gemm", "crt", "fallback")


class Oz2Error(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {STATUS.get(code, code)}")
        self.code = code


class oz2_stats(ctypes.Structure):
    _fields_ = [("status", ctypes.c_int32), ("fallback_rows", ctypes.c_int32), ("fallback_cols", ctypes.c_int32),
                ("u_max", ctypes.c_int32), ("s", ctypes.c_int32), ("d_min", ctypes.c_int32),
                ("d_max", ctypes.c_int32), ("e_min", ctypes.c_int32), ("e_max", ctypes.c_int32),
                ("k_slab", ctypes.c_int32), ("stage_ms", ctypes.c_float * 8), ("timed_calls", ctypes.c_int32),
                ("kernel_launches", ctypes.c_int64)]


class oz2_ws_layout(ctypes.Structure):
    _fields_ = [(name, ctypes.c_size_t) for name in
                ("ra", "cb", "row_flag", "col_flag", "d", "e", "urow", "misc",
                 "mag_a", "mag_b", "planes_a", "planes_b", "residues", "total")] + \
               [("k_pad", ctypes.c_int64), ("num_planes", ctypes.c_int32), ("res_ld", ctypes.c_int64)]


class oz2_plan_info(ctypes.Structure):
    _fields_ = [("kparts", ctypes.c_int64), ("host_blocks", ctypes.c_int32),
                ("host_widths", ctypes.c_int64 * 8), ("host_kparts", ctypes.c_int64 * 8),
                ("mag_kparts", ctypes.c_int64)]


_I64, _P, _I, _U, _SZ = ctypes.c_int64, ctypes.c_void_p, ctypes.c_int, ctypes.c_uint, ctypes.c_size_t
_SIGS = {
    "oz2_dgemm": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _P, _I64, _I, _P]),
    "oz2_workspace_size": (_SZ, [_I64, _I64, _I64, _I]),
    "oz2_dgemm_host": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _P, _I64, _I, _P]),
    "oz2_dgemm_noalloc": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _P, _I64, _I, _P]),
    "oz2_dgemm_ex": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _P, _I64, _I, _I, _I, _U, _P, _SZ, _P]),
    "oz2_workspace_layout": (_I, [_I64, _I64, _I64, _I, ctypes.POINTER(oz2_ws_layout)]),
    "oz2_plane_layout": (_I, [_I, _P]),
    "oz2_plan": (_I, [_I64, _I64, _I64, _I, _I, ctypes.POINTER(oz2_plan_info)]),
    "oz2_get_stats": (_I, [ctypes.POINTER(oz2_stats)]),
    "oz2_trim_memory": (_I, []),
    "oz2_selftest_timeout": (_I, [ctypes.c_longlong, _P]),
    "oz2_check_device_status": (_I, []),
    "oz2_probe_mma_rate": (_I, [_I64, _P, _P]),
    "oz2_status_string": (ctypes.c_char_p, [_I]),
    "oz2_scan": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _U, _P, _P, _P, _P, _P]),
    "oz2_scale": (_I, [_I64, _I64, _I64, _I, _P, _I64, _P, _I64, _P, _P, _P, _P, _I, _I, _P, _P, _P, _P, _P, _P]),
    "oz2_deconstruct": (_I, [_I64, _I64, _I64, _I, _P, _I64, _P, _I64, _P, _P, _P, _P, _I, _P, _P, _P]),
    "oz2_residue_gemm": (_I, [_I64, _I64, _I64, _I, _P, _P, _P, _I64, _P]),
    "oz2_residue_gemm_simt": (_I, [_I64, _I64, _I64, _I, _P, _P, _P, _I64, _P]),
    "oz2_reconstruct": (_I, [_I64, _I64, _I, _P, _I64, _P, _P, _P, _I64, _P]),
    "oz2_fallback": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _P, _P, _P, _I64, _P]),
    "oz2_native_dgemm": (_I, [_I64, _I64, _I64, _P, _I64, _P, _I64, _P, _I64, _P]),
}
_LIB = None


def lib() -> ctypes.CDLL:
    """The loaded liboz2.so (raises if it has not been built)."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run `python -m paper_2606_06510_gb300.build` "
                               "(or __graft_entry__.build()) first")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _LIB = L
    return _LIB


def exported_symbols():
    return list(_SIGS)


def _check(code: int, what: str):
    if code != OZ2_OK:
        raise Oz2Error(code, what)


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def colmajor(t: torch.Tensor) -> torch.Tensor:
    """Column-major copy (stride(0) == 1) of a 2-D tensor, same device/dtype."""
    return t.t().contiguous().t()


def _ld(t: torch.Tensor) -> int:
    assert t.dim() == 2, "expected a matrix"
    if t.numel() == 0:
        return max(t.shape[0], 1)
    if t.shape[1] > 1 or t.shape[0] > 1:
        assert t.stride(0) == 1 or t.shape[0] == 1, "matrices must be column-major (stride(0) == 1)"
    return max(t.stride(1), t.shape[0], 1)


def _dev(*ts):
    for t in ts:
        if t is not None:
            assert t.is_cuda, "oz2 operates on CUDA tensors"
            assert t.is_contiguous() or t.stride(0) == 1 or t.dim() == 1


# ----------------------------------------------------------------- production
def oz2_dgemm(A: torch.Tensor, B: torch.Tensor, C: torch.Tensor = None, num_moduli: int = 12, stream=None):
    """C = A·B by Ozaki Scheme II (TZ, R2); allocates its workspace on the stream."""
    m, k = A.shape
    k2, n = B.shape
    assert k == k2 and A.dtype == B.dtype == torch.float64
    if C is None:
        C = torch.empty((n, m), dtype=torch.float64, device=A.device).t()
    _dev(A, B, C)
    _check(lib().oz2_dgemm(m, n, k, _ptr(A), _ld(A), _ptr(B), _ld(B), _ptr(C), _ld(C), num_moduli,
                           _stream(stream)), "oz2_dgemm")
    return C


def oz2_dgemm_host(A, B, C=None, num_moduli: int = 12, stream=None):
    """C = A·B with A, B, C in host memory (column-major float64 numpy arrays or
    CPU tensors; pinned CPU tensors transfer fastest).  Synchronises."""
    import numpy as np
    def host_ptr(x):
        if isinstance(x, torch.Tensor):
            return ctypes.c_void_p(x.data_ptr()), (max(x.stride(1), x.shape[0], 1))
        assert x.flags.f_contiguous or x.ndim == 2 and x.shape[1] == 1
        return ctypes.c_void_p(x.ctypes.data), max(x.shape[0], 1)
    m, k = A.shape
    n = B.shape[1]
    if C is None:
        C = np.empty((m, n), order="F")
    pa, lda = host_ptr(A)
    pb, ldb = host_ptr(B)
    pc, ldc = host_ptr(C)
    _check(lib().oz2_dgemm_host(m, n, k, pa, lda, pb, ldb, pc, ldc, num_moduli, _stream(stream)), "oz2_dgemm_host")
    return C


def oz2_workspace_size(m: int, n: int, k: int, num_moduli: int) -> int:
    return lib().oz2_workspace_size(m, n, k, num_moduli)


def oz2_workspace_layout(m: int, n: int, k: int, num_moduli: int) -> dict:
    L = oz2_ws_layout()
    _check(lib().oz2_workspace_layout(m, n, k, num_moduli, ctypes.byref(L)), "oz2_workspace_layout")
    return {name: getattr(L, name) for name, _ in L._fields_}


def oz2_plan(m: int, n: int, k: int, num_moduli: int = 12, cta_pairs: int = 76) -> dict:
    """How the library runs an m×n×k problem on cta_pairs CTA pairs (host
    arithmetic only): the residue GEMM's parts of k, the column blocks of
    oz2_dgemm_host with each block's parts of k, and the "+1" magnitude
    GEMM's parts of k."""
    P = oz2_plan_info()
    _check(lib().oz2_plan(m, n, k, num_moduli, cta_pairs, ctypes.byref(P)), "oz2_plan")
    nb = P.host_blocks
    return {"kparts": P.kparts, "host_widths": list(P.host_widths[:nb]), "host_kparts": list(P.host_kparts[:nb]),
            "mag_kparts": P.mag_kparts}


def oz2_plane_layout(num_moduli: int):
    offs = (ctypes.c_int32 * 16)()
    total = lib().oz2_plane_layout(num_moduli, ctypes.cast(offs, ctypes.c_void_p))
    if total < 0:
        raise Oz2Error(total, "oz2_plane_layout")
    return list(offs[:num_moduli]), total


def oz2_dgemm_ex(A, B, C=None, num_moduli=12, quant="tz", scale="r2", flags=0, workspace=None, stream=None):
    """oz2_dgemm with explicit variant, flags and workspace (a uint8 CUDA tensor).

    Returns (C, workspace); the workspace holds the intermediates at the
    offsets given by oz2_workspace_layout.
    """
    m, k = A.shape
    k2, n = B.shape
    assert k == k2
    if C is None:
        C = torch.empty((n, m), dtype=torch.float64, device=A.device).t()
    size = oz2_workspace_size(m, n, k, num_moduli)
    if workspace is None:
        workspace = torch.empty(max(size, 1), dtype=torch.uint8, device=A.device)
    _dev(A, B, C)
    _check(lib().oz2_dgemm_ex(m, n, k, _ptr(A), _ld(A), _ptr(B), _ld(B), _ptr(C), _ld(C), num_moduli,
                              QUANT[quant], SCALE[scale], flags, _ptr(workspace), workspace.numel(),
                              _stream(stream)), "oz2_dgemm_ex")
    return C, workspace


def oz2_selftest_timeout(limit_cycles: int = 2_000_000, stream=None):
    _check(lib().oz2_selftest_timeout(limit_cycles, _stream(stream)), "oz2_selftest_timeout")


def oz2_trim_memory():
    _check(lib().oz2_trim_memory(), "oz2_trim_memory")


def oz2_get_stats() -> dict:
    s = oz2_stats()
    _check(lib().oz2_get_stats(ctypes.byref(s)), "oz2_get_stats")
    out = {name: getattr(s, name) for name, _ in s._fields_ if name != "stage_ms"}
    out["stage_ms"] = dict(zip(STAGES, list(s.stage_ms)))
    return out


def oz2_probe_mma_rate(iters: int, stream=None) -> int:
    """Launch the tensor-pipe rate probe (iters MMAs of 256x256x32 FP8 per
    CTA pair) on the stream; returns the number of CTA pairs it runs on."""
    pairs = ctypes.c_int(0)
    _check(lib().oz2_probe_mma_rate(iters, ctypes.cast(ctypes.pointer(pairs), ctypes.c_void_p), _stream(stream)),
           "oz2_probe_mma_rate")
    return pairs.value


def oz2_check_device_status() -> int:
    return lib().oz2_check_device_status()


def oz2_status_string(code: int) -> str:
    return lib().oz2_status_string(code).decode()


# ----------------------------------------------------------------- stages
def oz2_scan(A, B, flags=0, stream=None):
    m, k = A.shape
    n = B.shape[1]
    dev = A.device
    ra = torch.empty(m, dtype=torch.int32, device=dev)
    cb = torch.empty(n, dtype=torch.int32, device=dev)
    rf = torch.empty(m, dtype=torch.uint8, device=dev)
    cf = torch.empty(n, dtype=torch.uint8, device=dev)
    _check(lib().oz2_scan(m, n, k, _ptr(A), _ld(A), _ptr(B), _ld(B), flags, _ptr(ra), _ptr(cb), _ptr(rf), _ptr(cf),
                          _stream(stream)), "oz2_scan")
    return ra, cb, rf, cf


def oz2_scale(A, B, ra, cb, rf, cf, num_moduli=12, quant="tz", scale="r2", stream=None):
    m, k = A.shape
    n = B.shape[1]
    dev = A.device
    k_pad = (k + 127) // 128 * 128
    mag_a = torch.empty((m, k_pad), dtype=torch.uint8, device=dev)
    mag_b = torch.empty((n, k_pad), dtype=torch.uint8, device=dev)
    urow = torch.empty(m, dtype=torch.float32, device=dev)
    d = torch.empty(m, dtype=torch.int32, device=dev)
    e = torch.empty(n, dtype=torch.int32, device=dev)
    _check(lib().oz2_scale(m, n, k, num_moduli, _ptr(A), _ld(A), _ptr(B), _ld(B), _ptr(ra), _ptr(cb), _ptr(rf),
                           _ptr(cf), QUANT[quant], SCALE[scale], _ptr(mag_a), _ptr(mag_b), _ptr(urow), _ptr(d),
                           _ptr(e), _stream(stream)), "oz2_scale")
    return mag_a, mag_b, urow, d, e


def plane_storage_shape(rows: int, k_pad: int, num_planes: int) -> tuple:
    """Shape of the digit-plane storage of an operand with `rows` rows:
    (row blocks, k-blocks, planes, 128 rows, 128 bytes), rows padded to 128."""
    return ((rows + 127) // 128, k_pad // 128, num_planes, 128, 128)


def oz2_deconstruct(A, B, d, e, rf, cf, num_moduli=12, quant="tz", stream=None):
    m, k = A.shape
    n = B.shape[1]
    k_pad = (k + 127) // 128 * 128
    _, P = oz2_plane_layout(num_moduli)
    pa = torch.empty(plane_storage_shape(m, k_pad, P), dtype=torch.uint8, device=A.device)
    pb = torch.empty(plane_storage_shape(n, k_pad, P), dtype=torch.uint8, device=A.device)
    _check(lib().oz2_deconstruct(m, n, k, num_moduli, _ptr(A), _ld(A), _ptr(B), _ld(B), _ptr(d), _ptr(e), _ptr(rf),
                                 _ptr(cf), QUANT[quant], _ptr(pa), _ptr(pb), _stream(stream)), "oz2_deconstruct")
    return pa, pb


def residue_ld(m: int) -> int:
    """Leading dimension of the column-major residue matrices (m rounded up to 8)."""
    return (m + 7) // 8 * 8


def oz2_residue_gemm(planes_a, planes_b, m, n, k, num_moduli=12, simt=False, stream=None):
    """planes: uint8 CUDA tensors in the storage layout oz2_deconstruct returns
    (plane_storage_shape).  Returns an int16 view of
    shape (r, m, n) over column-major storage (r, n, ldr), ldr = residue_ld(m)."""
    ldr = residue_ld(m)
    res = torch.empty((num_moduli, n, ldr), dtype=torch.int16, device=planes_a.device)
    fn = lib().oz2_residue_gemm_simt if simt else lib().oz2_residue_gemm
    _check(fn(m, n, k, num_moduli, _ptr(planes_a), _ptr(planes_b), _ptr(res), ldr, _stream(stream)),
           "oz2_residue_gemm")
    return res[:, :, :m].transpose(1, 2)


def _residue_storage(residues, m, n):
    """(tensor, ldr) of column-major residue storage for a (r, m, n) tensor:
    the tensor's own storage when it already has that layout (as the views
    oz2_residue_gemm returns do), else a column-major copy."""
    r = residues.shape[0]
    st = residues.stride()
    if residues.shape[1:] == (m, n) and st[1] == 1 and st[2] >= max(1, m) and st[0] == n * st[2]:
        return residues, st[2]
    ldr = residue_ld(m)
    buf = torch.zeros((r, n, ldr), dtype=torch.int16, device=residues.device)
    buf[:, :, :m].copy_(residues.transpose(1, 2))
    return buf, ldr


def oz2_reconstruct(residues, d, e, m, n, num_moduli=12, C=None, stream=None):
    """residues: int16 CUDA tensor (r, m, n); column-major storage per modulus
    is used as is, any other layout is copied into it first."""
    if C is None:
        C = torch.empty((n, m), dtype=torch.float64, device=residues.device).t()
    res, ldr = _residue_storage(residues, m, n)
    _check(lib().oz2_reconstruct(m, n, num_moduli, _ptr(res), ldr, _ptr(d), _ptr(e), _ptr(C), _ld(C),
                                 _stream(stream)), "oz2_reconstruct")
    return C


def oz2_fallback(A, B, rf, cf, C, stream=None):
    m, k = A.shape
    n = B.shape[1]
    _check(lib().oz2_fallback(m, n, k, _ptr(A), _ld(A), _ptr(B), _ld(B), _ptr(rf), _ptr(cf), _ptr(C), _ld(C),
                              _stream(stream)), "oz2_fallback")
    return C


def oz2_native_dgemm(A, B, C=None, stream=None):
    m, k = A.shape
    n = B.shape[1]
    if C is None:
        C = torch.empty((n, m), dtype=torch.float64, device=A.device).t()
    _check(lib().oz2_native_dgemm(m, n, k, _ptr(A), _ld(A), _ptr(B), _ld(B), _ptr(C), _ld(C), _stream(stream)),
           "oz2_native_dgemm")
    return C


def workspace_views(ws: torch.Tensor, m: int, n: int, k: int, num_moduli: int) -> dict:
    """Typed views of the intermediates in an oz2_dgemm_ex workspace."""
    L = oz2_workspace_layout(m, n, k, num_moduli)
    k_pad, P = L["k_pad"], L["num_planes"]

    def view(off, count, dtype, shape):
        nbytes = count * torch.empty((), dtype=dtype).element_size()
        return ws[off:off + nbytes].view(dtype).view(shape)

    return {
        "ra": view(L["ra"], m, torch.int32, (m,)), "cb": view(L["cb"], n, torch.int32, (n,)),
        "row_flag": view(L["row_flag"], m, torch.uint8, (m,)), "col_flag": view(L["col_flag"], n, torch.uint8, (n,)),
        "d": view(L["d"], m, torch.int32, (m,)), "e": view(L["e"], n, torch.int32, (n,)),
        "urow": view(L["urow"], m, torch.float32, (m,)),
        "mag_a": view(L["mag_a"], m * k_pad, torch.uint8, (m, k_pad)),
        "mag_b": view(L["mag_b"], n * k_pad, torch.uint8, (n, k_pad)),
        "planes_a": view(L["planes_a"], P * ((m + 127) // 128 * 128) * k_pad, torch.uint8,
                         plane_storage_shape(m, k_pad, P)),
        "planes_b": view(L["planes_b"], P * ((n + 127) // 128 * 128) * k_pad, torch.uint8,
                         plane_storage_shape(n, k_pad, P)),
        "residues": view(L["residues"], num_moduli * n * L["res_ld"], torch.int16,
                         (num_moduli, n, L["res_ld"]))[:, :, :m].transpose(1, 2),
    }
