"""GB300-native ExTernD: ternary expanded-rank factorization A ~ B diag(D) C on one GPU.

Thin Python binding of libexternd.so (the C ABI in include/externd.h). Every function here only marshals
arguments: it allocates result tensors with PyTorch on the current CUDA device, passes raw pointers and the current
stream to the library, and raises ``ExterndError`` on a non-zero status. All arithmetic runs in the library's CUDA
kernels; there is no CPU fallback. If the library has not been built, the first call raises ``ExterndError``
(build it with ``python -m paper_2607_13511_gb300.build`` or ``__graft_entry__.build()``).
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

__all__ = [
    "ExterndError", "Decomposition", "library_path", "load", "rank", "block_width", "decompose", "decompose_traced",
    "decompose_host",
    "energy", "ternarize", "vstep_product", "ustep_product", "vstep_target", "ustep_target", "block_scales",
    "deflate", "profile", "profile_read", "kernel_launches", "PROFILE_KINDS", "Packed", "pack_ternary",
    "ternary_apply", "block_boundaries", "rank_for_energy", "allocate_ranks", "decompose_safeguarded", "refine",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB: Optional[ctypes.CDLL] = None

_c_i64, _c_int, _c_double, _c_void = ctypes.c_int64, ctypes.c_int, ctypes.c_double, ctypes.c_void_p
_c_dptr = ctypes.POINTER(ctypes.c_double)

# name -> (restype, argtypes); mirrors include/externd.h
_SIGNATURES = {
    "externd_strerror": (ctypes.c_char_p, [_c_int]),
    "externd_last_cuda_error": (ctypes.c_char_p, []),
    "externd_version": (ctypes.c_char_p, []),
    "externd_set_stream": (_c_int, [_c_void]),
    "externd_rank": (_c_int, [_c_i64, _c_i64, _c_double, ctypes.POINTER(_c_i64)]),
    "externd_block_width": (_c_int, [_c_i64, _c_i64, _c_int, ctypes.POINTER(_c_int)]),
    "externd_decompose": (_c_int, [_c_void, _c_i64, _c_i64, _c_double, _c_double, _c_int, _c_int, _c_void,
                                   _c_void, _c_void, _c_void, _c_dptr]),
    "externd_decompose_traced": (_c_int, [_c_void, _c_i64, _c_i64, _c_double, _c_double, _c_int, _c_int,
                                          _c_void, _c_void, _c_void, _c_void, _c_dptr, _c_dptr]),
    "externd_decompose_host": (_c_int, [_c_void, _c_i64, _c_i64, _c_double, _c_double, _c_int, _c_int, _c_void,
                                        _c_void, _c_void, _c_void, _c_dptr]),
    "externd_energy": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_void, _c_void, _c_i64, _c_void, _c_dptr]),
    "externd_energy_noalloc": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_void, _c_void, _c_i64, _c_void,
                                        _c_dptr]),
    "externd_profile": (_c_int, [_c_int]),
    "externd_profile_read": (_c_int, [_c_dptr, ctypes.POINTER(_c_i64)]),
    "externd_kernel_launches": (_c_int, [ctypes.POINTER(_c_i64)]),
    "externd_ternarize": (_c_int, [_c_void, _c_i64, _c_i64, _c_int, _c_double, _c_void]),
    "externd_vstep_product": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_i64, _c_void]),
    "externd_ustep_product": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_i64, _c_void, _c_void]),
    "externd_vstep_target": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_i64, _c_void]),
    "externd_ustep_target": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_i64, _c_void, _c_void]),
    "externd_block_scales": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_void, _c_i64, _c_void, _c_void]),
    "externd_deflate": (_c_int, [_c_void, _c_i64, _c_i64, _c_void, _c_void, _c_void, _c_i64, _c_void, _c_dptr]),
    "externd_decompose_safeguarded": (_c_int, [_c_void, _c_i64, _c_i64, _c_double, _c_double, _c_int, _c_int,
                                               _c_void, _c_void, _c_void, _c_void, _c_dptr, _c_dptr,
                                               ctypes.POINTER(_c_i64)]),
    "externd_refine": (_c_int, [_c_void, _c_i64, _c_i64, _c_double, _c_int, _c_int, _c_int, _c_void, _c_void,
                                _c_void, _c_void, _c_i64, _c_dptr, _c_dptr, ctypes.POINTER(_c_i64)]),
    "externd_block_boundaries": (_c_int, [_c_i64, _c_i64, _c_double, _c_int, ctypes.POINTER(_c_i64),
                                          ctypes.POINTER(_c_i64)]),
    "externd_rank_for_energy": (_c_int, [_c_i64, _c_i64, _c_double, _c_int, _c_dptr, _c_i64, _c_double,
                                         ctypes.POINTER(_c_i64)]),
    "externd_allocate_ranks": (_c_int, [_c_i64, ctypes.POINTER(_c_i64), ctypes.POINTER(_c_i64), _c_dptr, _c_dptr,
                                        _c_dptr, _c_double, ctypes.POINTER(_c_i64)]),
    "externd_pack_ternary": (_c_int, [_c_void, _c_i64, _c_i64, _c_i64, _c_void, ctypes.POINTER(_c_i64)]),
    "externd_ternary_apply": (_c_int, [_c_void, _c_void, _c_void, _c_i64, _c_i64, _c_i64, _c_void, _c_void]),
}


class ExterndError(RuntimeError):
    """A non-zero status from libexternd, or the library missing."""


def library_path() -> str:
    return os.path.join(_HERE, "_build", "libexternd.so")


def load() -> ctypes.CDLL:
    """Loads libexternd.so (once) and declares the C signatures."""
    global _LIB
    if _LIB is None:
        path = library_path()
        if not os.path.exists(path):
            raise ExterndError(f"libexternd.so is not built ({path}); run python -m paper_2607_13511_gb300.build")
        lib = ctypes.CDLL(path)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype, fn.argtypes = res, args
        _LIB = lib
    return _LIB


def _check(status: int) -> None:
    if status != 0:
        lib = load()
        msg = lib.externd_strerror(status).decode()
        if status == -4:
            msg += ": " + lib.externd_last_cuda_error().decode()
        raise ExterndError(f"libexternd status {status}: {msg}")


def _torch():
    import torch
    return torch


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _prep(t, dtype, name):
    torch = _torch()
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ExterndError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ExterndError(f"{name} must be {dtype}, got {t.dtype}")
    return t.contiguous()


def _stream(lib, device) -> None:
    torch = _torch()
    lib.externd_set_stream(ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream))


PROFILE_KINDS = {"off": 0, "vstep": 1, "ustep": 2, "deflate": 3, "decorrelate": 4, "apply": 5, "gram": 6,
                 "solve": 7, "start": 8, "products": 9}


def profile(kind: str) -> None:
    """Times one kernel class inside later decompose calls with CUDA events (see profile_read)."""
    _check(load().externd_profile(PROFILE_KINDS[kind]))


def profile_read() -> tuple[float, int]:
    """(device ms, launches) of the profiled kernel class during the last decompose call."""
    ms, n = _c_double(), _c_i64()
    _check(load().externd_profile_read(ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def kernel_launches() -> int:
    """Kernels launched by the last decompose call."""
    n = _c_i64()
    _check(load().externd_kernel_launches(ctypes.byref(n)))
    return n.value


def rank(m: int, n: int, mu: float) -> int:
    """§2.1 inner rank k = floor(mu * min(m, n) + 0.5)."""
    k = _c_i64()
    _check(load().externd_rank(m, n, mu, ctypes.byref(k)))
    return k.value


def block_width(m: int, n: int, block: int) -> int:
    """§2.4 block width min(block, floor(min(m, n)/8)), at least 1."""
    b = _c_int()
    _check(load().externd_block_width(m, n, block, ctypes.byref(b)))
    return b.value


@dataclass
class Decomposition:
    B: "object"          # m x k int8 {-1, 0, 1}
    D: "object"          # k float32
    C: "object"          # k x n int8 {-1, 0, 1}
    energy: float        # 1 - ||A - B diag(D) C||_H^2 / ||A||_H^2 (tracked residual)
    trace: Optional[list] = None   # energy after each block (decompose_traced, the extension entry points)


def _decompose_call(fn_name, A, mu, tau, block, iters, weights, out, traced):
    torch = _torch()
    lib = load()
    A = _prep(A, torch.float32, "A")
    m, n = A.shape
    k = rank(m, n, mu)
    h = None if weights is None else _prep(weights, torch.float32, "weights")
    if out is None:
        B = torch.empty((m, k), dtype=torch.int8, device=A.device)
        D = torch.empty((k,), dtype=torch.float32, device=A.device)
        C = torch.empty((k, n), dtype=torch.int8, device=A.device)
    else:
        B, D, C = out
    e = _c_double()
    args = [_ptr(A), m, n, mu, tau, block, iters, _ptr(h), _ptr(B), _ptr(D), _ptr(C), ctypes.byref(e)]
    tr = None
    if traced:
        tr = (_c_double * -(-k // block_width(m, n, block)))()
        args.append(tr)
    with torch.cuda.device(A.device):
        _stream(lib, A.device)
        _check(getattr(lib, fn_name)(*args))
    return Decomposition(B, D, C, e.value, None if tr is None else list(tr))


def decompose(A, mu: float, tau: float, block: int, iters: int, weights=None, out=None) -> Decomposition:
    """ExTernD of a CUDA float32 matrix A (m x n): §2.3 (block 1) / §2.4 block ALS, §2.5 when weights is given.

    ``out`` may pass preallocated (B, D, C) tensors to reuse. The result carries no per-block trace (see
    ``decompose_traced``)."""
    return _decompose_call("externd_decompose", A, mu, tau, block, iters, weights, out, False)


def decompose_traced(A, mu: float, tau: float, block: int, iters: int, weights=None, out=None) -> Decomposition:
    """``decompose`` that also returns the energy after every block (``trace``): E(k) at k = b, 2b, ..., k."""
    return _decompose_call("externd_decompose_traced", A, mu, tau, block, iters, weights, out, True)


def decompose_safeguarded(A, mu: float, tau: float, block: int, iters: int, weights=None, out=None):
    """``decompose`` with Prop. 2's safeguard; returns (Decomposition, blocks replaced by a single-entry pair).
    ``out`` may pass preallocated (B, D, C) tensors to reuse."""
    torch = _torch()
    lib = load()
    A = _prep(A, torch.float32, "A")
    m, n = A.shape
    k = rank(m, n, mu)
    nblocks = -(-k // block_width(m, n, block))
    h = None if weights is None else _prep(weights, torch.float32, "weights")
    if out is None:
        B = torch.empty((m, k), dtype=torch.int8, device=A.device)
        D = torch.empty((k,), dtype=torch.float32, device=A.device)
        C = torch.empty((k, n), dtype=torch.int8, device=A.device)
    else:
        B, D, C = out
    e = _c_double()
    tr = (_c_double * nblocks)()
    act = _c_i64()
    with torch.cuda.device(A.device):
        _stream(lib, A.device)
        _check(lib.externd_decompose_safeguarded(_ptr(A), m, n, mu, tau, block, iters, _ptr(h), _ptr(B), _ptr(D),
                                                 _ptr(C), ctypes.byref(e), tr, ctypes.byref(act)))
    return Decomposition(B, D, C, e.value, list(tr)), act.value


def refine(A, dec: Decomposition, tau: float, block: int, iters: int, sweeps: int, weights=None, out=None):
    """§2.4 refinement sweeps of ``dec``'s factors (same block layout as the run that made them). Returns
    (Decomposition with new factors, blocks replaced per sweep); ``dec``'s tensors are left untouched. ``out`` may
    pass preallocated (B, D, C) tensors that receive the factors (they are copied from ``dec`` first)."""
    torch = _torch()
    lib = load()
    A = _prep(A, torch.float32, "A")
    m, n = A.shape
    if out is None:
        B, D, C = dec.B.clone(), dec.D.clone(), dec.C.clone()
    else:
        B, D, C = out
        B.copy_(dec.B)
        D.copy_(dec.D)
        C.copy_(dec.C)
    k = B.shape[1]
    h = None if weights is None else _prep(weights, torch.float32, "weights")
    e = _c_double()
    tr = (_c_double * sweeps)()
    rep = (_c_i64 * sweeps)()
    with torch.cuda.device(A.device):
        _stream(lib, A.device)
        _check(lib.externd_refine(_ptr(A), m, n, tau, block, iters, sweeps, _ptr(h), _ptr(B), _ptr(D), _ptr(C), k,
                                  ctypes.byref(e), tr, rep))
    return Decomposition(B, D, C, e.value, list(tr)), list(rep)


def decompose_host(A, mu: float, tau: float, block: int, iters: int, weights=None, out=None) -> Decomposition:
    """Same as ``decompose`` for a host (CPU) float32 tensor: copies in and out happen inside the library call."""
    torch = _torch()
    lib = load()
    if A.is_cuda or A.dtype != torch.float32:
        raise ExterndError("A must be a CPU float32 tensor")
    A = A.contiguous()
    m, n = A.shape
    k = rank(m, n, mu)
    h = None if weights is None else weights.contiguous()
    if out is None:
        pin = torch.cuda.is_available()
        B = torch.empty((m, k), dtype=torch.int8, pin_memory=pin)
        D = torch.empty((k,), dtype=torch.float32, pin_memory=pin)
        C = torch.empty((k, n), dtype=torch.int8, pin_memory=pin)
    else:
        B, D, C = out
    e = _c_double()
    _stream(lib, torch.cuda.current_device())
    _check(lib.externd_decompose_host(_ptr(A), m, n, mu, tau, block, iters, _ptr(h), _ptr(B), _ptr(D), _ptr(C),
                                      ctypes.byref(e)))
    return Decomposition(B, D, C, e.value)


def energy(A, B, D, C, weights=None) -> float:
    """Eq. 1 (weighted per §2.5): 1 - ||A - B diag(D) C||_H^2 / ||A||_H^2 computed from the factors."""
    torch = _torch()
    lib = load()
    A = _prep(A, torch.float32, "A")
    B, D, C = _prep(B, torch.int8, "B"), _prep(D, torch.float32, "D"), _prep(C, torch.int8, "C")
    h = None if weights is None else _prep(weights, torch.float32, "weights")
    m, n = A.shape
    e = _c_double()
    with torch.cuda.device(A.device):
        _stream(lib, A.device)
        _check(lib.externd_energy(_ptr(A), m, n, _ptr(B), _ptr(D), _ptr(C), D.numel(), _ptr(h), ctypes.byref(e)))
    return e.value


def ternarize(X, tau: float, axis: int = 1):
    """Eq. 2 on each row (axis=1) or column (axis=0) of a CUDA float32 matrix; returns int8."""
    torch = _torch()
    lib = load()
    X = _prep(X, torch.float32, "X")
    T = torch.empty(X.shape, dtype=torch.int8, device=X.device)
    with torch.cuda.device(X.device):
        _stream(lib, X.device)
        _check(lib.externd_ternarize(_ptr(X), X.shape[0], X.shape[1], axis, tau, _ptr(T)))
    return T


def _step(fn_name, R, F, w_from, out_shape, weights=None, extra=()):
    torch = _torch()
    lib = load()
    R = _prep(R, torch.float32, "R")
    F = _prep(F, torch.int8, "factor")
    m, n = R.shape
    out = torch.empty(out_shape(m, n, w_from(F)), dtype=torch.float32, device=R.device)
    with torch.cuda.device(R.device):
        _stream(lib, R.device)
        args = [_ptr(R), m, n, _ptr(F), w_from(F)]
        if weights is not False:
            args.append(_ptr(None if weights is None else _prep(weights, torch.float32, "weights")))
        _check(getattr(lib, fn_name)(*args, _ptr(out)))
    return out


def vstep_product(R, U):
    """U^T R (w x n) for U m x w int8 (§2.3 step 1, §2.4)."""
    return _step("externd_vstep_product", R, U, lambda F: F.shape[1], lambda m, n, w: (w, n), weights=False)


def ustep_product(R, Cb, weights=None):
    """R diag(h) Cb^T (m x w) for Cb w x n int8 (§2.3 step 1, §2.5)."""
    return _step("externd_ustep_product", R, Cb, lambda F: F.shape[0], lambda m, n, w: (m, w), weights=weights)


def vstep_target(R, U):
    """Eq. 3 left: (U^T U + eps I)^-1 U^T R (w x n)."""
    return _step("externd_vstep_target", R, U, lambda F: F.shape[1], lambda m, n, w: (w, n), weights=False)


def ustep_target(R, Cb, weights=None):
    """Eq. 3 right with §2.5: R H V (V^T H V + eps I)^-1 (m x w), V = Cb^T."""
    return _step("externd_ustep_target", R, Cb, lambda F: F.shape[0], lambda m, n, w: (m, w), weights=weights)


def block_scales(R, U, Cb, weights=None):
    """Eq. 4 (§2.5 weighted): the joint scales d of the block (U, Cb) against residual R."""
    torch = _torch()
    lib = load()
    R = _prep(R, torch.float32, "R")
    U, Cb = _prep(U, torch.int8, "U"), _prep(Cb, torch.int8, "Cb")
    h = None if weights is None else _prep(weights, torch.float32, "weights")
    m, n = R.shape
    w = U.shape[1]
    d = torch.empty((w,), dtype=torch.float32, device=R.device)
    with torch.cuda.device(R.device):
        _stream(lib, R.device)
        _check(lib.externd_block_scales(_ptr(R), m, n, _ptr(U), _ptr(Cb), w, _ptr(h), _ptr(d)))
    return d


def deflate(R, U, d, Cb, weights=None) -> float:
    """In place R <- R - U diag(d) Cb (§2.3 step 3, §2.4); returns sum_ij h_j R_ij^2 afterwards."""
    torch = _torch()
    lib = load()
    if not (R.is_cuda and R.dtype == torch.float32 and R.is_contiguous()):
        raise ExterndError("R must be a contiguous CUDA float32 tensor (updated in place)")
    U, Cb, d = _prep(U, torch.int8, "U"), _prep(Cb, torch.int8, "Cb"), _prep(d, torch.float32, "d")
    h = None if weights is None else _prep(weights, torch.float32, "weights")
    m, n = R.shape
    out = _c_double()
    with torch.cuda.device(R.device):
        _stream(lib, R.device)
        _check(lib.externd_deflate(_ptr(R), m, n, _ptr(U), _ptr(d), _ptr(Cb), U.shape[1], _ptr(h),
                                   ctypes.byref(out)))
    return out.value


@dataclass
class Packed:
    """A ternary matrix in the library's packed form (§2.6): ``words`` is a (ceil(rows/16), ceil(cols/128), 32, 4)
    int32 tensor of 2-bit codes (bit 0 nonzero, bit 1 negative) in tensor-core fragment order (layout in
    include/externd.h); ``nnz`` is the number of nonzeros."""
    words: object
    rows: int
    cols: int
    nnz: int


def pack_ternary(T) -> Packed:
    """Packs a CUDA int8 ternary matrix; ``nnz`` gives Eq. 5's storage (rows*cols mask bits + nnz sign bits)."""
    torch = _torch()
    lib = load()
    T = _prep(T, torch.int8, "T")
    rows, cols = T.shape
    words = torch.empty(((rows + 15) // 16, (cols + 127) // 128, 32, 4), dtype=torch.int32, device=T.device)
    nnz = _c_i64()
    with torch.cuda.device(T.device):
        _stream(lib, T.device)
        _check(lib.externd_pack_ternary(_ptr(T), rows, cols, cols, _ptr(words), ctypes.byref(nnz)))
    return Packed(words, rows, cols, nnz.value)


def ternary_apply(Bp: Packed, D, Cp: Packed, x):
    """§2.6: y = B diag(D) (C x) from the packed factors; x is a CUDA float32 vector of length n."""
    torch = _torch()
    lib = load()
    m, k, n = Bp.rows, Bp.cols, Cp.cols
    if Cp.rows != k:
        raise ExterndError(f"inner ranks differ: B has {k} columns, C has {Cp.rows} rows")
    D, x = _prep(D, torch.float32, "D"), _prep(x, torch.float32, "x")
    if D.numel() != k or x.numel() != n:
        raise ExterndError("D must have k entries and x n entries")
    y = torch.empty((m,), dtype=torch.float32, device=x.device)
    with torch.cuda.device(x.device):
        _stream(lib, x.device)
        _check(lib.externd_ternary_apply(_ptr(Bp.words), _ptr(D), _ptr(Cp.words), m, k, n, _ptr(x), _ptr(y)))
    return y


def block_boundaries(m: int, n: int, mu: float, block: int) -> list[int]:
    """The inner ranks b, 2b, ..., k at which a run finishes a block: the ranks of the decompose trace."""
    lib = load()
    cnt = _c_i64()
    _check(lib.externd_block_boundaries(m, n, mu, block, None, ctypes.byref(cnt)))
    arr = (_c_i64 * cnt.value)()
    _check(lib.externd_block_boundaries(m, n, mu, block, arr, ctypes.byref(cnt)))
    return list(arr)


def rank_for_energy(trace, m: int, n: int, mu: float, block: int, target: float) -> Optional[int]:
    """Smallest block-boundary rank reaching ``target`` from one run's trace (None if never); mu = k / min(m, n)."""
    lib = load()
    tr = (_c_double * len(trace))(*trace)
    k = _c_i64()
    _check(lib.externd_rank_for_energy(m, n, mu, block, tr, len(trace), target, ctypes.byref(k)))
    return None if k.value == 0 else k.value


def allocate_ranks(curves, costs, budget: float, weights=None) -> list[int]:
    """Ranks per matrix under a storage budget: ``curves[j]`` lists (k, E_j(k)) at block boundaries, choosing
    rank k of matrix j costs ``costs[j] * k``."""
    lib = load()
    nm = len(curves)
    npts = (_c_i64 * nm)(*[len(c) for c in curves])
    flat = [p for c in curves for p in c]
    ks = (_c_i64 * max(1, len(flat)))(*[int(k) for k, _ in flat])
    es = (_c_double * max(1, len(flat)))(*[float(e) for _, e in flat])
    cs = (_c_double * nm)(*[float(c) for c in costs])
    ws = None if weights is None else (_c_double * nm)(*[float(w) for w in weights])
    out = (_c_i64 * nm)()
    _check(lib.externd_allocate_ranks(nm, npts, ks, es, cs, ws, budget, out))
    return list(out)
