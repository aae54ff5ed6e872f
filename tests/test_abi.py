"""The C-ABI library builds, loads and exports every entry point include/externd.h declares (no GPU needed).

Only host-side functions (rank, block width, status strings) are called here: no compute call without a GPU.
"""
import ctypes
import os
import re
import shutil

import pytest

from oracle import externd_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "externd.h")


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(externd_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2607_13511_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ("externd_decompose", "externd_energy", "externd_rank", "externd_set_stream", "externd_strerror",
                 "externd_ternarize", "externd_vstep_product", "externd_ustep_product", "externd_block_scales",
                 "externd_deflate"):
        assert name in syms


def test_library_exports_every_declared_symbol(lib):
    missing = [s for s in declared_symbols() if not hasattr(lib, s)]
    assert not missing, missing


def prototypes():
    """name -> (return type, [(parameter type, parameter name), ...]) for every declaration in the header."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    text = re.sub(r"#.*", "", text)
    out = {}
    for ret, name, params in re.findall(r"([A-Za-z_][\w \t*]*?)\b(externd_\w+)\s*\(([^)]*)\)\s*;", text):
        plist = []
        params = " ".join(params.split())
        if params not in ("", "void"):
            for p in params.split(","):
                m = re.match(r"^\s*(.*?)\s*\b(\w+)\s*$", p)
                plist.append((re.sub(r"\s*\*\s*", "*", m.group(1)).strip(), m.group(2)))
        out[name] = (re.sub(r"\s*\*\s*", "*", " ".join(ret.split())).strip(), plist)
    return out


# The boundary calls exactly as the problem statement of §2.1 (Eq. 1), Eq. 2 and §2.5 fix them:
# A (m x n), mu, tau, block, iters, optional weights, factors B, D, C, and the energy.
BOUNDARY = {
    "externd_decompose": ("int", [("const float*", "A"), ("int64_t", "m"), ("int64_t", "n"), ("double", "mu"),
                                  ("double", "tau"), ("int", "block"), ("int", "iters"),
                                  ("const float*", "weights"), ("int8_t*", "B"), ("float*", "D"),
                                  ("int8_t*", "C"), ("double*", "energy")]),
    "externd_energy": ("int", [("const float*", "A"), ("int64_t", "m"), ("int64_t", "n"), ("const int8_t*", "B"),
                               ("const float*", "D"), ("const int8_t*", "C"), ("int64_t", "k"),
                               ("const float*", "weights"), ("double*", "energy")]),
    "externd_rank": ("int", [("int64_t", "m"), ("int64_t", "n"), ("double", "mu"), ("int64_t*", "k")]),
    "externd_set_stream": ("int", [("void*", "cuda_stream")]),
    "externd_strerror": ("const char*", [("int", "status")]),
}


def test_boundary_prototypes_are_exact():
    protos = prototypes()
    for name, want in BOUNDARY.items():
        assert protos[name] == want, (name, protos[name])
    # the host variant takes the same twelve parameters
    assert protos["externd_decompose_host"] == BOUNDARY["externd_decompose"]
    # the traced variant appends the per-block energies and nothing else
    ret, params = protos["externd_decompose_traced"]
    assert (ret, params[:-1]) == BOUNDARY["externd_decompose"] and params[-1] == ("double*", "trace")


def test_binding_declares_every_symbol():
    import paper_2607_13511_gb300 as X
    assert sorted(X._SIGNATURES) == declared_symbols()


def test_binding_argument_counts_match_the_header():
    import paper_2607_13511_gb300 as X
    protos = prototypes()
    for name, (_, args) in X._SIGNATURES.items():
        assert len(args) == len(protos[name][1]), name


def test_host_side_rank_and_block_width_match_the_oracle(lib):
    rank = lib.externd_rank
    rank.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_double, ctypes.POINTER(ctypes.c_int64)]
    bw = lib.externd_block_width
    bw.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.POINTER(ctypes.c_int)]
    k = ctypes.c_int64()
    b = ctypes.c_int()
    for m, n, mu in [(256, 256, 2.0), (2048, 2048, 3.0), (2560, 9728, 3.0), (4096, 4096, 2.5), (10, 7, 0.5),
                     (10, 7, 0.2), (3, 1000, 1.7), (1, 1, 1.0)]:
        assert rank(m, n, mu, ctypes.byref(k)) == 0
        assert k.value == O.inner_rank(m, n, mu)
    for m, n, block in [(2048, 2048, 64), (2560, 1024, 256), (256, 256, 1), (12, 40, 64), (7, 7, 16), (9, 9, 200)]:
        assert bw(m, n, block, ctypes.byref(b)) == 0
        assert b.value == O.block_width(m, n, block)


def test_host_side_argument_errors(lib):
    rank = lib.externd_rank
    rank.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_double, ctypes.POINTER(ctypes.c_int64)]
    k = ctypes.c_int64()
    assert rank(0, 5, 1.0, ctypes.byref(k)) == -1
    assert rank(5, 5, 0.0, ctypes.byref(k)) == -1
    assert rank(5, 5, float("nan"), ctypes.byref(k)) == -1
    assert rank(5, 5, 1.0, None) == -1
    bw = lib.externd_block_width
    bw.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.POINTER(ctypes.c_int)]
    b = ctypes.c_int()
    assert bw(5, 5, 0, ctypes.byref(b)) == -1
    assert bw(5000, 5000, 257, ctypes.byref(b)) == -1     # widest supported block is 256
    se = lib.externd_strerror
    se.restype = ctypes.c_char_p
    for code in (0, -1, -2, -3, -4, -5, 7):
        assert se(code)


C_CALLER = r"""
#include <stdio.h>
#include <stdint.h>
#include "externd.h"

int main(void) {
    int64_t k = 0;
    double energy = 0.0;
    if (externd_rank(2560, 9728, 3.0, &k) != EXTERND_OK || k != 7680) return 1;
    /* the decomposition with the twelve parameters of the boundary: an empty matrix is rejected on the host */
    if (externd_decompose((const float*)0, 0, 9728, 3.0, 1.0, 128, 4, (const float*)0, (int8_t*)0, (float*)0,
                          (int8_t*)0, &energy) != EXTERND_EINVAL) return 2;
    if (externd_energy((const float*)0, 0, 9728, (const int8_t*)0, (const float*)0, (const int8_t*)0, 7680,
                       (const float*)0, &energy) != EXTERND_EINVAL) return 3;
    if (externd_strerror(EXTERND_EINVAL) == 0) return 4;
    printf("ok %lld\n", (long long)k);
    return 0;
}
"""


def test_c_caller_compiles_links_and_runs(lib, tmp_path):
    """A plain C99 program written to the boundary compiles against the header, links and runs its host-side
    checks (no GPU needed)."""
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    from paper_2607_13511_gb300 import build
    libdir = os.path.dirname(build.LIB)
    src = tmp_path / "caller.c"
    src.write_text(C_CALLER)
    exe = tmp_path / "caller"
    res = subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src), "-o",
                          str(exe), "-L", libdir, "-lexternd", f"-Wl,-rpath,{libdir}"], capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert run.returncode == 0 and run.stdout.strip() == "ok 7680", (run.returncode, run.stdout, run.stderr)
