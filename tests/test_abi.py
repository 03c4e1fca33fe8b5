"""The C-ABI library builds for sm_103a, loads, and exports every symbol the
header declares; host-side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

from paper_2608_28726_gb300 import build as prbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pro_router.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pr_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    path = prbuild.build()
    return ctypes.CDLL(path)


def test_header_declares_the_three_verifier_calls():
    names = declared_functions()
    for n in ("pr_token_features", "pr_aggregate_score", "pr_route"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_binding_covers_the_header(lib):
    from paper_2608_28726_gb300 import binding
    assert sorted(binding.EXPORTS) == declared_functions()


def test_header_is_plain_c(tmp_path):
    """The boundary is a C ABI: the header compiles as strict C99 with no
    CUDA or C++ header behind it."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "use.c"
    src.write_text('#include "pro_router.h"\nint main(void) { return pr_launch_count() > 0; }\n')
    subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I",
                    os.path.dirname(HEADER), "-c", str(src), "-o", str(tmp_path / "use.o")],
                   check=True)


def test_library_targets_sm_103a_only():
    assert prbuild.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


def test_status_strings(lib):
    lib.pr_status_string.restype = ctypes.c_char_p
    lib.pr_status_string.argtypes = [ctypes.c_int]
    assert lib.pr_status_string(0) == b"ok"
    assert lib.pr_status_string(-1) == b"invalid argument"
    assert lib.pr_status_string(-3) == b"CUDA error"
    assert lib.pr_status_string(12345) == b"unknown status"


def test_null_context_is_rejected(lib):
    P = ctypes.c_void_p
    lib.pr_launch_count.restype = ctypes.c_uint64
    n0 = lib.pr_launch_count()
    lib.pr_route.argtypes = [P, P, ctypes.c_int, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                             ctypes.c_int64, P, P, ctypes.c_int32, P, ctypes.c_float,
                             ctypes.c_float, P, P, P, P, P]
    assert lib.pr_route(None, None, 1, 0, 0, 1, 1, None, None, 1, None, 0.0, 0.5, None, None, None,
                        None, None) == -1
    lib.pr_ctx_create.argtypes = [ctypes.POINTER(P), ctypes.c_int, ctypes.c_int64, ctypes.c_int32]
    assert lib.pr_ctx_create(None, 0, 1, 1) == -1
    h = P()
    assert lib.pr_ctx_create(ctypes.byref(h), 0, -5, 1) == -1
    lib.pr_ctx_set_option.argtypes = [P, ctypes.c_int32, ctypes.c_int32]
    assert lib.pr_ctx_set_option(None, 0, 20) == -1
    # the LM-head calls and the wait self-test check their arguments on the host
    lib.pr_lmhead_features.argtypes = [P, P, P, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, P,
                                       ctypes.c_int32, P, ctypes.c_int32, P, P, P, P]
    assert lib.pr_lmhead_features(None, None, None, 8, 64, 256, None, 20, None, 0, None, None,
                                  None, None) == -1
    lib.pr_lmhead_decode_step.argtypes = [P, P, P, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64,
                                          P, P, P, P, ctypes.c_float, ctypes.c_float, P, P, P, P,
                                          P]
    assert lib.pr_lmhead_decode_step(None, None, None, 4, 64, 256, None, None, None, None, 0.0, 0.5,
                                     None, None, None, None, None) == -1
    lib.pr_selftest_wait.argtypes = [P, ctypes.c_int64, ctypes.POINTER(ctypes.c_int32)]
    done = ctypes.c_int32(7)
    assert lib.pr_selftest_wait(None, 1000, ctypes.byref(done)) == -1 and done.value == 7
    # the flag word, with and without a stream
    lib.pr_last_error.argtypes = [P, ctypes.POINTER(ctypes.c_uint32)]
    word = ctypes.c_uint32(9)
    assert lib.pr_last_error(None, ctypes.byref(word)) == -1 and word.value == 9
    lib.pr_ctx_flags.argtypes = [P, P, ctypes.c_int32, ctypes.POINTER(ctypes.c_uint32)]
    assert lib.pr_ctx_flags(None, None, 0, ctypes.byref(word)) == -1 and word.value == 9
    assert lib.pr_launch_count() == n0  # nothing was launched


def test_no_gpu_means_no_context(lib):
    """Without a device the context cannot be made, and says so (no fallback)."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    P = ctypes.c_void_p
    lib.pr_ctx_create.argtypes = [ctypes.POINTER(P), ctypes.c_int, ctypes.c_int64, ctypes.c_int32]
    h = P()
    assert lib.pr_ctx_create(ctypes.byref(h), 0, 16, 4) == -1
    assert not h.value


def test_head_parameter_count_matches_the_oracle_layout(lib):
    """The library's weight count for the scorer head is the oracle's layout size."""
    from oracle import head
    lib.pr_head_param_count.argtypes = [ctypes.c_int32]
    lib.pr_head_param_count.restype = ctypes.c_int64
    assert lib.pr_head_param_count(2) == 67329 == head.n_params(2)
    for n in (1, 4, 8):
        assert lib.pr_head_param_count(n) == head.n_params(n)
    assert lib.pr_head_param_count(0) == -1
    assert lib.pr_head_param_count(9) == -1
    P = ctypes.c_void_p
    lib.pr_head_score.argtypes = [P, P, P, ctypes.c_int64, P, ctypes.c_int32, P, ctypes.c_int32,
                                  ctypes.c_float, P, P, P, P]
    assert lib.pr_head_score(None, None, None, 0, None, 1, None, 2, 0.5, None, None, None,
                             None) == -1
