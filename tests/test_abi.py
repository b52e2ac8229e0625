"""The C-ABI library builds, loads and exports every symbol include/adapm.h declares.

No compute call is made here (no GPU needed).
"""
import ctypes
import os
import re

import pytest

from paper_2206_00470_gb300 import adapm
from paper_2206_00470_gb300 import build as libbuild

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "adapm.h")


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:adapm_status|const char\*)\s+(adapm_\w+)\s*\(", text, re.M)))


@pytest.fixture(scope="module")
def lib_path():
    return libbuild.build()


def test_header_declares_the_method_calls():
    names = declared_functions()
    for n in ("adapm_create", "adapm_intent", "adapm_advance_clock", "adapm_pull", "adapm_push",
              "adapm_sync"):
        assert n in names


def test_library_exports_every_declared_symbol(lib_path):
    lib = ctypes.CDLL(lib_path)
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_binding_covers_every_declared_symbol(lib_path):
    assert sorted(adapm.EXPORTS) == declared_functions()
    adapm.load(lib_path)


def test_binding_fails_loudly_without_the_library(tmp_path):
    saved = adapm._lib
    adapm._lib = None
    try:
        with pytest.raises(RuntimeError):
            adapm.load(str(tmp_path / "missing.so"))
    finally:
        adapm._lib = saved


def test_create_rejects_bad_configs_without_touching_the_gpu(lib_path):
    lib = adapm.load(lib_path)
    h = ctypes.c_void_p()
    bad = [
        adapm.Config(0, 4, 1, 0, None, None),          # no keys
        adapm.Config(10, 6, 1, 0, None, None),         # value_len not a multiple of 4
        adapm.Config(10, 4, 0, 0, None, None),         # no workers
        adapm.Config(10, 4, 33, 0, None, None),        # more than 32 workers
        adapm.Config(2 ** 32 - 1, 4, 1, 0, None, None),
        adapm.Config(10, 4, 1, 0, None, None, 2),                    # relocate is 0 or 1
        adapm.Config(10, 4, 1, 0, None, None, 0, 3),                 # unknown action timing
        adapm.Config(10, 4, 1, 0, None, None, 0, 1, 1.5),            # smoothing factor above 1
        adapm.Config(10, 4, 1, 0, None, None, 0, 1, 0.1, 1.0),       # quantile must be below 1
        adapm.Config(10, 4, 1, 0, None, None, 0, 1, 0.1, 0.9, -1.0),  # negative initial rate
        adapm.Config(10, 4, 1, 0, None, None, 0, 0, 0.0, 0.0, 0.0, 5),  # delta_refresh is 0 or 1
    ]
    for cfg in bad:
        assert lib.adapm_create(ctypes.byref(cfg), ctypes.byref(h)) == adapm.EINVAL
    assert lib.adapm_intent(None, 0, None, 0, 0, 1) == adapm.EINVAL
    assert lib.adapm_wait(None) == adapm.EINVAL


def test_poisson_quantile_of_the_library_equals_the_oracle(lib_path):
    # the host rule of adaptive action timing (Algorithm 1) against the oracle's, which is pinned to scipy
    from oracle.timing import poisson_quantile
    adapm.load(lib_path)
    for lam in (0.05, 0.7, 1.0, 2.0, 2.8, 9.5, 20.0, 111.1, 2500.0):
        for p in (0.001, 0.5, 0.9, 0.9999, 1 - 1e-10):
            assert adapm.poisson_quantile(lam, p) == poisson_quantile(lam, p), (lam, p)
    with pytest.raises(adapm.AdaPMError):
        adapm.poisson_quantile(0.0, 0.5)
    with pytest.raises(adapm.AdaPMError):
        adapm.poisson_quantile(1.0, 1.0)


def test_header_is_plain_c(tmp_path):
    # the boundary is a C ABI: the header must compile as C (no C++ constructs) and link against the library
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    src = tmp_path / "use_adapm.c"
    src.write_text(
        '#include "adapm.h"\n'
        "int main(void) {\n"
        "  adapm_config cfg = {0};\n"
        "  adapm_ctx* ctx = 0;\n"
        "  int64_t q = 0;\n"
        "  cfg.num_keys = 0;  /* invalid: rejected before any GPU work */\n"
        "  if (adapm_create(&cfg, &ctx) != ADAPM_EINVAL) return 1;\n"
        "  if (adapm_poisson_quantile(20.0, 0.9999, &q) != ADAPM_OK || q != 39) return 2;\n"
        "  return 0;\n"
        "}\n")
    lib = libbuild.build()
    exe = tmp_path / "use_adapm"
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe),
                        lib, "-Wl,-rpath," + os.path.dirname(lib)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, (r.returncode, r.stderr)
