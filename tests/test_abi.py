"""CPU checks of the C ABI: libw8a8.so builds for sm_103a, loads, exports every function that
include/*.h declares, and rejects bad arguments on the host before touching a GPU."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_28003_gb300 import build
    path = build.build()
    from paper_2608_28003_gb300 import binding
    assert os.path.samefile(path, binding.LIB_PATH)
    return binding


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?[A-Za-z_][\w]*\s*\**\s*(w8a8_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 15
    L = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in sorted(names) if not hasattr(L, n)]
    assert not missing, missing
    # the binding describes exactly the declared functions
    assert set(lib.SIGNATURES) == names


def test_abi_version_and_error_channel(lib):
    assert lib.abi_version() == 2
    assert isinstance(lib.lib().w8a8_last_error(), bytes)


def _qw(n, k, base=0x10000):
    return lib_mod().QWeightC(n, k, base, base + 0x1000, base + 0x2000, None)


def lib_mod():
    from paper_2608_28003_gb300 import binding
    return binding


def test_host_side_argument_errors(lib):
    L = lib.lib()
    ws = ctypes.c_void_p(0x200000)
    # null descriptor
    assert L.w8a8_linear(None, ctypes.c_void_p(0x1000), 4, None, ctypes.c_void_p(0x2000), None, ws, 1 << 20, None) == 1
    assert b"descriptor" in L.w8a8_last_error()
    # K not a multiple of 16
    w = _qw(64, 100)
    assert L.w8a8_linear(ctypes.byref(w), ctypes.c_void_p(0x1000), 4, None, ctypes.c_void_p(0x2000), None, ws,
                         1 << 20, None) == 2
    # misaligned activation pointer
    w = _qw(64, 128)
    assert L.w8a8_linear(ctypes.byref(w), ctypes.c_void_p(0x1001), 4, None, ctypes.c_void_p(0x2000), None, ws,
                         1 << 20, None) == 3
    # negative M
    assert L.w8a8_linear(ctypes.byref(w), ctypes.c_void_p(0x1000), -1, None, ctypes.c_void_p(0x2000), None, ws,
                         1 << 20, None) == 1
    # M == 0 is a no-op that succeeds without a device
    assert L.w8a8_linear(ctypes.byref(w), None, 0, None, None, None, None, 0, None) == 0
    # bad precision enum
    f = lib.FfnC(1152, 6912, _qw(13824, 1152), _qw(1152, 6912), None, None)
    assert L.w8a8_ffn_block(ctypes.byref(f), 7, ctypes.c_void_p(0x1000), 1, ctypes.c_void_p(0x2000), None, ws,
                            1 << 20, None) == 1
    # gate/up with F not a multiple of 8
    assert L.w8a8_prepare_gate_up(ctypes.c_void_p(0x1000), ctypes.c_void_p(0x2000), 12, 64, ctypes.c_void_p(0x3000),
                                  0.5, 1, ctypes.c_void_p(0x4000), ctypes.c_void_p(0x5000), ctypes.c_void_p(0x6000),
                                  ctypes.c_void_p(0x7000), None, None) == 2
    # alpha outside [0, 1]
    assert L.w8a8_prepare_weights(ctypes.c_void_p(0x1000), 8, 64, ctypes.c_void_p(0x3000), 1.5, 1,
                                  ctypes.c_void_p(0x4000), ctypes.c_void_p(0x5000), ctypes.c_void_p(0x6000),
                                  ctypes.c_void_p(0x7000), None, None) == 1
    # lm_head with too many tokens for one call
    h = lib.HeadC(262144, 1152, _qw(262144, 1152), None)
    assert L.w8a8_lm_head(ctypes.byref(h), 1, ctypes.c_void_p(0x1000), 100000, None, ctypes.c_void_p(0x2000), ws,
                          1 << 30, None) == 2


def test_product_path_fails_loudly_without_library(tmp_path, monkeypatch):
    from paper_2608_28003_gb300 import binding
    monkeypatch.setattr(binding, "_LIB", None)
    monkeypatch.setattr(binding, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        binding.lib()


def test_header_is_plain_c(tmp_path):
    """The boundary is a C ABI: every header compiles as strict C99 (no C++ constructs), and its
    structs are usable from C."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "use_header.c"
    src.write_text('#include "w8a8.h"\n'
                   "int main(void) {\n"
                   "  w8a8_mask m = {0u, 0u, 0};\n"
                   "  w8a8_layer_alloc_report r;\n"
                   "  r.chosen = m;\n"
                   "  return (int)r.chosen.lm;\n"
                   "}\n")
    out = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I",
                          os.path.join(ROOT, "include"), "-c", str(src), "-o", str(tmp_path / "use_header.o")],
                         capture_output=True, text=True)
    assert out.returncode == 0, out.stderr
