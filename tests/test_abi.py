"""Host-side checks of the C ABI (no GPU): the library builds, loads and exports every function
include/sd2.h declares, and the Python mirrors of its structs have the C layout."""
import ctypes
import os
import re
import subprocess

import pytest

from conftest import ROOT
from paper_2511_09844_gb300 import build, sd2

HEADER = os.path.join(ROOT, "include", "sd2.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sd2_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return ctypes.CDLL(build.LIB)


def test_every_declared_function_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(names) == sorted(sd2.EXPORTS)


def test_struct_layout_matches_header(tmp_path):
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "sd2.h"\n'
                   'int main(void){printf("%zu %zu %zu %zu %zu %zu\\n", sizeof(sd2_lm_config), sizeof(sd2_config),'
                   ' sizeof(sd2_lm_weights), sizeof(sd2_weights), offsetof(sd2_config, k),'
                   ' offsetof(sd2_weights, w_s)); return 0;}\n')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    want = [ctypes.sizeof(sd2.LMConfig), ctypes.sizeof(sd2.Config), ctypes.sizeof(sd2.LMWeights),
            ctypes.sizeof(sd2.Weights), sd2.Config.k.offset, sd2.Weights.w_s.offset]
    assert got == want


def test_context_free_errors_without_gpu(lib):
    """Argument checks happen on the host before any device work."""
    L = sd2.load_library()
    assert L.sd2_accept_workspace_bytes(0, 4) == 0
    assert L.sd2_accept_workspace_bytes(2, 4) % 256 == 0 and L.sd2_accept_workspace_bytes(2, 4) > 0
    st = L.sd2_accept_logits(None, None, 0, None, None, 1, 1, 8, 0, 0, None, None, None, 0, None)
    assert st == sd2.SD2_EINVAL and b"null" in L.sd2_last_error(None)
    cfg = sd2.Config()
    w = sd2.Weights()
    ctx = ctypes.c_void_p()
    assert L.sd2_init(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == sd2.SD2_EINVAL
    assert L.sd2_step(None) == sd2.SD2_EINVAL
    assert L.sd2_free(None) == sd2.SD2_OK


def test_product_path_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(sd2, "_LIB", None)
    with pytest.raises(RuntimeError, match="missing"):
        sd2.load_library(str(tmp_path / "nope.so"))
