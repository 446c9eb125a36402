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


def test_standalone_entry_points_check_arguments_on_the_host(lib):
    """Each standalone kernel entry rejects bad arguments with SD2_EINVAL before any device work
    (the pointers below are never dereferenced: every call fails a host check first)."""
    L = sd2.load_library()
    P = ctypes.c_void_p(1 << 20)                      # a 256-byte-aligned stand-in address
    U = ctypes.c_void_p((1 << 20) + 4)                # a misaligned one

    def err_is(st, word):
        return st == sd2.SD2_EINVAL and word in L.sd2_last_error(None)

    # steering (a1): workspace size, then argument checks in order
    assert L.sd2_steer_workspace_bytes(0, 4096, 2048) == 0
    sizes = [L.sd2_steer_workspace_bytes(B, 4096, 2048) for B in (1, 16, 256)]
    for B, n in zip((1, 16, 256), sizes):
        assert n % 256 == 0 and n >= B * (3 * 4096 * 2 + 2048 * 4 + 2048 * 2) + 4
    assert sizes == sorted(sizes)
    ws = L.sd2_steer_workspace_bytes(2, 64, 32)

    def steer(taps=P, B=2, dv=64, w_hml=P, dg=32, w_s=P, work=P, nbytes=ws):
        return L.sd2_steer(taps, B, dv, w_hml, P, P, 1e-5, dg, w_s, 96, P, P, work, nbytes, None)
    assert err_is(steer(taps=None), b"null")
    assert err_is(steer(w_hml=U), b"unaligned")
    assert err_is(steer(dv=60), b"multiples of 8")
    assert err_is(steer(B=0), b"B >= 1")
    assert err_is(steer(nbytes=ws - 1), b"workspace too small")
    assert err_is(steer(work=U), b"256-byte")

    # GEMM on caller buffers
    def gemm(x=P, ldx=64, M=2, K=64, w=P, w_up=None, N=128, epi=0, out=P, ldo=128, h=None, impl=0):
        return L.sd2_gemm(x, ldx, M, K, w, w_up, N, epi, out, ldo, h, None, None, 0, impl, None)
    assert err_is(gemm(K=60, ldx=60), b"bad GEMM shape")
    assert err_is(gemm(x=None), b"bad GEMM shape")
    assert err_is(gemm(epi=99), b"unknown epilogue")
    assert err_is(gemm(epi=2), b"missing output")           # SwiGLU without W_up and h
    assert err_is(gemm(ldo=64), b"missing output")          # f32 output narrower than N
    assert err_is(gemm(impl=3), b"impl")

    # Eq. 2 activation alone
    assert err_is(L.sd2_swiglu_steered(None, P, None, None, 2, 64, P, None), b"bad argument")
    assert err_is(L.sd2_swiglu_steered(P, P, None, None, 2, 0, P, None), b"bad argument")

    # paged attention
    def attn(q=P, M=6, H=32, Hkv=8, hd=128, max_rows=6):
        return L.sd2_attention(q, M, H, Hkv, hd, P, 64, P, 8, 0, P, P, P, P, 1, max_rows, 2, 128,
                               None, 0, 0, P, None, None)
    assert err_is(attn(q=None), b"null")
    assert err_is(attn(hd=96), b"bad attention shape")
    assert err_is(attn(H=30), b"bad attention shape")       # H not a multiple of Hkv
    assert err_is(attn(max_rows=17), b"bad attention shape")  # 17 rows x 4 heads > 64 query vectors

    # flat-mode attention: workspace size, then the host's rejections
    assert L.sd2_attention_flat_workspace_bytes(0, 38, 128) == 0
    assert L.sd2_attention_flat_workspace_bytes(8, 38, 128) == 8 * 38 * 64 * (128 * 4 + 8) + 64 * 8 * 4

    def flat(q=P, H=32, Hkv=8, hd=128, n_groups=2, max_rows=6, slots=38, max_ctx=1024, pre_len=P, work=P):
        return L.sd2_attention_flat(q, 12, H, Hkv, hd, P, 64, P, 8, 0, P, P, P, P, n_groups, max_rows, slots,
                                    max_ctx, pre_len, 0, 6, work, P, None, None)
    assert err_is(flat(q=None), b"null")
    assert err_is(flat(pre_len=None), b"null")
    assert err_is(flat(work=None), b"null")
    assert err_is(flat(work=U), b"16-byte")
    assert err_is(flat(hd=96), b"bad attention shape")
    assert err_is(flat(max_rows=17), b"bad attention shape")
    assert err_is(flat(n_groups=0), b"flat mode")
    assert err_is(flat(n_groups=65, slots=100), b"flat mode")
    assert err_is(flat(n_groups=3, slots=2), b"flat mode")
    assert err_is(flat(max_ctx=64), b"flat mode")
