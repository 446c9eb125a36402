"""sd2_accept_logits_noalloc: acceptance without any device allocation, for callers that cannot
call cudaMalloc (for example a plugin whose process gives it no allocator handle, or a loop that
must not risk the device-wide synchronisation of cudaMalloc/cudaFree).

It must give exactly the tokens of sd2_accept_logits (the existing entry point with a caller
workspace) on the same inputs, on consecutive calls that share its fixed scratch array, including
calls whose shapes move the tables around inside it and a call at its size limit. This file is
named so that pytest collects it last.
"""
from ctypes import c_int32, c_uint32, c_uint64, c_void_p

import pytest
import torch

from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

pytestmark = pytest.mark.gpu

LIMIT_K = 16
LIMIT_B = 470      # 16*B*(2k+1) + 28*B + 64 <= 261888 bytes of tables at k = 16


def _fn(lib):
    fn = lib.sd2_accept_logits_noalloc
    fn.argtypes = [c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_int32, c_int32, c_int32, c_uint64, c_uint32,
                   c_void_p, c_void_p, c_void_p]
    fn.restype = c_int32
    return fn


def _noalloc(lib, target, draft, xhat, temps, seed, step):
    B, k1, V = target.shape
    dtype = sd2.DTYPE_BF16 if target.dtype == torch.bfloat16 else sd2.DTYPE_F32
    tok = torch.full((B, k1), -7, dtype=torch.int32, device="cuda")
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    st = _fn(lib)(target.data_ptr(), draft.data_ptr(), dtype, xhat.data_ptr(), temps.data_ptr(), B, k1 - 1, V,
                  seed, step, tok.data_ptr(), n.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == sd2.SD2_OK, lib.sd2_last_error(None)
    return tok, n


def _check(lib):
    fn = lib.sd2_accept_logits_noalloc_check
    fn.argtypes = [c_void_p]
    fn.restype = c_int32
    return fn(torch.cuda.current_stream().cuda_stream)


def _emitted(tok, n):
    tok, n = tok.cpu(), n.cpu()
    return [tok[b, :int(n[b])].tolist() for b in range(tok.shape[0])]


def _inputs(B, k, V, dtype, seed):
    target, draft, xhat = W.make_sweep_logits(B, k, V, seed=seed, std=1.0)
    temps = torch.tensor([[0.0, 0.7, 1.0][b % 3] for b in range(B)], dtype=torch.float32, device="cuda")
    return target.to(dtype).cuda(), draft.to(dtype).cuda(), xhat.cuda(), temps


def _same_as_workspace_entry(lib, inputs, seed, step):
    target, draft, xhat, temps = inputs
    ref_tok, ref_n = sd2.accept_logits(target, draft, xhat, temps, seed, step)
    tok, n = _noalloc(lib, target, draft, xhat, temps, seed, step)
    torch.cuda.synchronize()
    assert torch.equal(n.cpu(), ref_n.cpu())
    assert _emitted(tok, n) == _emitted(ref_tok, ref_n)
    assert _check(lib) == sd2.SD2_OK


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(dtype):
    """Calls in a row with shapes that move the tables (small, largest sweep point, small again):
    rows left behind by one call must not leak into the next."""
    lib = sd2.load_library()
    small = _inputs(24, 6, 32000, dtype, seed=21)
    big = _inputs(256, 16, 1024, dtype, seed=22)
    for step, inp in ((5, small), (6, big), (7, small), (8, small)):
        _same_as_workspace_entry(lib, inp, 77, step)


def test_noalloc_at_its_size_limit():
    lib = sd2.load_library()
    inp = _inputs(LIMIT_B, LIMIT_K, 64, torch.float32, seed=23)
    _same_as_workspace_entry(lib, inp, 78, 1)


def test_noalloc_rejects_oversized_requests():
    lib = sd2.load_library()
    t = torch.zeros((1,), dtype=torch.float32, device="cuda")
    for B, k in ((LIMIT_B + 1, LIMIT_K), (1024, 16)):
        st = _fn(lib)(t.data_ptr(), t.data_ptr(), sd2.DTYPE_F32, t.data_ptr(), t.data_ptr(), B, k, 8, 1, 1,
                      t.data_ptr(), t.data_ptr(), None)
        assert st == sd2.SD2_ECAPACITY and b"scratch" in lib.sd2_last_error(None)


def test_noalloc_reports_nonfinite_logits():
    lib = sd2.load_library()
    target, draft, xhat, temps = _inputs(4, 3, 512, torch.float32, seed=24)
    target[2, 1, 17] = float("nan")
    _noalloc(lib, target, draft, xhat, torch.ones_like(temps), 79, 1)
    assert _check(lib) == sd2.SD2_ENUMERIC
    assert _check(lib) == sd2.SD2_OK          # the check cleared the word
