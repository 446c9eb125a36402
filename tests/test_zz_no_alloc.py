"""sd2_accept_logits_noalloc: acceptance without any device allocation, for callers that cannot
call cudaMalloc (for example a plugin whose process gives it no allocator handle, or a loop that
must not risk the device-wide synchronisation of cudaMalloc/cudaFree).

It must give exactly the tokens of sd2_accept_logits (the existing entry point with a caller
workspace) on the same inputs, on consecutive calls that share its fixed scratch array. This file
is named so that pytest collects it last.
"""
import ctypes
from ctypes import c_int32, c_uint32, c_uint64, c_void_p

import pytest
import torch

from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _noalloc(lib, target, draft, xhat, temps, seed, step):
    fn = lib.sd2_accept_logits_noalloc
    fn.argtypes = [c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_int32, c_int32, c_int32, c_uint64, c_uint32,
                   c_void_p, c_void_p, c_void_p]
    fn.restype = c_int32
    B, k1, V = target.shape
    dtype = sd2.DTYPE_BF16 if target.dtype == torch.bfloat16 else sd2.DTYPE_F32
    tok = torch.full((B, k1), -7, dtype=torch.int32, device="cuda")
    n = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    st = fn(target.data_ptr(), draft.data_ptr(), dtype, xhat.data_ptr(), temps.data_ptr(), B, k1 - 1, V,
            seed, step, tok.data_ptr(), n.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == sd2.SD2_OK, lib.sd2_last_error(None)
    return tok, n


def _emitted(tok, n):
    tok, n = tok.cpu(), n.cpu()
    return [tok[b, :int(n[b])].tolist() for b in range(tok.shape[0])]


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(dtype):
    lib = sd2.load_library()
    B, k, V = 24, 6, 32000
    target, draft, xhat = W.make_sweep_logits(B, k, V, seed=21, std=1.0)
    target, draft, xhat = target.to(dtype).cuda(), draft.to(dtype).cuda(), xhat.cuda()
    temps = torch.tensor([[0.0, 0.7, 1.0][b % 3] for b in range(B)], dtype=torch.float32, device="cuda")
    for step in (5, 6):                                   # two calls in a row share the scratch
        ref_tok, ref_n = sd2.accept_logits(target, draft, xhat, temps, 77, step)
        tok, n = _noalloc(lib, target, draft, xhat, temps, 77, step)
        torch.cuda.synchronize()
        assert torch.equal(n.cpu(), ref_n.cpu())
        assert _emitted(tok, n) == _emitted(ref_tok, ref_n)


def test_noalloc_rejects_oversized_requests():
    lib = sd2.load_library()
    B, k, V = 1024, 16, 8
    t = torch.zeros((1,), dtype=torch.float32, device="cuda")
    fn = lib.sd2_accept_logits_noalloc
    fn.argtypes = [c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_int32, c_int32, c_int32, c_uint64, c_uint32,
                   c_void_p, c_void_p, c_void_p]
    fn.restype = c_int32
    st = fn(t.data_ptr(), t.data_ptr(), sd2.DTYPE_F32, t.data_ptr(), t.data_ptr(), B, k, V, 1, 1, t.data_ptr(),
            t.data_ptr(), None)
    assert st == sd2.SD2_ECAPACITY and b"scratch" in lib.sd2_last_error(None)
