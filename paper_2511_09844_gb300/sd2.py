"""Python binding of libsd2.so (ctypes): argument marshalling only.

Every step of the SD^2 hot path runs in the library's CUDA kernels; this module turns torch
tensors into device pointers and mirrors the C structs of include/sd2.h. If the library has not
been built, importing the engine raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int32, c_int64, c_size_t, c_uint32, c_uint64, c_void_p
from typing import List, Optional, Sequence

import torch

from .workloads import LAYER_SLOTS, PairWorkload

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libsd2.so")

SD2_OK, SD2_EINVAL, SD2_ENOMEM, SD2_ECUDA, SD2_ECAPACITY, SD2_ESTATE, SD2_ENUMERIC, SD2_ETIMEOUT = range(8)
STATUS_NAMES = ["OK", "EINVAL", "ENOMEM", "ECUDA", "ECAPACITY", "ESTATE", "ENUMERIC", "ETIMEOUT"]
DTYPE_F32, DTYPE_BF16 = 0, 1
# sd2_debug_buffer ids
BUF_TARGET, BUF_DRAFT, BUF_XHAT, BUF_TAPS, BUF_G, BUF_BIAS, BUF_COMMITTED, BUF_STATE, BUF_ITER = range(9)
PROFILE_CLASSES = ["gemm", "attention", "accept", "sample", "other", "verify", "draft", "steer"]

EXPORTS = ["sd2_init", "sd2_prefill", "sd2_step", "sd2_accept", "sd2_check", "sd2_free", "sd2_last_error",
           "sd2_set_graphs", "sd2_debug_buffer", "sd2_profile", "sd2_profile_read", "sd2_accept_workspace_bytes",
           "sd2_accept_logits", "sd2_steer_workspace_bytes", "sd2_steer", "sd2_swiglu_steered",
           "sd2_accept_logits_noalloc", "sd2_gemm", "sd2_set_gemm_impl", "sd2_stage_timing", "sd2_stage_read",
           "sd2_set_drafter_chain", "sd2_attention", "sd2_set_fused_attention",
           "sd2_accept_logits_noalloc_check", "sd2_debug_fail_alloc", "sd2_debug_expire_wait",
           "sd2_gemm_timing", "sd2_gemm_timing_read", "sd2_generate", "sd2_attention_flat_workspace_bytes",
           "sd2_attention_flat"]


class LMConfig(ctypes.Structure):
    _fields_ = [("n_layers", c_int32), ("d_model", c_int32), ("n_heads", c_int32), ("n_kv_heads", c_int32),
                ("head_dim", c_int32), ("d_ffn", c_int32), ("vocab", c_int32), ("rope_theta", c_float),
                ("norm_eps", c_float)]


class Config(ctypes.Structure):
    _fields_ = [("verifier", LMConfig), ("drafter", LMConfig), ("d_steer", c_int32), ("tap_layers", c_int32 * 3),
                ("steer_ln_eps", c_float), ("k", c_int32), ("max_batch", c_int32), ("max_ctx", c_int32),
                ("max_prefill_tokens", c_int32), ("kv_block", c_int32), ("no_steering", c_int32),
                ("steering_site", c_int32)]


class LMWeights(ctypes.Structure):
    _fields_ = [("embed", c_void_p), ("final_norm", c_void_p), ("lm_head", c_void_p), ("layers", POINTER(c_void_p))]


class Weights(ctypes.Structure):
    _fields_ = [("verifier", LMWeights), ("drafter", LMWeights), ("w_hml", c_void_p), ("steer_ln_gamma", c_void_p),
                ("steer_ln_beta", c_void_p), ("w_s", c_void_p), ("w_c1x", c_void_p), ("w_c1g", c_void_p),
                ("w_c2", c_void_p)]


_LIB = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libsd2.so and declare its prototypes. Raises if it is missing."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2511_09844_gb300.build.build()")
    lib = ctypes.CDLL(path)
    lib.sd2_init.argtypes = [POINTER(Config), POINTER(Weights), c_void_p, POINTER(c_void_p)]
    lib.sd2_prefill.argtypes = [c_void_p, c_int32, c_void_p, POINTER(c_int32), POINTER(c_float), c_uint64, c_void_p]
    lib.sd2_step.argtypes = [c_void_p]
    lib.sd2_accept.argtypes = [c_void_p, c_void_p, c_void_p]
    lib.sd2_check.argtypes = [c_void_p]
    lib.sd2_free.argtypes = [c_void_p]
    lib.sd2_last_error.argtypes = [c_void_p]
    lib.sd2_last_error.restype = ctypes.c_char_p
    lib.sd2_set_graphs.argtypes = [c_void_p, c_int32]
    lib.sd2_debug_buffer.argtypes = [c_void_p, c_int32, POINTER(c_void_p), POINTER(c_int64), POINTER(c_int32)]
    lib.sd2_profile.argtypes = [c_void_p, c_int32]
    lib.sd2_profile_read.argtypes = [c_void_p, POINTER(c_int64), POINTER(c_double), POINTER(c_double), c_int32]
    lib.sd2_stage_timing.argtypes = [c_void_p, c_int32]
    lib.sd2_stage_read.argtypes = [c_void_p, POINTER(c_double)]
    lib.sd2_accept_workspace_bytes.argtypes = [c_int32, c_int32]
    lib.sd2_accept_workspace_bytes.restype = c_size_t
    lib.sd2_accept_logits.argtypes = [c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_int32, c_int32, c_int32,
                                      c_uint64, c_uint32, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]
    lib.sd2_steer_workspace_bytes.argtypes = [c_int32, c_int32, c_int32]
    lib.sd2_steer_workspace_bytes.restype = c_size_t
    lib.sd2_steer.argtypes = [c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p, c_float, c_int32, c_void_p,
                              c_int32, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]
    lib.sd2_swiglu_steered.argtypes = [c_void_p, c_void_p, c_void_p, c_void_p, c_int32, c_int32, c_void_p, c_void_p]
    lib.sd2_gemm.argtypes = [c_void_p, c_int32, c_int32, c_int32, c_void_p, c_void_p, c_int32, c_int32, c_void_p,
                             c_int32, c_void_p, c_void_p, c_void_p, c_int32, c_int32, c_void_p]
    lib.sd2_set_gemm_impl.argtypes = [c_void_p, c_int32]
    lib.sd2_attention.argtypes = [c_void_p, c_int32, c_int32, c_int32, c_int32, c_void_p, c_int32, c_void_p, c_int32,
                                  c_int32, c_void_p, c_void_p, c_void_p, c_void_p, c_int32, c_int32, c_int32, c_int32,
                                  c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p]
    lib.sd2_attention_flat_workspace_bytes.argtypes = [c_int32, c_int32, c_int32]
    lib.sd2_attention_flat_workspace_bytes.restype = c_size_t
    lib.sd2_attention_flat.argtypes = [c_void_p, c_int32, c_int32, c_int32, c_int32, c_void_p, c_int32, c_void_p,
                                       c_int32, c_int32, c_void_p, c_void_p, c_void_p, c_void_p, c_int32, c_int32,
                                       c_int32, c_int32, c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p,
                                       c_void_p]
    lib.sd2_set_drafter_chain.argtypes = [c_void_p, c_int32]
    lib.sd2_set_fused_attention.argtypes = [c_void_p, c_int32]
    lib.sd2_accept_logits_noalloc.argtypes = [c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_int32, c_int32,
                                              c_int32, c_uint64, c_uint32, c_void_p, c_void_p, c_void_p]
    lib.sd2_accept_logits_noalloc_check.argtypes = [c_void_p]
    lib.sd2_debug_fail_alloc.argtypes = [c_int32]
    lib.sd2_gemm_timing.argtypes = [c_void_p, c_int32]
    lib.sd2_generate.argtypes = [c_void_p, c_int32, POINTER(c_int32), POINTER(c_int32), POINTER(c_float), c_uint64,
                                 c_int32, POINTER(c_int32), POINTER(c_int32)]
    lib.sd2_gemm_timing_read.argtypes = [c_void_p, c_int32, POINTER(c_int32), POINTER(c_uint64), POINTER(c_double),
                                         POINTER(c_int32)]
    lib.sd2_debug_expire_wait.argtypes = [c_void_p, c_int64]
    for name in EXPORTS:
        if name not in ("sd2_last_error", "sd2_accept_workspace_bytes", "sd2_steer_workspace_bytes",
                        "sd2_attention_flat_workspace_bytes"):
            getattr(lib, name).restype = c_int32
    _LIB = lib
    return lib


class SD2Error(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"SD2_{STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else status}: {msg}")
        self.status = status


def _check(lib, status: int, ctx=None):
    if status != SD2_OK:
        raise SD2Error(status, lib.sd2_last_error(ctx).decode(errors="replace"))


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return c_void_p(s.cuda_stream)


def lm_config(shape) -> LMConfig:
    return LMConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.d_ffn,
                    shape.vocab, shape.rope_theta, shape.norm_eps)


class _DeviceView:
    """A __cuda_array_interface__ wrapper so torch can view a library-owned device buffer."""

    def __init__(self, ptr: int, n: int, typestr: str):
        self.__cuda_array_interface__ = {"shape": (n,), "typestr": typestr, "data": (ptr, False), "version": 3}


class SD2Engine:
    """One SD^2 context: borrowed weights, device-resident state, and the four hot-path calls."""

    def __init__(self, work: PairWorkload, verifier_w: dict, drafter_w: dict, steer_w: dict, max_batch: int,
                 max_ctx: int, max_prefill_tokens: int, stream=None, steering: bool = True):
        self.lib = load_library()
        self.work = work
        self.k = work.k
        self.vocab = work.verifier.vocab
        self._keep = [verifier_w, drafter_w, steer_w]
        cfg = Config()
        cfg.verifier = lm_config(work.verifier)
        cfg.drafter = lm_config(work.drafter)
        cfg.d_steer = work.d_steer
        cfg.tap_layers = (c_int32 * 3)(*work.tap_layers)
        cfg.steer_ln_eps = work.steer_ln_eps
        cfg.k = work.k
        cfg.max_batch = max_batch
        cfg.max_ctx = max_ctx
        cfg.max_prefill_tokens = max_prefill_tokens
        cfg.kv_block = work.kv_block
        cfg.no_steering = 0 if steering else 1     # False: the pretrained drafter, no steering stage
        cfg.steering_site = {"mlp_up": 0, "after_mlp": 1, "cond_mlp": 2}[work.steering_site]
        self.cfg = cfg
        w = Weights()
        w.verifier = self._lm_weights(verifier_w)
        w.drafter = self._lm_weights(drafter_w)
        if steer_w is not None:
            w.w_hml = _ptr(steer_w["w_hml"])
            w.steer_ln_gamma = _ptr(steer_w["ln_gamma"])
            w.steer_ln_beta = _ptr(steer_w["ln_beta"])
            w.w_s = _ptr(steer_w.get("w_s"))
            w.w_c1x = _ptr(steer_w.get("w_c1x"))
            w.w_c1g = _ptr(steer_w.get("w_c1g"))
            w.w_c2 = _ptr(steer_w.get("w_c2"))
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        ctx = c_void_p()
        _check(self.lib, self.lib.sd2_init(ctypes.byref(cfg), ctypes.byref(w), _stream(self.stream), ctypes.byref(ctx)))
        self.ctx = ctx
        self.batch = 0

    def _lm_weights(self, w: dict) -> LMWeights:
        ptrs = []
        for lw in w["layers"]:
            for slot in LAYER_SLOTS:
                ptrs.append(lw[slot].data_ptr())
        arr = (c_void_p * len(ptrs))(*ptrs)
        self._keep.append(arr)
        return LMWeights(w["embed"].data_ptr(), w["final_norm"].data_ptr(), w["lm_head"].data_ptr(),
                         ctypes.cast(arr, POINTER(c_void_p)))

    def _call(self, status):
        _check(self.lib, status, self.ctx)

    def prefill(self, prompts: Sequence[Sequence[int]], temps: Sequence[float], seed: int) -> torch.Tensor:
        flat = [t for p in prompts for t in p]
        cu = [0]
        for p in prompts:
            cu.append(cu[-1] + len(p))
        self._prompt_dev = torch.tensor(flat, dtype=torch.int32, device="cuda")
        first = torch.empty(len(prompts), dtype=torch.int32, device="cuda")
        cu_arr = (c_int32 * len(cu))(*cu)
        t_arr = (c_float * len(temps))(*[float(t) for t in temps])
        self._call(self.lib.sd2_prefill(self.ctx, len(prompts), _ptr(self._prompt_dev), cu_arr, t_arr, c_uint64(seed),
                                        _ptr(first)))
        self.batch = len(prompts)
        self.tokens_out = torch.empty((self.batch, self.k + 1), dtype=torch.int32, device="cuda")
        self.n_out = torch.empty(self.batch, dtype=torch.int32, device="cuda")
        return first

    def generate(self, prompts: Sequence[Sequence[int]], temps: Sequence[float], seed: int, max_new: int):
        """A whole request through sd2_generate on host buffers: returns each sequence's new tokens."""
        flat = [t for p in prompts for t in p]
        cu = [0]
        for p in prompts:
            cu.append(cu[-1] + len(p))
        B = len(prompts)
        tok = (c_int32 * len(flat))(*flat)
        cu_arr = (c_int32 * len(cu))(*cu)
        t_arr = (c_float * B)(*[float(t) for t in temps])
        out = (c_int32 * (B * max_new))()
        n = (c_int32 * B)()
        self._call(self.lib.sd2_generate(self.ctx, B, tok, cu_arr, t_arr, c_uint64(seed), max_new, out, n))
        self.batch = B
        self.tokens_out = torch.empty((B, self.k + 1), dtype=torch.int32, device="cuda")
        self.n_out = torch.empty(B, dtype=torch.int32, device="cuda")
        return [[out[b * max_new + t] for t in range(n[b])] for b in range(B)]

    def step(self):
        self._call(self.lib.sd2_step(self.ctx))

    def accept(self, tokens: Optional[torch.Tensor] = None, n: Optional[torch.Tensor] = None):
        tokens = self.tokens_out if tokens is None else tokens
        n = self.n_out if n is None else n
        self._call(self.lib.sd2_accept(self.ctx, _ptr(tokens), _ptr(n)))
        return tokens, n

    def check(self):
        self._call(self.lib.sd2_check(self.ctx))

    def set_graphs(self, enable: bool):
        self._call(self.lib.sd2_set_graphs(self.ctx, 1 if enable else 0))

    def buffer(self, which: int) -> torch.Tensor:
        """A copy of one of the context's device buffers (see sd2_debug_buffer)."""
        p, n, dt = c_void_p(), c_int64(), c_int32()
        self._call(self.lib.sd2_debug_buffer(self.ctx, which, ctypes.byref(p), ctypes.byref(n), ctypes.byref(dt)))
        typestr = "<f4" if dt.value == DTYPE_F32 else "<i4"
        torch.cuda.synchronize()
        return torch.as_tensor(_DeviceView(p.value, n.value, typestr), device="cuda").clone()

    def set_gemm_impl(self, impl: int):
        """0: tensor-core GEMM where the shape allows (default); 1: CUDA-core GEMM."""
        self._call(self.lib.sd2_set_gemm_impl(self.ctx, impl))

    def profile(self, enable: bool):
        self._call(self.lib.sd2_profile(self.ctx, 1 if enable else 0))

    def profile_read(self):
        n = len(PROFILE_CLASSES)
        la, ms, by = (c_int64 * n)(), (c_double * n)(), (c_double * n)()
        self._call(self.lib.sd2_profile_read(self.ctx, la, ms, by, n))
        return {name: {"launches": la[i], "ms": ms[i], "bytes": by[i]} for i, name in enumerate(PROFILE_CLASSES)}

    def set_drafter_chain(self, enable: bool):
        """Drafter steps as one persistent kernel, or one kernel per projection (the default)."""
        self._call(self.lib.sd2_set_drafter_chain(self.ctx, 1 if enable else 0))

    def set_fused_attention(self, enable: bool):
        """Batch-1 decode: attention inside the O projection, or its own kernel (the default)."""
        self._call(self.lib.sd2_set_fused_attention(self.ctx, 1 if enable else 0))

    def stage_timing(self, enable: bool):
        """Record stage events inside the captured step (steering, k drafter steps, verify)."""
        self._call(self.lib.sd2_stage_timing(self.ctx, 1 if enable else 0))

    def stage_read(self):
        """Milliseconds of the last timed step: (steering, all k drafter steps, verify)."""
        ms = (c_double * 3)()
        self._call(self.lib.sd2_stage_read(self.ctx, ms))
        return {"steer": ms[0], "draft": ms[1], "verify": ms[2]}

    def gemm_timing(self, enable: bool):
        """In-graph GEMM timing: globaltimer stamps of every tensor-core GEMM launch of a step."""
        self._call(self.lib.sd2_gemm_timing(self.ctx, 1 if enable else 0))

    def gemm_timing_read(self, cap: int = 8192):
        """Launches of the last timed step in stream order: dicts with entry/wait/exit ns, bytes, stage."""
        n = c_int32()
        st, by, sg = (c_uint64 * (3 * cap))(), (c_double * cap)(), (c_int32 * cap)()
        self._call(self.lib.sd2_gemm_timing_read(self.ctx, cap, ctypes.byref(n), st, by, sg))
        return [{"entry": st[3 * i], "wait": st[3 * i + 1], "exit": st[3 * i + 2], "bytes": by[i], "stage": sg[i]}
                for i in range(min(n.value, cap))]

    def close(self):
        if getattr(self, "ctx", None) is not None and self.ctx.value:
            self.lib.sd2_free(self.ctx)
            self.ctx = c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def accept_logits(target: torch.Tensor, draft: torch.Tensor, xhat: torch.Tensor, temperature: torch.Tensor, seed: int,
                  step: int, workspace: Optional[torch.Tensor] = None, stream=None):
    """Standalone speculative acceptance of B blocks (sd2_accept_logits); returns (tokens, n)."""
    lib = load_library()
    B, k1, V = target.shape
    k = k1 - 1
    dtype = DTYPE_BF16 if target.dtype == torch.bfloat16 else DTYPE_F32
    tokens = torch.empty((B, k + 1), dtype=torch.int32, device=target.device)
    n = torch.empty(B, dtype=torch.int32, device=target.device)
    need = lib.sd2_accept_workspace_bytes(B, k)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=target.device)
    _check(lib, lib.sd2_accept_logits(_ptr(target), _ptr(draft), dtype, _ptr(xhat), _ptr(temperature), B, k, V,
                                      c_uint64(seed), c_uint32(step), _ptr(tokens), _ptr(n), _ptr(workspace),
                                      workspace.numel(), _stream(stream)))
    return tokens, n


def steer(taps: torch.Tensor, st: dict, eps: float, n_bias: int, stream=None):
    """Standalone steering step (sd2_steer): taps [B, 3, d_v] f32 -> (g [B, d_g], biases [B, n_bias])."""
    lib = load_library()
    B, _, dv = taps.shape
    dg = st["w_hml"].shape[0]
    g = torch.empty((B, dg), dtype=torch.float32, device=taps.device)
    bias = torch.empty((B, n_bias), dtype=torch.float32, device=taps.device)
    ws = torch.empty(lib.sd2_steer_workspace_bytes(B, dv, dg), dtype=torch.uint8, device=taps.device)
    _check(lib, lib.sd2_steer(_ptr(taps.contiguous()), B, dv, _ptr(st["w_hml"]), _ptr(st["ln_gamma"]),
                              _ptr(st["ln_beta"]), c_float(eps), dg, _ptr(st["w_s"]), n_bias, _ptr(g), _ptr(bias),
                              _ptr(ws), ws.numel(), _stream(stream)))
    return g, bias


def swiglu_steered(gate: torch.Tensor, up: torch.Tensor, bias: Optional[torch.Tensor], seq: Optional[torch.Tensor],
                   stream=None) -> torch.Tensor:
    """Standalone Eq. 2 activation (sd2_swiglu_steered): bf16 (up + bias[seq]) * SiLU(gate)."""
    lib = load_library()
    M, F = gate.shape
    h = torch.empty((M, F), dtype=torch.bfloat16, device=gate.device)
    _check(lib, lib.sd2_swiglu_steered(_ptr(gate), _ptr(up), _ptr(bias), _ptr(seq), M, F, _ptr(h), _stream(stream)))
    return h


def attention(q: torch.Tensor, pool: torch.Tensor, table: torch.Tensor, layer: int, row_pos: torch.Tensor,
              grp_row0: torch.Tensor, grp_nrows: torch.Tensor, grp_seq: torch.Tensor, max_rows: int,
              n_splits: int, chunk: int, pre_len: Optional[torch.Tensor] = None, pre_stable: int = 0,
              pre_fresh: int = 0, err: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Standalone paged causal attention (sd2_attention). q [M, H, hd] f32; pool bf16
    [L, n_blocks, 2, Hkv, 16, hd]; table int32 [n_seq, bt_stride]; returns bf16 [M, H * hd]. `err`, a
    one-element int32 device tensor, collects the device error bits."""
    lib = load_library()
    M, H, hd = q.shape
    Hkv, n_blocks = pool.shape[3], pool.shape[1]
    out = torch.empty((M, H * hd), dtype=torch.bfloat16, device=q.device)
    _check(lib, lib.sd2_attention(_ptr(q), M, H, Hkv, hd, _ptr(pool), n_blocks, _ptr(table), table.shape[1], layer,
                                  _ptr(row_pos), _ptr(grp_row0), _ptr(grp_nrows), _ptr(grp_seq), grp_row0.numel(),
                                  max_rows, n_splits, chunk, _ptr(pre_len), pre_stable, pre_fresh, _ptr(out),
                                  _ptr(err), _stream(stream)))
    return out


def attention_flat(q: torch.Tensor, pool: torch.Tensor, table: torch.Tensor, layer: int, row_pos: torch.Tensor,
                   grp_row0: torch.Tensor, grp_nrows: torch.Tensor, grp_seq: torch.Tensor, max_rows: int,
                   slots: int, max_ctx: int, pre_len: torch.Tensor, pre_stable: int = 0, pre_fresh: int = 0,
                   workspace: Optional[torch.Tensor] = None, err: Optional[torch.Tensor] = None,
                   stream=None) -> torch.Tensor:
    """Standalone flat-mode attention (sd2_attention_flat): `slots` CTAs per KV head shared out over
    the groups by length; arguments as attention(), plus the workspace (zeroed uint8, allocated here
    when not given). Returns bf16 [M, H * hd]."""
    lib = load_library()
    M, H, hd = q.shape
    Hkv, n_blocks = pool.shape[3], pool.shape[1]
    if workspace is None:
        workspace = torch.zeros(lib.sd2_attention_flat_workspace_bytes(Hkv, slots, hd), dtype=torch.uint8,
                                device=q.device)
    out = torch.empty((M, H * hd), dtype=torch.bfloat16, device=q.device)
    _check(lib, lib.sd2_attention_flat(_ptr(q), M, H, Hkv, hd, _ptr(pool), n_blocks, _ptr(table), table.shape[1],
                                       layer, _ptr(row_pos), _ptr(grp_row0), _ptr(grp_nrows), _ptr(grp_seq),
                                       grp_row0.numel(), max_rows, slots, max_ctx, _ptr(pre_len), pre_stable,
                                       pre_fresh, _ptr(workspace), _ptr(out), _ptr(err), _stream(stream)))
    return out


def gemm(x: torch.Tensor, w: torch.Tensor, epilogue: int = 0, out: Optional[torch.Tensor] = None,
         w_up: Optional[torch.Tensor] = None, bias: Optional[torch.Tensor] = None,
         seq: Optional[torch.Tensor] = None, impl: int = 0, stream=None):
    """Standalone weight-streaming GEMM (sd2_gemm). epilogue 0: returns X W^T (f32); 1: adds it into
    `out` (plus bias[seq] if given); 2: steered SwiGLU with w = W_gate, w_up = W_up, returns bf16
    [M, N]; 4: returns bf16(SiLU(X W^T + bias[seq]))."""
    lib = load_library()
    M, K = x.shape
    N = w.shape[0]
    h = None
    if epilogue == 0 and out is None:
        out = torch.empty((M, N), dtype=torch.float32, device=x.device)
    if epilogue in (2, 4):
        h = torch.empty((M, N), dtype=torch.bfloat16, device=x.device)
    _check(lib, lib.sd2_gemm(_ptr(x), x.stride(0), M, K, _ptr(w), _ptr(w_up), N, epilogue, _ptr(out),
                             0 if out is None else out.stride(0), _ptr(h), _ptr(bias), _ptr(seq),
                             0 if bias is None else bias.stride(0), impl, _stream(stream)))
    return h if epilogue in (2, 4) else out
