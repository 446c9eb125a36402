"""Decoder forward in fp32 on the CPU (oracle; test infrastructure only).

A Llama-style pre-norm decoder, the "SwiGLU" model family of every pair in the paper (Sec. 3.2,
Sec. 6), with the drafter's MLP steered as in Eq. 2:

    x = Embed[token]
    per layer:  a = RMSNorm(x) * gamma_attn
                q, k, v = a W_q^T, a W_k^T, a W_v^T;  rotary embedding on q and k
                x = x + Attn(q, k, v) W_o^T       (causal, GQA, scale 1/sqrt(head_dim))
                a = RMSNorm(x) * gamma_mlp
                x = x + W_d((W_u a + b^(l)) * SiLU(W_g a))          (Eq. 2; b^(l) = 0: Eq. 1)
    logits = (RMSNorm(x) * gamma_final) W_lm^T

Readings where the paper is silent: no projection biases, untied lm_head, rotate-half rotary
embedding with frequencies theta^(-2i/d_head) and no frequency scaling, sigma of Eq. 1/2 read as
SiLU (the paper calls the MLP SwiGLU). Taps: the residual stream after 1-based layer l, before the
final norm (App. A.2 names layers 3, L/2, L-2).

This is the full-sequence definition: position t sees exactly tokens 0..t, so a KV cache is not
needed here; the GPU's cached computation must agree with it.

Pinned in tests/test_oracle_model.py: each block against a library routine (F.rms_norm,
F.scaled_dot_product_attention, F.silu) or a closed form (rotary embedding preserves norms and
makes q.k depend only on the position difference), causality (appending tokens leaves earlier
logits unchanged), and Eq. 2 against a hand-worked example (tests/golden/eq2_swiglu.txt).
"""
from __future__ import annotations

import math
from typing import Dict, Optional, Sequence

import torch
import torch.nn.functional as F


def rms_norm(x: torch.Tensor, gamma: torch.Tensor, eps: float) -> torch.Tensor:
    """x / sqrt(mean(x^2) + eps) * gamma over the last dim."""
    return x * torch.rsqrt((x * x).mean(dim=-1, keepdim=True) + eps) * gamma.float()


def rotary(x: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """Rotate-half rotary embedding. x: [T, H, hd]; pos: [T] integer positions.

    Pair (i, i + hd/2) is rotated by angle pos * theta^(-2i/hd); angles in fp64.
    """
    hd = x.shape[-1]
    half = hd // 2
    freq = theta ** (-(torch.arange(half, dtype=torch.float64) * 2.0 / hd))
    ang = pos.to(torch.float64)[:, None] * freq[None, :]
    cos = torch.cos(ang).to(torch.float32)[:, None, :]
    sin = torch.sin(ang).to(torch.float32)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], dim=-1)


def causal_attention(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, row_block: int = 1024) -> torch.Tensor:
    """softmax(q k^T / sqrt(hd) + causal mask) v with grouped KV heads.

    q: [T, H, hd], k and v: [T, H_kv, hd]; query head h reads KV head h // (H / H_kv).
    Query rows are independent by this definition, so they are taken `row_block` at a time (row
    r attends to keys 0..r; each block reads the keys up to its last row), which bounds the score
    matrix at long context without changing any row's softmax.
    """
    T, H, hd = q.shape
    rep = H // k.shape[1]
    k = k.repeat_interleave(rep, dim=1)
    v = v.repeat_interleave(rep, dim=1)
    out = torch.empty(T, H, hd, dtype=q.dtype)
    for r0 in range(0, T, row_block):
        r1 = min(T, r0 + row_block)
        scores = torch.einsum("thd,shd->hts", q[r0:r1], k[:r1]) / math.sqrt(hd)
        mask = torch.arange(r1)[None, :] > torch.arange(r0, r1)[:, None]    # key after the query row
        scores = scores.masked_fill(mask[None], float("-inf"))
        probs = torch.softmax(scores, dim=-1)
        out[r0:r1] = torch.einsum("hts,shd->thd", probs, v[:r1])
    return out


def silu(x: torch.Tensor) -> torch.Tensor:
    return x * torch.sigmoid(x)


def steered_swiglu(a: torch.Tensor, w_gate, w_up, w_down, bias: Optional[torch.Tensor]) -> torch.Tensor:
    """Eq. 2: W_d((W_u a + b) * SiLU(W_g a)); with bias None it is Eq. 1."""
    up = a @ w_up.float().T
    if bias is not None:
        up = up + bias
    return (up * silu(a @ w_gate.float().T)) @ w_down.float().T


def cond_bias(f: torch.Tensor, g: torch.Tensor, st: Dict, layer: int) -> torch.Tensor:
    """The "Cond. Bias in MLP" variant (Sec. 5): b = W_c2 SiLU(W_c1 [f; g]) per position, with f the
    layer's input f^(l-1) [T, d_D] and g [T, d_g]; W_c1 = [W_c1x | W_c1g] split by input block."""
    dg = st["w_c1g"].shape[1]
    F = st["w_c2"].shape[0] // (st["w_c1x"].shape[0] // dg)
    w1x = st["w_c1x"][layer * dg:(layer + 1) * dg].float()
    w1g = st["w_c1g"][layer * dg:(layer + 1) * dg].float()
    w2 = st["w_c2"][layer * F:(layer + 1) * F].float()
    return silu(f @ w1x.T + g @ w1g.T) @ w2.T


def forward(shape, w: Dict, tokens: Sequence[int], bias: Optional[torch.Tensor] = None,
            tap_layers: Optional[Sequence[int]] = None, logit_rows: Optional[Sequence[int]] = None,
            bias_site: str = "mlp_up", cond: Optional[tuple] = None):
    """Run the decoder over `tokens` (positions 0..T-1).

    bias: None, or [T, L, w] fp32 steering biases b^(l) per position. bias_site "mlp_up": w = d_ffn,
      added to W_u a before the gating (Eq. 2); "after_mlp": w = d_model, added to the layer's output
      f^(l) = x + MLP(...) (the "Inv. Bias after MLP" variant of Sec. 5).
    cond: with bias_site "cond_mlp", (g [T, d_g] per position, steering weights): the bias of layer l
      at each position is cond_bias(f^(l-1), g) and enters as in Eq. 2 ("Cond. Bias in MLP", Sec. 5).
    tap_layers: 1-based layers whose output residual stream is returned (App. A.2 order h, m, l).
    logit_rows: positions whose logits are computed (default: all).
    Returns (logits [R, V] fp32, taps [T, len(tap_layers), d] fp32 or None).
    """
    tok = torch.as_tensor(list(tokens), dtype=torch.long)
    T = tok.numel()
    pos = torch.arange(T)
    x = w["embed"][tok].float()
    taps = {}
    H, Hkv, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    for li, lw in enumerate(w["layers"]):
        f_in = x                                             # f^(l-1): this layer's input
        a = rms_norm(x, lw["attn_norm"], shape.norm_eps)
        q = (a @ lw["wq"].float().T).view(T, H, hd)
        k = (a @ lw["wk"].float().T).view(T, Hkv, hd)
        v = (a @ lw["wv"].float().T).view(T, Hkv, hd)
        q = rotary(q, pos, shape.rope_theta)
        k = rotary(k, pos, shape.rope_theta)
        o = causal_attention(q, k, v).reshape(T, H * hd)
        x = x + o @ lw["wo"].float().T
        a = rms_norm(x, lw["mlp_norm"], shape.norm_eps)
        b = None if bias is None else bias[:, li, :]
        if bias_site == "cond_mlp" and cond is not None:
            b = cond_bias(f_in, cond[0], cond[1], li)
        if bias_site in ("mlp_up", "cond_mlp"):
            x = x + steered_swiglu(a, lw["w_gate"], lw["w_up"], lw["w_down"], b)
        else:
            x = x + steered_swiglu(a, lw["w_gate"], lw["w_up"], lw["w_down"], None)
            if b is not None:
                x = x + b
        taps[li + 1] = x
    hN = rms_norm(x, w["final_norm"], shape.norm_eps)
    if logit_rows is not None:
        hN = hN[torch.as_tensor(list(logit_rows), dtype=torch.long)]
    logits = hN @ w["lm_head"].float().T
    tap_out = None
    if tap_layers is not None:
        tap_out = torch.stack([taps[l] for l in tap_layers], dim=1)
    return logits, tap_out
