"""Workload shapes and seeded synthetic inputs for SD^2 (steered speculative decoding).

This module is the single source of inputs for both the CUDA path and the CPU
oracle. It holds shapes and random-number draws only: no step of the method's
arithmetic (no norm, projection, softmax, sampling or acceptance) lives here.

Shapes follow the paper's model families: Llama/Qwen-style pre-norm decoders
with SwiGLU feed-forward layers (Sec. 3.2, "Drafting"; Sec. 6 notes every model
in the study uses SwiGLU). Tap layers follow App. A.2 (layers 3, L/2, L-2).
Weights are random (the paper's trained checkpoints are not available), drawn
N(0, 0.02^2) and rounded to bf16, so both sides consume identical values.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence, Tuple

import torch

# Slot order of one decoder layer's tensors; the C header uses the same order.
LAYER_SLOTS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")


@dataclass(frozen=True)
class LMShape:
    """One Llama-style decoder (no projection biases, untied lm_head)."""
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    rope_theta: float
    norm_eps: float

    def layer_shapes(self) -> Dict[str, Tuple[int, ...]]:
        d, hd = self.d_model, self.head_dim
        return {
            "attn_norm": (d,),
            "wq": (self.n_heads * hd, d),
            "wk": (self.n_kv_heads * hd, d),
            "wv": (self.n_kv_heads * hd, d),
            "wo": (d, self.n_heads * hd),
            "mlp_norm": (d,),
            "w_gate": (self.d_ffn, d),
            "w_up": (self.d_ffn, d),
            "w_down": (d, self.d_ffn),
        }

    def param_count(self, include_embed: bool = False) -> int:
        per_layer = sum(_numel(s) for s in self.layer_shapes().values())
        n = self.n_layers * per_layer + self.d_model + self.vocab * self.d_model  # + final norm + lm_head
        if include_embed:
            n += self.vocab * self.d_model
        return n


def _numel(shape: Sequence[int]) -> int:
    n = 1
    for s in shape:
        n *= int(s)
    return n


def default_tap_layers(n_layers: int) -> Tuple[int, int, int]:
    """(h, m, l) = 1-based layer outputs (L-2, L/2, 3), clamped to [1, L] (App. A.2)."""
    clamp = lambda x: max(1, min(n_layers, x))
    return (clamp(n_layers - 2), clamp(n_layers // 2), clamp(3))


@dataclass(frozen=True)
class PairWorkload:
    """A verifier/drafter pair plus the decoding setup of one benchmark configuration."""
    name: str
    verifier: LMShape
    drafter: LMShape
    d_steer: int
    k: int
    batch: int
    prompt_len: Tuple[int, int]          # (min, max) inclusive; equal for fixed length
    gen_tokens: int
    temperatures: Tuple[float, ...]
    kv_block: int = 16
    steer_ln_eps: float = 1e-5
    description: str = ""
    # where the steering bias enters the drafter: "mlp_up" is Eq. 2 (added to W_u a before the
    # gating, F_D wide per layer); "after_mlp" is the "Inv. Bias after MLP" ablation of Sec. 5
    # (added to each layer's output, d_D wide per layer); "cond_mlp" is its "Cond. Bias in MLP"
    # ablation (per position, a 2-layer MLP of the layer input f^(l-1) and g gives the bias used
    # as in Eq. 2)
    steering_site: str = "mlp_up"

    @property
    def tap_layers(self) -> Tuple[int, int, int]:
        return default_tap_layers(self.verifier.n_layers)

    @property
    def bias_width(self) -> int:
        """Steering bias entries per drafter layer."""
        return self.drafter.d_model if self.steering_site == "after_mlp" else self.drafter.d_ffn


TINY_V = LMShape(4, 256, 4, 4, 64, 1024, 4096, 10000.0, 1e-5)
TINY_D = LMShape(2, 128, 2, 2, 64, 512, 4096, 10000.0, 1e-5)
LLAMA8B = LMShape(32, 4096, 32, 8, 128, 14336, 128256, 500000.0, 1e-5)
LLAMA1B = LMShape(16, 2048, 32, 8, 64, 8192, 128256, 500000.0, 1e-5)
QWEN32B = LMShape(64, 5120, 40, 8, 128, 27648, 152064, 1000000.0, 1e-6)
QWEN05B = LMShape(24, 896, 14, 2, 64, 4864, 152064, 1000000.0, 1e-6)

WORKLOADS: Dict[str, PairWorkload] = {
    "tiny": PairWorkload(
        "tiny", TINY_V, TINY_D, d_steer=128, k=4, batch=1, prompt_len=(32, 32), gen_tokens=64,
        temperatures=(0.0, 1.0),
        description="tiny 4L/d256 verifier, 2L/d128 drafter, vocab 4096, B=1, prompt 32, k=4, 64 new"),
    "llama8b_1b": PairWorkload(
        "llama8b_1b", LLAMA8B, LLAMA1B, d_steer=2048, k=5, batch=1, prompt_len=(512, 512),
        gen_tokens=256, temperatures=(1.0,),
        description="Llama-3-8B-shaped verifier / Llama-3.2-1B-shaped drafter, B=1, prompt 512, k=5, T=1"),
    "llama8b_1b_b16": PairWorkload(
        "llama8b_1b_b16", LLAMA8B, LLAMA1B, d_steer=2048, k=8, batch=16, prompt_len=(128, 1024),
        gen_tokens=256, temperatures=(0.0, 0.7, 1.0),
        description="8B/1B pair, B=16 ragged prompts 128-1024, k=8, T in {0,0.7,1}, paged KV block 16"),
    "qwen32b_05b": PairWorkload(
        "qwen32b_05b", QWEN32B, QWEN05B, d_steer=896, k=6, batch=4, prompt_len=(2048, 2048),
        gen_tokens=512, temperatures=(1.0,),
        description="Qwen2.5-32B-shaped verifier / 0.5B-shaped drafter, B=4, prompt 2048, k=6, T=1"),
}


def shrink(shape: LMShape, **kw) -> LMShape:
    """Copy of a shape with some fields replaced (used to build small test shapes)."""
    return dataclasses.replace(shape, **kw)


# ----------------------------------------------------------------------------------------------
# Seeded tensors
# ----------------------------------------------------------------------------------------------

def _gen(seed: int, device: str) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _normal(shape, std: float, seed: int, device: str) -> torch.Tensor:
    t = torch.randn(tuple(shape), generator=_gen(seed, device), device=device, dtype=torch.float32)
    return (t * std).to(torch.bfloat16)


def _norm_weight(n: int, jitter: float, seed: int, device: str) -> torch.Tensor:
    if jitter == 0.0:
        return torch.ones(n, dtype=torch.bfloat16, device=device)
    t = torch.randn(n, generator=_gen(seed, device), device=device, dtype=torch.float32)
    return (1.0 + jitter * t).to(torch.bfloat16)


def make_lm_weights(shape: LMShape, seed: int, device: str = "cpu", std: float = 0.02,
                    norm_jitter: float = 0.0) -> dict:
    """Random bf16 weights of one decoder: {'embed','final_norm','lm_head','layers':[{slot: tensor}]}.

    Tensor i of the model is drawn from its own generator seeded with seed*1000+i, so any one
    tensor can be regenerated alone. norm_jitter > 0 gives RMSNorm gains 1 + jitter*N(0,1)
    (tests use it so that a dropped gain is visible); 0 gives gains of exactly 1.
    """
    idx = 0

    def nxt():
        nonlocal idx
        idx += 1
        return seed * 1000 + idx

    w = {"embed": _normal((shape.vocab, shape.d_model), std, nxt(), device)}
    layers = []
    for _ in range(shape.n_layers):
        lw = {}
        for slot, shp in shape.layer_shapes().items():
            if slot.endswith("norm"):
                lw[slot] = _norm_weight(shp[0], norm_jitter, nxt(), device)
            else:
                lw[slot] = _normal(shp, std, nxt(), device)
        layers.append(lw)
    w["layers"] = layers
    w["final_norm"] = _norm_weight(shape.d_model, norm_jitter, nxt(), device)
    w["lm_head"] = _normal((shape.vocab, shape.d_model), std, nxt(), device)
    return w


def make_steering_weights(work: PairWorkload, seed: int, device: str = "cpu", std: float = 0.02,
                          ln_jitter: float = 0.0, zero_ws: bool = False) -> dict:
    """Random steering parameters: W_hml [d_g, 3 d_v], LayerNorm gain/shift [d_g], W_s [L_D*w, d_g]
    with w = work.bias_width (F_D for Eq. 2, d_D for the after-MLP ablation).

    W_s is one stacked matrix: rows l*w .. (l+1)*w-1 give the bias of drafter layer l.
    zero_ws=True gives the paper's W_s = 0 initialisation (Sec. 3.3).
    """
    dv, dg = work.verifier.d_model, work.d_steer
    n_out = work.drafter.n_layers * work.bias_width
    st = {"w_hml": _normal((dg, 3 * dv), std, seed * 1000 + 901, device)}
    if ln_jitter == 0.0:
        st["ln_gamma"] = torch.ones(dg, dtype=torch.bfloat16, device=device)
        st["ln_beta"] = torch.zeros(dg, dtype=torch.bfloat16, device=device)
    else:
        st["ln_gamma"] = _norm_weight(dg, ln_jitter, seed * 1000 + 902, device)
        st["ln_beta"] = _normal((dg,), ln_jitter, seed * 1000 + 903, device)
    if work.steering_site == "cond_mlp":
        # the conditional bias MLP of every drafter layer: hidden width d_g, input [f^(l-1); g]
        # split into its two column blocks W_c1 = [W_c1x | W_c1g]; W_c2 maps back to F_D
        L, dd = work.drafter.n_layers, work.drafter.d_model
        st["w_c1x"] = _normal((L * dg, dd), std, seed * 1000 + 905, device)
        st["w_c1g"] = _normal((L * dg, dg), std, seed * 1000 + 906, device)
        st["w_c2"] = (torch.zeros((n_out, dg), dtype=torch.bfloat16, device=device) if zero_ws
                      else _normal((n_out, dg), std, seed * 1000 + 907, device))
        return st
    if zero_ws:
        st["w_s"] = torch.zeros((n_out, dg), dtype=torch.bfloat16, device=device)
    else:
        st["w_s"] = _normal((n_out, dg), std, seed * 1000 + 904, device)
    return st


def make_prompts(vocab: int, batch: int, length: Tuple[int, int], seed: int = 7) -> List[List[int]]:
    """Uniform-random token ids; lengths uniform in [length[0], length[1]] (ragged batches)."""
    g = _gen(seed, "cpu")
    lo, hi = length
    if lo == hi:
        lens = [lo] * batch
    else:
        lens = torch.randint(lo, hi + 1, (batch,), generator=g).tolist()
    return [torch.randint(0, vocab, (n,), generator=g).tolist() for n in lens]


def make_sweep_logits(batch: int, k: int, vocab: int, seed: int, device: str = "cpu",
                      std: float = 3.0, boost: float = 8.0, share_prob: float = 0.5):
    """Acceptance-kernel inputs: bf16 logits N(0, std^2) with one boosted token per row.

    Returns (target [B, k+1, V] bf16, draft [B, k, V] bf16, xhat [B, k] int32). With
    probability share_prob a draft row boosts the same token as the target row it is checked
    against; each draft token is that draft row's boosted token with probability 1/2 and a
    uniform-random token otherwise.
    """
    g = _gen(seed, device)
    target = torch.randn((batch, k + 1, vocab), generator=g, device=device) * std
    draft = torch.randn((batch, k, vocab), generator=g, device=device) * std
    t_idx = torch.randint(0, vocab, (batch, k + 1), generator=g, device=device)
    own = torch.randint(0, vocab, (batch, k), generator=g, device=device)
    share = torch.rand((batch, k), generator=g, device=device) < share_prob
    d_idx = torch.where(share, t_idx[:, :k], own)
    target.scatter_add_(2, t_idx[..., None], torch.full_like(t_idx[..., None], boost, dtype=target.dtype))
    draft.scatter_add_(2, d_idx[..., None], torch.full_like(d_idx[..., None], boost, dtype=draft.dtype))
    pick = torch.rand((batch, k), generator=g, device=device) < 0.5
    rnd = torch.randint(0, vocab, (batch, k), generator=g, device=device)
    xhat = torch.where(pick, d_idx, rnd).to(torch.int32)
    return target.to(torch.bfloat16), draft.to(torch.bfloat16), xhat


def make_taps(batch: int, d_v: int, seed: int, device: str = "cpu") -> torch.Tensor:
    """Random verifier hidden states [B, 3, d_v] fp32 ~ N(0,1) for the steering sweep."""
    return torch.randn((batch, 3, d_v), generator=_gen(seed, device), device=device)
