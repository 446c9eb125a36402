"""Steering vector and per-layer biases (oracle; test infrastructure only).

Sec. 3.1: g_t = W_hml [h_t, m_t, l_t]^T, the concatenation of the verifier's high, middle and
low hidden states (layers L-2, L/2, 3 per App. A.2), read at the position of the last returned
token. App. A.2: a layer norm is applied right after computing the steering vector.
Eq. 2 / Sec. 3.2: every drafter MLP layer l receives the bias b^(l) = W_s^(l) g_t, computed once
per drafting stage because it does not depend on the draft position.

Readings: LayerNorm is a true layer norm (mean removed, biased variance, eps, affine gain and
shift); W_s is per layer (Fig. 2: "a set of biases ... added to all MLP hidden states"), stored as
one stacked [L_D * F_D, d_g] matrix whose rows l*F_D..(l+1)*F_D-1 give layer l.

Pinned in tests/test_oracle_model.py: LayerNorm against F.layer_norm, and the paper's own
initialisation identity (Sec. 3.3): with W_hml = [I I I], g = LN(h + m + l) on a hand-worked
vector (tests/golden/steering_identity.txt).
"""
from __future__ import annotations

import torch


def layer_norm(x: torch.Tensor, gamma: torch.Tensor, beta: torch.Tensor, eps: float) -> torch.Tensor:
    mu = x.mean(dim=-1, keepdim=True)
    var = ((x - mu) ** 2).mean(dim=-1, keepdim=True)
    return (x - mu) / torch.sqrt(var + eps) * gamma.float() + beta.float()


def steering_vector(taps_hml: torch.Tensor, st: dict, eps: float) -> torch.Tensor:
    """g = LN(W_hml [h; m; l]). taps_hml: [..., 3, d_v] in the order (h, m, l)."""
    cat = taps_hml.reshape(*taps_hml.shape[:-2], -1).float()
    return layer_norm(cat @ st["w_hml"].float().T, st["ln_gamma"], st["ln_beta"], eps)


def steering_bias(g: torch.Tensor, st: dict, n_layers: int, width: int) -> torch.Tensor:
    """b^(l) = W_s^(l) g for every drafter layer: [..., L_D, width] (width F_D for Eq. 2, d_D for the
    after-MLP variant of Sec. 5)."""
    return (g.float() @ st["w_s"].float().T).reshape(*g.shape[:-1], n_layers, width)
