"""Pins for the oracle's decoder forward and steering (CPU only).

Each block is checked against a library routine or a closed form, Eq. 2 and the steering
initialisation identity against hand-worked examples (tests/golden/), and causality by appending
tokens.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from conftest import golden_rows
from oracle import model, steering
from paper_2511_09844_gb300 import workloads as W


def test_rms_norm_matches_library():
    g = torch.Generator().manual_seed(0)
    x = torch.randn(7, 96, generator=g)
    gamma = 1 + 0.1 * torch.randn(96, generator=g)
    ref = F.rms_norm(x, (96,), weight=gamma, eps=1e-5)
    assert torch.allclose(model.rms_norm(x, gamma, 1e-5), ref, atol=1e-6, rtol=1e-5)


def test_silu_and_layer_norm_match_library():
    g = torch.Generator().manual_seed(1)
    x = torch.randn(5, 33, generator=g) * 3
    assert torch.allclose(model.silu(x), F.silu(x), atol=1e-6)
    gamma, beta = torch.randn(33, generator=g), torch.randn(33, generator=g)
    ref = F.layer_norm(x, (33,), gamma, beta, eps=1e-5)
    assert torch.allclose(steering.layer_norm(x, gamma, beta, 1e-5), ref, atol=1e-5, rtol=1e-5)


@pytest.mark.parametrize("H,Hkv", [(4, 4), (8, 2), (14, 2)])
def test_attention_matches_library(H, Hkv):
    g = torch.Generator().manual_seed(H * 10 + Hkv)
    T, hd = 9, 16
    q, k, v = (torch.randn(T, h, hd, generator=g) for h in (H, Hkv, Hkv))
    ref = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.transpose(0, 1)[None],
                                         v.transpose(0, 1)[None], is_causal=True,
                                         enable_gqa=True)[0].transpose(0, 1)
    assert torch.allclose(model.causal_attention(q, k, v), ref, atol=1e-5, rtol=1e-5)


def test_attention_uniform_keys_average_values():
    """All keys equal -> every allowed position weighs the same: row t is the mean of v[0..t]."""
    T, hd = 6, 8
    q = torch.randn(T, 2, hd)
    k = torch.ones(T, 1, hd)
    v = torch.arange(T, dtype=torch.float32)[:, None, None].expand(T, 1, hd).contiguous()
    out = model.causal_attention(q, k, v)
    for t in range(T):
        assert torch.allclose(out[t], torch.full((2, hd), t / 2.0), atol=1e-6)


def test_rotary_closed_forms():
    theta = 10000.0
    x = torch.tensor([[[1.0, 0.0]]])           # hd = 2: one pair, frequency 1
    for p in (0, 1, 5):
        r = model.rotary(x, torch.tensor([p]), theta)[0, 0]
        assert torch.allclose(r, torch.tensor([math.cos(p), math.sin(p)]), atol=1e-6)
    g = torch.Generator().manual_seed(2)
    q = torch.randn(1, 3, 64, generator=g)
    kk = torch.randn(1, 3, 64, generator=g)
    assert torch.allclose(model.rotary(q, torch.tensor([0]), theta), q)             # position 0
    r = model.rotary(q, torch.tensor([1234]), theta)
    assert torch.allclose(r.norm(dim=-1), q.norm(dim=-1), rtol=1e-5)               # a rotation
    dots = []
    for m, n in [(7, 3), (107, 103), (1007, 1003)]:                                 # relative only
        dots.append((model.rotary(q, torch.tensor([m]), theta) *
                     model.rotary(kk, torch.tensor([n]), theta)).sum(-1))
    assert torch.allclose(dots[0], dots[1], atol=1e-4) and torch.allclose(dots[0], dots[2], atol=1e-4)


def _closed(expr):
    silu = lambda x: x / (1 + math.exp(-x))
    return eval(expr, {"silu": silu, "sqrt": math.sqrt})


def test_eq2_hand_worked():
    rows = {r[0]: r[1:] for r in golden_rows("eq2_swiglu.txt")}
    t = lambda name, shp: torch.tensor([float(x) for x in rows[name]]).reshape(shp)
    a, wg, wu, wd, b = t("a", (1, 2)), t("w_gate", (2, 2)), t("w_up", (2, 2)), t("w_down", (2, 2)), t("bias", (1, 2))
    eq2 = torch.tensor([_closed(e) for e in rows["eq2"]])
    eq1 = torch.tensor([_closed(e) for e in rows["eq1"]])
    assert torch.allclose(model.steered_swiglu(a, wg, wu, wd, b)[0], eq2, atol=1e-6)
    assert torch.allclose(model.steered_swiglu(a, wg, wu, wd, None)[0], eq1, atol=1e-6)


def test_steering_identity_init():
    rows = {r[0]: r[1:] for r in golden_rows("steering_identity.txt")}
    v = lambda n: torch.tensor([float(x) for x in rows[n]])
    d = 4
    st = {"w_hml": torch.cat([torch.eye(d)] * 3, dim=1), "ln_gamma": v("gamma"), "ln_beta": v("beta"),
          "w_s": torch.zeros(6, d)}
    taps = torch.stack([v("h"), v("m"), v("l")])
    g = steering.steering_vector(taps, st, 1e-5)
    assert torch.allclose(g, torch.tensor([_closed(e) for e in rows["g"]]), atol=1e-6)
    # W_s = 0 -> zero biases for every layer (Sec. 3.3 / App. A.2: drafter initially unchanged)
    assert torch.count_nonzero(steering.steering_bias(g, st, 2, 3)) == 0
    # the stacked W_s: rows l*F..(l+1)*F-1 belong to layer l
    st["w_s"] = torch.arange(6 * d, dtype=torch.float32).reshape(6, d)
    b = steering.steering_bias(torch.tensor([1.0, 0, 0, 0]), st, 2, 3)
    assert torch.equal(b, torch.tensor([[0.0, 4, 8], [12, 16, 20]]))


def _small_pair():
    vs = W.shrink(W.TINY_V, n_layers=3, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16, d_ffn=96, vocab=97)
    return vs


def test_causality_and_taps():
    vs = _small_pair()
    w = W.make_lm_weights(vs, seed=3, norm_jitter=0.2)
    toks = W.make_prompts(vs.vocab, 1, (12, 12), seed=4)[0]
    full, taps = model.forward(vs, w, toks, tap_layers=(2, 1, 3))
    part, taps_p = model.forward(vs, w, toks[:5], tap_layers=(2, 1, 3))
    assert torch.allclose(full[:5], part, atol=1e-5, rtol=1e-4)
    assert torch.allclose(taps[:5], taps_p, atol=1e-5, rtol=1e-4)
    assert taps.shape == (12, 3, vs.d_model)
    # the last tap (layer 3 = L) is the residual stream before the final norm
    z = model.rms_norm(taps[:, 2], w["final_norm"], vs.norm_eps) @ w["lm_head"].float().T
    assert torch.allclose(z, full, atol=1e-5, rtol=1e-4)
    rows, _ = model.forward(vs, w, toks, logit_rows=[3, 11])
    assert torch.allclose(rows, full[[3, 11]])


def test_bias_enters_every_layer():
    vs = _small_pair()
    w = W.make_lm_weights(vs, seed=5)
    toks = [1, 2, 3, 4]
    base, _ = model.forward(vs, w, toks)
    zero = torch.zeros(4, vs.n_layers, vs.d_ffn)
    same, _ = model.forward(vs, w, toks, bias=zero)
    assert torch.equal(base, same)
    for l in range(vs.n_layers):
        b = zero.clone()
        b[:, l, :] = 0.5
        moved, _ = model.forward(vs, w, toks, bias=b)
        assert (moved - base).abs().max() > 1e-4
    # a bias at position t leaves earlier positions unchanged (causal)
    b = zero.clone()
    b[2] = 0.5
    moved, _ = model.forward(vs, w, toks, bias=b)
    assert torch.equal(moved[:2], base[:2]) and (moved[2:] - base[2:]).abs().max() > 1e-4


def test_rotary_pairing_and_frequency_order():
    """hd = 4: element 0 pairs with 2 at frequency 1, element 1 with 3 at theta^(-1/2)."""
    theta, p = 100.0, 3
    x = torch.tensor([[[1.0, 0.0, 0.0, 0.0], [0.0, 1.0, 0.0, 0.0]]])
    r = model.rotary(x, torch.tensor([p]), theta)[0]
    f1 = theta ** -0.5
    assert torch.allclose(r[0], torch.tensor([math.cos(p), 0.0, math.sin(p), 0.0]), atol=1e-6)
    assert torch.allclose(r[1], torch.tensor([0.0, math.cos(p * f1), 0.0, math.sin(p * f1)]), atol=1e-6)


def test_tap_layers_follow_appendix():
    """App. A.2: h, m, l are layers L-2, L/2 and 3 (1-based), clamped for shallow models."""
    assert W.default_tap_layers(32) == (30, 16, 3)
    assert W.default_tap_layers(64) == (62, 32, 3)
    assert W.default_tap_layers(4) == (2, 2, 3)
    assert W.default_tap_layers(2) == (1, 1, 2)


def test_attention_row_blocks_do_not_change_rows():
    """Query rows are independent: any row blocking gives the same output as one block."""
    g = torch.Generator().manual_seed(3)
    q = torch.randn(97, 4, 16, generator=g)
    k = torch.randn(97, 2, 16, generator=g)
    v = torch.randn(97, 2, 16, generator=g)
    whole = model.causal_attention(q, k, v, row_block=10 ** 9)
    for blk in (1, 13, 64):
        assert torch.allclose(model.causal_attention(q, k, v, row_block=blk), whole, atol=1e-6, rtol=0)


def test_after_mlp_bias_site():
    """The "Inv. Bias after MLP" variant (Sec. 5): b^(l) (d_model wide) is added to layer l's output
    f^(l). A zero bias changes nothing; at the last layer the residual stream (the tap before the
    final norm) moves by exactly b; a bias at layer l changes the input of every later layer; and
    with Eq. 2's site the same d_model-wide tensor would not fit the MLP (widths differ)."""
    vs = _small_pair()
    w = W.make_lm_weights(vs, seed=8, norm_jitter=0.1)
    toks = [5, 6, 7, 8, 9]
    L = vs.n_layers
    base, taps0 = model.forward(vs, w, toks, tap_layers=(1, 2, L))
    zero = torch.zeros(len(toks), L, vs.d_model)
    same, taps_z = model.forward(vs, w, toks, tap_layers=(1, 2, L), bias=zero, bias_site="after_mlp")
    assert torch.equal(base, same) and torch.equal(taps0, taps_z)
    g = torch.Generator().manual_seed(9)
    b = zero.clone()
    b[:, L - 1, :] = torch.randn(len(toks), vs.d_model, generator=g)
    _, taps_b = model.forward(vs, w, toks, tap_layers=(1, 2, L), bias=b, bias_site="after_mlp")
    assert torch.equal(taps_b[:, :2], taps0[:, :2])                      # earlier layers untouched
    assert torch.allclose(taps_b[:, 2] - taps0[:, 2], b[:, L - 1], atol=1e-5, rtol=0)
    b1 = zero.clone()
    b1[:, 0, :] = 0.25
    _, taps_1 = model.forward(vs, w, toks, tap_layers=(1, 2, L), bias=b1, bias_site="after_mlp")
    assert torch.allclose(taps_1[:, 0] - taps0[:, 0], b1[:, 0], atol=1e-5, rtol=0)
    assert (taps_1[:, 1] - taps0[:, 1] - b1[:, 0]).abs().max() > 1e-4   # layer 2 saw the shifted input
    assert vs.d_model != vs.d_ffn


def test_cond_bias_site():
    """The "Cond. Bias in MLP" variant (Sec. 5): b = W_c2 SiLU(W_c1 [f^(l-1); g]) per position,
    used as in Eq. 2. W_c2 = 0 leaves the drafter unsteered; with W_c1x = 0 the bias no longer
    depends on the position's input and the pass equals Eq. 2 with the stage bias
    W_c2 SiLU(W_c1g g); the bias reads this layer's input (a change of f changes it)."""
    vs = _small_pair()
    dg = 8
    w = W.make_lm_weights(vs, seed=10, norm_jitter=0.1)
    toks = [3, 1, 4, 1, 5, 9]
    T, L = len(toks), vs.n_layers
    g = torch.Generator().manual_seed(11)
    st = {"w_c1x": torch.randn(L * dg, vs.d_model, generator=g) * 0.1,
          "w_c1g": torch.randn(L * dg, dg, generator=g) * 0.1,
          "w_c2": torch.zeros(L * vs.d_ffn, dg)}
    g_rows = torch.randn(T, dg, generator=g)
    base, _ = model.forward(vs, w, toks)
    zero, _ = model.forward(vs, w, toks, bias_site="cond_mlp", cond=(g_rows, st))
    assert torch.equal(base, zero)
    st["w_c2"] = torch.randn(L * vs.d_ffn, dg, generator=g) * 0.1
    st_nox = dict(st, w_c1x=torch.zeros_like(st["w_c1x"]))
    cond, _ = model.forward(vs, w, toks, bias_site="cond_mlp", cond=(g_rows, st_nox))
    stage = torch.stack([model.silu(g_rows @ st["w_c1g"][l * dg:(l + 1) * dg].T) @
                         st["w_c2"][l * vs.d_ffn:(l + 1) * vs.d_ffn].T for l in range(L)], dim=1)
    eq2, _ = model.forward(vs, w, toks, bias=stage)
    assert torch.allclose(cond, eq2, atol=1e-5, rtol=1e-4)
    full, _ = model.forward(vs, w, toks, bias_site="cond_mlp", cond=(g_rows, st))
    assert (full - cond).abs().max() > 1e-4
    # the hand-evaluated bias of layer 0 at one position (f^(-1) = the embedding row)
    f0 = w["embed"][toks[2]].float()
    b0 = model.cond_bias(f0[None], g_rows[2:3], st, 0)[0]
    ref = model.silu(f0 @ st["w_c1x"][:dg].T + g_rows[2] @ st["w_c1g"][:dg].T) @ st["w_c2"][:vs.d_ffn].T
    assert torch.allclose(b0, ref)
